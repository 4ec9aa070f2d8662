"""Seeded input generator (CPU): determinism, random access, moments, recipes."""
import numpy as np


def test_counter_random_access(wl):
    full = wl.normal_bf16(5, wl.stream_id(wl.K_X, 0, 3), 1000)
    part = wl.normal_bf16(5, wl.stream_id(wl.K_X, 0, 3), 100, first=451)
    np.testing.assert_array_equal(full[451:551], part)
    # odd start inside a Box-Muller pair
    part = wl.normal_bf16(5, wl.stream_id(wl.K_X, 0, 3), 3, first=7)
    np.testing.assert_array_equal(full[7:10], part)


def test_threads_do_not_change_values(wl):
    a = wl.normal_bf16(1, 2, 300_000)
    b = np.concatenate([wl.normal_bf16(1, 2, 150_000), wl.normal_bf16(1, 2, 150_000, first=150_000)])
    np.testing.assert_array_equal(a, b)


def test_normal_moments(wl):
    v = wl.bf16_bits_to_float(wl.normal_bf16(3, 9, 400_000, sigma=0.5)).astype(np.float64)
    assert abs(v.mean()) < 0.005
    assert abs(v.std() - 0.5) < 0.005
    assert abs(((v / 0.5) ** 4).mean() - 3.0) < 0.05


def test_streams_differ(wl):
    a = wl.normal_bf16(1, wl.stream_id(1, 0, 0), 64)
    b = wl.normal_bf16(1, wl.stream_id(1, 0, 1), 64)
    c = wl.normal_bf16(2, wl.stream_id(1, 0, 0), 64)
    assert (a != b).mean() > 0.9 and (a != c).mean() > 0.9


def test_bf16_round_trip(wl):
    x = np.array([1.0, -2.5, 1.00390625, 3.0e38, 1e-40], dtype=np.float32)
    b = wl.float_to_bf16_bits(x)
    assert wl.bf16_bits_to_float(b)[0] == 1.0 and wl.bf16_bits_to_float(b)[1] == -2.5
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7: round to even -> 1.0
    assert wl.bf16_bits_to_float(b)[2] == 1.0


def test_config_recipes(wl):
    w0 = wl.config0()
    assert w0.T == 16 and sorted(np.bincount(w0.slot_ids).tolist()) == [4, 4, 4, 4]
    assert (w0.dom_ids == w0.slot_ids % 2).all()
    w1 = wl.config1()
    assert w1.T == 64 and w1.slot_ids.max() < 64 and (w1.dom_ids == w1.slot_ids % 4).all()
    w2 = wl.config2()
    lens = np.bincount(w2.slot_ids)
    assert w2.T == 8192 and lens.min() >= 128 and lens.max() <= 1024 + 127
    assert (np.diff(w2.slot_ids) >= 0).all()
    w3 = wl.config3()
    assert w3.T == 256 and np.bincount(w3.slot_ids).argmax() == 0  # Zipf head
    for step in (1, 2, 3):
        dom, slot = wl.config4_ids(4, step)
        filling = wl.config4_region(step)
        assert not ((slot >= filling) & (slot < filling + 64)).any()
        assert slot.max() < 512 and (dom == slot % 8).all()


def test_zipf_probabilities(wl):
    u = wl.uniform(0, 123, 200_000)
    k = wl.zipf_draw(u, 10, 1.1)
    p = np.arange(1, 11) ** -1.1
    p /= p.sum()
    freq = np.bincount(k, minlength=11)[1:] / k.size
    assert np.abs(freq - p).max() < 0.005


def test_algorithmic_bytes_config3(wl):
    w = wl.config3()
    b = sum(w.algorithmic_bytes(l) for l in range(7))
    # x 19.9 MB, y 44.0 MB, centroids 83.9 MB, residuals from the distinct slots present
    n_slots = len(np.unique(w.slot_ids))
    exp = 256 * 38912 * 2 + 256 * 43008 * 4 + 8 * 64 * 81920 * 2 + n_slots * 2 * 81920 * 2
    assert b == exp
