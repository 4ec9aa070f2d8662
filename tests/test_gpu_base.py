"""salt_lora_apply_with_base: the base-weight GEMM fused with the SALT delta
(y = x W_base + s_c (x A_c) B_c + s_u (x a_u) b_u, y written), against the
fp64 oracle's W_final evaluation, for both weight layouts."""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_close, guarded_like, guards_intact, oracle_tables

pytestmark = pytest.mark.gpu


def _weight(wl, seed, d_in, d_out, layout):
    W = wl.normal_bf16(seed, wl.stream_id(wl.K_AUX, 40, d_in, d_out), d_in * d_out, 1.0 / np.sqrt(d_in))
    W = W.reshape(d_in, d_out)
    return W if layout == 0 else np.ascontiguousarray(W.T)


def _run(salt, r, w, l, W, layout):
    from paper_2608_03579_gb300.runner import bf16_bits, bf16_tensor
    x = bf16_tensor(w.x(l))
    Wd = bf16_tensor(W)
    y0 = torch.full((w.T, int(w.d_out[l])), float("nan"), dtype=torch.bfloat16, device="cuda")  # never read
    y, buf = guarded_like(y0)
    salt.salt_lora_apply_with_base(r.ctx, r.seg, l, x, Wd, layout, y)
    torch.cuda.synchronize()
    assert guards_intact(buf), "a store ran past y"
    return bf16_bits(y)


def _ref(oracle_mod, w, l, W, layout, rows=None):
    cents, res = oracle_tables(w, l)
    dom = w.dom_ids if rows is None else w.dom_ids[rows]
    slot = w.slot_ids if rows is None else w.slot_ids[rows]
    return oracle_mod.apply(w.x(l), None, w.dom_ids, w.slot_ids, cents, res, rows=rows, w_base=W, w_layout=layout)


@pytest.mark.parametrize("layout", [0, 1])
def test_with_base_config0(salt_lib, oracle_mod, wl, layout):
    from paper_2608_03579_gb300.runner import SaltRunner
    w = wl.config0()
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        r.build()
        W = _weight(wl, 0, 512, 512, layout)
        got = _run(salt_lib, r, w, 0, W, layout)
        assert r.device_error() == 0
        assert salt_lib.salt_guard_check(r.ctx, r.seg) == 0
    assert_close(got, _ref(oracle_mod, w, 0, W, layout), f"with base, config 0, layout {layout}")


@pytest.mark.parametrize("layout", [0, 1])
def test_with_base_ragged_and_absent_ids(salt_lib, oracle_mod, wl, layout):
    """d_in, d_out not multiples of the tiles, tokens with no term (x W_base
    alone), a batch that is not a multiple of 128 tokens."""
    from paper_2608_03579_gb300.runner import SaltRunner
    T, n_users = 200, 12
    u = (wl.uniform(21, 1, T) * n_users).astype(np.int32) % n_users
    dom = (u % 3).astype(np.int32)
    slot = u.copy()
    none = wl.uniform(21, 2, T) < 0.2
    dom[none], slot[none] = -1, -1
    dom[wl.uniform(21, 3, T) < 0.1] = -1
    w = wl.Workload("ragged_base", 21, [("p", 72, 520)], 3, [8, 16, 5], n_users, [1, 2] * (n_users // 2),
                    dom_ids=dom, slot_ids=slot)
    w.y_mode = "zeros"
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        r.build()
        W = _weight(wl, 21, 72, 520, layout)
        got = _run(salt_lib, r, w, 0, W, layout)
        assert r.device_error() == 0
    assert_close(got, _ref(oracle_mod, w, 0, W, layout), f"with base, ragged, layout {layout}")


@pytest.mark.parametrize("layout", [0, 1])
def test_with_base_config3(salt_lib, oracle_mod, wl, layout):
    """One Llama-3.1-8B layer's q (4096 -> 4096) and down (14336 -> 4096) at
    256 decode tokens; rows at every 128-token tile edge, every row block's
    first and last token and a spread sample."""
    from paper_2608_03579_gb300.runner import SaltRunner
    w = wl.config3()
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        r.build()
        exp = r.export()
        starts = exp["blocks"][:, 0]
        ends = starts + exp["blocks"][:, 1]
        pos = np.unique(np.concatenate([starts, ends - 1, [0, 127, 128, w.T - 1]]))
        rows = np.unique(np.concatenate([exp["perm"][pos[(pos >= 0) & (pos < w.T)]],
                                         (wl.uniform(3, 77, 24) * w.T).astype(int)]))
        for l in (0, 6):
            W = _weight(wl, 3, int(w.d_in[l]), int(w.d_out[l]), layout)
            got = _run(salt_lib, r, w, l, W, layout)
            assert r.device_error() == 0
            assert_close(got[rows], _ref(oracle_mod, w, l, W, layout, rows=rows),
                         f"with base, config 3 {w.layers[l][0]}, layout {layout}")
