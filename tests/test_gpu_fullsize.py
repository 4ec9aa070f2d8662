"""Full-size parity in the launch configuration bench.py times.

The Llama-3.1-8B 32-layer decode step (512 tokens, 8 rank-64 centroids, a
512-slot pool of rank-2 residuals, 64 swaps per step on a side stream, 128
grouped applies replayed from one CUDA graph) runs for several steps; then y
is cleared and one more step is run.  Every output row of 21 projections
(five fixed ones, and one of each launch group in every 8th layer) is checked
against the fp64 oracle with the slot contents that step actually read (fixed
slots: the initial residuals; the region swapped in by the previous step:
that step's blobs).
"""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_close

pytestmark = pytest.mark.gpu


class _Args:
    layers = 32
    mode = "salt"


@pytest.fixture(scope="module")
def step(salt_lib):
    import bench
    st = bench.Step(_Args(), 0)
    st.capture()
    yield st
    st.close()


def test_config4_step_full_projections(step, oracle_mod, wl):
    st = step
    s_last = 5
    for s in range(s_last):
        st.step(s)
    st.join_side()
    torch.cuda.synchronize()
    st.y_all.zero_()
    torch.cuda.synchronize()
    st.step(s_last)
    st.join_side()
    torch.cuda.synchronize()
    assert st.runner.device_error() == 0
    # no store or swap ran past the arenas, the slot pool, the V tiles or the partials
    assert st.salt.salt_guard_check(st.runner.ctx, st.runner.seg) == 0

    dom, slot = st.ids[s_last % st.N_ID_SETS]
    prev_region = wl.config4_region(s_last - 1)
    prev_version = 1 + ((s_last - 1) % 2)
    w = st.w
    from paper_2608_03579_gb300.runner import bf16_bits
    rows = np.arange(st.T)
    # every row of: q, v and down of layer 1, gate of layer 14, down of layer 31;
    # and one projection of each launch group (q/k/v, o, gate/up, down) in every
    # 8th layer: every row block and every K split of every launch shape
    checks = [0, 2, 13, 100, 223]
    for layer in (0, 8, 16, 24):
        checks += [7 * layer + 1, 7 * layer + 3, 7 * layer + 5, 7 * layer + 6]
    used = sorted(set(int(u) for u in slot if u >= 0))
    for l in sorted(set(checks)):
        din, dout = w.layers[l][1], w.layers[l][2]
        cents = [(w.centroid_At(d, l), w.centroid_B(d, l), 1.0) for d in range(w.n_domains)]
        res = [None] * w.n_slots
        for u in used:
            v = prev_version if prev_region <= u < prev_region + wl.C4_REGION else 0
            res[u] = (w.residual_At(u, l, v), w.residual_B(u, l, v), 1.0)
        ref = oracle_mod.apply(w.x(l), np.zeros((st.T, dout), np.uint16), dom, slot, cents, res)
        got = bf16_bits(st.ys[l].view(st.T, dout))
        assert_close(got, ref, f"32-layer step, projection {w.layers[l][0]}")
