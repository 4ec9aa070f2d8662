"""The factored alignment regulariser (Eq. 2) on the GPU against the dense
fp64 oracle.

Tolerance.  Each Gram entry G_ij = sum_t F_it F_jt is an fp32 sum of d exact
products (a product of two bf16 is exact in fp32), so its error is at most
about d u sum_t |F_it F_jt| with u = 2^-24; the test allows 4 d u.  The
trace and the squared norms are block sums of G_in o G_out, so their errors
are bounded by the same sums with |G| and the entry bounds, plus the fp32
rounding of the products and of the sums themselves (fixed order, at most 64
additions deep: 66 u times the block's sum of |G_in o G_out|);
the cosine's error follows to first order.  The bound is computed from the
factors of each case, with a floor of 1e-6 (float output)."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _f(wl, bits):
    return wl.bf16_bits_to_float(bits).astype(np.float64)


def _bound(wl, At, B, Atc, Bc, s, s_c, cos_ref):
    r = At.shape[0]
    Fi, Fo = np.vstack([_f(wl, At), _f(wl, Atc)]), np.vstack([_f(wl, B), _f(wl, Bc)])
    Gi, Go = Fi @ Fi.T, Fo @ Fo.T
    Ei = 4 * Fi.shape[1] * 2.0 ** -24 * (np.abs(Fi) @ np.abs(Fi).T)
    Eo = 4 * Fo.shape[1] * 2.0 ** -24 * (np.abs(Fo) @ np.abs(Fo).T)
    E = Ei * np.abs(Go) + np.abs(Gi) * Eo + Ei * Eo + 66 * 2.0 ** -24 * np.abs(Gi * Go)
    num_e = E[:r, r:].sum()
    na, nc = (Gi * Go)[:r, :r].sum(), (Gi * Go)[r:, r:].sum()
    na_e, nc_e = E[:r, :r].sum(), E[r:, r:].sum()
    den = np.sqrt(max(na, 1e-300)) * np.sqrt(max(nc, 1e-300))
    return num_e / den + abs(cos_ref) * (na_e / (2 * max(na, 1e-300)) + nc_e / (2 * max(nc, 1e-300))) + 1e-6


def _pair(wl, seed, r, rc, din, dout):
    sid = wl.stream_id
    At = wl.normal_bf16(seed, sid(93, 1), r * din, 1 / np.sqrt(din)).reshape(r, din)
    B = wl.normal_bf16(seed, sid(93, 2), r * dout, 1 / np.sqrt(r)).reshape(r, dout)
    Atc = wl.normal_bf16(seed, sid(93, 3), rc * din, 1 / np.sqrt(din)).reshape(rc, din)
    Bc = wl.normal_bf16(seed, sid(93, 4), rc * dout, 1 / np.sqrt(rc)).reshape(rc, dout)
    return At, B, Atc, Bc


def _run(salt, cases, eps=1e-8):
    from paper_2608_03579_gb300.runner import bf16_tensor
    keep, pairs = [], []
    for (At, B, Atc, Bc, s, s_c) in cases:
        t = [bf16_tensor(a) for a in (At, B, Atc, Bc)]
        keep.append(t)
        pairs.append(dict(At=t[0], B=t[1], At_c=t[2], B_c=t[3], r=At.shape[0], rc=Atc.shape[0],
                          d_in=At.shape[1], d_out=B.shape[1], s=s, s_c=s_c))
    loss = torch.full((len(cases),), float("nan"), device="cuda")
    cos = torch.full((len(cases),), float("nan"), device="cuda")
    salt.salt_align_loss(pairs, eps, loss, cos)
    torch.cuda.synchronize()
    return loss.cpu().numpy().astype(np.float64), cos.cpu().numpy().astype(np.float64)


SHAPES = [(2, 8, 64, 40, 1.0, 1.0), (1, 16, 520, 136, 2.0, -0.5), (16, 64, 4096, 1024, 1.0, 0.8),
          (3, 5, 8, 8, 0.25, 3.0), (64, 64, 264, 4104, 1.0, 1.0), (1, 127, 72, 16, 1.0, 1.0)]


def test_align_matches_dense_oracle(salt_lib, oracle_mod, wl):
    cases = []
    for i, (r, rc, din, dout, s, s_c) in enumerate(SHAPES):
        cases.append((*_pair(wl, i, r, rc, din, dout), s, s_c))
    loss, cos = _run(salt_lib, cases)
    for i, c in enumerate(cases):
        ref = oracle_mod.align_loss(*c[:2], c[4], *c[2:4], c[5])
        tol = _bound(wl, c[0], c[1], c[2], c[3], c[4], c[5], ref["cosine"])
        assert abs(cos[i] - ref["cosine"]) <= tol, (i, cos[i], ref["cosine"], tol)
        assert abs(loss[i] - ref["loss"]) <= tol, (i, loss[i], ref["loss"], tol)


def test_align_special_cases(salt_lib, wl):
    At, B, Atc, Bc = _pair(wl, 9, 4, 4, 256, 128)
    neg = Bc ^ np.uint16(0x8000)  # -B_c, exactly
    zero = np.zeros_like(Atc)
    loss, cos = _run(salt_lib, [(Atc, Bc, Atc, Bc, 1.0, 1.0), (Atc, neg, Atc, Bc, 1.0, 1.0),
                                (At, B, zero, Bc, 1.0, 1.0)])
    assert abs(loss[0]) <= 1e-5 and abs(loss[1] - 2.0) <= 1e-5
    assert loss[2] == 1.0 and cos[2] == 0.0


def test_align_many_pairs_across_launches(salt_lib, oracle_mod, wl):
    """More pairs than one launch takes (32), with mixed shapes."""
    cases = []
    for i in range(41):
        r, rc = 1 + i % 3, 4 + (i * 7) % 29
        din, dout = 8 * (1 + (i * 5) % 40), 8 * (1 + (i * 3) % 50)
        cases.append((*_pair(wl, 100 + i, r, rc, din, dout), 1.0, 1.0))
    loss, cos = _run(salt_lib, cases)
    for i, c in enumerate(cases):
        ref = oracle_mod.align_loss(*c[:2], 1.0, *c[2:4], 1.0)
        assert abs(cos[i] - ref["cosine"]) <= _bound(wl, *c[:4], 1.0, 1.0, ref["cosine"]), i


@pytest.mark.parametrize("din,dout", [(4096, 4096), (4096, 14336), (14336, 4096)])
def test_align_llama8b_projection(salt_lib, oracle_mod, wl, din, dout):
    """A Llama-3.1-8B projection: rank-16 task update against the rank-64
    centroid (the dense oracle forms both d_in x d_out matrices)."""
    c = (*_pair(wl, din + dout, 16, 64, din, dout), 1.0, 1.0)
    loss, cos = _run(salt_lib, [c])
    ref = oracle_mod.align_loss(*c[:2], 1.0, *c[2:4], 1.0)
    assert abs(cos[0] - ref["cosine"]) <= _bound(wl, *c[:4], 1.0, 1.0, ref["cosine"])


def test_align_argument_errors(salt_lib, wl):
    from paper_2608_03579_gb300.runner import bf16_tensor
    At, B, Atc, Bc = _pair(wl, 1, 2, 4, 64, 64)
    t = [bf16_tensor(a) for a in (At, B, Atc, Bc)]
    loss = torch.zeros(1, device="cuda")
    base = dict(At=t[0], B=t[1], At_c=t[2], B_c=t[3], r=2, rc=4, d_in=64, d_out=64, s=1.0, s_c=1.0)
    for kw, name in [(dict(r=0), "SALT_ERR_RANK"), (dict(rc=127), "SALT_ERR_RANK"),
                     (dict(d_in=60), "SALT_ERR_INVALID_ARG"), (dict(At=t[0].data_ptr() + 2), "SALT_ERR_ALIGN")]:
        q = dict(base)
        q.update(kw)
        with pytest.raises(salt_lib.SaltError) as e:
            salt_lib.salt_align_loss([q], 1e-8, loss)
        assert e.value.name == name
