"""salt_lora_apply_host: applies on page-locked host activations through the
library's staging pipe (copies in, apply, copies out on their own streams),
against the fp64 oracle and bit for bit against the same grouped apply on
device buffers (one launch configuration, a deterministic kernel)."""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_close, oracle_tables

pytestmark = pytest.mark.gpu


def _host_views(salt, shapes):
    """One salt_host_alloc region carved into bf16 host tensors of the given shapes."""
    sizes = [int(np.prod(s)) * 2 for s in shapes]
    offs = np.cumsum([0] + [(n + 255) // 256 * 256 for n in sizes])
    buf = salt.salt_host_alloc(int(offs[-1]))
    views = [buf.tensor[int(o):int(o) + n].view(torch.bfloat16).view(*s) for o, n, s in zip(offs, sizes, shapes)]
    return buf, views


def test_host_pipe_config3_layer(salt_lib, oracle_mod, wl):
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_bits, bf16_tensor
    salt = salt_lib
    w = wl.config3()
    w.y_mode = "normal"
    T = w.T
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        r.build()
        shapes = []
        for l in range(7):
            shapes += [(T, int(w.d_in[l])), (T, int(w.d_out[l]))]
        buf, views = _host_views(salt, shapes)
        xh, yh = views[0::2], views[1::2]
        for l in range(7):
            xh[l].copy_(bf16_tensor(w.x(l), "cpu"))
            yh[l].copy_(bf16_tensor(w.y_in(l), "cpu"))
        # two stages for four groups: the stages are reused while copies are in flight
        pipe = salt.salt_host_pipe_create(r.ctx, 2)
        stream = torch.cuda.Stream()
        for grp in w.group:
            salt.salt_lora_apply_host(pipe, r.seg, grp, [xh[l] for l in grp], [yh[l] for l in grp], stream)
        salt.salt_host_pipe_wait(pipe, stream)
        stream.synchronize()
        got = [yh[l].clone() for l in range(7)]
        assert r.device_error() == 0
        # the same groups on device buffers
        xs, ys = r.alloc_xy(range(7))
        for grp in w.group:
            r.apply(grp, [xs[l] for l in grp], [ys[l] for l in grp])
        torch.cuda.synchronize()
        for l in range(7):
            g = got[l].view(torch.int16).numpy().view(np.uint16)
            np.testing.assert_array_equal(g, bf16_bits(ys[l]), err_msg=f"host pipe vs device apply, layer {l}")
            cents, res = oracle_tables(w, l)
            ref = oracle_mod.apply(w.x(l), w.y_in(l), w.dom_ids, w.slot_ids, cents, res)
            assert_close(g, ref, f"host pipe {w.layers[l][0]}")
        pipe.close()
        buf.close()


def test_host_pipe_rejects_pageable_and_oversize(salt_lib, wl):
    from paper_2608_03579_gb300.runner import SaltRunner
    salt = salt_lib
    w = wl.config0()
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        r.build()
        pipe = salt.salt_host_pipe_create(r.ctx, 2)
        x = torch.zeros(w.T, 512, dtype=torch.bfloat16)   # ordinary pageable host memory
        y = torch.zeros(w.T, 512, dtype=torch.bfloat16)
        with pytest.raises(salt.SaltError) as e:
            salt.salt_lora_apply_host(pipe, r.seg, [0], [x], [y])
        assert e.value.status == 3  # SALT_ERR_NOT_PINNED_HOST
        pipe.close()
        small = salt.salt_host_pipe_create(r.ctx, 2, 4096)  # smaller than one token batch's x and y
        buf, (xp, yp) = _host_views(salt, [(w.T, 512), (w.T, 512)])
        with pytest.raises(salt.SaltError) as e:
            salt.salt_lora_apply_host(small, r.seg, [0], [xp], [yp])
        assert e.value.status == 1  # SALT_ERR_INVALID_ARG
        small.close()
        buf.close()
