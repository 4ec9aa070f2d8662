"""C-ABI library on the CPU: it builds, loads and exports every declared
symbol; host-only entry points (blob sizing and packing, config checks)
behave as specified.  No compute call is made without a GPU."""
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "salt.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(salt_[a-z_0-9]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(salt_lib):
    import ctypes
    lib = ctypes.CDLL(salt_lib.LIB_PATH)
    names = _declared_functions()
    assert len(names) >= 14
    for n in names:
        assert hasattr(lib, n), n
    # and the binding exposes the same names
    for n in names:
        assert hasattr(salt_lib, n), n


def test_abi_version_and_status_strings(salt_lib):
    assert salt_lib.salt_abi_version() == 1
    assert salt_lib.salt_status_string(0) == "ok"
    assert "reloaded" in salt_lib.salt_status_string(16)


def test_blob_bytes_match_oracle(salt_lib, oracle_mod, wl):
    for shapes, layers in ((wl.MISTRAL7B_QV, 32), (wl.LLAMA3B_ALL, 28), (wl.PYTHIA12B_ATTN, 36), (wl.LLAMA8B_LAYER, 32)):
        din = [a for (_, a, b) in shapes] * layers
        dout = [b for (_, a, b) in shapes] * layers
        for r in (1, 2, 4, 16):
            assert salt_lib.salt_residual_blob_bytes(din, dout, r) == 256 + oracle_mod.adapter_bytes(din, dout, r)
    assert salt_lib.salt_residual_blob_bytes([8], [8], 0) == -1


def test_blob_pack_layout(salt_lib, wl):
    din, dout, r = [16, 24], [8, 32], 2
    A = np.arange(r * sum(din), dtype=np.uint16)
    B = (np.arange(r * sum(dout), dtype=np.uint16) + 1000)
    n = salt_lib.salt_residual_blob_bytes(din, dout, r)
    blob = np.zeros(n, dtype=np.uint8)
    salt_lib.salt_residual_blob_pack(din, dout, r, 0.75, A, B, blob, n)
    hdr = blob[:256]
    assert hdr[:8].view(np.uint64)[0] == 0x3153455254414C53
    assert hdr[8:12].view(np.uint32)[0] == 1
    assert hdr[12:16].view(np.int32)[0] == r
    assert hdr[16:20].view(np.int32)[0] == 2
    assert hdr[20:24].view(np.float32)[0] == np.float32(0.75)
    assert hdr[24:32].view(np.uint64)[0] == 2 * r * (sum(din) + sum(dout))
    pay = blob[256:].view(np.uint16)
    # layer 0: At [r][16] then B [r][8]; layer 1: At [r][24] then B [r][32]
    np.testing.assert_array_equal(pay[0:32], A[0:32])
    np.testing.assert_array_equal(pay[32:48], B[0:16])
    np.testing.assert_array_equal(pay[48:96], A[32:80])
    np.testing.assert_array_equal(pay[96:160], B[16:80])
    with pytest.raises(salt_lib.SaltError):
        salt_lib.salt_residual_blob_pack(din, dout, r, 1.0, A, B, blob, n - 1)


@pytest.mark.parametrize("kw,status", [
    (dict(d_in=[12], d_out=[8]), "SALT_ERR_INVALID_ARG"),           # not a multiple of 8
    (dict(rc_max=65), "SALT_ERR_RANK"),
    (dict(r_max=0), "SALT_ERR_RANK"),
    (dict(r_max=81), "SALT_ERR_RANK"),
    (dict(r_max=65), "SALT_ERR_RANK"),                             # rc_max 16 + 65 > 80
    (dict(n_slots=1 << 17), "SALT_ERR_INVALID_ARG"),
    (dict(max_tokens=16385), "SALT_ERR_TOO_MANY_TOKENS"),
    (dict(max_tokens=0), "SALT_ERR_TOO_MANY_TOKENS"),
])
def test_config_rejected_before_any_cuda_call(salt_lib, kw, status):
    args = dict(d_in=[64], d_out=[64], n_domains=2, rc_max=16, n_slots=4, r_max=2, max_tokens=16, device=0)
    args.update(kw)
    with pytest.raises(salt_lib.SaltError) as e:
        salt_lib.salt_ctx_create(**args)
    assert e.value.name == status


def test_binding_fails_loudly_without_library(tmp_path, monkeypatch):
    """The binding raises ImportError when libsalt.so is absent: no fallback."""
    import importlib.util
    src = os.path.join(ROOT, "paper_2608_03579_gb300", "salt.py")
    fake = tmp_path / "salt.py"
    fake.write_text(open(src).read())
    spec = importlib.util.spec_from_file_location("salt_nolib", str(fake))
    mod = importlib.util.module_from_spec(spec)
    with pytest.raises(ImportError):
        spec.loader.exec_module(mod)


def test_align_loss_checks_arguments_before_any_cuda_call(salt_lib):
    """salt_align_loss validates every pair on the host first; n = 0 is a no-op."""
    base = dict(At=4096, B=8192, At_c=12288, B_c=16384, r=2, rc=8, d_in=64, d_out=64, s=1.0, s_c=1.0)
    for kw, name in [(dict(r=0), "SALT_ERR_RANK"), (dict(rc=0), "SALT_ERR_RANK"), (dict(r=64, rc=65), "SALT_ERR_RANK"),
                     (dict(d_in=60), "SALT_ERR_INVALID_ARG"), (dict(d_out=0), "SALT_ERR_INVALID_ARG"),
                     (dict(B_c=0), "SALT_ERR_INVALID_ARG"), (dict(At=4098), "SALT_ERR_ALIGN")]:
        q = dict(base)
        q.update(kw)
        with pytest.raises(salt_lib.SaltError) as e:
            salt_lib.salt_align_loss([q], 1e-8, 256, None, 0)
        assert e.value.name == name, (kw, e.value.name)
    salt_lib.salt_align_loss([], 1e-8, 256, None, 0)
