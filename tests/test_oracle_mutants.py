"""The oracle pins must catch plausible mistakes (CPU only).

Each case plants one mistake in a copy of ``oracle/salt_oracle.c`` (a dropped
term, a wrong sign, a transposed operand, an ignored index, a broken tie
order, a wrong element size), builds it with the host C compiler into a
temporary directory, binds a fresh copy of the oracle module to it and runs
the pin checks of ``test_oracle_pins.py``: at least one must fail.
"""
import importlib.util
import os
import subprocess

import pytest

import test_oracle_pins as pins

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "salt_oracle.c")

MUTANTS = {
    "residual_scale_dropped": ("out[j] += s_u[u] * acc;", "out[j] += acc;"),
    "centroid_sign": ("out[j] += s_c[d] * acc;", "out[j] -= s_c[d] * acc;"),
    "centroid_A_transposed": ("oracle_bf16_value(At_c[d][k * d_in + i])", "oracle_bf16_value(At_c[d][i * R + k])"),
    "residual_B_rank_ignored": ("oracle_bf16_value(B_u[u][k * d_out + j])", "oracle_bf16_value(B_u[u][j])"),
    "y_in_dropped": ("out[j] = y_in ? oracle_bf16_value(y_in[t * d_out + j]) : 0.0;", "out[j] = 0.0;"),
    "x_row_index": ("const uint16_t *xt = x + t * d_in;", "const uint16_t *xt = x + (t / 2) * d_in;"),
    "tie_order_reversed": ("if (a->t != b->t) return a->t < b->t ? -1 : 1;", "if (a->t != b->t) return a->t < b->t ? 1 : -1;"),
    "user_run_ignores_domain": ("if (i == 0 || keys[i].d != keys[i - 1].d || keys[i].u != keys[i - 1].u) {",
                                "if (i == 0 || keys[i].u != keys[i - 1].u) {"),
    "adapter_bytes_fp32": ("return params * 2;", "return params * 4;"),
}


def _checks(orc, wl):
    """Run every pin; return the names of those that fail."""
    failed = []
    cases = [
        ("hand_example", lambda: pins.test_hand_example(orc)),
        ("dense", lambda: [pins.test_dense_closed_form(orc, wl, s) for s in (0, 1, 2)]),
        ("concat", lambda: pins.test_concatenation_identity(orc, wl, 3)),
        ("zero_residual", lambda: pins.test_zero_residual_is_centroid_only(orc, wl)),
        ("multi_lora", lambda: pins.test_no_centroid_is_plain_multi_lora(orc, wl)),
        ("absent", lambda: pins.test_both_ids_absent_leave_y(orc, wl)),
        ("segments_hand", lambda: pins.test_segments_hand_example(orc)),
        ("segments_sort", lambda: pins.test_segments_match_library_sort(orc, wl, 100, 5, 40)),
        ("segments_tiny", lambda: pins.test_segments_exhaustive_tiny(orc)),
        ("footprints", lambda: pins.test_adapter_bytes_match_paper_tables(orc)),
    ]
    for name, fn in cases:
        try:
            fn()
        except Exception:  # an assertion or a rejected call both count as caught
            failed.append(name)
    return failed


def test_unmodified_oracle_passes_every_pin(oracle_mod, wl):
    assert _checks(oracle_mod, wl) == []


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, wl, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not found exactly once"
    mutant_c = tmp_path / "mutant.c"
    mutant_c.write_text(src.replace(old, new))
    so = tmp_path / "libmutant.so"
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-o", str(so), str(mutant_c)], check=True)
    spec = importlib.util.spec_from_file_location(f"oracle_mutant_{name}", os.path.join(ROOT, "oracle", "__init__.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    mod.use_library(str(so))
    failed = _checks(mod, wl)
    assert failed, f"mutant {name} passed every pin"
