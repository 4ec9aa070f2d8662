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
    "centroid_sign": ("out[j] += gt * s_c[d] * acc;", "out[j] -= gt * s_c[d] * acc;"),
    "centroid_A_transposed": ("oracle_bf16_value(At_c[d][k * d_in + i])", "oracle_bf16_value(At_c[d][i * R + k])"),
    "residual_B_rank_ignored": ("oracle_bf16_value(B_u[u][k * d_out + j])", "oracle_bf16_value(B_u[u][j])"),
    "y_in_dropped": ("out[j] = y_in ? oracle_bf16_value(y_in[t * d_out + j]) : 0.0;", "out[j] = 0.0;"),
    "x_row_index": ("const uint16_t *xt = x + t * d_in;", "const uint16_t *xt = x + (t / 2) * d_in;"),
    "tie_order_reversed": ("if (a->t != b->t) return a->t < b->t ? -1 : 1;", "if (a->t != b->t) return a->t < b->t ? 1 : -1;"),
    "user_run_ignores_domain": ("if (new_dom || keys[i].u != keys[i - 1].u) {",
                                "if (i == 0 || keys[i].u != keys[i - 1].u) {"),
    "adapter_bytes_fp32": ("return params * 2;", "return params * 4;"),
    "gamma_dropped": ("out[j] += gt * s_c[d] * acc;", "out[j] += s_c[d] * acc;"),
    "gamma_wrong_token": ("double gt = gamma ? gamma[t] : 1.0;", "double gt = gamma ? gamma[0] : 1.0;"),
    "gbin_ignored_in_runs": ("int new_dom = i == 0 || keys[i].d != keys[i - 1].d || keys[i].g != keys[i - 1].g;",
                             "int new_dom = i == 0 || keys[i].d != keys[i - 1].d;"),
    "gbin_kept_without_centroid": ("keys[t].g = (gbin && dom[t] >= 0) ? gbin[t] : -1;",
                                   "keys[t].g = gbin ? gbin[t] : -1;"),
    "gbin_sorted_after_slot": ("    if (a->g != b->g) return a->g < b->g ? -1 : 1;\n    if (a->u != b->u) return a->u < b->u ? -1 : 1;",
                               "    if (a->u != b->u) return a->u < b->u ? -1 : 1;\n    if (a->g != b->g) return a->g < b->g ? -1 : 1;"),
    "align_B_rank_ignored": ("dw[j] += a * oracle_bf16_value(B[k * d_out + j]);",
                             "dw[j] += a * oracle_bf16_value(B[j]);"),
    "align_centroid_scale_dropped": ("wb[j] *= s_c;", "wb[j] *= 1.0;"),
    "align_eps_in_numerator": ("double cosine = tr / (n_dw * n_wb + eps);",
                               "double cosine = (tr + eps) / (n_dw * n_wb + eps);"),
    "align_norm_not_rooted": ("double n_dw = sqrt(nn_dw), n_wb = sqrt(nn_wb);",
                              "double n_dw = nn_dw, n_wb = sqrt(nn_wb);"),
    "fold_layout_ignored": ("int64_t idx = layout ? j * d_in + i : i * d_out + j;", "int64_t idx = i * d_out + j;"),
    "fold_A_transposed": ("double a = oracle_bf16_value(At_c[k * d_in + i]);\n            for (int64_t j = 0; j < d_out; ++j) row[j]",
                          "double a = oracle_bf16_value(At_c[i * rc + k]);\n            for (int64_t j = 0; j < d_out; ++j) row[j]"),
    "base_term_dropped": ("                out[j] += base;", "                out[j] += 0.0 * base;"),
    "base_layout_ignored": ("oracle_bf16_value(W_base[w_layout ? j * d_in + i : i * d_out + j])",
                            "oracle_bf16_value(W_base[i * d_out + j])"),
    "base_x_column": ("base += oracle_bf16_value(xt[i])", "base += oracle_bf16_value(xt[j % d_in])"),
    "fold_scale_dropped": ("W_out[idx] = oracle_bf16_value(W[idx]) + scale * row[j];",
                           "W_out[idx] = oracle_bf16_value(W[idx]) + row[j];"),
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
        ("gamma_dense", lambda: [pins.test_dense_closed_form_with_gamma(orc, wl, s) for s in (20, 21)]),
        ("gamma_segments_sort", lambda: pins.test_gamma_segments_match_library_sort(orc, wl, 2000, 8, 4, 300)),
        ("gamma_segments_plain", lambda: pins.test_gamma_segments_without_bins_are_plain(orc, wl)),
        ("align_dense", lambda: [pins.test_align_dense_brute_force(orc, wl, *a) for a in
                                 ((0, 2, 8, 24, 40, 1.0, 1.0), (1, 1, 16, 64, 16, 2.0, -0.5))]),
        ("align_rank_one", lambda: pins.test_align_rank_one_closed_form(orc, wl)),
        ("align_special", lambda: pins.test_align_special_cases(orc, wl)),
        ("fold_dense", lambda: [pins.test_fold_dense_brute_force(orc, wl, lay) for lay in (0, 1)]),
        ("fold_special", lambda: pins.test_fold_special_cases(orc, wl)),
        ("w_final_dense", lambda: [pins.test_w_final_dense_closed_form(orc, wl, s, lay) for s, lay in ((30, 0), (31, 1))]),
        ("w_final_layouts", lambda: pins.test_w_final_zero_base_and_layouts(orc, wl)),
        ("w_final_fold", lambda: pins.test_w_final_fold_then_residual_only(orc, wl)),
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
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-o", str(so), str(mutant_c), "-lm"], check=True)
    spec = importlib.util.spec_from_file_location(f"oracle_mutant_{name}", os.path.join(ROOT, "oracle", "__init__.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    mod.use_library(str(so))
    failed = _checks(mod, wl)
    assert failed, f"mutant {name} passed every pin"
