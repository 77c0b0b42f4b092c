"""The pins catch plausible mistakes planted in a copy of the oracle.

Each mutant is one textual edit of ``oracle/oracle.c`` (a dropped term, a
wrong sign or index, a confused leading dimension, a lost compensation
term, a truncated integer product, an off-by-one trim).  The copy is built
with the same flags in a temporary directory and must fail at least one pin
from ``oracle_pins``.  The real oracle is never modified.
"""
import os

import pytest

import oracle
import oracle_pins as P

SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")

# (name, text to replace, replacement, which occurrence (0-based))
MUTANTS = [
    ("f32_dropped_last_term", "for (int64_t j = 0; j < N; ++j) {\n            const double a = (double)A",
     "for (int64_t j = 0; j + 1 < N; ++j) {\n            const double a = (double)A", 0),
    ("f32_lda_as_N", "const double a = (double)A[i * lda + j];",
     "const double a = (double)A[i * N + j];", 0),
    ("f32_wrong_sign_s", "s[j] += a * ri;", "s[j] -= a * ri;", 0),
    ("f32_r_for_p", "qi += a * (double)p[j];", "qi += a * (double)r[i];", 0),
    ("f64_lost_product_error_q", "q_lo = q_lo + (perr + serr);", "q_lo = q_lo + serr;", 0),
    ("f64_lost_sum_error_s", "s_lo[j] = s_lo[j] + (perr + serr);",
     "s_lo[j] = s_lo[j] + perr;", 0),
    ("f64_twosum_sign", "*err = (x - (t - z)) + (y - z);", "*err = (x - (t - z)) - (y - z);", 0),
    ("f64_row_index", "const double ri = r[i];", "const double ri = r[M - 1 - i];", 0),
    ("i32_truncated_product", "qi += (uint64_t)(a * (int64_t)p[j]);",
     "qi += (uint64_t)(uint32_t)(a * (int64_t)p[j]);", 0),
    ("i32_column_uses_p", "s_acc[j] += (uint64_t)(a * ri);",
     "s_acc[j] += (uint64_t)(a * (int64_t)p[j]);", 0),
    ("absdot_missing_abs", "acc += a * fabs((double)p[j]);", "acc += a * (double)p[j];", 0),
    ("trim_off_by_one", "for (int64_t i = k; i < R - k; ++i)",
     "for (int64_t i = k; i <= R - k; ++i)", 0),
    ("trim_wrong_count", "*out = sum / (double)(R - 2 * k);", "*out = sum / (double)(R - k);", 0),
    ("gesummv_swapped_scalars", "y[i] = alpha * ta + beta * tb;",
     "y[i] = beta * ta + alpha * tb;", 0),
    ("gesummv_lda_for_ldb", "tb += (double)B[i * ldb + j] * (double)x[j];",
     "tb += (double)B[i * lda + j] * (double)x[j];", 0),
    ("gesummv_f64_lost_compensation", "y[i] = alpha * (a_hi + a_lo) + beta * (b_hi + b_lo);",
     "y[i] = alpha * a_hi + beta * (b_hi + b_lo);", 0),
    ("atax_second_pass_uses_x", "for (int64_t j = 0; j < N; ++j) y[j] += (double)A[i * lda + j] * tmp;",
     "for (int64_t j = 0; j < N; ++j) y[j] += (double)A[i * lda + j] * (double)x[j];", 0),
    ("atax_dropped_x", "for (int64_t j = 0; j < N; ++j) tmp += (double)A[i * lda + j] * (double)x[j];",
     "for (int64_t j = 0; j < N; ++j) tmp += (double)A[i * lda + j];", 0),
    ("atax_f64_tmp_uncompensated", "const double tmp = t_hi + t_lo;", "const double tmp = t_hi;", 0),
    ("gemver_wrong_v", "+ (double)u1[i] * (double)v1[j]", "+ (double)u1[i] * (double)v2[j]", 0),
    ("gemver_x_without_z", "xo[j] = (double)x[j] + beta * acc + (double)z[j];",
     "xo[j] = (double)x[j] + beta * acc;", 0),
    ("gemver_w_uses_old_x", "for (int64_t j = 0; j < N; ++j) acc += ahat[i * N + j] * xo[j];",
     "for (int64_t j = 0; j < N; ++j) acc += ahat[i * N + j] * (double)x[j];", 0),
    ("gemver_alpha_beta_swapped", "wo[i] = (double)w[i] + alpha * acc;",
     "wo[i] = (double)w[i] + beta * acc;", 0),
    ("gemver_f64_dropped_update_error", "ahat[i * N + j] = s2 + ((t1 + t2) + (e1 + e2));",
     "ahat[i * N + j] = s2;", 0),
]


def _mutate(text, old, new, occurrence):
    start = -1
    for _ in range(occurrence + 1):
        start = text.find(old, start + 1)
        assert start >= 0, f"mutation site not found: {old!r}"
    return text[:start] + new + text[start + len(old):]


def test_real_oracle_passes_every_pin():
    assert P.failing_pins(oracle.load()) == []


@pytest.mark.parametrize("name,old,new,occ", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(tmp_path, name, old, new, occ):
    text = open(SRC).read()
    src = tmp_path / "oracle_mutant.c"
    src.write_text(_mutate(text, old, new, occ))
    so = oracle.build(str(src), str(tmp_path / f"liboracle_{name}.so"))
    failed = P.failing_pins(oracle.load(so))
    assert failed, f"mutant {name} passed every pin"
