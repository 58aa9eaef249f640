"""The oracle's pins must catch plausible mistakes.

Each case below plants one mistake in a copy of the oracle's C source (on the CPU,
never in the CUDA path), builds it, and runs the pin suite against the broken build
in a subprocess.  The suite must fail for every mutant.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "bandlu_oracle.c")

# (name, text to replace, replacement): each text occurs in the source; the first occurrence is replaced
MUTANTS = [
    ("ipiv_zero_based", "ipiv[j] = (int)(j + p + 1);\n        if (AB_", "ipiv[j] = (int)(j + p);\n        if (AB_"),
    ("last_max_tie_break", "if (v > best) { best = v; p = t; }", "if (v >= best) { best = v; p = t; }"),
    ("update_sign", "fma(-AB_(kv + t, j), u,", "fma(AB_(kv + t, j), u,"),
    ("short_swap_range", "for (int64_t c = j; c <= ju; ++c) {", "for (int64_t c = j; c < ju; ++c) {"),
    ("km_not_clamped", "int64_t km = (int64_t)kl < n - 1 - j ? (int64_t)kl : n - 1 - j;\n        /* pivot",
     "int64_t km = (int64_t)kl;\n        /* pivot"),
    ("reach_ignores_pivot_row", "int64_t reach = j + ku + p < n - 1 ? j + ku + p : n - 1;",
     "int64_t reach = j + ku < n - 1 ? j + ku : n - 1;"),
    ("divide_instead_of_reciprocal", "for (int64_t t = 1; t <= km; ++t) AB_(kv + t, j) *= rcp;",
     "for (int64_t t = 1; t <= km; ++t) AB_(kv + t, j) /= AB_(kv, j);"),
    ("pivot_search_misses_last_row", "for (int64_t t = 1; t <= km; ++t) {\n            double v",
     "for (int64_t t = 1; t < km; ++t) {\n            double v"),
    ("detect_lower_upper_swapped", "if (i - j > best_l) best_l = i - j;", "if (j - i > best_l) best_l = j - i;"),
    ("convert_drops_last_subdiagonal", "int64_t i1 = j + kl < n - 1 ? j + kl : n - 1;\n        for (int64_t i = i0; i <= i1; ++i) AB[(kv + i - j) + j * ldab] = A",
     "int64_t i1 = j + kl - 1 < n - 1 ? j + kl - 1 : n - 1;\n        for (int64_t i = i0; i <= i1; ++i) AB[(kv + i - j) + j * ldab] = A"),
    ("residual_drops_interchange", "if (p != j) {\n            for (int64_t c = j; c <= c1; ++c) {",
     "if (0) {\n            for (int64_t c = j; c <= c1; ++c) {"),
    ("fill_rows_not_cleared", "for (int64_t r = 0; r < kl; ++r) AB_(r, c) = 0.0;", "for (int64_t r = 0; r < 0; ++r) AB_(r, c) = 0.0;"),
    ("info_reports_last_zero_pivot", "} else if (info == 0) {\n            info = (int)(j + 1);\n        }\n    }\n#undef AB_",
     "} else {\n            info = (int)(j + 1);\n        }\n    }\n#undef AB_"),
    ("predicate_drops_conversion_cost", "return 3 * (I + C + f) < F3 ? 1 : 0;", "return 3 * (I + f) < F3 ? 1 : 0;"),
    ("predicate_dense_cost_n_cubed", "__int128 F3 = 2 * N * N * N; /* 3*F */", "__int128 F3 = 3 * N * N * N; /* 3*F */"),
    ("predicate_fill_width_kl_plus_ku", "__int128 f = N * L * (2 * (L + U) + 1);", "__int128 f = N * L * (L + U + 1);"),
    ("flops_drop_reciprocal", "fl += 1 + km + 2 * km * (ju - j);", "fl += km + 2 * km * (ju - j);"),
    ("dense_lu_swaps_whole_row", "for (int64_t c = j; c < n; ++c) {\n                    double t0 = A[j * lda + c];",
     "for (int64_t c = 0; c < n; ++c) {\n                    double t0 = A[j * lda + c];"),
    ("gbtrs_no_interchange", "if (l != j) {\n                    const double t0 = b[l];",
     "if (0) {\n                    const double t0 = b[l];"),
    ("gbtrs_update_sign", "b[j + t] = fma(-AB_(kv + t, j), bj, b[j + t]);", "b[j + t] = fma(AB_(kv + t, j), bj, b[j + t]);"),
    ("gbtrs_drops_last_multiplier", "for (int64_t t = 1; t <= km; ++t) b[j + t]", "for (int64_t t = 1; t < km; ++t) b[j + t]"),
    ("gbtrs_drops_top_superdiagonal", "const int64_t i0 = j - kv > 0 ? j - kv : 0;", "const int64_t i0 = j - kv + 1 > 0 ? j - kv + 1 : 0;"),
    ("tbsv_lower_drops_last_band_entry", "const int64_t i1 = j + k < n - 1 ? j + k : n - 1;",
     "const int64_t i1 = j + k - 1 < n - 1 ? j + k - 1 : n - 1;"),
    ("tbsv_upper_update_sign", "for (int64_t i = i0; i < j; ++i) b[i] = fma(-x, A[i * lda + j], b[i]);",
     "for (int64_t i = i0; i < j; ++i) b[i] = fma(x, A[i * lda + j], b[i]);"),
    ("tbsv_lower_transposed_operand", "for (int64_t i = j + 1; i <= i1; ++i) b[i] = fma(-x, A[i * lda + j], b[i]);",
     "for (int64_t i = j + 1; i <= i1; ++i) b[i] = fma(-x, A[j * lda + i], b[i]);"),
    ("tbsv_lower_skips_division", "b[j] = b[j] / A[j * lda + j];\n                    const double x = b[j];\n                    const int64_t i1",
     "const double x = b[j];\n                    const int64_t i1"),
    ("tbsv_info_reports_last_zero", "*info = (int)(i + 1);\n            return 0;\n        }\n    for (int64_t c = 0; c < nrhs; ++c) {\n        double *b",
     "*info = (int)(i + 1);\n        }\n    for (int64_t c = 0; c < nrhs; ++c) {\n        double *b"),
    ("diag_multiplies_by_reciprocal", "B[c * ldb + i] = B[c * ldb + i] / A[i * lda + i];",
     "B[c * ldb + i] = B[c * ldb + i] * (1.0 / A[i * lda + i]);"),
    ("cm_detect_reads_row_major", "if (is_nonzero(A[i + j * lda])) {", "if (is_nonzero(A[j + i * lda])) {"),
    ("cm_convert_drops_top_superdiagonal", "const int64_t i0 = j - ku > 0 ? j - ku : 0;\n        const int64_t i1 = j + kl < n - 1 ? j + kl : n - 1;\n        for (int64_t i = i0; i <= i1; ++i) AB[(kv + i - j) + j * ldab] = A[i + j * lda];",
     "const int64_t i0 = j - ku + 1 > 0 ? j - ku + 1 : 0;\n        const int64_t i1 = j + kl < n - 1 ? j + kl : n - 1;\n        for (int64_t i = i0; i <= i1; ++i) AB[(kv + i - j) + j * ldab] = A[i + j * lda];"),
    ("classify_lower_upper_swapped", "if (ku == 0) return kl == 0 ? ORACLE_KIND_DIAGONAL : ORACLE_KIND_LOWER;",
     "if (ku == 0) return kl == 0 ? ORACLE_KIND_DIAGONAL : ORACLE_KIND_UPPER;"),
]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_mutant(tmp_path, name, old, new):
    src = open(SRC).read()
    assert old in src, f"mutation site for {name} not found"
    mutated = src.replace(old, new, 1)
    c_path = tmp_path / "mutant.c"
    so_path = tmp_path / "libmutant.so"
    c_path.write_text(mutated)
    sys.path.insert(0, ROOT)
    import oracle
    subprocess.run(["gcc", *oracle.CFLAGS, "-o", str(so_path), str(c_path), "-lm"], check=True)
    env = dict(os.environ, BANDLU_ORACLE_LIB=str(so_path))
    r = subprocess.run([sys.executable, "-m", "pytest", os.path.join(ROOT, "tests", "test_oracle.py"), "-x", "-q"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"pins did not catch mutant {name}:\n{r.stdout[-2000:]}"
