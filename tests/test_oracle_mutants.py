"""The oracle's pins have power: planted mistakes fail them (CPU only).

Each case compiles a copy of oracle.cpp with one plausible mistake (a wrong row index, a
dropped clamp, a flipped comparison, a reused uniform) and runs the exact-enumeration
losslessness check on it; every mutant must break the target distribution.
"""

import numpy as np
import pytest

from test_oracle_accept import GENERIC_P, GENERIC_Q, exact_output_distribution, target_product
from test_oracle_filtered import P_FILT, filtered_output_distribution

MUTANTS = {
    # the draft is scored against p_{i+1} instead of p_i
    "wrong_target_row": ("const double* p_i = p_rows + static_cast<int64_t>(i - 1) * vocab;",
                         "const double* p_i = p_rows + static_cast<int64_t>(i) * vocab;"),
    # the residual is not clamped at zero
    "unclamped_residual": ("w[x] = std::max(0.0, p_last[x] - q_n[x]);",
                           "w[x] = std::fabs(p_last[x] - q_n[x]);"),
    # accept and reject swapped
    "flipped_test": ("if (uniforms[i - 1] > thresh) { n = i; break; }",
                     "if (uniforms[i - 1] < thresh) { n = i; break; }"),
    # the residual subtracts the previous drafter row
    "wrong_drafter_row": ("const double* q_n = q_rows + static_cast<int64_t>(n) * vocab;",
                          "const double* q_n = q_rows + static_cast<int64_t>(n - 1) * vocab;"),
    # the rejecting uniform is reused for the residual draw
    "reused_uniform": ("const double u = uniforms[gamma - 1];",
                       "const double u = uniforms[n - 1];"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_breaks_losslessness(oracle_mod, name):
    before, after = MUTANTS[name]
    src = oracle_mod.source_text()
    assert src.count(before) == 1, f"mutation site for {name} not found in oracle.cpp"
    lib = oracle_mod.load_variant(src.replace(before, after), name)
    P, _ = exact_output_distribution(oracle_mod, GENERIC_P, GENERIC_Q, 16, lib=lib)
    assert np.abs(P - target_product(GENERIC_P)).max() > 1e-4


FILTER_MUTANTS = {
    # equal probabilities ranked by the higher token id
    "ties_to_higher_id": ("for (int64_t x = 0; x < vocab; ++x) order[x] = x;",
                          "for (int64_t x = 0; x < vocab; ++x) order[x] = vocab - 1 - x;"),
    # the token whose mass crosses top_p is dropped
    "crossing_token_dropped": ("      keep = j + 1;\n", "      keep = std::max<int64_t>(j, 1);\n"),
    # top-p compared against the mass of the whole row, not of the top-k
    "top_p_not_renormalised": ("c += p[order[j]] / mass_k;", "c += p[order[j]];"),
    # top-k ignored
    "top_k_ignored": ("const int64_t k = std::min<int64_t>(top_k, vocab);",
                      "const int64_t k = vocab;"),
    # the drafter distribution left unfiltered
    "drafter_unfiltered": (
        "oracle_filter_row(sm_row.data(), vocab, k, tp, &q_rows[j * vocab], &m);",
        "std::copy(sm_row.begin(), sm_row.end(), q_rows.begin() + j * vocab);"),
    # the target distribution left unfiltered
    "target_unfiltered": (
        "oracle_filter_row(sm_row.data(), vocab, k, tp, &p_rows[j * vocab], &m);",
        "std::copy(sm_row.begin(), sm_row.end(), p_rows.begin() + j * vocab);"),
}


@pytest.mark.parametrize("name", sorted(FILTER_MUTANTS))
def test_filter_mutant_breaks_filtered_losslessness(oracle_mod, name):
    before, after = FILTER_MUTANTS[name]
    src = oracle_mod.source_text()
    assert src.count(before) == 1, f"mutation site for {name} not found in oracle.cpp"
    lib = oracle_mod.load_variant(src.replace(before, after), "f_" + name)
    P, _ = filtered_output_distribution(oracle_mod, 1.0, lib=lib)
    assert np.abs(P - target_product(P_FILT)).max() > 1e-4
