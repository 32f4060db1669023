"""The oracle's pins have power: planted mistakes fail them (CPU only).

Each case compiles a copy of oracle.cpp with one plausible mistake (a wrong row index, a
dropped clamp, a flipped comparison, a reused uniform) and runs the exact-enumeration
losslessness check on it; every mutant must break the target distribution.
"""

import numpy as np
import pytest

from test_oracle_accept import GENERIC_P, GENERIC_Q, exact_output_distribution, target_product

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
