"""The oracle's pins have power: planted mistakes fail them (CPU only).

Each case plants one plausible mistake (a wrong row index, a dropped clamp, a flipped
comparison, a reused uniform, a transposed layout, a tie broken the other way) in a copy
of the oracle and runs, on that copy, a pin that checks the oracle against something
other than itself; every mutant must fail it. The acceptance mutants break the exact
enumeration of losslessness; the others fail the pins of test_oracle_attention,
test_oracle_draft, test_oracle_tree and test_oracle_lm_head.
"""

import types

import numpy as np
import pytest

import test_oracle_accept as ACC
import test_oracle_attention as ATT
import test_oracle_draft as DRAFT
import test_oracle_lm_head as LM
import test_oracle_tree as TREE

from test_oracle_accept import (GENERIC8_P, GENERIC8_Q, GENERIC_P, GENERIC_Q,
                                exact_output_distribution, target_product)
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
    # caught by the enumeration at vocabulary 4 (1/16 rows) and at vocabulary 8 (1/8 rows)
    for p_rows, q_rows, denom in ((GENERIC_P, GENERIC_Q, 16), (GENERIC8_P, GENERIC8_Q, 8)):
        P, _ = exact_output_distribution(oracle_mod, p_rows, q_rows, denom, lib=lib)
        assert np.abs(P - target_product(p_rows)).max() > 1e-4, (name, p_rows.shape)


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


# ---------------------------------------------------------------------------------
# the rest of the oracle: a mutated copy of the whole package, run through its pins
# ---------------------------------------------------------------------------------
def mutant_oracle(oracle_mod, tag, cpp=None, py=None):
    """A fresh copy of the oracle package with one planted mistake: cpp = (before, after)
    in oracle.cpp, py = (before, after) in the package's Python source."""
    with open(oracle_mod.__file__) as f:
        text = f.read()
    if py is not None:
        assert text.count(py[0]) == 1, f"mutation site for {tag} not found in the oracle package"
        text = text.replace(*py)
    mod = types.ModuleType(f"oracle_mutant_{tag}")
    mod.__file__ = oracle_mod.__file__
    exec(compile(text, oracle_mod.__file__, "exec"), mod.__dict__)
    if cpp is not None:
        src = oracle_mod.source_text()
        assert src.count(cpp[0]) == 1, f"mutation site for {tag} not found in oracle.cpp"
        path = oracle_mod.load_variant(src.replace(*cpp), tag)._name
        mod.build = lambda force=False: path
    return mod


def _dense_attention_pin(m):
    for case in ATT.CASES:
        ATT.test_matches_dense_restatement(m, case)


def _commit_pins(m):
    DRAFT.test_commit_worked_example(m)
    DRAFT.test_commit_flags_bad_input_and_exhaustion(m)


PACKAGE_MUTANTS = {
    # --- the building blocks (oracle.cpp) ---
    # equal maxima go to the highest token id
    "argmax_ties_to_last": (dict(cpp=("if (row[x] > row[best]) best = x;",
                                      "if (row[x] >= row[best]) best = x;")),
                            DRAFT.test_sample_greedy_is_lowest_argmax),
    # the exponent drops the temperature (the maximum keeps it)
    "softmax_temperature_dropped": (dict(cpp=("p[x] = std::exp(logits[x] / temperature - m);",
                                              "p[x] = std::exp(logits[x] - m);")),
                                    ACC.test_softmax_matches_scipy),
    # the draw compares unnormalised cumulative weights with u instead of u * S
    "inverse_cdf_unscaled_target": (dict(cpp=("const double target = u * S;",
                                              "const double target = u;")),
                                    ACC.test_inverse_cdf_matches_searchsorted),
    # --- verify attention (oracle.cpp) ---
    # a block query does not see its own key
    "attn_query_misses_own_key": (dict(cpp=(": i <= j;", ": i < j;")), _dense_attention_pin),
    # query head h reads kv head h mod Hkv instead of its group's
    "attn_head_modulo": (dict(cpp=("const int32_t g = h / group;",
                                   "const int32_t g = h % num_kv_heads;")), _dense_attention_pin),
    # the softmax scale is dropped
    "attn_scale_dropped": (dict(cpp=("s[k] = dot * softmax_scale;", "s[k] = dot;")),
                           _dense_attention_pin),
    # the cache read as [page][slot][head] instead of [page][head][slot]
    "attn_cache_layout": (dict(cpp=(
        "return ((static_cast<int64_t>(pg) * num_kv_heads + g) * page_size + k % page_size) * D;",
        "return ((static_cast<int64_t>(pg) * page_size + k % page_size) * num_kv_heads + g) * D;")),
        _dense_attention_pin),
    # lse without the running maximum
    "attn_lse_without_max": (dict(cpp=("if (lse) lse[orow] = m + std::log(l);",
                                       "if (lse) lse[orow] = std::log(l);")), _dense_attention_pin),
    # the tree mask read transposed (node j sees its descendants)
    "tree_mask_transposed": (dict(cpp=("(tree_mask[static_cast<int64_t>(b) * gamma + j] >> i)",
                                       "(tree_mask[static_cast<int64_t>(b) * gamma + i] >> j)")),
                             TREE.test_tree_attention_dense_restatement),
    # --- draft-side sampling (oracle.cpp) ---
    # every block token of a sequence drawn with the first uniform
    "sample_shared_uniform": (dict(cpp=("const double u = static_cast<double>(uniforms[row]);",
                                        "const double u = static_cast<double>(uniforms[b * gamma]);")),
                              DRAFT.test_sample_matches_searchsorted_per_row),
    # the drafter row sampled at T = 1 whatever the temperature
    "sample_untempered": (dict(cpp=("if (oracle_softmax(raw.data(), vocab, T, q.data())) { code = 1; break; }",
                                    "if (oracle_softmax(raw.data(), vocab, 1.0, q.data())) { code = 1; break; }")),
                          DRAFT.test_sample_matches_searchsorted_per_row),
    # the filter computed but the unfiltered row sampled
    "sample_filter_skipped": (dict(cpp=("w = qf.data();", "w = q.data();")),
                              DRAFT.test_sample_filtered_law),
    # --- noise tokens and KV commit (Python) ---
    # z = x mod V instead of the multiply-shift map
    "noise_modulo": (dict(py=("return ((w * np.uint64(vocab)) >> np.uint64(32)).astype(np.int32)",
                              "return (w % np.uint64(vocab)).astype(np.int32)")),
                     DRAFT.test_noise_tokens_closed_forms),
    # a refused request does not count against the later ones
    "commit_refusal_not_counted": (dict(py=(
        "                flags[b] = 2\n                asked += need\n                continue",
        "                flags[b] = 2\n                continue")), _commit_pins),
    # the new length drops the free token x^{L+1}
    "commit_length_off_by_one": (dict(py=(
        "new[b] = kv[b] - gamma + (na[b] + 1 if na[b] >= 0 else 0)",
        "new[b] = kv[b] - gamma + (na[b] if na[b] >= 0 else 0)")), _commit_pins),
    # release frees a partly used page (floor instead of ceiling)
    "commit_frees_partial_page": (dict(py=("keep = -(-int(new[b]) // page_size)",
                                           "keep = int(new[b]) // page_size")), _commit_pins),
    # --- the tree sampler, tree acceptance and compaction (Python) ---
    # equal candidates ranked by the higher token id
    "tree_ties_to_higher_id": (dict(py=(
        "order = sorted(range(V), key=lambda x: (-lq[x], x))[:min(top_k, V)]",
        "order = sorted(range(V), key=lambda x: (-lq[x], -x))[:min(top_k, V)]")),
        TREE.test_tie_rules_worked_example),
    # equal offers go to the higher parent index
    "tree_parent_ties_to_higher_index": (dict(py=(
        "best = max(offers, key=lambda o: (o[0], -o[1]))",
        "best = max(offers, key=lambda o: (o[0], o[1]))")), TREE.test_tie_rules_worked_example),
    # an offer scored by its own log q, not the path's sum
    "tree_scores_not_summed": (dict(py=("offers.append((score[u] + logq[d][c], u, c))",
                                        "offers.append((logq[d][c], u, c))")),
                               lambda m: TREE.test_tree_is_the_best_prefixes(m, 3, 4, 12)),
    # position d ranked by drafter row d - 1
    "tree_wrong_drafter_row": (dict(py=("z = dl[b, d] / T", "z = dl[b, d - 1] / T")),
                               lambda m: TREE.test_tree_is_the_best_prefixes(m, 3, 4, 12)),
    # log q at T = 1 whatever the temperature
    "tree_untempered": (dict(py=("z = dl[b, d] / T", "z = dl[b, d]")),
                        lambda m: TREE.test_tree_is_the_best_prefixes(m, 3, 4, 12)),
    # a node's mask without its own bit
    "tree_mask_without_self": (dict(py=("bits, a = 0, j", "bits, a = 0, parents[j]")),
                               TREE.test_tree_structure),
    # a child checked against its own target row instead of its parent's
    "tree_walk_child_row": (dict(py=(
        "if parents[b, c] == cur and tokens[b, c] == a), None)",
        "if parents[b, c] == cur and tokens[b, c] == int(np.argmax(tl[b, c]))), None)")),
        TREE.test_greedy_walk_is_the_deepest_matching_path),
    # the final token taken from the root's row
    "tree_final_from_root": (dict(py=(
        "toks = [int(tokens[b, x]) for x in walk] + [int(np.argmax(tl[b, cur]))]",
        "toks = [int(tokens[b, x]) for x in walk] + [int(np.argmax(tl[b, 0]))]")),
        TREE.test_greedy_walk_is_the_deepest_matching_path),
    # the sampled walk's final draw reuses the last node's test uniform
    "tree_sampled_draw_reuses_uniform": (dict(py=("final, margin = inverse_cdf(w, u[b, 0])",
                                                  "final, margin = inverse_cdf(w, u[b, N - 1])")),
                                         lambda m: TREE.test_sampled_tree_acceptance_is_lossless(m, "tree4")),
    # every node's children tested against the root's target row
    "tree_sampled_root_row_only": (dict(py=("prob = softmax(tl[b, cur], float(T[b]))",
                                            "prob = softmax(tl[b, 0], float(T[b]))")),
                                   lambda m: TREE.test_sampled_tree_acceptance_is_lossless(m, "tree4")),
    # path rows moved one slot too low (over the root)
    "compact_destination_shifted": (dict(py=("src, dst = ctx + int(path[b, d]), ctx + d",
                                             "src, dst = ctx + int(path[b, d]), ctx + d - 1")),
                                    TREE.test_compaction_moves_the_path),
    # kv_len keeps the final token's slot
    "compact_length_off_by_one": (dict(py=("kl[b] = ctx + n", "kl[b] = ctx + n + 1")),
                                  TREE.test_compaction_moves_the_path),
    # --- the LM head and its row statistics (Python) ---
    # equal maxima go to the highest index
    "lm_ties_to_last": (dict(py=('out["row_argmax"][i] = int(np.argmax(l))',
                                 'out["row_argmax"][i] = len(l) - 1 - int(np.argmax(l[::-1]))')),
                        LM.test_ties_go_to_the_lowest_index_and_temperature_rule),
    # the temperature multiplies instead of divides
    "lm_temperature_multiplies": (dict(py=('out["row_sum"][i] = np.exp((l - m) / T).sum()',
                                           'out["row_sum"][i] = np.exp((l - m) * T).sum()')),
                                  LM.test_temperature_scales_the_sum),
    # row r takes temperature r mod (sequences) instead of its sequence's
    "lm_temperature_of_row": (dict(py=(
        "T = float(np.float32(temperature[r // rows_per_seq]))",
        "T = float(np.float32(temperature[r % len(temperature)]))")),
        LM.test_each_row_takes_its_sequence_temperature),
    # the token logit indexed by the selected row's position, not the row
    "lm_token_of_position": (dict(py=('out["token_logit"][i] = l[int(tokens[r])]',
                                      'out["token_logit"][i] = l[int(tokens[i])]')),
                             LM.test_token_logit_and_row_subset),
}


@pytest.mark.parametrize("name", sorted(PACKAGE_MUTANTS))
def test_package_mutant_fails_its_pin(oracle_mod, name):
    edit, pin = PACKAGE_MUTANTS[name]
    m = mutant_oracle(oracle_mod, name, **edit)
    with pytest.raises(AssertionError):
        pin(m)


def test_unmutated_copy_passes_every_pin(oracle_mod):
    # the harness itself: an unchanged copy passes the same pins
    m = mutant_oracle(oracle_mod, "none", cpp=("const int32_t g = h / group;",
                                               "const int32_t g = h / group;"))
    pins = {id(p): p for _, p in PACKAGE_MUTANTS.values()}
    for pin in pins.values():
        pin(m)
