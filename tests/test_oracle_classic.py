"""The classic speculative-decoding convention (k drafts from q_1..q_k, k + 1 target rows,
the last the bonus row) through the acceptance call with gamma = k + 1, block token 0 the
last emitted token and an unused leading drafter row: the exact law of the emitted
tokens is the target chain p_1 x .. x p_{k+1} (the classic rule's losslessness), and the
unused drafter row is never read (NaN there changes nothing)."""

import numpy as np

from paper_2609_04010_gb300 import workloads as W
from test_oracle_accept import exact_output_distribution, rows16, target_product


def test_classic_convention_is_lossless_with_an_unread_row(oracle_mod):
    # k = 2 drafts; target rows p_1, p_2, p_3; drafter rows q_1, q_2
    p_c = rows16([5, 3, 6, 2], [1, 7, 4, 4], [8, 2, 3, 3])
    q_c = rows16([4, 4, 2, 6], [2, 6, 6, 2])
    q_rows = np.vstack([np.full(4, np.nan), q_c])  # the leading row: never read
    P, _ = exact_output_distribution(oracle_mod, p_c, q_rows, 16)
    np.testing.assert_allclose(P, target_product(p_c), rtol=0, atol=1e-12)


def test_unused_drafter_row_does_not_change_the_outputs(oracle_mod):
    inp = W.make_accept_inputs(6, 9, 500, "f32", 3.0, 1.0, [1.0, 0.0, 0.7], seed=11)
    base = oracle_mod.accept_block(inp.target_logits, inp.drafter_logits, inp.block_tokens,
                                   inp.temperature, inp.uniforms)
    dl = inp.drafter_logits.copy()
    dl[:, 0, :] = np.nan
    other = oracle_mod.accept_block(inp.target_logits, dl, inp.block_tokens, inp.temperature,
                                    inp.uniforms)
    assert np.all(other["status"] == 0)
    for k in ("num_accepted", "out_tokens", "num_emitted"):
        np.testing.assert_array_equal(other[k], base[k])
    # out_tokens[0] echoes block token 0 (the last emitted token in the classic convention)
    np.testing.assert_array_equal(base["out_tokens"][:, 0], inp.block_tokens[:, 0])
