"""Pins of oracle.lm_head_stats (the LM head and the acceptance's row statistics):
closed forms of the logits for one-hot weight rows and for identity hidden states,
the logsumexp definition of the sum, ties to the lowest index, the temperature rule
and the token logit."""

import numpy as np
from scipy import special

from paper_2609_04010_gb300 import workloads as W


def bf16(x):
    return W.f32_to_bf16_bits(np.asarray(x, np.float32)).reshape(np.shape(x))


def dec(bits):
    return (np.asarray(bits).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def test_one_hot_weight_rows_select_hidden_columns(oracle_mod):
    # weight row v = c_v * e_{pi(v)}: logit (r, v) = c_v * h[r, pi(v)], exactly
    rng = np.random.default_rng(1)
    R, H, V = 5, 24, 40
    h = bf16(rng.standard_normal((R, H)))
    pi = rng.integers(0, H, V)
    c = bf16(rng.choice([0.5, -1.0, 2.0, 0.25], V))
    w = np.zeros((V, H), np.uint16)
    w[np.arange(V), pi] = c
    want = dec(h)[:, pi] * dec(c)[None, :]
    o = oracle_mod.lm_head_stats(h, w, np.ones(R, np.float32), 1)
    np.testing.assert_array_equal(o["logits"], want)
    np.testing.assert_array_equal(o["row_max"], want.max(axis=1))


def test_identity_hidden_states_read_weight_columns(oracle_mod):
    # hidden = I (rows = H): logits (r, v) = weight[v, r]; a transposed operand fails
    rng = np.random.default_rng(2)
    H, V = 16, 50
    h = bf16(np.eye(H))
    w = bf16(rng.standard_normal((V, H)) * 3)
    T = np.float32(0.7)
    o = oracle_mod.lm_head_stats(h, w, np.array([T], np.float32), H)
    wt = dec(w).T
    np.testing.assert_array_equal(o["logits"], wt)
    # sum of exp((l - max) / T) = exp(logsumexp(l / T) - max / T)
    lse = special.logsumexp(wt / np.float64(T), axis=1)
    np.testing.assert_allclose(o["row_sum"], np.exp(lse - wt.max(axis=1) / np.float64(T)), rtol=1e-12)
    np.testing.assert_array_equal(o["row_argmax"], np.argmax(wt, axis=1))


def test_ties_go_to_the_lowest_index_and_temperature_rule(oracle_mod):
    H, V = 8, 12
    h = bf16(np.eye(H)[:3])
    w = np.zeros((V, H), np.uint16)
    w[[3, 7, 9], 0] = bf16(2.0)      # row 0: three equal maxima
    w[5, 1] = bf16(-1.0)             # row 1: all others zero, the max is 0 at index 0
    o = oracle_mod.lm_head_stats(h, w, np.array([0.0, -1.0, 2.0], np.float32), 1)
    assert list(o["row_argmax"]) == [3, 0, 0]
    # T <= 0 sums at T = 1: row 0 = 3 + 9 e^-2, row 1 = 11 + e^-1
    np.testing.assert_allclose(o["row_sum"][0], 3 + 9 * np.exp(-2.0), rtol=1e-14)
    np.testing.assert_allclose(o["row_sum"][1], 11 + np.exp(-1.0), rtol=1e-14)
    # T = 2 on a row of zeros: V
    np.testing.assert_allclose(o["row_sum"][2], V, rtol=1e-14)


def test_temperature_scales_the_sum(oracle_mod):
    rng = np.random.default_rng(3)
    h, w, _, _ = W.make_lm_inputs(6, 64, 300, 2, seed=3)
    o1 = oracle_mod.lm_head_stats(h, w, np.ones(3, np.float32), 2)
    o2 = oracle_mod.lm_head_stats(h, w, np.full(3, 0.5, np.float32), 2)
    l = o1["logits"]
    # the T = 0.5 sum equals the T = 1 sum of the doubled logits
    np.testing.assert_allclose(o2["row_sum"], np.exp(2 * (l - l.max(axis=1, keepdims=True))).sum(axis=1),
                               rtol=1e-13)
    assert np.all(o2["row_sum"] < o1["row_sum"])


def test_token_logit_and_row_subset(oracle_mod):
    h, w, T, tok = W.make_lm_inputs(9, 32, 500, 3, seed=4)
    tok = tok.copy()
    tok[2] = -1
    tok[5] = 500
    o = oracle_mod.lm_head_stats(h, w, T, 3, tokens=tok)
    for r in range(9):
        if r in (2, 5):
            assert np.isnan(o["token_logit"][r])
        else:
            assert o["token_logit"][r] == o["logits"][r, tok[r]]
    sub = oracle_mod.lm_head_stats(h, w, T, 3, tokens=tok, rows=[7, 1], chunk=64)
    for key in ("row_max", "row_sum", "row_argmax", "token_logit"):
        np.testing.assert_array_equal(sub[key], o[key][[7, 1]])
    # the bound on a logit's accumulation error dominates every logit
    assert np.all(np.abs(o["logits"]).max(axis=1) <= o["abs_bound"] + 1e-12)


def test_each_row_takes_its_sequence_temperature(oracle_mod):
    # rows_per_seq = 2: rows 2s and 2s + 1 use temperature[s]; the sum is the closed form
    # exp(logsumexp(l / T) - max / T) at that T (T <= 0 at T = 1)
    h, w, _, _ = W.make_lm_inputs(6, 32, 200, 2, seed=5)
    T = np.array([1.0, 0.5, 0.0], np.float32)
    o = oracle_mod.lm_head_stats(h, w, T, 2)
    l = o["logits"]
    for r in range(6):
        t = float(T[r // 2]) if T[r // 2] > 0 else 1.0
        want = np.exp(special.logsumexp(l[r] / t) - l[r].max() / t)
        np.testing.assert_allclose(o["row_sum"][r], want, rtol=1e-12)
