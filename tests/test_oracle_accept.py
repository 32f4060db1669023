"""Pins of the oracle's acceptance rule (CPU only, no GPU).

Each test checks the oracle against something other than itself:
  * exact losslessness, by enumerating every draft and every cell of the uniforms on
    probability rows whose entries are multiples of 1/8 (vocabulary 8, gamma 3) or of
    1/16 (vocabulary 4, gamma 3) (the paper's claim that the
    verify step "preserves the base model's target distribution", Sec. 4.2);
  * the closed-form acceptance rate alpha_i = sum_x min(p_i(x), q_i(x)) = 1 - TV
    (the Total Variation link the paper cites in Sec. 3.2, Eq. "tv-loss");
  * a chi-square test of 10^6 seeded draws against the target product distribution;
  * special cases that reduce to textbook or library routines (gamma = 1 is plain
    inverse-CDF sampling; softmax against scipy; the T -> 0 limit is greedy decoding);
  * a negative control: greedy drafting verified by the stochastic rule is not
    lossless (the I-DLM finding, Appendix "Uno-Qwen vs I-DLM"), and the tests detect it.
"""

import itertools
from fractions import Fraction

import numpy as np
import pytest
from scipy import special, stats


# ---------------------------------------------------------------------------------
# exact enumeration
# ---------------------------------------------------------------------------------
def farey(n):
    return sorted({Fraction(a, b) for b in range(1, n + 1) for a in range(0, b + 1)})


def uniform_cells(denom):
    """Cells of (0, 1] between consecutive fractions with denominator <= denom.

    Every threshold the rule compares a uniform with (min(1, p/q) and the cumulative
    sums C(k)/S of the residual or bonus weights) is such a fraction when the
    probabilities are multiples of 1/denom, so the rule's output is constant on each
    cell and the cell midpoint stands for the whole cell."""
    fr = farey(denom)
    mids = np.array([float((a + b) / 2) for a, b in zip(fr[:-1], fr[1:])])
    widths = np.array([float(b - a) for a, b in zip(fr[:-1], fr[1:])])
    return mids, widths


def exact_output_distribution(oracle_mod, p_rows, q_rows, denom, draft_weights=None, lib=None):
    """Exact probability of every completed tuple (x_1 .. x_gamma) of one verify step.

    Drafts t_i (i >= 1) are enumerated with weight q_i(t_i) (or ``draft_weights``), the
    uniforms over all cells; an output with n tokens after t_0 is completed by drawing
    positions n+1 .. gamma from their target rows."""
    gamma, V = p_rows.shape
    mids, widths = uniform_cells(denom)
    C = len(mids)
    idx = np.stack([g.ravel() for g in np.meshgrid(*([np.arange(C)] * gamma), indexing="ij")], 1)
    U = mids[idx]
    W = np.prod(widths[idx], axis=1)
    dw = q_rows if draft_weights is None else draft_weights
    A = [None] + [np.zeros(V ** n) for n in range(1, gamma + 1)]
    for drafts in itertools.product(range(V), repeat=gamma - 1):
        wd = 1.0
        for i, t in enumerate(drafts, start=1):
            wd *= dw[i][t]
        if wd == 0.0:
            continue
        tokens = np.tile(np.array([0, *drafts], np.int32), (U.shape[0], 1))
        n, out, ne = oracle_mod.accept_probs_many(p_rows, q_rows, tokens, U, lib=lib)
        assert np.all(ne == n + 1)
        emitted = out[:, 1:]
        for nn in range(1, gamma + 1):
            sel = n == nn
            if not sel.any():
                continue
            flat = np.ravel_multi_index(tuple(emitted[sel, k] for k in range(nn)), (V,) * nn)
            A[nn] += np.bincount(flat, weights=wd * W[sel], minlength=V ** nn)
    P = np.zeros((V,) * gamma)
    for nn in range(1, gamma + 1):
        term = A[nn].reshape((V,) * nn)
        for k in range(nn + 1, gamma + 1):
            term = np.multiply.outer(term, p_rows[k - 1])
        P += term
    return P, A


def target_product(p_rows):
    P = p_rows[0]
    for r in p_rows[1:]:
        P = np.multiply.outer(P, r)
    return P


def rows16(*rows):
    a = np.array(rows, dtype=np.float64) / 16.0
    assert np.allclose(a.sum(axis=1), 1.0)
    return a


def rows8(*rows):
    a = np.array(rows, dtype=np.float64) / 8.0
    assert np.allclose(a.sum(axis=1), 1.0)
    return a


# vocabulary 8, gamma 3: rows whose entries are multiples of 1/8, so that every
# threshold of the rule is a fraction with denominator <= 8 and Farey(8) cells suffice
GENERIC8_P = rows8([2, 1, 0, 1, 1, 0, 2, 1], [0, 1, 3, 1, 0, 1, 1, 1], [1, 1, 1, 1, 1, 1, 1, 1])
GENERIC8_Q = rows8([1, 1, 1, 1, 1, 1, 1, 1], [1, 2, 0, 1, 2, 1, 0, 1], [3, 0, 1, 1, 0, 1, 1, 1])
SPARSE8_P = rows8([0, 4, 0, 0, 4, 0, 0, 0], [8, 0, 0, 0, 0, 0, 0, 0], [0, 0, 3, 0, 0, 0, 0, 5])
SPARSE8_Q = rows8([0, 0, 0, 8, 0, 0, 0, 0], [1, 1, 1, 0, 0, 0, 0, 5], [0, 2, 2, 0, 0, 4, 0, 0])

GENERIC_P = rows16([5, 3, 6, 2], [1, 7, 4, 4], [8, 2, 3, 3])
GENERIC_Q = rows16([4, 4, 4, 4], [4, 4, 2, 6], [2, 6, 6, 2])
SPARSE_P = rows16([0, 8, 8, 0], [16, 0, 0, 0], [3, 0, 0, 13])
SPARSE_Q = rows16([1, 1, 1, 13], [2, 2, 12, 0], [0, 4, 4, 8])


@pytest.mark.parametrize("p_rows,q_rows", [(GENERIC_P, GENERIC_Q), (SPARSE_P, SPARSE_Q)],
                         ids=["generic", "sparse"])
def test_lossless_exact_enumeration(oracle_mod, p_rows, q_rows):
    P, _ = exact_output_distribution(oracle_mod, p_rows, q_rows, 16)
    assert abs(P.sum() - 1.0) < 1e-12
    np.testing.assert_allclose(P, target_product(p_rows), rtol=0, atol=1e-12)


@pytest.mark.parametrize("p_rows,q_rows", [(GENERIC8_P, GENERIC8_Q), (SPARSE8_P, SPARSE8_Q)],
                         ids=["generic", "sparse"])
def test_lossless_exact_enumeration_vocab8(oracle_mod, p_rows, q_rows):
    # every one of the 8^2 draft pairs and every Farey(8) cell of the three uniforms
    P, A = exact_output_distribution(oracle_mod, p_rows, q_rows, 8)
    assert abs(P.sum() - 1.0) < 1e-12
    np.testing.assert_allclose(P, target_product(p_rows), rtol=0, atol=1e-12)
    # an immediate rejection and a later one are both taken; on the generic rows also
    # the full acceptance (the sparse q_2 has no mass where p_1 has any)
    assert A[1].sum() > 0 and A[2].sum() > 0
    assert (A[3].sum() > 0) == (p_rows is GENERIC8_P)


def test_negative_control_vocab8(oracle_mod):
    greedy = np.zeros_like(GENERIC8_Q)
    for i in range(GENERIC8_Q.shape[0]):
        greedy[i, int(np.argmax(GENERIC8_Q[i]))] = 1.0
    P, _ = exact_output_distribution(oracle_mod, GENERIC8_P, GENERIC8_Q, 8, draft_weights=greedy)
    assert np.abs(P - target_product(GENERIC8_P)).max() > 1e-2


def test_identical_drafter_accepts_everything(oracle_mod):
    # q_i = p_i for every draft: min(1, p/q) = 1, so every draft is accepted and the
    # step emits gamma + 1 tokens, the last one a bonus draw from p_gamma.
    p = GENERIC_P
    q = np.vstack([p[0], p[0], p[1]])  # q_1 = p_1 (row 0), q_2 = p_2 (row 1)
    P, A = exact_output_distribution(oracle_mod, p, q, 16)
    assert A[1].sum() == 0.0 and A[2].sum() == 0.0
    np.testing.assert_allclose(P, target_product(p), rtol=0, atol=1e-12)


def test_disjoint_supports_reject_first_draft(oracle_mod):
    # Drafts never land where the target has mass: the first draft is always rejected
    # and the replacement is drawn from [p_1 - q_1]_+ = p_1.
    p = rows16([8, 8, 0, 0], [4, 12, 0, 0], [0, 16, 0, 0])
    q = rows16([4, 4, 4, 4], [0, 0, 8, 8], [0, 0, 2, 14])
    P, A = exact_output_distribution(oracle_mod, p, q, 16)
    assert A[2].sum() == 0.0 and A[3].sum() == 0.0
    np.testing.assert_allclose(A[1], p[0], rtol=0, atol=1e-12)
    np.testing.assert_allclose(P, target_product(p), rtol=0, atol=1e-12)


def test_negative_control_greedy_drafting_is_not_lossless(oracle_mod):
    # Greedy drafting (t_i = argmax q_i) verified with the stochastic rule: the rule
    # assumes t_i ~ q_i, so the output distribution is biased. The enumeration must see it.
    p, q = GENERIC_P, GENERIC_Q
    greedy = np.zeros_like(q)
    for i in range(q.shape[0]):
        greedy[i, int(np.argmax(q[i]))] = 1.0
    P, _ = exact_output_distribution(oracle_mod, p, q, 16, draft_weights=greedy)
    assert np.abs(P - target_product(p)).max() > 1e-2


# ---------------------------------------------------------------------------------
# closed form: expected accepted length
# ---------------------------------------------------------------------------------
def _rows_from_logits(logits, T):
    return special.softmax(logits.astype(np.float64) / T, axis=-1)


def _mc_inputs(rng, target, drafter, T, trials):
    """Drafts t_i ~ q_i and uniforms in (0, 1] for ``trials`` independent steps."""
    gamma, V = target.shape
    q = _rows_from_logits(drafter, T)
    tokens = np.zeros((trials, gamma), np.int32)
    for i in range(1, gamma):
        tokens[:, i] = rng.choice(V, size=trials, p=q[i])
    tokens[:, 0] = rng.choice(V, size=trials, p=q[0])
    u = (1.0 - rng.random((trials, gamma))).astype(np.float32)
    tl = np.broadcast_to(target, (trials, gamma, V)).copy()
    dl = np.broadcast_to(drafter, (trials, gamma, V)).copy()
    return tl, dl, tokens, u


@pytest.mark.parametrize("T", [1.0, 0.7])
def test_closed_form_expected_accepted(oracle_mod, T):
    rng = np.random.default_rng(11)
    gamma, V, trials = 6, 16, 40000
    target = (rng.standard_normal((gamma, V)) * 2.0).astype(np.float32)
    drafter = np.empty_like(target)
    drafter[0] = rng.standard_normal(V).astype(np.float32)
    drafter[1:] = target[:-1] + (rng.standard_normal((gamma - 1, V)) * 0.8).astype(np.float32)
    p = _rows_from_logits(target, T)
    q = _rows_from_logits(drafter, T)
    alpha = np.array([np.minimum(p[i - 1], q[i]).sum() for i in range(1, gamma)])
    surv = np.cumprod(alpha)              # P(a >= k), k = 1 .. gamma-1
    expected = surv.sum()
    tl, dl, tok, u = _mc_inputs(rng, target, drafter, T, trials)
    r = oracle_mod.accept_block(tl, dl, tok, np.full(trials, T, np.float32), u)
    a = r["num_accepted"].astype(np.float64)
    assert np.all(r["num_emitted"] == a + 2)
    assert a.min() >= 0 and a.max() <= gamma - 1
    se = a.std() / np.sqrt(trials)
    assert abs(a.mean() - expected) < 5 * se + 1e-12
    for k in range(1, gamma):
        pk = surv[k - 1]
        emp = (a >= k).mean()
        assert abs(emp - pk) < 5 * np.sqrt(pk * (1 - pk) / trials) + 1e-9


# ---------------------------------------------------------------------------------
# chi-square over 10^6 seeded draws
# ---------------------------------------------------------------------------------
def _complete(rng, out, ne, p):
    """Completed tuples: emitted tokens after t_0, then fresh draws from target rows."""
    gamma, V = p.shape
    N = out.shape[0]
    x = np.empty((N, gamma), np.int64)
    n = ne - 1
    for k in range(1, gamma + 1):
        fresh = rng.choice(V, size=N, p=p[k - 1])
        x[:, k - 1] = np.where(k <= n, out[:, k], fresh)
    return x


def _chi2_pvalue(x, p):
    gamma, V = p.shape
    N = x.shape[0]
    flat = np.ravel_multi_index(tuple(x[:, k] for k in range(gamma)), (V,) * gamma)
    obs = np.bincount(flat, minlength=V ** gamma).astype(np.float64)
    exp = target_product(p).ravel() * N
    small = exp < 5
    o = np.append(obs[~small], obs[small].sum())
    e = np.append(exp[~small], exp[small].sum())
    if e[-1] == 0:
        o, e = o[:-1], e[:-1]
    return stats.chisquare(o, e).pvalue


def _chi2_run(oracle_mod, greedy_drafts, seed=5, N=1_000_000, chunk=250_000):
    rng = np.random.default_rng(seed)
    gamma, V, T = 3, 8, 1.0
    target = (rng.standard_normal((gamma, V)) * 1.5).astype(np.float32)
    drafter = np.empty_like(target)
    drafter[0] = rng.standard_normal(V).astype(np.float32)
    drafter[1:] = target[:-1] + rng.standard_normal((gamma - 1, V)).astype(np.float32)
    p = _rows_from_logits(target, T)
    q = _rows_from_logits(drafter, T)
    xs, firsts = [], []
    for _ in range(N // chunk):
        tl, dl, tok, u = _mc_inputs(rng, target, drafter, T, chunk)
        if greedy_drafts:
            for i in range(1, gamma):
                tok[:, i] = int(np.argmax(q[i]))
        r = oracle_mod.accept_block(tl, dl, tok, np.full(chunk, T, np.float32), u)
        xs.append(_complete(rng, r["out_tokens"], r["num_emitted"], p))
        firsts.append(r["out_tokens"][:, 1])
    x = np.concatenate(xs)
    first = np.concatenate(firsts)
    p_first = stats.chisquare(np.bincount(first, minlength=V), p[0] * N).pvalue
    return _chi2_pvalue(x, p), p_first


def test_chi_square_million_draws(oracle_mod):
    p_joint, p_first = _chi2_run(oracle_mod, greedy_drafts=False)
    assert p_joint > 1e-3
    assert p_first > 1e-3


def test_chi_square_rejects_greedy_drafting(oracle_mod):
    p_joint, _ = _chi2_run(oracle_mod, greedy_drafts=True, N=250_000)
    assert p_joint < 1e-6


# ---------------------------------------------------------------------------------
# special cases and library routines
# ---------------------------------------------------------------------------------
def test_softmax_matches_scipy(oracle_mod):
    rng = np.random.default_rng(3)
    for T in (1.0, 0.7, 2.5):
        l = rng.standard_normal(1000) * 4
        np.testing.assert_allclose(oracle_mod.softmax(l, T), special.softmax(l / T),
                                   rtol=1e-13, atol=0)
    np.testing.assert_allclose(oracle_mod.softmax(np.full(7, 3.25), 1.0), np.full(7, 1 / 7),
                               rtol=1e-15)
    l = rng.standard_normal(50)
    np.testing.assert_allclose(oracle_mod.softmax(l + 123.0, 0.5), oracle_mod.softmax(l, 0.5),
                               rtol=1e-12)
    with pytest.raises(ValueError):
        oracle_mod.softmax(np.array([0.0, np.nan]), 1.0)
    with pytest.raises(ValueError):
        oracle_mod.softmax(np.array([-np.inf, -np.inf]), 1.0)


def test_inverse_cdf_matches_searchsorted(oracle_mod):
    rng = np.random.default_rng(4)
    for _ in range(200):
        w = rng.random(37) * (rng.random(37) < 0.6)
        if w.sum() == 0:
            continue
        u = 1.0 - rng.random()
        c = np.cumsum(w)
        expect = int(np.searchsorted(c, u * c[-1], side="left"))
        if np.min(np.abs(c - u * c[-1])) < 1e-12:
            continue
        x, margin = oracle_mod.inverse_cdf(w, u)
        assert x == expect
        assert w[x] > 0
        assert margin >= 0 and margin <= w[x]


def test_gamma_one_is_categorical_sampling(oracle_mod):
    # gamma = 1: no drafts; the step emits t_0 and one draw from p_1 by inverse CDF.
    rng = np.random.default_rng(6)
    V, N = 50, 2000
    target = (rng.standard_normal((1, V)) * 2).astype(np.float32)
    drafter = rng.standard_normal((1, V)).astype(np.float32)
    p = special.softmax(target[0].astype(np.float64))
    c = np.cumsum(p)
    u = (1.0 - rng.random((N, 1))).astype(np.float32)
    tok = rng.integers(0, V, (N, 1)).astype(np.int32)
    r = oracle_mod.accept_block(np.broadcast_to(target, (N, 1, V)).copy(),
                                np.broadcast_to(drafter, (N, 1, V)).copy(), tok,
                                np.ones(N, np.float32), u)
    assert np.all(r["num_accepted"] == 0) and np.all(r["num_emitted"] == 2)
    assert np.all(r["out_tokens"][:, 0] == tok[:, 0])
    expect = np.searchsorted(c, u[:, 0].astype(np.float64) * c[-1], side="left")
    clear = np.min(np.abs(c[None, :] - u.astype(np.float64) * c[-1]), axis=1) > 1e-9
    assert np.all(r["out_tokens"][clear, 1] == expect[clear])


def test_greedy_is_the_small_temperature_limit(oracle_mod):
    # With well-separated logits and drafts taken as the drafter's argmax, the
    # stochastic rule at T = 1e-3 makes the same decisions and emits the same tokens
    # as the greedy (T = 0) rule.
    rng = np.random.default_rng(7)
    B, gamma, V = 300, 6, 40
    base = rng.permutation(V).astype(np.float32) * 0.25
    target = np.stack([np.stack([rng.permutation(base) for _ in range(gamma)]) for _ in range(B)])
    drafter = np.empty_like(target)
    for b in range(B):
        drafter[b, 0] = rng.permutation(base)
        for j in range(1, gamma):
            # agree with the target row most of the time, so chains of accepts occur
            drafter[b, j] = target[b, j - 1] if rng.random() < 0.7 else rng.permutation(base)
    tok = np.argmax(drafter, axis=-1).astype(np.int32)
    u = (1.0 - rng.random((B, gamma))).astype(np.float32)
    g = oracle_mod.accept_block(target, drafter, tok, np.zeros(B, np.float32), u)
    s = oracle_mod.accept_block(target, drafter, tok, np.full(B, 1e-3, np.float32), u)
    np.testing.assert_array_equal(g["num_accepted"], s["num_accepted"])
    np.testing.assert_array_equal(g["out_tokens"], s["out_tokens"])
    assert len(set(g["num_accepted"].tolist())) > 2


def test_greedy_accepts_argmax_chain(oracle_mod):
    # Drafts equal to the target argmax chain are all accepted; the bonus is the
    # argmax of the last target row.
    rng = np.random.default_rng(8)
    B, gamma, V = 20, 5, 300
    target = rng.standard_normal((B, gamma, V)).astype(np.float32)
    drafter = rng.standard_normal((B, gamma, V)).astype(np.float32)
    tok = np.zeros((B, gamma), np.int32)
    tok[:, 0] = rng.integers(0, V, B)
    tok[:, 1:] = np.argmax(target[:, :-1], axis=-1)
    r = oracle_mod.accept_block(target, drafter, tok, np.zeros(B, np.float32),
                                np.full((B, gamma), 0.5, np.float32))
    assert np.all(r["num_accepted"] == gamma - 1)
    np.testing.assert_array_equal(r["out_tokens"][:, :gamma], tok)
    np.testing.assert_array_equal(r["out_tokens"][:, gamma], np.argmax(target[:, -1], axis=-1))


def test_diag_matches_scipy_softmax(oracle_mod):
    rng = np.random.default_rng(9)
    B, gamma, V = 6, 5, 500
    T = float(np.float32(0.8))  # the oracle divides by the fp32 temperature it is given
    target = (rng.standard_normal((B, gamma, V)) * 3).astype(np.float32)
    drafter = target + rng.standard_normal((B, gamma, V)).astype(np.float32)
    tok = rng.integers(0, V, (B, gamma)).astype(np.int32)
    u = np.full((B, gamma), 1e-7, np.float32)  # accept every draft with p > 0
    r = oracle_mod.accept_block(target, drafter, tok, np.full(B, T, np.float32), u)
    for b in range(B):
        for i in range(1, gamma):
            pe = special.softmax(target[b, i - 1].astype(np.float64) / T)[tok[b, i]]
            qe = special.softmax(drafter[b, i].astype(np.float64) / T)[tok[b, i]]
            if i <= r["num_accepted"][b] + 1:
                np.testing.assert_allclose(r["diag"][b, i], [pe, qe], rtol=1e-12)


def test_bf16_logits_decode_exactly(oracle_mod):
    from paper_2609_04010_gb300.workloads import f32_to_bf16_bits, bf16_bits_to_f32
    rng = np.random.default_rng(10)
    B, gamma, V = 3, 4, 200
    t32 = (rng.standard_normal((B, gamma, V)) * 3).astype(np.float32)
    d32 = (rng.standard_normal((B, gamma, V)) * 3).astype(np.float32)
    tb, db = f32_to_bf16_bits(t32).reshape(t32.shape), f32_to_bf16_bits(d32).reshape(d32.shape)
    tok = rng.integers(0, V, (B, gamma)).astype(np.int32)
    u = (1.0 - rng.random((B, gamma))).astype(np.float32)
    T = np.ones(B, np.float32)
    r16 = oracle_mod.accept_block(tb, db, tok, T, u)
    r32 = oracle_mod.accept_block(bf16_bits_to_f32(tb).reshape(t32.shape),
                                  bf16_bits_to_f32(db).reshape(d32.shape), tok, T, u)
    for k in ("num_accepted", "out_tokens", "num_emitted"):
        np.testing.assert_array_equal(r16[k], r32[k])


def test_invalid_inputs_are_flagged(oracle_mod):
    rng = np.random.default_rng(12)
    B, gamma, V = 4, 3, 20
    target = rng.standard_normal((B, gamma, V)).astype(np.float32)
    drafter = rng.standard_normal((B, gamma, V)).astype(np.float32)
    tok = rng.integers(0, V, (B, gamma)).astype(np.int32)
    tok[1, 2] = V          # token out of range
    target[2, 0, 5] = np.nan  # undefined softmax
    u = np.full((B, gamma), 0.5, np.float32)
    r = oracle_mod.accept_block(target, drafter, tok, np.ones(B, np.float32), u)
    assert list(r["status"]) == [0, 2, 1, 0]
    for b in (1, 2):
        assert r["num_accepted"][b] == -1 and r["num_emitted"][b] == 0
        assert np.all(r["out_tokens"][b] == -1)
    assert r["num_emitted"][0] >= 2
