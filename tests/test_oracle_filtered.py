"""Pins of the oracle's top-k / top-p filtered acceptance (CPU only, no GPU).

The paper samples with top-k 50 and top-p 0.95 for both drafting and verification
(Sec. 5.1, Sec. 5.2, Appendix C.1). Filtering turns p and q into the filtered,
renormalised distributions p' and q'; the acceptance rule is then the unfiltered one
applied to them, so that the output follows the filtered target exactly.

Each test checks the oracle against something other than itself:
  * a hand-worked example and a brute-force definition of the filter in exact rational
    arithmetic (a token is kept iff fewer than k tokens outrank it and the mass ranked
    strictly before it is below top_p times the top-k mass), including ties;
  * special cases: the filter is the identity when k >= V and top_p = 1; k = 1 is the
    argmax; the filtered block step equals the unfiltered one when filtering is off,
    and greedy sequences ignore the filter;
  * exact losslessness for the filtered target, by enumerating every draft from q' and
    every cell of the uniforms on rows whose filtered forms are multiples of 1/4;
  * the closed-form acceptance rate sum_x min(p'(x), q'(x)) over seeded draws.
"""

import itertools
from fractions import Fraction

import numpy as np
import pytest
from scipy import special

from test_oracle_accept import uniform_cells, target_product


# ---------------------------------------------------------------------------------
# the filter on one row
# ---------------------------------------------------------------------------------
def brute_filter(p, k, top_p):
    """Exact filtered row (as Fractions) from the definition, without sorting.

    Rank order: higher probability first, equal probabilities by lower token id."""
    P = [Fraction(x) for x in p]
    V = len(P)
    tp = Fraction(top_p)

    def outranks(y, x):
        return P[y] > P[x] or (P[y] == P[x] and y < x)

    topk = [x for x in range(V) if sum(outranks(y, x) for y in range(V)) < k]
    Mk = sum(P[x] for x in topk)
    kept = []
    for x in topk:
        before = sum(P[y] for y in topk if outranks(y, x))
        if tp >= 1 or before < tp * Mk:
            kept.append(x)
    S = sum(P[x] for x in kept)
    return [P[x] / S if x in kept else Fraction(0) for x in range(V)]


def test_filter_worked_example(oracle_mod):
    # p = (0.1, 0.4, 0.2, 0.3), k = 3: the top three are tokens 1, 3, 2 with mass 0.9,
    # renormalised 4/9, 3/9, 2/9. Cumulative 4/9 < 0.7 <= 7/9, so top-p 0.7 keeps
    # tokens 1 and 3; renormalised over 0.7: 4/7 and 3/7. The margin is the distance
    # from 0.7 to the nearer bracketing sum, min(0.7 - 4/9, 7/9 - 0.7) = 7/90.
    out, margin = oracle_mod.filter_row(np.array([0.1, 0.4, 0.2, 0.3]), 3, 0.7)
    np.testing.assert_allclose(out, [0.0, 4 / 7, 0.0, 3 / 7], rtol=1e-15, atol=0)
    assert out[0] == 0.0 and out[2] == 0.0
    assert abs(margin - 7 / 90) < 1e-15


def test_filter_matches_brute_force_definition(oracle_mod):
    rng = np.random.default_rng(21)
    checked = 0
    for trial in range(400):
        V = int(rng.integers(1, 9))
        if trial % 3 == 0:
            # small integer weights: many ties, at the top-k and at the top-p cut
            w = rng.integers(0, 5, V).astype(np.float64)
            if w.sum() == 0:
                w[rng.integers(V)] = 1.0
            p = w / w.sum()
        else:
            p = rng.dirichlet(np.full(V, 0.7))
        k = int(rng.integers(1, V + 2))
        top_p = float(rng.choice([1.0, 0.95, 0.9, 0.7, 0.5, 0.3, 0.05]))
        out, margin = oracle_mod.filter_row(p, k, top_p)
        if margin < 1e-12:
            continue  # the cut sits on a rounding tie: fp64 may go either way
        exact = brute_filter(p, k, top_p)
        np.testing.assert_allclose(out, [float(x) for x in exact], rtol=1e-14, atol=1e-300)
        assert all((out[x] == 0.0) == (exact[x] == 0) for x in range(V))
        checked += 1
    assert checked > 300


def test_filter_identity_and_point_mass(oracle_mod):
    rng = np.random.default_rng(22)
    p = rng.dirichlet(np.ones(50))
    out, margin = oracle_mod.filter_row(p, 50, 1.0)
    np.testing.assert_allclose(out, p, rtol=1e-14)
    assert margin == np.inf
    out, _ = oracle_mod.filter_row(p, 1000, 1.0)
    np.testing.assert_allclose(out, p, rtol=1e-14)
    # k = 1: a point mass on the argmax; a tie goes to the lower token id
    out, _ = oracle_mod.filter_row(p, 1, 0.95)
    assert out[np.argmax(p)] == 1.0 and out.sum() == 1.0
    q = np.array([0.1, 0.3, 0.2, 0.3, 0.1])
    out, _ = oracle_mod.filter_row(q, 1, 1.0)
    np.testing.assert_array_equal(out, [0, 1, 0, 0, 0])
    # tiny top_p: only the most probable token survives
    out, _ = oracle_mod.filter_row(q, 5, 1e-6)
    np.testing.assert_array_equal(out, [0, 1, 0, 0, 0])


def test_filter_invariants(oracle_mod):
    rng = np.random.default_rng(23)
    for _ in range(100):
        V = int(rng.integers(2, 400))
        p = special.softmax(rng.standard_normal(V) * 3)
        k = int(rng.integers(1, V + 1))
        tp = float(rng.uniform(0.05, 1.0))
        out, margin = oracle_mod.filter_row(p, k, tp)
        kept = np.flatnonzero(out > 0)
        assert 1 <= kept.size <= k
        assert abs(out.sum() - 1.0) < 1e-12
        # kept tokens keep their relative odds, and outrank every dropped token
        np.testing.assert_allclose(out[kept] / out[kept].sum(), p[kept] / p[kept].sum(),
                                   rtol=1e-12)
        dropped = np.setdiff1d(np.arange(V), kept)
        if dropped.size:
            assert p[kept].min() >= p[dropped].max()
        if margin > 1e-12:
            # the kept mass reaches top_p of the top-k mass; without its least token it does not
            mk = np.sort(p)[::-1][:k].sum()
            assert p[kept].sum() >= tp * mk * (1 - 1e-12)
            assert p[kept].sum() - p[kept].min() < tp * mk


@pytest.mark.parametrize("k,tp", [(0, 0.9), (-3, 0.9), (5, 0.0), (5, 1.5), (5, float("nan"))])
def test_filter_rejects_bad_parameters(oracle_mod, k, tp):
    with pytest.raises(ValueError):
        oracle_mod.filter_row(np.array([0.5, 0.5]), k, tp)


# ---------------------------------------------------------------------------------
# the block step with filtering
# ---------------------------------------------------------------------------------
def _random_block(rng, B, gamma, V, T):
    target = (rng.standard_normal((B, gamma, V)) * 2.5).astype(np.float32)
    drafter = np.empty_like(target)
    drafter[:, 0] = rng.standard_normal((B, V)).astype(np.float32)
    drafter[:, 1:] = target[:, :-1] + rng.standard_normal((B, gamma - 1, V)).astype(np.float32)
    tok = rng.integers(0, V, (B, gamma)).astype(np.int32)
    u = (1.0 - rng.random((B, gamma))).astype(np.float32)
    temps = np.resize(np.asarray(T, np.float32), B)
    return target, drafter, tok, temps, u


def test_filter_off_equals_unfiltered_rule(oracle_mod):
    rng = np.random.default_rng(24)
    B, gamma, V = 40, 5, 300
    target, drafter, tok, temps, u = _random_block(rng, B, gamma, V, [1.0, 0.7, 0.0, 1.3])
    r0 = oracle_mod.accept_block(target, drafter, tok, temps, u)
    for k in (V, V + 7, 1 << 30):
        r1 = oracle_mod.accept_block_filtered(target, drafter, tok, temps, k, 1.0, u)
        for key in ("num_accepted", "out_tokens", "num_emitted", "status"):
            np.testing.assert_array_equal(r1[key], r0[key])
        np.testing.assert_allclose(r1["diag"], r0["diag"], rtol=1e-12)


def test_greedy_sequences_ignore_the_filter(oracle_mod):
    rng = np.random.default_rng(25)
    B, gamma, V = 30, 6, 200
    target, drafter, tok, _, u = _random_block(rng, B, gamma, V, 0.0)
    tok[:, 1:] = np.argmax(target[:, :-1], axis=-1)
    tok[::3, 3] = (tok[::3, 3] + 1) % V
    temps = np.zeros(B, np.float32)
    r0 = oracle_mod.accept_block(target, drafter, tok, temps, u)
    r1 = oracle_mod.accept_block_filtered(target, drafter, tok, temps, 1, 0.01, u)
    for key in ("num_accepted", "out_tokens", "num_emitted", "status"):
        np.testing.assert_array_equal(r1[key], r0[key])
    # an out-of-range filter on a greedy sequence is not an error
    r2 = oracle_mod.accept_block_filtered(target, drafter, tok, temps, 0, 2.0, u)
    np.testing.assert_array_equal(r2["out_tokens"], r0["out_tokens"])


def test_per_sequence_filters(oracle_mod):
    rng = np.random.default_rng(26)
    B, gamma, V = 12, 4, 100
    target, drafter, tok, temps, u = _random_block(rng, B, gamma, V, 1.0)
    ks = rng.integers(1, 60, B).astype(np.int32)
    tps = rng.uniform(0.2, 1.0, B).astype(np.float32)
    r = oracle_mod.accept_block_filtered(target, drafter, tok, temps, ks, tps, u)
    for b in range(B):
        rb = oracle_mod.accept_block_filtered(target[b:b + 1], drafter[b:b + 1], tok[b:b + 1],
                                              temps[b:b + 1], ks[b], tps[b], u[b:b + 1])
        for key in ("num_accepted", "out_tokens", "num_emitted"):
            np.testing.assert_array_equal(r[key][b], rb[key][0])


def test_bad_filter_parameters_flag_tempered_sequences(oracle_mod):
    rng = np.random.default_rng(27)
    B, gamma, V = 4, 3, 50
    target, drafter, tok, temps, u = _random_block(rng, B, gamma, V, 1.0)
    r = oracle_mod.accept_block_filtered(target, drafter, tok, temps,
                                         np.array([5, 0, 5, 5], np.int32),
                                         np.array([0.9, 0.9, 0.0, 1.0], np.float32), u)
    assert list(r["status"]) == [0, 3, 3, 0]
    assert r["num_accepted"][1] == -1 and np.all(r["out_tokens"][2] == -1)


def test_draft_outside_the_filtered_proposal(oracle_mod):
    # A draft outside q's filtered support has q'(t) = 0: it is accepted when p'(t) > 0
    # and rejected when p'(t) = 0 (ratio 0 against a uniform in (0, 1]).
    p = np.array([[0.5, 0.5, 0.0], [0.25, 0.25, 0.5]])
    q = np.array([[1 / 3, 1 / 3, 1 / 3], [0.0, 1.0, 0.0]])
    for t, accept in ((0, True), (2, False)):
        r = oracle_mod.accept_probs(p, q, np.array([1, t], np.int32),
                                    np.array([1.0, 0.5], np.float32))
        assert (r["n"] == 2) == accept


# exact losslessness for the filtered target ------------------------------------
# Raw rows (relative weights, V = 5) and their filtered forms under k = 3, top-p 0.7:
#   p_1 [4, 12, 1, 4, 2]: top-3 = tokens 1, 0, 3 (0 and 3 tie; 0 ranks first), mass
#       20; cumulative 0.6, 0.8 -> keep {1, 0}: p'_1 = (1/4, 3/4, 0, 0, 0)
#   p_2 [1, 6, 2, 6, 4]: top-3 = 1, 3, 4, mass 16; cumulative 0.375, 0.75 -> keep
#       {1, 3}: p'_2 = (0, 1/2, 0, 1/2, 0)
#   p_3 [8, 8, 1, 2, 3]: top-3 = 0, 1, 4, mass 19; 8/19, 16/19 -> keep {0, 1}:
#       p'_3 = (1/2, 1/2, 0, 0, 0)
#   q_1 [6, 2, 1, 2, 1]: top-3 = 0, 1, 3, mass 10; 0.6, 0.8 -> keep {0, 1}:
#       q'_1 = (3/4, 1/4, 0, 0, 0)
#   q_2 [1, 3, 2, 5, 5]: top-3 = 3, 4, 1, mass 13; 5/13, 10/13 -> keep {3, 4}:
#       q'_2 = (0, 0, 0, 1/2, 1/2)
RAW_P = np.array([[4, 12, 1, 4, 2], [1, 6, 2, 6, 4], [8, 8, 1, 2, 3]], np.float64)
RAW_Q = np.array([[1, 1, 1, 1, 1], [6, 2, 1, 2, 1], [1, 3, 2, 5, 5]], np.float64)
P_FILT = np.array([[0.25, 0.75, 0, 0, 0], [0, 0.5, 0, 0.5, 0], [0.5, 0.5, 0, 0, 0]])
Q_FILT = np.array([[0.2] * 5, [0.75, 0.25, 0, 0, 0], [0, 0, 0, 0.5, 0.5]])


def test_worked_rows_filter_as_stated():
    for raw, filt in zip(np.vstack([RAW_P, RAW_Q[1:]]), np.vstack([P_FILT, Q_FILT[1:]])):
        exact = brute_filter(raw / raw.sum(), 3, 0.7)
        assert [float(x) for x in exact] == list(filt)


def filtered_output_distribution(oracle_mod, T, lib=None):
    """Exact distribution of the completed tuple (x_1, x_2, x_3) of one filtered verify
    step on the rows above (k = 3, top-p 0.7): drafts enumerated from q' with their
    weights, uniforms over every cell, positions after the emitted ones completed from
    their filtered target rows."""
    gamma, V = 3, 5
    mids, widths = uniform_cells(8)
    C = len(mids)
    cells = np.array(list(itertools.product(range(C), repeat=gamma)))
    drafts = [d for d in itertools.product(range(V), repeat=gamma - 1)
              if Q_FILT[1][d[0]] > 0 and Q_FILT[2][d[1]] > 0]
    N = len(drafts) * len(cells)
    tl = np.broadcast_to((np.log(RAW_P) * T).astype(np.float32), (N, gamma, V)).copy()
    dl = np.broadcast_to((np.log(RAW_Q) * T).astype(np.float32), (N, gamma, V)).copy()
    tok = np.zeros((N, gamma), np.int32)
    u = np.empty((N, gamma), np.float32)
    wt = np.empty(N)
    for di, d in enumerate(drafts):
        sl = slice(di * len(cells), (di + 1) * len(cells))
        tok[sl, 1:] = d
        u[sl] = mids[cells]
        wt[sl] = Q_FILT[1][d[0]] * Q_FILT[2][d[1]] * np.prod(widths[cells], axis=1)
    r = oracle_mod.accept_block_filtered(tl, dl, tok, np.full(N, T, np.float32), 3, 0.7, u,
                                         lib=lib)
    ne = r["num_emitted"]
    out = r["out_tokens"]
    Pout = np.zeros((V,) * gamma)
    for s in range(N):
        n = ne[s] - 1
        if n < 1:
            continue
        term = np.zeros((V,) * n)
        term[tuple(out[s, 1:n + 1])] = wt[s]
        for k in range(n + 1, gamma + 1):
            term = np.multiply.outer(term, P_FILT[k - 1])
        Pout += term
    return Pout, r


@pytest.mark.parametrize("T", [1.0, 0.5])
def test_filtered_lossless_exact_enumeration(oracle_mod, T):
    Pout, r = filtered_output_distribution(oracle_mod, T)
    assert np.all(r["status"] == 0)
    assert np.all(r["filter_margin"] > 1e-3)
    np.testing.assert_allclose(Pout, target_product(P_FILT), rtol=0, atol=1e-12)


def test_filtered_acceptance_rate_closed_form(oracle_mod):
    # E[accepted] = sum_k prod_{i<=k} alpha_i with alpha_i = sum_x min(p'_i, q'_i), the
    # rows filtered by the brute-force definition; drafts drawn from q'.
    rng = np.random.default_rng(28)
    gamma, V, T, k, tp, trials = 5, 24, 1.0, 6, 0.8, 40000
    target = (rng.standard_normal((gamma, V)) * 1.5).astype(np.float32)
    drafter = np.empty_like(target)
    drafter[0] = rng.standard_normal(V).astype(np.float32)
    drafter[1:] = target[:-1] + (rng.standard_normal((gamma - 1, V)) * 0.7).astype(np.float32)
    p = special.softmax(target.astype(np.float64) / T, axis=-1)
    q = special.softmax(drafter.astype(np.float64) / T, axis=-1)
    pf = np.array([[float(x) for x in brute_filter(r, k, tp)] for r in p])
    qf = np.array([[float(x) for x in brute_filter(r, k, tp)] for r in q])
    alpha = np.array([np.minimum(pf[i - 1], qf[i]).sum() for i in range(1, gamma)])
    surv = np.cumprod(alpha)
    tok = np.zeros((trials, gamma), np.int32)
    for i in range(1, gamma):
        tok[:, i] = rng.choice(V, size=trials, p=qf[i])
    u = (1.0 - rng.random((trials, gamma))).astype(np.float32)
    r = oracle_mod.accept_block_filtered(np.broadcast_to(target, (trials, gamma, V)).copy(),
                                         np.broadcast_to(drafter, (trials, gamma, V)).copy(),
                                         tok, np.full(trials, T, np.float32), k, tp, u)
    a = r["num_accepted"].astype(np.float64)
    se = a.std() / np.sqrt(trials)
    assert abs(a.mean() - surv.sum()) < 5 * se
    for j in range(1, gamma):
        emp = (a >= j).mean()
        assert abs(emp - surv[j - 1]) < 5 * np.sqrt(surv[j - 1] * (1 - surv[j - 1]) / trials) + 1e-9
    # every emitted token lies in the support of the filtered row it came from
    out, ne = r["out_tokens"], r["num_emitted"]
    for s in range(0, trials, 97):
        n = ne[s] - 1
        final = out[s, n]
        row = pf[n - 1] if n == gamma else np.maximum(pf[n - 1] - qf[n], 0)
        assert row[final] > 0
