"""Pins of the oracle's draft-side steps (CPU only, no GPU): sampling the block tokens
from the drafter rows (the free token x^{L+1} ~ q_0 and the drafts x~ ~ q of the
Algorithm, Appendix B.3), the noise tokens z ~ U[V] that start a draft pass, and the
roll-back of a paged KV cache to the accepted prefix.

Each test checks the oracle against something other than itself: exact probabilities
of an inverse-CDF draw over every cell of the uniform on dyadic rows, numpy's
searchsorted on scipy's softmax, a chi-square of seeded draws, the argmax special case,
the brute-force filter definition of test_oracle_filtered, closed forms of the noise
mapping, and conservation laws of the page pool on hand-worked and random cases.
"""

import numpy as np
import pytest
from scipy import special, stats

from paper_2609_04010_gb300 import workloads as W
from test_oracle_accept import uniform_cells
from test_oracle_filtered import brute_filter


# ---------------------------------------------------------------------------------
# sampling the block tokens
# ---------------------------------------------------------------------------------
def test_sample_exact_over_uniform_cells(oracle_mod):
    # Rows whose probabilities are multiples of 1/8: the token is constant on every cell
    # between fractions of denominator <= 8, so weighting each cell by its width gives
    # the exact law of the draw, which must be the row itself.
    rows = np.array([[1, 2, 0, 4, 1], [4, 4, 0, 0, 0], [0, 1, 1, 1, 5]], np.float64) / 8
    mids, widths = uniform_cells(8)
    C = len(mids)
    for T in (1.0, 0.5):
        logits = np.where(rows > 0, np.log(np.where(rows > 0, rows, 1)) * T, -np.inf)
        dl = np.broadcast_to(logits.astype(np.float32), (C, 3, 5)).copy()
        u = np.repeat(mids[:, None], 3, axis=1).astype(np.float32)
        r = oracle_mod.sample_block(dl, np.full(C, T, np.float32), u)
        assert np.all(r["status"] == 0)
        for j in range(3):
            law = np.bincount(r["tokens"][:, j], weights=widths, minlength=5)
            np.testing.assert_allclose(law, rows[j], rtol=0, atol=1e-12)


def test_sample_matches_searchsorted_per_row(oracle_mod):
    # Each block token j uses its own row and its own uniform u[b][j].
    rng = np.random.default_rng(31)
    B, G, V = 40, 6, 300
    dl = (rng.standard_normal((B, G, V)) * 2).astype(np.float32)
    T = np.resize(np.array([1.0, 0.7, 1.6], np.float32), B)
    u = (1.0 - rng.random((B, G))).astype(np.float32)
    r = oracle_mod.sample_block(dl, T, u)
    checked = 0
    for b in range(B):
        for j in range(G):
            p = special.softmax(dl[b, j].astype(np.float64) / float(T[b]))
            c = np.cumsum(p)
            target = float(u[b, j]) * c[-1]
            if np.min(np.abs(c - target)) < 1e-12:
                continue
            x = int(np.searchsorted(c, target, side="left"))
            assert r["tokens"][b, j] == x
            np.testing.assert_allclose(r["q_tok"][b, j], p[x], rtol=1e-12)
            checked += 1
    assert checked > 200


def test_sample_chi_square(oracle_mod):
    rng = np.random.default_rng(32)
    N, G, V = 200_000, 3, 12
    row_logits = (rng.standard_normal((G, V)) * 1.5).astype(np.float32)
    dl = np.broadcast_to(row_logits, (N, G, V)).copy()
    u = W.philox_uniforms(7, N * G).reshape(N, G)
    r = oracle_mod.sample_block(dl, np.ones(N, np.float32), u)
    for j in range(G):
        p = special.softmax(row_logits[j].astype(np.float64))
        obs = np.bincount(r["tokens"][:, j], minlength=V)
        assert stats.chisquare(obs, p * N).pvalue > 1e-3


def test_sample_greedy_is_lowest_argmax(oracle_mod):
    rng = np.random.default_rng(33)
    B, G, V = 30, 4, 50
    dl = rng.integers(-3, 3, (B, G, V)).astype(np.float32)  # many ties
    r = oracle_mod.sample_block(dl, np.zeros(B, np.float32), np.full((B, G), 0.5, np.float32))
    np.testing.assert_array_equal(r["tokens"], np.argmax(dl, axis=-1))
    assert np.all(r["q_tok"] == 1.0)


def test_sample_small_temperature_limit(oracle_mod):
    rng = np.random.default_rng(34)
    B, G, V = 20, 4, 64
    base = rng.permutation(V).astype(np.float32) * 0.25
    dl = np.stack([np.stack([rng.permutation(base) for _ in range(G)]) for _ in range(B)])
    u = (1.0 - rng.random((B, G))).astype(np.float32)
    g = oracle_mod.sample_block(dl, np.zeros(B, np.float32), u)
    s = oracle_mod.sample_block(dl, np.full(B, 1e-3, np.float32), u)
    np.testing.assert_array_equal(g["tokens"], s["tokens"])


def test_sample_filtered_law(oracle_mod):
    rng = np.random.default_rng(35)
    N, V, k, tp = 100_000, 20, 5, 0.8
    row = (rng.standard_normal((1, V)) * 1.5).astype(np.float32)
    dl = np.broadcast_to(row, (N, 1, V)).copy()
    u = W.philox_uniforms(8, N).reshape(N, 1)
    r = oracle_mod.sample_block(dl, np.ones(N, np.float32), u, top_k=k, top_p=tp)
    pf = np.array([float(x) for x in brute_filter(special.softmax(row[0].astype(np.float64)), k, tp)])
    obs = np.bincount(r["tokens"][:, 0], minlength=V)
    assert np.all(obs[pf == 0] == 0)
    keep = pf > 0
    assert stats.chisquare(obs[keep], pf[keep] * N).pvalue > 1e-3
    # filtering off: the unfiltered draw exactly
    a = oracle_mod.sample_block(dl[:1000], np.ones(1000, np.float32), u[:1000], top_k=V, top_p=1.0)
    b = oracle_mod.sample_block(dl[:1000], np.ones(1000, np.float32), u[:1000])
    np.testing.assert_array_equal(a["tokens"], b["tokens"])


def test_sample_flags_bad_inputs(oracle_mod):
    rng = np.random.default_rng(36)
    B, G, V = 5, 3, 40
    dl = rng.standard_normal((B, G, V)).astype(np.float32)
    dl[1, 2, 7] = np.nan
    dl[2, 0, :] = -np.inf
    T = np.array([1, 1, 1, 0, 1], np.float32)
    r = oracle_mod.sample_block(dl, T, np.full((B, G), 0.5, np.float32),
                                top_k=np.array([5, 5, 5, 0, 0], np.int32),
                                top_p=np.array([0.9, 0.9, 0.9, 0.9, 0.9], np.float32))
    assert list(r["status"]) == [0, 1, 1, 0, 3]  # greedy ignores the filter
    assert np.all(r["tokens"][[1, 2, 4]] == -1)


# ---------------------------------------------------------------------------------
# noise tokens
# ---------------------------------------------------------------------------------
def test_noise_tokens_closed_forms(oracle_mod):
    oracle = oracle_mod
    words = W.philox_words(11, 4096)
    for k in (1, 8, 17):
        np.testing.assert_array_equal(oracle.noise_tokens(words, 1 << k),
                                      (words >> np.uint32(32 - k)).astype(np.int32))
    t = oracle.noise_tokens(np.array([0, 2**32 - 1, 2**31], np.uint64), 128256)
    assert list(t) == [0, 128255, 64128]
    big = oracle.noise_tokens(W.philox_words(12, 600_000), 151936)
    assert big.min() >= 0 and big.max() < 151936
    obs = np.bincount(big // 1187, minlength=128)  # 128 equal bins of the vocabulary
    assert stats.chisquare(obs).pvalue > 1e-3


# ---------------------------------------------------------------------------------
# KV commit
# ---------------------------------------------------------------------------------
def test_commit_worked_example(oracle_mod):
    oracle = oracle_mod
    # page size 4, gamma 4; three sequences of ctx 5, 8, 3 (kv_len = ctx + 4).
    table = np.array([[10, 11, 12, -1], [20, 21, 22, -1], [30, 31, -1, -1]], np.int32)
    kv = np.array([9, 12, 7], np.int32)
    na = np.array([1, 3, -1], np.int32)  # n = 2, 4; the third step failed
    free = np.zeros(16, np.int32)
    free[:3] = [40, 41, 42]
    # reserve: lengths 7, 12, 3; the first needs pages for 11 keys (3 pages, has 3),
    # the second for 16 (4 pages, has 3: pops 42), the third for 7 (2 pages, has 2).
    new, t, f, c, fl = oracle.commit_kv(kv, na, table, 4, 4, free, 3, reserve=True)
    assert list(new) == [7, 12, 3] and c == 2 and list(fl) == [0, 0, 0]
    assert list(t[1]) == [20, 21, 22, 42] and list(t[0]) == [10, 11, 12, -1]
    # release: lengths 7 (2 pages: frees 12), 12 (3 pages), 3 (1 page: frees 31)
    new, t, f, c, fl = oracle.commit_kv(kv, na, table, 4, 4, free, 3, reserve=False)
    assert list(new) == [7, 12, 3] and c == 5 and list(f[3:5]) == [12, 31]
    assert list(t[0]) == [10, 11, -1, -1] and list(t[2]) == [30, -1, -1, -1]


def _random_pool(rng, B, P, max_pages, gamma, spare):
    ctx = rng.integers(0, max_pages * P - gamma + 1, B)
    kv = (ctx + gamma).astype(np.int32)
    npages = -(-kv // P)
    ids = rng.permutation(int(npages.sum()) + spare).astype(np.int32)
    table = np.full((B, max_pages), -1, np.int32)
    pos = 0
    for b in range(B):
        table[b, :npages[b]] = ids[pos:pos + npages[b]]
        pos += npages[b]
    free = np.zeros(len(ids), np.int32)
    free[:spare] = ids[pos:]
    return kv, table, free, spare, len(ids)


@pytest.mark.parametrize("reserve", [True, False])
def test_commit_conserves_pages(oracle_mod, reserve):
    oracle = oracle_mod
    rng = np.random.default_rng(37)
    for trial in range(50):
        B, P, gamma = int(rng.integers(1, 20)), int(rng.choice([4, 16])), int(rng.integers(1, 9))
        max_pages = int(rng.integers(2, 12))
        if max_pages * P < gamma:
            continue
        kv, table, free, count, total = _random_pool(rng, B, P, max_pages, gamma,
                                                     int(rng.integers(0, 6)))
        na = rng.integers(-1, gamma, B).astype(np.int32)
        new, t, f, c, fl = oracle.commit_kv(kv, na, table, P, gamma, free, count, reserve)
        # every page is held exactly once: by one table or by the free list
        held = np.concatenate([t[t >= 0], f[:c]])
        assert np.array_equal(np.sort(held), np.arange(total))
        for b in range(B):
            n = na[b] + 1 if na[b] >= 0 else 0
            assert new[b] == kv[b] - gamma + n
            pages = int((t[b] >= 0).sum())
            assert np.all(t[b, :pages] >= 0) and np.all(t[b, pages:] == -1)
            if reserve and fl[b] == 0:
                assert pages == -(-(new[b] + gamma) // P)
            elif fl[b] == 2:
                assert pages == -(-kv[b] // P)
            else:
                assert pages == -(-new[b] // P)
        if reserve:  # once the pool refuses a request, every later request is refused
            need = np.array([-(-(new[b] + gamma) // P) - -(-kv[b] // P) for b in range(B)])
            fits = np.array([-(-(new[b] + gamma) // P) <= max_pages for b in range(B)])
            pool_refused = np.flatnonzero((fl == 2) & fits)
            if pool_refused.size:
                later = np.arange(B) > pool_refused[0]
                assert np.all(fl[later & (fl == 0)] == 0)
                assert not np.any(later & (fl == 0) & (need > 0))


def test_commit_flags_bad_input_and_exhaustion(oracle_mod):
    oracle = oracle_mod
    table = np.array([[1, 2, -1], [3, -1, -1], [4, -1, -1]], np.int32)
    kv = np.array([6, 2, 3], np.int32)     # gamma 3: the second has kv_len < gamma
    na = np.array([2, 0, 5], np.int32)     # the third's num_accepted > gamma - 1
    free = np.array([9, 0, 0, 0], np.int32)
    new, t, f, c, fl = oracle.commit_kv(kv, na, table, 4, 3, free, 1, reserve=True)
    assert list(fl) == [0, 1, 1] and list(new) == [6, 2, 3]
    assert list(t[0]) == [1, 2, 9] and c == 0
    # two sequences that both need a page, one page free: batch order decides
    table = np.array([[1, -1], [2, -1]], np.int32)
    new, t, f, c, fl = oracle.commit_kv(np.array([4, 4]), np.array([3, 3]), table, 4, 4,
                                        np.array([7, 0]), 1, reserve=True)
    assert list(fl) == [0, 2] and list(t[0]) == [1, 7] and list(t[1]) == [2, -1]
    # batch order: the first two take the list's two pages, so the third's single page,
    # which would fit the list on its own, is refused
    table = np.array([[1, -1, -1], [2, -1, -1], [3, -1, -1]], np.int32)
    new, t, f, c, fl = oracle.commit_kv(np.array([4, 4, 4]), np.array([0, 3, 3]), table, 4, 4,
                                        np.array([7, 8, 0]), 2, reserve=True)
    # needs: 1 (ctx 0 + n 1 + 4 keys = 5 -> 2 pages), 1 (8 keys -> 2), 1
    assert list(fl) == [0, 0, 2] and list(t[0][:2]) == [1, 8] and list(t[1][:2]) == [2, 7]
    # a refused request still counts against the later ones (gamma 8, one free page): the
    # first asks for 2 pages (ctx 0 + n 8 + 8 keys -> 4 pages, has 2) and is refused; the
    # second's single page (ctx 0 + n 1 + 8 keys -> 3 pages) would fit, but the requests
    # of sequences 0 and 1 together do not
    table = np.array([[1, 2, -1, -1], [3, 4, -1, -1]], np.int32)
    new, t, f, c, fl = oracle.commit_kv(np.array([8, 8]), np.array([7, 0]), table, 4, 8,
                                        np.array([9, 0]), 1, reserve=True)
    assert list(fl) == [2, 2] and list(new) == [8, 1] and c == 1
    assert np.array_equal(t, table)
    # a request of zero pages after a refused one is served, and the list's top stays
    # where the last grant left it
    table = np.array([[1, -1, -1], [2, -1, -1], [3, 4, -1]], np.int32)
    new, t, f, c, fl = oracle.commit_kv(np.array([4, 4, 8]), np.array([3, 3, -1]), table, 4, 4,
                                        np.array([5, 0, 0]), 1, reserve=True)
    assert list(fl) == [0, 2, 0] and c == 0 and list(t[0]) == [1, 5, -1]
    # release with room for one more page: every step failed, so each sequence drops
    # back to its context and offers one page; the first fits, the other two do not
    table = np.array([[1, 2, 3], [4, 5, -1], [6, 7, -1]], np.int32)
    new, t, f, c, fl = oracle.commit_kv(np.array([12, 8, 8]), np.array([-1, -1, -1]), table, 4,
                                        4, np.array([9, 0]), 1, reserve=False)
    assert list(new) == [8, 4, 4] and list(fl) == [0, 2, 2] and c == 2 and list(f) == [9, 3]
    assert list(t[0]) == [1, 2, -1] and list(t[1]) == [4, 5, -1] and list(t[2]) == [6, 7, -1]
