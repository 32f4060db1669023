"""Pins of the oracle's tree verification (CPU only, no GPU): the tree sampler's
candidate tree (the top K tokens per block position, pruned to the best prefixes by
log-probability, Sec. 3.3 "Tree Sampler"), tree attention (every node sees the prefix
and its own ancestors, Sec. 4.2), greedy acceptance along the tree, and the compaction
of the accepted path's keys and values.

Each test checks the oracle against something other than itself: brute-force
enumeration of every prefix, structural invariants, the special case K = 1 (a chain:
the linear sampler and the linear greedy rule), a dense numpy restatement of masked
attention, causal masks against the block-causal attention oracle, invariance to keys a
node cannot see, and a depth-first search for the deepest argmax-matching path.
"""

import itertools

import numpy as np
import pytest
from scipy import special

from paper_2609_04010_gb300 import workloads as W


def _logq(row, T):
    return special.log_softmax(row.astype(np.float64) / T)


def brute_force_prefixes(dl_b, T, K, budget):
    """Every prefix of top-K candidates, scored; the best `budget` (as token tuples)."""
    G = dl_b.shape[0]
    lq = [None] + [_logq(dl_b[d], T) for d in range(1, G)]
    top = [None] + [sorted(range(dl_b.shape[1]), key=lambda x: (-lq[d][x], x))[:K] for d in range(1, G)]
    prefixes = []
    for depth in range(1, G):
        for combo in itertools.product(*[top[d] for d in range(1, depth + 1)]):
            score = sum(lq[d + 1][c] for d, c in enumerate(combo))
            prefixes.append((score, combo))
    prefixes.sort(key=lambda t: -t[0])
    return {c for _, c in prefixes[:budget]}, prefixes


def node_prefix(tree, b, j):
    out = []
    while j > 0:
        out.append(int(tree["tokens"][b, j]))
        j = int(tree["parents"][b, j])
    return tuple(reversed(out))


@pytest.mark.parametrize("K,G,budget", [(3, 4, 12), (2, 5, 20), (4, 3, 19), (5, 4, 30)])
def test_tree_is_the_best_prefixes(oracle_mod, K, G, budget):
    rng = np.random.default_rng(K * 100 + G)
    B, V = 6, 20
    dl = (rng.standard_normal((B, G, V)) * 1.5).astype(np.float32)
    T = np.resize(np.array([1.0, 0.7, 0.0], np.float32), B)
    tree = oracle_mod.build_tree(dl, T, rng.integers(0, V, B), K, budget)
    for b in range(B):
        t = float(T[b]) if T[b] > 0 else 1.0
        want, ranked = brute_force_prefixes(dl[b], t, K, budget)
        if budget < len(ranked) and ranked[budget - 1][0] - ranked[budget][0] < 1e-9:
            continue  # a tie at the cut
        got = {node_prefix(tree, b, j) for j in range(1, budget + 1)}
        assert got == want
        scores = {c: s for s, c in ranked}
        for j in range(1, budget + 1):
            np.testing.assert_allclose(tree["score"][b, j], scores[node_prefix(tree, b, j)], rtol=1e-12)


def test_tie_rules_worked_example(oracle_mod):
    # Worked by hand (K = 2, budget 6, T = 1). Position 1's tokens 0 and 1 tie at the
    # top, position 2's tokens 1 and 2 tie behind token 0. Equal candidates rank by the
    # lower token id; equal offers go to the lower parent index.
    #   step 1: root offers token 0 (the lower id of the tie)          -> node 1
    #   step 2: root's token 1 (same score) beats node 1's child       -> node 2
    #   step 3: nodes 1 and 2 offer token 0 at the same score; node 1  -> node 3
    #   step 4: node 2's token 0 beats node 1's token 1                -> node 4
    #   step 5: nodes 1 and 2 offer token 1 at the same score; node 1  -> node 5
    #   step 6: node 2's token 1                                       -> node 6
    dl = np.array([[[0, 0, 0], [0, 0, -10], [5, 0, 0]]], np.float32)
    tree = oracle_mod.build_tree(dl, np.ones(1, np.float32), np.array([2]), 2, 6)
    assert list(tree["tokens"][0]) == [2, 0, 1, 0, 0, 1, 1]
    assert list(tree["parents"][0]) == [-1, 0, 0, 1, 2, 1, 2]
    assert list(tree["cand_tokens"][0, 1]) == [0, 1] and list(tree["cand_tokens"][0, 2]) == [0, 1]
    assert tree["margin"][0] == 0.0


def test_tree_structure(oracle_mod):
    rng = np.random.default_rng(51)
    B, G, V, K, budget = 8, 16, 200, 8, 40
    dl = (rng.standard_normal((B, G, V)) * 2).astype(np.float32)
    tree = oracle_mod.build_tree(dl, np.ones(B, np.float32), rng.integers(0, V, B), K, budget)
    for b in range(B):
        par, dep, tok = tree["parents"][b], tree["depth"][b], tree["tokens"][b]
        assert par[0] == -1 and dep[0] == 0
        for j in range(1, budget + 1):
            assert 0 <= par[j] < j and dep[j] == dep[par[j]] + 1 <= G - 1
            # bit i of the mask: i is j or an ancestor of j
            anc, a = set(), j
            while a >= 0:
                anc.add(a)
                a = par[a]
            bits = int(tree["mask"][b, j])
            assert {i for i in range(budget + 1) if bits >> i & 1} == anc
            assert tree["score"][b, j] <= tree["score"][b, par[j]]
        for u in range(budget + 1):
            # a node's children are its best candidates, in order, with distinct tokens
            kids = [c for c in range(budget + 1) if par[c] == u]
            if kids:
                lq = _logq(dl[b, dep[u] + 1], 1.0)
                best = sorted(range(V), key=lambda x: (-lq[x], x))[:len(kids)]
                assert [int(tok[c]) for c in kids] == best


def test_k1_tree_is_the_greedy_chain(oracle_mod):
    # K = 1: one candidate per position, so the tree is the chain of the drafter's
    # argmaxes, and greedy tree acceptance is the linear greedy rule on that chain.
    rng = np.random.default_rng(52)
    B, G, V = 20, 8, 100
    inp = W.make_accept_inputs(B, G, V, "f32", 3.0, 1.0, 0.0, seed=52)
    root = inp.block_tokens[:, 0]
    tree = oracle_mod.build_tree(inp.drafter_logits, inp.temperature, root, 1, G - 1)
    np.testing.assert_array_equal(tree["tokens"][:, 1:], np.argmax(inp.drafter_logits[:, 1:], -1))
    np.testing.assert_array_equal(tree["parents"], np.tile(np.arange(-1, G - 1), (B, 1)))
    tokens = tree["tokens"]
    acc = oracle_mod.accept_tree_greedy(inp.target_logits, tokens, tree["parents"])
    lin = oracle_mod.accept_block(inp.target_logits, inp.drafter_logits, tokens, inp.temperature,
                                  inp.uniforms)
    np.testing.assert_array_equal(acc["num_accepted"], lin["num_accepted"])
    np.testing.assert_array_equal(acc["out_tokens"], lin["out_tokens"])
    assert len(set(acc["num_accepted"].tolist())) > 1


def test_greedy_walk_is_the_deepest_matching_path(oracle_mod):
    rng = np.random.default_rng(53)
    B, G, V, K, budget = 30, 6, 12, 3, 25
    dl = (rng.standard_normal((B, G, V)) * 1.0).astype(np.float32)
    tree = oracle_mod.build_tree(dl, np.ones(B, np.float32), rng.integers(0, V, B), K, budget)
    N = budget + 1
    # targets that often agree with the tree's tokens, so long paths occur
    tl = rng.standard_normal((B, N, V)).astype(np.float32)
    for b in range(B):
        for j in range(N):
            kids = [c for c in range(N) if tree["parents"][b, c] == j]
            if kids and rng.random() < 0.8:
                tl[b, j, tree["tokens"][b, rng.choice(kids)]] += 10.0
    acc = oracle_mod.accept_tree_greedy(tl, tree["tokens"], tree["parents"])
    depths = []
    for b in range(B):
        am = np.argmax(tl[b], axis=-1)
        # depth-first search over every root path whose steps all match the argmax
        best, stack = [0], [[0]]
        while stack:
            path = stack.pop()
            if len(path) > len(best):
                best = path
            for c in range(N):
                if tree["parents"][b, c] == path[-1] and tree["tokens"][b, c] == am[path[-1]]:
                    stack.append(path + [c])
        n = len(best)
        assert list(acc["path"][b, :n]) == best and np.all(acc["path"][b, n:] == -1)
        assert acc["num_accepted"][b] == n - 1 and acc["num_emitted"][b] == n + 1
        assert list(acc["out_tokens"][b, :n]) == [tree["tokens"][b, x] for x in best]
        assert acc["out_tokens"][b, n] == am[best[-1]]
        depths.append(n)
    assert max(depths) >= 3


def _attn_case(rng, B, N, Hq, Hkv, D, P, ctx_hi):
    ctx = rng.integers(0, ctx_hi, B)
    kv = (ctx + N).astype(np.int32)
    pages = -(-kv // P)
    num_pages = int(pages.sum()) + 2
    perm = rng.permutation(num_pages).astype(np.int32)
    table = np.zeros((B, int(pages.max())), np.int32)
    pos = 0
    for b in range(B):
        table[b, :pages[b]] = perm[pos:pos + pages[b]]
        pos += pages[b]
    bf = lambda a: W.f32_to_bf16_bits(a.astype(np.float32)).reshape(a.shape)
    q = bf(rng.standard_normal((B, N, Hq, D)))
    k = bf(rng.standard_normal((num_pages, Hkv, P, D)))
    v = bf(rng.standard_normal((num_pages, Hkv, P, D)))
    return q, k, v, table, kv


def _random_masks(rng, B, N):
    masks = np.zeros((B, N), np.uint64)
    for b in range(B):
        par = [-1] + [int(rng.integers(0, j)) for j in range(1, N)]
        for j in range(N):
            bits, a = 0, j
            while a >= 0:
                bits |= 1 << a
                a = par[a]
            masks[b, j] = np.uint64(bits)
    return masks


def test_tree_attention_dense_restatement(oracle_mod):
    rng = np.random.default_rng(54)
    B, N, Hq, Hkv, D, P = 3, 9, 4, 2, 16, 4
    q, k, v, table, kv = _attn_case(rng, B, N, Hq, Hkv, D, P, 20)
    masks = _random_masks(rng, B, N)
    out, lse, st = oracle_mod.verify_attention(q, k, v, table, kv, N, tree_mask=masks)
    f = lambda h: (h.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    for b in range(B):
        ctx = kv[b] - N
        keys = np.stack([f(k[table[b, t // P], :, t % P]) for t in range(kv[b])])  # [t][Hkv][D]
        vals = np.stack([f(v[table[b, t // P], :, t % P]) for t in range(kv[b])])
        for j in range(N):
            vis = [t for t in range(kv[b]) if t < ctx or (int(masks[b, j]) >> (t - ctx)) & 1]
            for h in range(Hq):
                g = h // (Hq // Hkv)
                s = keys[vis, g] @ f(q[b, j, h]) / np.sqrt(D)
                w = special.softmax(s)
                np.testing.assert_allclose(out[b, j, h], w @ vals[vis, g], rtol=1e-10, atol=1e-12)
                np.testing.assert_allclose(lse[b, j, h], special.logsumexp(s), rtol=1e-12)


def test_causal_masks_give_block_causal_attention(oracle_mod):
    rng = np.random.default_rng(55)
    B, N, Hq, Hkv, D, P = 4, 7, 8, 2, 32, 16
    q, k, v, table, kv = _attn_case(rng, B, N, Hq, Hkv, D, P, 60)
    causal = np.array([[(1 << (j + 1)) - 1 for j in range(N)]] * B, np.uint64)
    a = oracle_mod.verify_attention(q, k, v, table, kv, N, tree_mask=causal)
    c = oracle_mod.verify_attention(q, k, v, table, kv, N)
    np.testing.assert_array_equal(a[0], c[0])
    np.testing.assert_array_equal(a[1], c[1])


def test_tree_attention_ignores_unseen_keys(oracle_mod):
    rng = np.random.default_rng(56)
    B, N, Hq, Hkv, D, P = 2, 10, 4, 4, 16, 8
    q, k, v, table, kv = _attn_case(rng, B, N, Hq, Hkv, D, P, 30)
    masks = _random_masks(rng, B, N)
    base, _, _ = oracle_mod.verify_attention(q, k, v, table, kv, N, tree_mask=masks)
    k2, v2 = k.copy(), v.copy()
    for b in range(B):
        ctx = kv[b] - N
        for i in range(N):
            if not (int(masks[b, N - 1]) >> i) & 1:  # not an ancestor of the last node
                t = ctx + i
                k2[table[b, t // P], :, t % P] ^= np.uint16(0x1234)
                v2[table[b, t // P], :, t % P] ^= np.uint16(0x0F0F)
    other, _, _ = oracle_mod.verify_attention(q, k2, v2, table, kv, N, tree_mask=masks)
    np.testing.assert_array_equal(other[:, N - 1], base[:, N - 1])


def test_compaction_moves_the_path(oracle_mod):
    rng = np.random.default_rng(57)
    B, N, Hkv, D, P = 5, 12, 2, 8, 4
    _, k, v, table, kv = _attn_case(rng, B, N, 4, Hkv, D, P, 13)
    path = np.full((B, N), -1, np.int32)
    na = np.array([3, 0, 5, -1, 2], np.int32)
    for b in range(B):
        n = na[b] + 1 if na[b] >= 0 else 0
        if n:
            path[b, :n] = np.concatenate([[0], np.sort(rng.choice(np.arange(1, N), n - 1, replace=False))])
    k2, v2, kl = oracle_mod.compact_tree_kv(k, v, table, kv, N, path, na)
    for b in range(B):
        ctx = kv[b] - N
        n = na[b] + 1 if na[b] >= 0 else 0
        assert kl[b] == ctx + n
        for d in range(N):
            t = ctx + d
            got = k2[table[b, t // P], :, t % P]
            if 1 <= d < n:
                s = ctx + path[b, d]
                np.testing.assert_array_equal(got, k[table[b, s // P], :, s % P])
                np.testing.assert_array_equal(v2[table[b, t // P], :, t % P], v[table[b, s // P], :, s % P])
            else:  # the root's slot and the slots past the path keep their keys
                np.testing.assert_array_equal(got, k[table[b, t // P], :, t % P])
        # prefix keys untouched
        for t in range(ctx):
            np.testing.assert_array_equal(k2[table[b, t // P], :, t % P], k[table[b, t // P], :, t % P])


# ---------------------------------------------------------------------------------
# sampled (T > 0) tree acceptance
# ---------------------------------------------------------------------------------
from test_oracle_accept import uniform_cells  # noqa: E402


def tree_output_law(oracle_mod, p_rows, tokens, parents, denom, lib_mod=None):
    """Exact law of the emitted tokens (after the root) of one sampled tree verification:
    every combination of Farey(denom) cells of the N uniforms, weighted by the cells'
    widths, through the oracle (one sequence per combination). Rows are probability
    rows whose entries are multiples of 1/denom, given as log-probabilities at T = 1, so
    every threshold the rule compares a uniform with is such a fraction."""
    import itertools
    m = oracle_mod if lib_mod is None else lib_mod
    N, V = p_rows.shape
    mids, widths = uniform_cells(denom)
    combos = np.array(list(itertools.product(range(len(mids)), repeat=N)))
    U = mids[combos].astype(np.float32)
    Wt = np.prod(widths[combos], axis=1)
    with np.errstate(divide="ignore"):
        logits = np.log(p_rows).astype(np.float32)
    B = len(U)
    r = m.accept_tree_sampled(np.broadcast_to(logits, (B, N, V)).copy(),
                              np.broadcast_to(tokens, (B, N)).copy(),
                              np.broadcast_to(parents, (B, N)).copy(),
                              np.ones(B, np.float32), U)
    assert np.all(r["status"] == 0)
    law = {}
    for b in range(B):
        seq = tuple(int(x) for x in r["out_tokens"][b, 1:r["num_emitted"][b]])
        law[seq] = law.get(seq, 0.0) + Wt[b]
    return law


def target_tree_law(p_rows, tokens, parents):
    """The law the target model gives the emitted tokens: from the root, draw x ~ p of the
    current node; if x is the token of one of its children, move there and draw again,
    else stop."""
    N, V = p_rows.shape
    law = {}

    def walk(node, prefix, prob):
        for x in range(V):
            if p_rows[node, x] == 0.0:
                continue
            child = next((c for c in range(1, N) if parents[c] == node and tokens[c] == x), None)
            if child is None:
                law[prefix + (x,)] = law.get(prefix + (x,), 0.0) + prob * p_rows[node, x]
            else:
                walk(child, prefix + (x,), prob * p_rows[node, x])
    walk(0, (), 1.0)
    return law


def assert_same_law(a, b, tol=1e-12):
    keys = set(a) | set(b)
    for k in keys:
        assert abs(a.get(k, 0.0) - b.get(k, 0.0)) <= tol, (k, a.get(k, 0.0), b.get(k, 0.0))


# a root with two children, the first of which has a child (V = 4, rows in quarters)
TREE4_P = np.array([[1, 2, 1, 0], [2, 1, 1, 0], [0, 1, 1, 2], [1, 1, 1, 1]], np.float64) / 4
TREE4_TOK = np.array([3, 1, 0, 2], np.int32)    # root token, then the nodes' tokens
TREE4_PAR = np.array([-1, 0, 0, 1], np.int32)
# a root with three children covering most of its mass (V = 6, rows in sixths)
TREE6_P = np.array([[1, 2, 0, 2, 1, 0], [1, 1, 1, 1, 1, 1], [0, 0, 3, 3, 0, 0],
                    [6, 0, 0, 0, 0, 0]], np.float64) / 6
TREE6_TOK = np.array([0, 3, 1, 4], np.int32)
TREE6_PAR = np.array([-1, 0, 0, 0], np.int32)


@pytest.mark.parametrize("case", ["tree4", "tree6"])
def test_sampled_tree_acceptance_is_lossless(oracle_mod, case):
    p, tok, par, denom = ((TREE4_P, TREE4_TOK, TREE4_PAR, 4) if case == "tree4"
                          else (TREE6_P, TREE6_TOK, TREE6_PAR, 6))
    got = tree_output_law(oracle_mod, p, tok, par, denom)
    assert abs(sum(got.values()) - 1.0) < 1e-12
    assert_same_law(got, target_tree_law(p, tok, par))
    # every branch is reached: a child accepted at depth 2, a later sibling accepted, and
    # a final draw after rejections
    assert any(len(k) == 3 for k in got) or case == "tree6"
    assert any(len(k) == 2 for k in got) and any(len(k) == 1 for k in got)


def test_sampled_tree_without_renormalisation_is_caught(oracle_mod):
    # power check: the rule run on p instead of the renormalised residual p' (the rejected
    # candidates kept) must fail the same exact comparison
    import types
    src = open(oracle_mod.__file__).read()
    site = "                w[tok[b, c]] = 0.0  # the rejected candidate leaves the distribution\n"
    assert src.count(site) == 1
    mod = types.ModuleType("oracle_no_renorm")
    mod.__file__ = oracle_mod.__file__
    exec(compile(src.replace(site, ""), oracle_mod.__file__, "exec"), mod.__dict__)
    got = tree_output_law(oracle_mod, TREE6_P, TREE6_TOK, TREE6_PAR, 6, lib_mod=mod)
    want = target_tree_law(TREE6_P, TREE6_TOK, TREE6_PAR)
    assert max(abs(got.get(k, 0.0) - want.get(k, 0.0)) for k in set(got) | set(want)) > 1e-3


def test_sampled_chain_equals_linear_rule_with_point_mass_drafts(oracle_mod):
    # a chain tree (one child per node) proposes its tokens with certainty: the linear rule
    # with one-hot drafter rows (q = point mass at the draft) takes the same decisions;
    # the tree tests node c with uniforms[c] and draws with uniforms[0], the linear rule
    # tests draft i with uniforms[i - 1] and draws with uniforms[gamma - 1]
    rng = np.random.default_rng(5)
    B, N, V = 300, 5, 12
    tl = (rng.standard_normal((B, N, V)) * 1.5).astype(np.float32)
    T = rng.choice([1.0, 0.7, 1.6], size=B).astype(np.float32)
    tok = np.zeros((B, N), np.int32)
    for b in range(B):
        for c in range(N):
            tok[b, c] = rng.integers(V) if rng.random() < 0.5 else int(np.argmax(tl[b, max(c - 1, 0)]))
    par = np.broadcast_to(np.arange(-1, N - 1, dtype=np.int32), (B, N)).copy()
    u_tree = rng.random((B, N)).astype(np.float32)
    t = oracle_mod.accept_tree_sampled(tl, tok, par, T, u_tree)
    dl = np.full((B, N, V), -np.inf, np.float32)
    for b in range(B):
        for c in range(N):
            dl[b, c, tok[b, c]] = 0.0
    u_lin = np.concatenate([u_tree[:, 1:], u_tree[:, :1]], axis=1)
    lin = oracle_mod.accept_block(tl[:, :N], dl, tok, T, u_lin)
    np.testing.assert_array_equal(t["num_accepted"], lin["num_accepted"])
    np.testing.assert_array_equal(t["out_tokens"], lin["out_tokens"])
    np.testing.assert_array_equal(t["num_emitted"], lin["num_emitted"])


def test_sampled_tree_greedy_and_low_temperature_limits(oracle_mod):
    rng = np.random.default_rng(6)
    B, N, V = 40, 9, 30
    tl = (rng.standard_normal((B, N, V)) * 3).astype(np.float32)
    par = np.array([-1, 0, 0, 1, 1, 2, 3, 3, 5], np.int32)
    tok = np.zeros((B, N), np.int32)
    for b in range(B):
        for c in range(1, N):  # half the children match their parent's argmax
            p = par[c]
            tok[b, c] = int(np.argmax(tl[b, p])) if rng.random() < 0.6 else rng.integers(V)
    parents = np.broadcast_to(par, (B, N)).copy()
    g = oracle_mod.accept_tree_greedy(tl, tok, parents)
    u = rng.uniform(0.05, 0.95, (B, N)).astype(np.float32)
    for T in (0.0, -1.0, 1e-3):
        s = oracle_mod.accept_tree_sampled(tl, tok, parents, np.full(B, T, np.float32), u)
        assert np.all(s["status"] == 0)
        for k in ("path", "num_accepted", "out_tokens", "num_emitted"):
            np.testing.assert_array_equal(s[k], g[k], err_msg=f"T={T} {k}")


def test_sampled_tree_flags_bad_inputs(oracle_mod):
    rng = np.random.default_rng(7)
    B, N, V = 5, 4, 16
    tl = rng.standard_normal((B, N, V)).astype(np.float32)
    tok = rng.integers(0, V, (B, N)).astype(np.int32)
    par = np.broadcast_to(np.array([-1, 0, 0, 1], np.int32), (B, N)).copy()
    T = np.array([1.0, 1.0, 1.0, 0.0, 1.0], np.float32)
    tok[1, 2] = V                 # token outside the vocabulary
    par[2, 3] = 3                 # not a tree
    tl[3, 2, 5] = np.nan          # NaN row, greedy sequence
    tl[4, 1, :] = -np.inf         # no finite logit, tempered sequence
    r = oracle_mod.accept_tree_sampled(tl, tok, par, T, rng.random((B, N)).astype(np.float32))
    assert list(r["status"]) == [0, 2, 2, 1, 1]
    for b in (1, 2, 3, 4):
        assert r["num_accepted"][b] == -1 and r["num_emitted"][b] == 0
        assert np.all(r["out_tokens"][b] == -1) and np.all(r["path"][b] == -1)
    assert r["num_emitted"][0] == r["num_accepted"][0] + 2
