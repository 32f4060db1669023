"""GPU parity of tree verification with the oracle, through the C ABI: the tree sampler
(spec_build_tree), tree attention (spec_verify_attention with tree_mask, both kernels),
greedy acceptance along a tree (spec_accept_tree) and the compaction of the accepted
path (spec_commit_tree_kv).

The tree's structure, acceptance and compaction are integer results: bit-exact, except
a sequence whose tree construction met a near-tie of path scores in the oracle (two
offers within TREE_MARGIN = 1e-4 in log-probability; the kernel ranks by fp32 log q), which
may differ and is counted. Attention within the tolerances of the block-causal tests; a
causal mask reproduces the block-causal kernels bit for bit."""

import numpy as np
import pytest
import torch

from paper_2609_04010_gb300 import binding
from paper_2609_04010_gb300 import workloads as W

from helpers import bf16_dev, compare_attention, dev, logits_dev, sample_rows

pytestmark = pytest.mark.gpu

TREE_MARGIN = 1e-4


def gpu_build(dl, T, root, K, N, ws=None):
    r = binding.build_tree(logits_dev(dl), dev(np.asarray(T, np.float32)),
                           dev(np.asarray(root, np.int32)), K, N, ws=ws)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in r.items()}


def assert_valid_tree(g, o, b, tol):
    """The GPU's tree for sequence b is a best-first tree over the oracle's ranked
    candidates in which every step took an offer within tol of the best one: each
    node's token is its parent's next unused candidate, its depth and mask follow its
    parent's, and its score (fp64, from the oracle's log q) is at most tol below the
    best offer of that step."""
    tok, par, dep, msk = g["tokens"][b], g["parents"][b], g["depth"][b], g["mask"][b].view(np.uint64)
    ct, cq = o["cand_tokens"][b], o["cand_logq"][b]
    G, Kc = ct.shape
    N = len(tok)
    assert tok[0] == o["tokens"][b, 0] and par[0] == -1 and dep[0] == 0 and msk[0] == 1
    score, nxt = [0.0], [0]
    for i in range(1, N):
        offers = {u: score[u] + cq[dep[u] + 1, nxt[u]] for u in range(i)
                  if dep[u] + 1 < G and nxt[u] < Kc}
        u = int(par[i])
        assert u in offers, f"seq {b} node {i}: parent {u} had no offer"
        assert offers[u] >= max(offers.values()) - tol, f"seq {b} node {i}: not the best offer"
        assert tok[i] == ct[dep[u] + 1, nxt[u]] and dep[i] == dep[u] + 1, f"seq {b} node {i}"
        assert msk[i] == msk[u] | np.uint64(1 << i), f"seq {b} node {i}: mask"
        score.append(offers[u])
        nxt[u] += 1
        nxt.append(0)


def check_build(oracle_mod, dl, T, root, K, N, strict=False):
    """GPU trees equal the oracle's where its margin is at least TREE_MARGIN; elsewhere
    they are valid best-first trees within TREE_MARGIN (or equal, if strict)."""
    g = gpu_build(dl, T, root, K, N)
    o = oracle_mod.build_tree(dl, T, root, K, N - 1)
    for b in range(dl.shape[0]):
        same = all(np.array_equal(g[k][b], o[k][b]) for k in ("tokens", "parents", "depth")) and \
            np.array_equal(g["mask"][b].view(np.uint64), o["mask"][b])
        if not same:
            assert not strict and o["margin"][b] < TREE_MARGIN, (
                f"seq {b}: trees differ, oracle margin {o['margin'][b]:.3g}\n"
                f"GPU {g['tokens'][b]} {g['parents'][b]}\noracle {o['tokens'][b]} {o['parents'][b]}")
            assert_valid_tree(g, o, b, TREE_MARGIN)
    return g, o


@pytest.mark.parametrize("batch,G,V,dtype,K,N,temps", [
    (1, 16, 128256, "bf16", 32, 33, 1.0),        # (B, K, V) = (16, 32, 32)
    (1, 16, 151936, "bf16", 32, 64, 0.0),
    (8, 8, 32000, "f32", 8, 33, [1.0, 0.0, 0.5, 2.0]),
    (16, 6, 5000, "bf16", 4, 21, 1.0),
    (32, 8, 32000, "bf16", 16, 33, 0.8),
    (3, 4, 33, "f32", 50, 8, 1.0),               # top_k above the vocabulary, unaligned rows
    (2, 5, 100, "bf16", 3, 12, 0.7),
])
def test_build_tree(oracle_mod, batch, G, V, dtype, K, N, temps):
    inp = W.make_accept_inputs(batch, G, V, dtype, 3.0, 1.0, temps, seed=V + batch)
    check_build(oracle_mod, inp.drafter_logits, inp.temperature, inp.block_tokens[:, 0], K, N)


def test_build_tree_chain_and_root_only(oracle_mod):
    inp = W.make_accept_inputs(2, 40, 3000, "bf16", 3.0, 1.0, 1.0, seed=8)
    g, _ = check_build(oracle_mod, inp.drafter_logits, inp.temperature, inp.block_tokens[:, 0], 1, 33)
    assert np.array_equal(g["parents"][0], np.arange(-1, 32))
    g = gpu_build(inp.drafter_logits, inp.temperature, inp.block_tokens[:, 0], 5, 1)
    assert np.array_equal(g["tokens"][:, 0], inp.block_tokens[:, 0])
    assert np.all(g["parents"] == -1) and np.all(g["depth"] == 0) and np.all(g["mask"] == 1)


def test_build_tree_masked_rows(oracle_mod):
    # rows with fewer finite logits than K: the remaining candidates have log q = -inf
    inp = W.make_accept_inputs(3, 5, 1000, "f32", 3.0, 1.0, 1.0, seed=9)
    dl = inp.drafter_logits
    dl[0, 1:, 5:] = -np.inf
    dl[1, 2, :997] = -np.inf
    check_build(oracle_mod, dl, inp.temperature, inp.block_tokens[:, 0], 8, 30, strict=True)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_build_tree_ranks_structured_rows(oracle_mod, dtype):
    # One drafter position: the tree is the root and the top N-1 candidates in rank
    # order, so this compares the ranked candidate list itself. Sequences 0 and 1 put
    # their large logits in whole 16-byte groups with a period of 128 groups, so that a
    # row part's threads with the largest values hold many values above the threshold
    # (the exact ranking rounds); sequence 2 is a constant row (every candidate tied,
    # ranked by id).
    rng = np.random.default_rng(10)
    B, G, V, epv = 3, 2, 32768, (4 if dtype == "f32" else 8)
    x = rng.standard_normal((B, G, V)).astype(np.float32)
    for b, shift in ((0, 0), (1, 512)):
        grp = ((np.arange(V) + shift) // epv) % 128
        big = grp < 63
        vals = 100.0 + grp[big] * 4.0 + rng.random((G, int(big.sum()))) * 0.5
        x[b][:, big] = vals
    x[2] = 0.25
    dl = W.f32_to_bf16_bits(x).reshape(x.shape) if dtype == "bf16" else x
    g, o = check_build(oracle_mod, dl, np.ones(B, np.float32), np.array([3, 4, 5], np.int32), 63, 64,
                       strict=True)
    assert np.array_equal(g["tokens"][2, 1:], np.arange(63))


def test_build_tree_bad_inputs(oracle_mod):
    B, G, V = 6, 6, 2000
    inp = W.make_accept_inputs(B, G, V, "f32", 3.0, 1.0, 1.0, seed=12)
    dl, root = inp.drafter_logits, inp.block_tokens[:, 0].copy()
    dl[0, 0, 7] = np.nan          # row 0 is never read
    dl[1, 2, 9] = np.nan
    dl[2, 3, 1] = np.inf
    dl[3, 1, :] = -np.inf
    root[4] = V
    ws = binding.new_workspace(1 << 22)
    g = gpu_build(dl, inp.temperature, root, 4, 9, ws=ws)
    flags = binding.read_device_status(ws)[1]
    assert flags == binding.FLAG_BAD_LOGITS | binding.FLAG_BAD_TOKEN
    for b in (1, 2, 3, 4):
        assert np.all(g["tokens"][b] == -1) and np.all(g["parents"][b] == -1)
        assert np.all(g["depth"][b] == -1) and np.all(g["mask"][b] == 0)
    o = oracle_mod.build_tree(dl[[0, 5]], inp.temperature[[0, 5]], root[[0, 5]], 4, 8)
    for i, b in enumerate((0, 5)):
        assert np.array_equal(g["tokens"][b], o["tokens"][i]) or o["margin"][i] < TREE_MARGIN


def test_build_tree_capacity_is_checked():
    dl = torch.zeros(1, 2, 100, dtype=torch.float32, device="cuda")
    T = torch.ones(1, device="cuda")
    root = torch.zeros(1, dtype=torch.int32, device="cuda")
    binding.build_tree(dl, T, root, 3, 4)          # three children of the root
    with pytest.raises(binding.SpecError):
        binding.build_tree(dl, T, root, 3, 5)      # a fourth node has no place


def tree_case(oracle_mod, seed, batch, budget, K, gamma_draft, vocab, dtype="bf16", agree=0.8):
    """A tree built by the oracle from synthetic drafter rows, and target rows that often
    agree with one of each node's children (so long accepted paths occur)."""
    rng = np.random.default_rng(seed)
    inp = W.make_accept_inputs(batch, gamma_draft, vocab, dtype, 3.0, 1.0, 1.0, seed=seed)
    tree = oracle_mod.build_tree(inp.drafter_logits, inp.temperature, inp.block_tokens[:, 0], K,
                                 budget)
    N = budget + 1
    tl32 = rng.standard_normal((batch, N, vocab)).astype(np.float32) * 3
    for b in range(batch):
        for j in range(N):
            kids = [c for c in range(N) if tree["parents"][b, c] == j]
            if kids and rng.random() < agree:
                tl32[b, j, tree["tokens"][b, rng.choice(kids)]] = tl32[b, j].max() + 1.0
    tl = W.f32_to_bf16_bits(tl32).reshape(tl32.shape) if dtype == "bf16" else tl32
    return tree, tl


def attn_tree_inputs(seed, batch, N, hq, hkv, D, P, ctx):
    inp = W.make_attn_inputs(batch, N, hq, hkv, D, P, ctx, True, seed)
    return inp


@pytest.mark.parametrize("path", [binding.ATTN_TENSOR_CORES, binding.ATTN_CUDA_CORES])
# 132 rows per KV group (one M tile), 244 (two), 17, and 48 (two KV heads per block)
@pytest.mark.parametrize("N,hq,hkv,D,P,ctx,batch", [(33, 32, 8, 128, 16, 4096, 1),
                                                    (61, 32, 8, 128, 16, 2000, 2),
                                                    (17, 8, 8, 64, 64, (100, 900), 4),
                                                    (12, 32, 8, 128, 16, (300, 1500), 3)])
def test_tree_attention(oracle_mod, path, N, hq, hkv, D, P, ctx, batch):
    rng = np.random.default_rng(N * 7 + batch)
    inp = attn_tree_inputs(N + batch, batch, N, hq, hkv, D, P, ctx)
    masks = np.zeros((batch, N), np.uint64)
    for b in range(batch):
        par = [-1] + [int(rng.integers(max(0, j - 6), j)) for j in range(1, N)]
        for j in range(N):
            bits, a = 0, j
            while a >= 0:
                bits |= 1 << a
                a = par[a]
            masks[b, j] = np.uint64(bits)
    q, k, v, pt, kl = (bf16_dev(inp.q), bf16_dev(inp.k_cache), bf16_dev(inp.v_cache),
                       dev(inp.page_table), dev(inp.kv_len))
    tm = dev(masks.view(np.int64))
    out, lse = binding.verify_attention(q, k, v, pt, kl, path=path, tree_mask=tm)
    torch.cuda.synchronize()
    rows = sample_rows(inp, 200, seed=N)
    # every node of the first sequence, head 0
    rows = np.unique(np.concatenate([rows, np.array([[0, j, 0] for j in range(N)], np.int32)]), axis=0)
    o_out, o_lse, _ = oracle_mod.verify_attention(inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                                  inp.kv_len, N, rows=rows, tree_mask=masks)
    compare_attention(out.float().cpu().numpy(), lse.cpu().numpy(), o_out, o_lse, rows)


# tree attention runs on the row-tile tensor-core kernel (or the CUDA-core one); its
# block-causal mode is the reference for a causal mask
@pytest.mark.parametrize("path,causal_path", [
    (binding.ATTN_TENSOR_CORES, binding.ATTN_TENSOR_CORES),
    (binding.ATTN_CUDA_CORES, binding.ATTN_CUDA_CORES)])
def test_causal_mask_reproduces_block_attention(path, causal_path):
    inp = attn_tree_inputs(3, 2, 16, 32, 8, 128, 16, 1000)
    N = 16
    causal = np.array([[(1 << (j + 1)) - 1 for j in range(N)]] * 2, np.uint64)
    args = (bf16_dev(inp.q), bf16_dev(inp.k_cache), bf16_dev(inp.v_cache), dev(inp.page_table),
            dev(inp.kv_len))
    a, la = binding.verify_attention(*args, path=path, tree_mask=dev(causal.view(np.int64)))
    c, lc = binding.verify_attention(*args, path=causal_path)
    torch.cuda.synchronize()
    assert torch.equal(a, c) and torch.equal(la, lc)


def compare_tree_accept(g, o):
    for k in ("path", "num_accepted", "out_tokens", "num_emitted"):
        np.testing.assert_array_equal(g[k], o[k], err_msg=k)


def gpu_accept_tree(tl, tree):
    r = binding.accept_tree(logits_dev(tl), dev(tree["tokens"]), dev(tree["parents"]))
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in r.items()}


@pytest.mark.parametrize("batch,budget,K,G,vocab,dtype", [(1, 32, 32, 16, 128256, "bf16"),
                                                          (1, 60, 32, 16, 151936, "bf16"),
                                                          (8, 32, 8, 8, 32000, "f32"),
                                                          (16, 20, 4, 6, 5000, "bf16"),
                                                          (3, 7, 2, 4, 33, "f32")])
def test_tree_greedy_acceptance(oracle_mod, batch, budget, K, G, vocab, dtype):
    tree, tl = tree_case(oracle_mod, budget + batch, batch, budget, K, G, vocab, dtype)
    g = gpu_accept_tree(tl, tree)
    o = oracle_mod.accept_tree_greedy(tl, tree["tokens"], tree["parents"])
    compare_tree_accept(g, o)


def test_tree_full_chain_and_root_only(oracle_mod):
    # K = 1 makes the tree a chain; sequence 0's target follows it to the end (the longest
    # path, num_accepted = N - 1), sequence 1's root row prefers a token no child has
    # (num_accepted = 0), sequence 2 is a one-node tree
    B, G, V, N = 3, 40, 1000, 33
    inp = W.make_accept_inputs(B, G, V, "f32", 3.0, 1.0, 1.0, seed=5)
    tree = oracle_mod.build_tree(inp.drafter_logits, inp.temperature, inp.block_tokens[:, 0], 1, N - 1)
    assert np.array_equal(tree["parents"][0], np.arange(-1, N - 1))
    tl = np.random.default_rng(5).standard_normal((B, N, V)).astype(np.float32)
    for j in range(N - 1):
        tl[0, j, tree["tokens"][0, j + 1]] = 10.0
    tl[1, 0, (tree["tokens"][1, 1] + 1) % V] = 10.0
    g = gpu_accept_tree(tl, tree)
    o = oracle_mod.accept_tree_greedy(tl, tree["tokens"], tree["parents"])
    compare_tree_accept(g, o)
    assert list(o["num_accepted"][:2]) == [N - 1, 0]
    one = gpu_accept_tree(tl[2:, :1].copy(), {k: tree[k][2:, :1].copy() for k in ("tokens", "parents")})
    assert one["num_accepted"][0] == 0 and one["num_emitted"][0] == 1 + 1
    assert one["out_tokens"][0, 1] == int(np.argmax(tl[2, 0]))


def test_tree_acceptance_flags_bad_sequences(oracle_mod):
    tree, tl = tree_case(oracle_mod, 9, 4, 10, 3, 5, 3000, "f32")
    tree["parents"][1, 5] = 7           # a parent after its child
    tree["tokens"][2, 3] = 3000         # a token outside the vocabulary
    tl[3, 4, 11] = np.nan
    ws = binding.new_workspace(1 << 20)
    r = binding.accept_tree(logits_dev(tl), dev(tree["tokens"]), dev(tree["parents"]), ws=ws)
    torch.cuda.synchronize()
    code, flags = binding.read_device_status(ws)
    assert flags & binding.FLAG_BAD_TREE and flags & binding.FLAG_BAD_TOKEN
    assert flags & binding.FLAG_BAD_LOGITS
    g = {k: v.cpu().numpy() for k, v in r.items()}
    for b in (1, 2, 3):
        assert g["num_accepted"][b] == -1 and g["num_emitted"][b] == 0
        assert np.all(g["out_tokens"][b] == -1) and np.all(g["path"][b] == -1)
    o = oracle_mod.accept_tree_greedy(tl[:1], tree["tokens"][:1], tree["parents"][:1])
    np.testing.assert_array_equal(g["out_tokens"][0], o["out_tokens"][0])


def commit_case(oracle_mod, inp, N, path, na, expect_flags=0):
    k2, v2, kl2 = oracle_mod.compact_tree_kv(inp.k_cache, inp.v_cache, inp.page_table, inp.kv_len, N,
                                             path, na)
    dk, dv, dkl = bf16_dev(inp.k_cache), bf16_dev(inp.v_cache), dev(inp.kv_len)
    ws = binding.new_workspace(1024)
    binding.commit_tree_kv(dk, dv, dev(inp.page_table), dkl, dev(path), dev(na), status_ws=ws)
    torch.cuda.synchronize()
    assert binding.read_device_status(ws)[1] == expect_flags
    np.testing.assert_array_equal(dkl.cpu().numpy(), kl2)
    np.testing.assert_array_equal(dk.view(torch.int16).cpu().numpy().view(np.uint16), k2)
    np.testing.assert_array_equal(dv.view(torch.int16).cpu().numpy().view(np.uint16), v2)


@pytest.mark.parametrize("D,P", [(128, 16), (64, 64)])
def test_tree_commit(oracle_mod, D, P):
    rng = np.random.default_rng(61 + D)
    batch, N = 6, 33
    inp = attn_tree_inputs(61, batch, N, 32, 8, D, P, (40, 300))
    path = np.full((batch, N), -1, np.int32)
    na = np.array([5, -1, 12, 0, 5, 32], np.int32)
    for b in range(batch):
        n = na[b] + 1 if na[b] >= 0 else 0
        if n:
            path[b, :n] = np.concatenate([[0], np.sort(rng.choice(np.arange(1, N), n - 1, replace=False))])
    # a source that is a later position's destination (slot 2 is read by position 1 and
    # written by position 2), and the whole block kept
    path[4, :6] = [0, 2, 3, 4, 5, 7]
    path[5] = np.arange(N)
    commit_case(oracle_mod, inp, N, path, na)


def test_tree_commit_bad_inputs_leave_the_sequence(oracle_mod):
    batch, N = 4, 9
    inp = attn_tree_inputs(62, batch, N, 8, 8, 64, 16, 50)
    path = np.tile(np.arange(N, dtype=np.int32), (batch, 1))
    path[:, 1:4] = [[2, 5, 7]] * batch
    na = np.array([3, 3, 3, 3], np.int32)
    ok = np.array([True, False, False, True])
    path[1, 2] = 1                   # not rising
    inp.page_table[2, :] = 10 ** 6   # a page outside the cache
    expect = oracle_mod.compact_tree_kv(inp.k_cache, inp.v_cache, inp.page_table, inp.kv_len, N,
                                        np.where(ok[:, None], path, -1), np.where(ok, na, -1))
    dk, dv, dkl = bf16_dev(inp.k_cache), bf16_dev(inp.v_cache), dev(inp.kv_len)
    ws = binding.new_workspace(1024)
    binding.commit_tree_kv(dk, dv, dev(inp.page_table), dkl, dev(path), dev(na), status_ws=ws)
    torch.cuda.synchronize()
    flags = binding.read_device_status(ws)[1]
    assert flags == binding.FLAG_BAD_TREE | binding.FLAG_BAD_PAGE
    kl = dkl.cpu().numpy()
    np.testing.assert_array_equal(kl[ok], expect[2][ok])
    np.testing.assert_array_equal(kl[~ok], inp.kv_len[~ok])
    np.testing.assert_array_equal(dk.view(torch.int16).cpu().numpy().view(np.uint16), expect[0])


def test_tree_step_end_to_end(oracle_mod):
    # the tree sampler, tree attention over its nodes, greedy acceptance, then the
    # compaction, all on the GPU: the results match the oracle's chain of the same steps
    batch, budget, K, G, V = 1, 32, 32, 16, 128256
    N = budget + 1
    tree, tl = tree_case(oracle_mod, 71, batch, budget, K, G, V)
    inp_d = W.make_accept_inputs(batch, G, V, "bf16", 3.0, 1.0, 1.0, seed=71)
    gt = gpu_build(inp_d.drafter_logits, inp_d.temperature, inp_d.block_tokens[:, 0], K, N)
    if tree["margin"][0] >= TREE_MARGIN:
        for k in ("tokens", "parents", "depth"):
            np.testing.assert_array_equal(gt[k], tree[k])
        tree["mask"] = gt["mask"].view(np.uint64)
    inp = attn_tree_inputs(71, batch, N, 32, 8, 128, 16, 4096)
    args = (bf16_dev(inp.q), bf16_dev(inp.k_cache), bf16_dev(inp.v_cache), dev(inp.page_table),
            dev(inp.kv_len))
    out, lse = binding.verify_attention(*args, tree_mask=dev(tree["mask"].view(np.int64)))
    g = gpu_accept_tree(tl, tree)
    o = oracle_mod.accept_tree_greedy(tl, tree["tokens"], tree["parents"])
    compare_tree_accept(g, o)
    dk, dv, dkl = args[1], args[2], args[4]
    binding.commit_tree_kv(dk, dv, args[3], dkl, dev(g["path"]), dev(g["num_accepted"]))
    torch.cuda.synchronize()
    k2, v2, kl2 = oracle_mod.compact_tree_kv(inp.k_cache, inp.v_cache, inp.page_table, inp.kv_len,
                                             N, o["path"], o["num_accepted"])
    np.testing.assert_array_equal(dkl.cpu().numpy(), kl2)
    np.testing.assert_array_equal(dk.view(torch.int16).cpu().numpy().view(np.uint16), k2)
    rows = sample_rows(inp, 100, seed=3)
    o_out, o_lse, _ = oracle_mod.verify_attention(inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                                  inp.kv_len, N, rows=rows, tree_mask=tree["mask"])
    compare_attention(out.float().cpu().numpy(), lse.cpu().numpy(), o_out, o_lse, rows)


# ---------------------------------------------------------------------------------
# sampled (T > 0) tree acceptance
# ---------------------------------------------------------------------------------
def random_tree(rng, tl, T, N, branch=3):
    """A tree whose children are distinct tokens drawn from their parent's target row (so
    that acceptance happens), parents chosen among the first nodes with room."""
    V = tl.shape[1]
    par = np.full(N, -1, np.int32)
    tok = np.zeros(N, np.int32)
    tok[0] = rng.integers(V)
    kids = {0: set()}
    for c in range(1, N):
        cands = [u for u in range(c) if len(kids[u]) < branch]
        u = int(cands[min(len(cands) - 1, int(rng.integers(0, min(4, len(cands)))))])
        z = tl[u].astype(np.float64) / (T if T > 0 else 1.0)
        pr = np.exp(z - z.max())
        for t in kids[u]:
            pr[t] = 0.0
        pr /= pr.sum()
        t = int(rng.choice(V, p=pr)) if rng.random() < 0.8 else int(rng.integers(V))
        par[c], tok[c] = u, t
        kids[u].add(t)
        kids[c] = set()
    return tok, par


def compare_tree_sampled(g, o):
    """Bit-exact but for ties: a sequence may differ only where one of the oracle's
    decisions or its final draw lay within TIE_MARGIN of its threshold."""
    from helpers import TIE_MARGIN
    ties = []
    for b in range(len(o["num_accepted"])):
        if o["status"][b] != 0:
            assert g["num_accepted"][b] == -1 and g["num_emitted"][b] == 0, b
            assert np.all(g["out_tokens"][b] == -1) and np.all(g["path"][b] == -1), b
            continue
        same = all(np.array_equal(g[k][b], o[k][b])
                   for k in ("path", "num_accepted", "out_tokens", "num_emitted"))
        if not same:
            fin = o["accept_margin"][b][np.isfinite(o["accept_margin"][b])]
            m = min(fin.min() if fin.size else np.inf, o["sample_margin"][b])
            assert m < TIE_MARGIN, (b, g["out_tokens"][b], o["out_tokens"][b], m)
            ties.append((b, float(m)))
    return ties


def gpu_accept_tree_sampled(tl, tok, par, T=None, u=None):
    r = binding.accept_tree(logits_dev(tl), dev(tok), dev(par),
                            temperature=None if T is None else dev(np.asarray(T, np.float32)),
                            uniforms=None if u is None else dev(np.asarray(u, np.float32)))
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in r.items()}


@pytest.mark.parametrize("V,dtype,B,N", [(128256, "bf16", 4, 33), (32000, "f32", 6, 33),
                                         (1000, "bf16", 16, 17), (65, "f32", 24, 9),
                                         (8193, "bf16", 8, 64)])
def test_sampled_tree_acceptance_matches_oracle(oracle_mod, V, dtype, B, N):
    rng = np.random.default_rng(V + N)
    T = np.resize(np.array([1.0, 0.7, 0.0, 1.3], np.float32), B)
    tl32 = (rng.standard_normal((B, N, V)) * 3.0).astype(np.float32)
    tl = W.f32_to_bf16_bits(tl32) if dtype == "bf16" else tl32
    seen = W.bf16_bits_to_f32(tl) if dtype == "bf16" else tl32
    tok = np.zeros((B, N), np.int32)
    par = np.zeros((B, N), np.int32)
    for b in range(B):
        tok[b], par[b] = random_tree(rng, seen[b], float(T[b]), N)
    if N >= 3:  # a repeated sibling token: the second occurrence has probability 0
        kids = [c for c in range(1, N) if par[0, c] == par[0, 1]]
        if len(kids) >= 2:
            tok[0, kids[1]] = tok[0, kids[0]]
    u = (1.0 - rng.random((B, N))).astype(np.float32)
    g = gpu_accept_tree_sampled(tl, tok, par, T, u)
    o = oracle_mod.accept_tree_sampled(tl, tok, par, T, u)
    assert np.all(o["status"] == 0)
    ties = compare_tree_sampled(g, o)
    assert len(ties) <= max(1, B // 20), ties
    assert np.all(g["num_emitted"] == g["num_accepted"] + 2)
    print(f"V={V} N={N}: mean accepted {g['num_accepted'].mean():.2f}, ties {len(ties)}")


def test_sampled_tree_output_law_chi_square():
    """200,000 GPU verifications of one small tree (V = 4, rows in quarters) against the
    target's own law of the emitted tokens."""
    from scipy import stats
    import test_oracle_tree as OT
    p, tok, par = OT.TREE4_P, OT.TREE4_TOK, OT.TREE4_PAR
    N, V = p.shape
    want = OT.target_tree_law(p, tok, par)
    keys = sorted(want)
    with np.errstate(divide="ignore"):
        logits = np.log(p).astype(np.float32)
    chunk, total = 50_000, 200_000
    counts = dict.fromkeys(keys, 0)
    tl = torch.from_numpy(np.broadcast_to(logits, (chunk, N, V)).copy()).cuda()
    tk = torch.from_numpy(np.broadcast_to(tok, (chunk, N)).copy()).cuda()
    pr = torch.from_numpy(np.broadcast_to(par, (chunk, N)).copy()).cuda()
    T = torch.ones(chunk, dtype=torch.float32, device="cuda")
    for c in range(total // chunk):
        u = binding.philox_uniforms(W.uniform_seed(7000 + c), chunk * N).view(chunk, N)
        r = binding.accept_tree(tl, tk, pr, temperature=T, uniforms=u)
        out, ne = r["out_tokens"].cpu().numpy(), r["num_emitted"].cpu().numpy()
        for b in range(chunk):
            counts[tuple(int(x) for x in out[b, 1:ne[b]])] += 1
    obs = np.array([counts[k] for k in keys], np.float64)
    exp = np.array([want[k] for k in keys]) * total
    assert stats.chisquare(obs, exp).pvalue > 1e-3


def test_sampled_tree_bad_inputs_are_flagged():
    rng = np.random.default_rng(9)
    B, N, V = 6, 5, 300
    tl = rng.standard_normal((B, N, V)).astype(np.float32)
    tok = rng.integers(0, V, (B, N)).astype(np.int32)
    par = np.broadcast_to(np.array([-1, 0, 0, 1, 1], np.int32), (B, N)).copy()
    T = np.ones(B, np.float32)
    tl[1, 2, 7] = np.inf        # +inf in a tempered row
    tl[2, 3, :] = -np.inf       # no finite logit in a tempered row
    tok[3, 4] = V               # token outside the vocabulary
    tl[4, 0, 3] = np.nan        # NaN
    u = (1.0 - rng.random((B, N))).astype(np.float32)
    r = binding.accept_tree(dev(tl), dev(tok), dev(par), temperature=dev(T), uniforms=dev(u))
    torch.cuda.synchronize()
    g = {k: v.cpu().numpy() for k, v in r.items()}
    for b in (1, 2, 3, 4):
        assert g["num_accepted"][b] == -1 and g["num_emitted"][b] == 0
        assert np.all(g["out_tokens"][b] == -1)
    for b in (0, 5):
        assert g["num_emitted"][b] == g["num_accepted"][b] + 2
