"""GPU parity of the draft-side steps with the oracle, through the C ABI: sampling the
block tokens from the drafter rows (spec_sample_block, unfiltered and top-k / top-p
filtered), the noise tokens (spec_noise_tokens) and the KV commit (spec_commit_kv).

Tokens must match bit for bit except a draw whose uniform lies within 1e-6 of a CDF step
in the oracle (or, filtered, whose top-p cut lies within 1e-9 of a rounding tie); such
draws are counted as ties. q_tok within 1e-5 relative. Noise tokens and the commit are
integer results: bit-exact."""

import numpy as np
import pytest
import torch

from paper_2609_04010_gb300 import binding
from paper_2609_04010_gb300 import workloads as W

from helpers import DIAG_RTOL, TIE_MARGIN, dev, logits_dev

pytestmark = pytest.mark.gpu


def draft_inputs(batch, gamma, vocab, dtype, temps, seed, sigma=3.0):
    inp = W.make_accept_inputs(batch, gamma, vocab, dtype, sigma, 1.0, temps, seed=seed)
    return inp.drafter_logits, inp.temperature, inp.uniforms


def gpu_sample(dl, T, u, top_k=None, top_p=None, max_top_k=None):
    B = dl.shape[0]
    kw = {}
    if top_k is not None:
        kw = dict(top_k=dev(np.broadcast_to(np.asarray(top_k, np.int32), (B,)).copy()),
                  top_p=dev(np.broadcast_to(np.asarray(top_p, np.float32), (B,)).copy()),
                  max_top_k=max_top_k)
    r = binding.sample_block(logits_dev(dl), dev(T), dev(u), **kw)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in r.items()}


def check(oracle_mod, dl, T, u, top_k=None, top_p=None, max_top_k=None, max_tie_frac=0.01):
    g = gpu_sample(dl, T, u, top_k, top_p, max_top_k)
    o = oracle_mod.sample_block(dl, T, u, top_k=top_k, top_p=top_p)
    B, G = u.shape
    ties = 0
    for b in range(B):
        if o["status"][b] != 0:
            assert np.all(g["block_tokens"][b] == -1), b
            continue
        for j in range(G):
            if g["block_tokens"][b, j] == o["tokens"][b, j]:
                np.testing.assert_allclose(g["q_tok"][b, j], o["q_tok"][b, j], rtol=DIAG_RTOL,
                                           err_msg=f"q_tok b={b} j={j}")
                continue
            assert o["margin"][b, j] < TIE_MARGIN or o["filter_margin"][b, j] < 1e-9, (
                f"b={b} j={j}: GPU {g['block_tokens'][b, j]} oracle {o['tokens'][b, j]}, "
                f"margin {o['margin'][b, j]:.3g}")
            ties += 1
    assert ties <= max(1, int(max_tie_frac * B * G)), ties
    return g, o


@pytest.mark.parametrize("name", ["tiny", "llama8b", "serve64", "long70b"])
def test_named_workloads(oracle_mod, name):
    inp = W.workload(name).accept_inputs(seed=1)
    check(oracle_mod, inp.drafter_logits, inp.temperature, inp.uniforms)


@pytest.mark.parametrize("vocab,dtype", [(1, "f32"), (7, "f32"), (8, "bf16"), (33, "bf16"),
                                         (4095, "bf16"), (8193, "bf16"), (24577, "f32"),
                                         (40000, "f32"), (151936, "bf16")])
def test_vocab_edges(oracle_mod, vocab, dtype):
    dl, T, u = draft_inputs(12, 5, vocab, dtype, [1.0, 0.0, 0.5, 2.0], seed=vocab)
    check(oracle_mod, dl, T, u)


def test_large_batch_without_row_splits(oracle_mod):
    dl, T, u = draft_inputs(160, 8, 32000, "bf16", [1.0, 0.7], seed=5)
    check(oracle_mod, dl, T, u)


@pytest.mark.parametrize("k,tp", [(1, 1.0), (50, 0.95), (200, 0.9), (1024, 1.0), (3, 0.3)])
def test_filtered(oracle_mod, k, tp):
    dl, T, u = draft_inputs(16, 6, 50000, "bf16", [1.0, 0.0, 0.8], seed=k)
    check(oracle_mod, dl, T, u, top_k=k, top_p=tp, max_top_k=1024)


def test_extreme_uniforms_and_masked_rows(oracle_mod):
    dl, T, u = draft_inputs(8, 4, 20000, "bf16", 1.0, seed=6)
    u[0] = np.float32(1.0)                     # the last positive token
    u[1] = np.float32(2.0 ** -24)              # the first positive token
    ninf = np.uint16(0xFF80)
    dl[2, :, :19000] = ninf                    # mass only at the end of the row
    dl[3, 1, 1000:] = ninf                     # mass only at the start
    check(oracle_mod, dl, T, u)
    check(oracle_mod, dl, T, u, top_k=20, top_p=0.9, max_top_k=20)


def test_bad_rows_flag_their_sequence(oracle_mod):
    dl, T, u = draft_inputs(5, 4, 3000, "f32", [1.0, 1.0, 0.0, 1.0, 1.0], seed=7)
    dl[1, 3, 17] = np.nan
    dl[3, 0, :] = -np.inf
    dl[4, 2, 5] = np.inf
    ws = binding.new_workspace(1 << 22)
    r = binding.sample_block(logits_dev(dl), dev(T), dev(u), ws=ws)
    torch.cuda.synchronize()
    code, flags = binding.read_device_status(ws)
    assert flags & binding.FLAG_BAD_LOGITS
    tok = r["block_tokens"].cpu().numpy()
    for b in (1, 3, 4):
        assert np.all(tok[b] == -1)
    o = oracle_mod.sample_block(dl, T, u)
    assert list(o["status"]) == [0, 1, 0, 1, 1]
    np.testing.assert_array_equal(tok[[0, 2]], o["tokens"][[0, 2]])


def test_sampled_drafts_feed_the_verify_step(oracle_mod):
    # The drafts drawn on the GPU are the block tokens of a verify step; the verify step
    # on them matches the oracle's.
    from helpers import compare_accept
    inp = W.workload("llama8b").accept_inputs(seed=2)
    g = gpu_sample(inp.drafter_logits, inp.temperature, inp.uniforms)
    inp.block_tokens[:] = g["block_tokens"]
    r = binding.accept_block(logits_dev(inp.target_logits), logits_dev(inp.drafter_logits),
                             dev(inp.block_tokens), dev(inp.temperature), dev(inp.uniforms))
    torch.cuda.synchronize()
    gv = {k: v.cpu().numpy() for k, v in r.items() if v is not None}
    o = oracle_mod.accept_block(inp.target_logits, inp.drafter_logits, inp.block_tokens,
                                inp.temperature, inp.uniforms)
    compare_accept(gv, o, inp.gamma)


def test_noise_tokens_bit_exact(oracle_mod):
    for seed, n, vocab, offset in [(1, 1, 2, 0), (7, 4097, 128256, 3), (9, 100000, 151936, 12345),
                                   (2**40 + 5, 513, 32000, 2**33)]:
        g = binding.noise_tokens(seed, n, vocab, offset=offset).cpu().numpy()
        words = W.philox_words(seed, n, offset)
        np.testing.assert_array_equal(g, oracle_mod.noise_tokens(words, vocab))


@pytest.mark.parametrize("reserve", [True, False])
def test_commit_matches_oracle(oracle_mod, reserve):
    rng = np.random.default_rng(41 + reserve)
    for trial in range(30):
        B = int(rng.integers(1, 3000)) if trial % 10 == 0 else int(rng.integers(1, 64))
        P, gamma = int(rng.choice([16, 64])), int(rng.integers(1, 33))
        max_pages = int(rng.integers(3, 40))
        if max_pages * P < gamma:
            continue
        ctx = rng.integers(0, max_pages * P - gamma + 1, B)
        kv = (ctx + gamma).astype(np.int32)
        npages = -(-kv // P)
        spare = int(rng.integers(0, 3 * B))
        ids = rng.permutation(int(npages.sum()) + spare).astype(np.int32)
        table = np.full((B, max_pages), -1, np.int32)
        pos = 0
        for b in range(B):
            table[b, :npages[b]] = ids[pos:pos + npages[b]]
            pos += npages[b]
        capacity = len(ids) - (int(rng.integers(0, 3)) if not reserve else 0)
        free = np.zeros(capacity, np.int32)
        count = min(spare, capacity)
        free[:count] = ids[pos:pos + count]
        na = rng.integers(-1, gamma, B).astype(np.int32)
        if trial % 7 == 0:
            na[rng.integers(0, B)] = gamma + 3  # bad input
        new, t, f, c, fl = oracle_mod.commit_kv(kv, na, table, P, gamma, free, count, reserve)
        d_kv, d_table, d_free = dev(kv), dev(table), dev(free)
        d_count = dev(np.array([count], np.int32))
        d_flags = dev(np.zeros(B, np.int32))
        binding.commit_kv(d_kv, dev(na), d_table, P, gamma, d_free, d_count, reserve, d_flags)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(d_kv.cpu().numpy(), new)
        np.testing.assert_array_equal(d_table.cpu().numpy(), t)
        np.testing.assert_array_equal(d_flags.cpu().numpy(), fl)
        assert int(d_count.cpu().numpy()[0]) == c
        np.testing.assert_array_equal(d_free.cpu().numpy()[:c], f[:c])


def test_commit_worked_examples_on_gpu(oracle_mod):
    # the hand-worked cases of the oracle's pins, including a request of zero pages after
    # a refused one (it is served, and the list's top stays at the last grant) and a
    # request that fits only if an earlier refused one is not counted (it is refused)
    cases = [
        (np.array([[10, 11, 12, -1], [20, 21, 22, -1], [30, 31, -1, -1]]), [9, 12, 7], [1, 3, -1],
         4, 4, [40, 41, 42] + [0] * 13, 3),
        (np.array([[1, -1, -1], [2, -1, -1], [3, -1, -1]]), [4, 4, 4], [0, 3, 3], 4, 4, [7, 8, 0], 2),
        (np.array([[1, 2, 3], [4, 5, -1], [6, 7, -1]]), [12, 8, 8], [-1, -1, -1], 4, 4, [9, 0], 1),
        (np.array([[1, -1, -1], [2, -1, -1], [3, 4, -1]]), [4, 4, 8], [3, 3, -1], 4, 4, [5, 0, 0], 1),
        (np.array([[1, 2, -1, -1], [3, 4, -1, -1]]), [8, 8], [7, 0], 4, 8, [9, 0], 1),
    ]
    for table, kv, na, P, G, free, count in cases:
        for reserve in (True, False):
            table = np.asarray(table, np.int32)
            kv, na, free = (np.asarray(x, np.int32) for x in (kv, na, free))
            new, t, f, c, fl = oracle_mod.commit_kv(kv, na, table, P, G, free, count, reserve)
            d_kv, d_table, d_free = dev(kv), dev(table), dev(free)
            d_count, d_flags = dev(np.array([count], np.int32)), dev(np.zeros(len(kv), np.int32))
            binding.commit_kv(d_kv, dev(na), d_table, P, G, d_free, d_count, reserve, d_flags)
            torch.cuda.synchronize()
            np.testing.assert_array_equal(d_kv.cpu().numpy(), new)
            np.testing.assert_array_equal(d_table.cpu().numpy(), t)
            np.testing.assert_array_equal(d_flags.cpu().numpy(), fl)
            assert int(d_count.cpu().numpy()[0]) == c
            np.testing.assert_array_equal(d_free.cpu().numpy()[:c], f[:c])
