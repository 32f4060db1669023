"""Pins of the oracle's block-causal paged GQA attention (CPU only, no GPU).

The verify pass scores the whole block [x^{L+1}, x~] in one causal forward pass while
the prefix stays in the KV cache (Sec. 4.1; Alg. "Lossless Psi-Spec", the verifier
pass).  The oracle is checked against a dense restatement with scipy's softmax, against
closed forms (one key, zero query, identical keys), and against invariances (keys a
query cannot see, physical page order, grouped heads).
"""

import numpy as np
import pytest
from scipy import special

from paper_2609_04010_gb300.workloads import bf16_bits_to_f32, f32_to_bf16_bits, make_attn_inputs


def dense_attention(inp, scale=None):
    """Dense restatement: gather each sequence's keys in logical order, then
    softmax(q k^T * scale) over keys 0 .. ctx + j for block position j."""
    B, G, Hq, D = inp.q.shape
    Hkv, P = inp.num_kv_heads, inp.page_size
    grp = Hq // Hkv
    scale = 1.0 / np.sqrt(D) if scale is None else scale
    q = bf16_bits_to_f32(inp.q).reshape(inp.q.shape).astype(np.float64)
    k = bf16_bits_to_f32(inp.k_cache).reshape(inp.k_cache.shape).astype(np.float64)
    v = bf16_bits_to_f32(inp.v_cache).reshape(inp.v_cache.shape).astype(np.float64)
    out = np.zeros((B, G, Hq, D))
    lse = np.zeros((B, G, Hq))
    for b in range(B):
        L = int(inp.kv_len[b])
        pages = inp.page_table[b, :(L + P - 1) // P]
        kd = k[pages].transpose(1, 0, 2, 3).reshape(Hkv, -1, D)[:, :L]  # [Hkv][L][D]
        vd = v[pages].transpose(1, 0, 2, 3).reshape(Hkv, -1, D)[:, :L]
        ctx = L - G
        for j in range(G):
            n = ctx + j + 1
            for h in range(Hq):
                s = kd[h // grp, :n] @ q[b, j, h] * scale
                out[b, j, h] = special.softmax(s) @ vd[h // grp, :n]
                lse[b, j, h] = special.logsumexp(s)
    return out, lse


def run(oracle_mod, inp, **kw):
    return oracle_mod.verify_attention(inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                       inp.kv_len, inp.gamma, **kw)


CASES = [
    dict(batch=2, gamma=3, num_q_heads=4, num_kv_heads=2, head_dim=16, page_size=4, ctx=(5, 17)),
    dict(batch=3, gamma=5, num_q_heads=8, num_kv_heads=2, head_dim=8, page_size=16, ctx=(0, 40)),
    dict(batch=1, gamma=1, num_q_heads=2, num_kv_heads=2, head_dim=32, page_size=8, ctx=23),
    dict(batch=2, gamma=8, num_q_heads=6, num_kv_heads=1, head_dim=64, page_size=64, ctx=(60, 70)),
]


@pytest.mark.parametrize("case", CASES, ids=[str(i) for i in range(len(CASES))])
def test_matches_dense_restatement(oracle_mod, case):
    inp = make_attn_inputs(seed=3, **case)
    out, lse, st = run(oracle_mod, inp)
    ref, ref_lse = dense_attention(inp)
    assert np.all(st == 0)
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, ref_lse, rtol=1e-13, atol=1e-13)


def test_single_key_returns_its_value(oracle_mod):
    inp = make_attn_inputs(2, 1, 4, 2, 16, 8, 0, seed=1)  # kv_len = 1
    out, lse, _ = run(oracle_mod, inp)
    v = bf16_bits_to_f32(inp.v_cache).reshape(inp.v_cache.shape).astype(np.float64)
    for b in range(2):
        pg = inp.page_table[b, 0]
        for h in range(4):
            np.testing.assert_array_equal(out[b, 0, h], v[pg, h // 2, 0])


def test_zero_query_averages_visible_values(oracle_mod):
    inp = make_attn_inputs(2, 4, 4, 4, 16, 8, (3, 30), seed=2)
    inp.q[...] = 0
    out, lse, _ = run(oracle_mod, inp)
    v = bf16_bits_to_f32(inp.v_cache).reshape(inp.v_cache.shape).astype(np.float64)
    for b in range(2):
        L = int(inp.kv_len[b])
        pages = inp.page_table[b, :(L + 7) // 8]
        vd = v[pages].transpose(1, 0, 2, 3).reshape(4, -1, 16)[:, :L]
        for j in range(4):
            n = L - 4 + j + 1
            np.testing.assert_allclose(lse[b, j], np.log(n), rtol=1e-14)
            for h in range(4):
                np.testing.assert_allclose(out[b, j, h], vd[h, :n].mean(axis=0), atol=1e-13)


def test_identical_keys_average_visible_values(oracle_mod):
    inp = make_attn_inputs(1, 3, 2, 1, 8, 4, 9, seed=4)
    inp.k_cache[...] = inp.k_cache[0, 0, 0]
    out, _, _ = run(oracle_mod, inp)
    zq = make_attn_inputs(1, 3, 2, 1, 8, 4, 9, seed=4)
    zq.q[...] = 0
    ref, _, _ = run(oracle_mod, zq)
    np.testing.assert_allclose(out, ref, atol=1e-13)


def test_keys_a_query_cannot_see_do_not_matter(oracle_mod):
    inp = make_attn_inputs(2, 6, 4, 2, 16, 4, (10, 20), seed=5)
    base, _, _ = run(oracle_mod, inp)
    rng = np.random.default_rng(0)
    for b in range(2):
        L = int(inp.kv_len[b])
        ctx = L - 6
        for pos in range(ctx + 1, inp.page_table.shape[1] * 4):
            if pos // 4 >= (L + 3) // 4:
                break
            pg, slot = inp.page_table[b, pos // 4], pos % 4
            inp.k_cache[pg, :, slot] = f32_to_bf16_bits(rng.standard_normal((2, 16)) * 50).reshape(2, 16)
            inp.v_cache[pg, :, slot] = f32_to_bf16_bits(rng.standard_normal((2, 16)) * 50).reshape(2, 16)
    pert, _, _ = run(oracle_mod, inp)
    # block position 0 sees only the prefix and its own key (position ctx); the
    # perturbed keys start at ctx + 1.
    np.testing.assert_array_equal(pert[:, 0], base[:, 0])
    assert np.abs(pert[:, 1:] - base[:, 1:]).max() > 1e-3


def test_physical_page_order_does_not_matter(oracle_mod):
    inp = make_attn_inputs(3, 4, 4, 2, 16, 8, (5, 40), permute_pages=False, seed=6)
    base, base_lse, _ = run(oracle_mod, inp)
    perm = np.random.default_rng(1).permutation(inp.num_pages)
    inv = np.argsort(perm)
    k2 = inp.k_cache[perm]
    v2 = inp.v_cache[perm]
    pt2 = np.where(inp.page_table >= 0, inv[np.maximum(inp.page_table, 0)], -1).astype(np.int32)
    out, lse, _ = oracle_mod.verify_attention(inp.q, k2, v2, pt2, inp.kv_len, 4)
    np.testing.assert_array_equal(out, base)
    np.testing.assert_array_equal(lse, base_lse)


def test_heads_of_one_group_share_keys(oracle_mod):
    inp = make_attn_inputs(1, 2, 8, 2, 16, 4, 13, seed=7)
    inp.q[:, :, 1] = inp.q[:, :, 0]   # heads 0, 1 in group 0
    inp.q[:, :, 4] = inp.q[:, :, 0]   # head 4 in group 1
    out, _, _ = run(oracle_mod, inp)
    np.testing.assert_array_equal(out[:, :, 1], out[:, :, 0])
    assert np.abs(out[:, :, 4] - out[:, :, 0]).max() > 1e-3


def test_sampled_rows_equal_full_rows(oracle_mod):
    inp = make_attn_inputs(2, 3, 4, 2, 16, 4, (5, 17), seed=8)
    full, full_lse, _ = run(oracle_mod, inp)
    rows = np.array([[0, 0, 3], [1, 2, 0], [1, 1, 2]], np.int32)
    part, part_lse, _ = run(oracle_mod, inp, rows=rows)
    for b, j, h in rows:
        np.testing.assert_array_equal(part[b, j, h], full[b, j, h])
        assert part_lse[b, j, h] == full_lse[b, j, h]
    assert np.isnan(part[0, 1, 0, 0])


def test_bad_pages_and_lengths_are_flagged(oracle_mod):
    inp = make_attn_inputs(4, 2, 2, 1, 8, 4, 9, seed=9)
    inp.page_table[1, 1] = inp.num_pages        # out of range page id
    inp.kv_len[2] = 1                            # shorter than the block
    inp.kv_len[3] = inp.page_table.shape[1] * 4 + 1  # longer than the page table
    out, lse, st = run(oracle_mod, inp)
    assert list(st) == [0, 1, 1, 1]
    for b in (1, 2, 3):
        assert np.all(out[b] == 0) and np.all(np.isneginf(lse[b]))
    assert np.all(np.isfinite(out[0]))
