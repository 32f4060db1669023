"""The seeded input generator (CPU only): Philox against its published known-answer
vectors, bf16 rounding against torch's, and the shapes and ranges of the workloads."""

import os

import numpy as np
import torch

from paper_2609_04010_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def test_philox_known_answers():
    rows = [l.split() for l in open(GOLDEN) if l.strip() and not l.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        out = W.philox4x32_10(np.array(v[:4], np.uint32), (v[4], v[5]))
        assert [int(x) for x in out] == v[6:]


def test_uniforms_are_in_half_open_unit_interval():
    u = W.philox_uniforms(W.uniform_seed(0), 100000)
    assert u.dtype == np.float32 and u.min() > 0 and u.max() <= 1
    assert abs(u.mean() - 0.5) < 0.005
    # offsets address the same stream
    np.testing.assert_array_equal(W.philox_uniforms(7, 10, offset=5), W.philox_uniforms(7, 15)[5:])


def test_bf16_rounding_matches_torch():
    x = (np.random.default_rng(0).standard_normal(100000) * 10).astype(np.float32)
    x[:4] = [1.00390625, 1.01171875, -2.00390625, 0.0]  # exact ties
    ours = W.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(ours, ref)


def test_accept_inputs_shapes_and_drafts():
    inp = W.make_accept_inputs(3, 4, 1000, "bf16", 3.0, 0.5, [0.0, 1.0, 0.7], seed=1)
    assert inp.target_logits.shape == (3, 4, 1000) and inp.target_logits.dtype == np.uint16
    assert inp.block_tokens.min() >= 0 and inp.block_tokens.max() < 1000
    d = W.bf16_bits_to_f32(inp.drafter_logits).reshape(3, 4, 1000)
    # greedy sequence: drafts are the drafter argmax
    np.testing.assert_array_equal(inp.block_tokens[0], np.argmax(d[0], axis=-1))
    again = W.make_accept_inputs(3, 4, 1000, "bf16", 3.0, 0.5, [0.0, 1.0, 0.7], seed=1)
    np.testing.assert_array_equal(inp.block_tokens, again.block_tokens)
    np.testing.assert_array_equal(inp.uniforms, again.uniforms)


def test_attn_inputs_page_tables():
    inp = W.make_attn_inputs(5, 4, 8, 2, 64, 16, (10, 100), seed=2)
    pages = (inp.kv_len + 15) // 16
    used = np.concatenate([inp.page_table[b, :pages[b]] for b in range(5)])
    assert sorted(used.tolist()) == list(range(inp.num_pages))
    for b in range(5):
        assert np.all(inp.page_table[b, pages[b]:] == -1)
    assert np.all(inp.kv_len >= 14) and np.all(inp.kv_len <= 104)


def test_named_workloads():
    w = W.workload("llama8b")
    assert (w.batch, w.gamma, w.vocab, w.num_q_heads, w.num_kv_heads, w.head_dim) == \
        (8, 8, 128256, 32, 8, 128)
    s = W.workload("sweep_g16_b32_s3_t0")
    assert (s.gamma, s.batch, s.drafter_sigma, s.temperatures) == (16, 32, 3.0, (0.0,))
