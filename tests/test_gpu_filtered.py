"""GPU parity of the top-k / top-p filtered acceptance (spec_accept_block_filtered) with
the oracle, through the C ABI, on the same seeded inputs.

The bar is that of the unfiltered path: accepted lengths and emitted tokens bit-exact,
except decisions and draws whose uniform lies within 1e-6 of its threshold in the oracle
(counted as ties); p'_i(t_i), q'_i(t_i) within 1e-5 relative. A sequence whose top-p cut
lies within 1e-9 of a rounding tie in the oracle (filter_margin) may keep a different
set on either side, and is counted as a tie as well."""

import numpy as np
import pytest
import torch

from paper_2609_04010_gb300 import binding
from paper_2609_04010_gb300 import workloads as W

from helpers import accept_tensors, compare_accept, dev

pytestmark = pytest.mark.gpu

FILTER_TIE = 1e-9


def per_sequence(x, B, dtype):
    return np.broadcast_to(np.asarray(x, dtype), (B,)).copy()


def gpu_filtered(inp, top_k, top_p, max_top_k=None, ws=None):
    tl, dl, tok, T, u = accept_tensors(inp)
    B = inp.batch
    r = binding.accept_block_filtered(tl, dl, tok, T, dev(per_sequence(top_k, B, np.int32)),
                                      dev(per_sequence(top_p, B, np.float32)), u,
                                      max_top_k=max_top_k, ws=ws)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in r.items() if v is not None}


def oracle_filtered(oracle_mod, inp, top_k, top_p):
    return oracle_mod.accept_block_filtered(inp.target_logits, inp.drafter_logits,
                                            inp.block_tokens, inp.temperature, top_k, top_p,
                                            inp.uniforms)


def same_outputs(g, o, b):
    return all(np.array_equal(g[k][b], o[k][b]) for k in ("num_accepted", "out_tokens",
                                                          "num_emitted"))


def check(oracle_mod, inp, top_k, top_p, max_tie_frac=0.02, max_top_k=None):
    B = inp.batch
    top_k = per_sequence(top_k, B, np.int32)
    top_p = per_sequence(top_p, B, np.float32)
    g = gpu_filtered(inp, top_k, top_p, max_top_k)
    o = oracle_filtered(oracle_mod, inp, top_k, top_p)
    # a top-p cut on a rounding tie may keep different sets: such a sequence may differ
    # (an exact tie, e.g. two equal top logits under top_p = 0.5, is computed exactly on
    # both sides and must not)
    skip = {b for b in range(B) if o["status"][b] == 0 and o["filter_margin"][b] < FILTER_TIE
            and not same_outputs(g, o, b)}
    ties = compare_accept(g, o, inp.gamma, skip=skip)
    assert len(ties) + len(skip) <= max(1, int(max_tie_frac * B)), (ties, skip)
    ok = o["status"] == 0
    assert np.all(g["num_emitted"][ok] == g["num_accepted"][ok] + 2)
    return g, o


@pytest.mark.parametrize("name", ["llama8b_topk", "serve64_topk"])
def test_named_filtered_workloads(oracle_mod, name):
    wl = W.workload(name)
    inp = wl.accept_inputs(seed=0)
    k, p = wl.filter_params()
    g, o = check(oracle_mod, inp, k, p)
    print(f"{name}: mean accepted {g['num_accepted'].mean():.3f}")


@pytest.mark.parametrize("k,tp", [(1, 1.0), (2, 0.5), (50, 0.95), (50, 1.0), (200, 0.9),
                                  (1024, 0.95), (1024, 1.0), (7, 0.3)])
def test_filter_parameters(oracle_mod, k, tp):
    inp = W.make_accept_inputs(24, 6, 50000, "bf16", 3.0, 1.0, [1.0, 0.7, 1.5], seed=k,
                               draft_top_k=k)
    check(oracle_mod, inp, k, tp, max_top_k=1024)


@pytest.mark.parametrize("vocab,dtype", [(1, "f32"), (7, "f32"), (8, "bf16"), (4095, "bf16"),
                                         (8193, "bf16"), (24577, "f32"), (40000, "f32"),
                                         (151936, "bf16")])
def test_vocab_edges(oracle_mod, vocab, dtype):
    inp = W.make_accept_inputs(12, 5, vocab, dtype, 3.0, 1.0, [1.0, 0.0, 0.5], seed=vocab,
                               draft_top_k=50)
    check(oracle_mod, inp, 50, 0.95, max_tie_frac=0.1, max_top_k=64)


def test_mixed_parameters_and_greedy(oracle_mod):
    B = 32
    inp = W.make_accept_inputs(B, 8, 32000, "bf16", 3.0, 1.0, [1.0, 0.0, 0.8, 1.2], seed=11,
                               draft_top_k=20)
    rng = np.random.default_rng(11)
    ks = rng.integers(1, 100, B).astype(np.int32)
    tps = rng.choice([0.3, 0.8, 0.95, 1.0], B).astype(np.float32)
    g, o = check(oracle_mod, inp, ks, tps, max_top_k=100)
    greedy = inp.temperature == 0
    assert greedy.any() and (~greedy).any()


def test_tied_logits_take_the_exact_path(oracle_mod):
    # Constant rows (every logit ties: the candidates overflow the bounded set and the
    # exact whole-row selection runs) and rows of a few distinct values.
    B, gamma, V = 6, 4, 30000
    inp = W.make_accept_inputs(B, gamma, V, "bf16", 3.0, 1.0, 1.0, seed=12)
    rng = np.random.default_rng(12)
    inp.target_logits[0] = W.f32_to_bf16_bits(np.zeros((gamma, V), np.float32)).reshape(gamma, V)
    inp.drafter_logits[0] = inp.target_logits[0]
    small = rng.integers(0, 4, (gamma, V)).astype(np.float32)
    inp.target_logits[1] = W.f32_to_bf16_bits(small).reshape(gamma, V)
    inp.drafter_logits[1] = W.f32_to_bf16_bits(small + rng.integers(0, 2, (gamma, V))).reshape(gamma, V)
    inp.block_tokens[0] = rng.integers(0, 100, gamma)
    inp.block_tokens[1] = rng.integers(0, V, gamma)
    # top_p chosen off the multiples of 1/k, where a tie of the cumulative sum could fall
    check(oracle_mod, inp, [100, 1000, 50, 50, 3, 1000], [0.555, 0.95, 0.95, 1.0, 0.9, 0.5],
          max_tie_frac=0.0, max_top_k=1000)


def test_k_above_vocab(oracle_mod):
    inp = W.make_accept_inputs(8, 4, 300, "f32", 2.0, 1.0, 1.0, seed=13)
    check(oracle_mod, inp, 1000, 0.9, max_top_k=1024)
    check(oracle_mod, inp, 300, 1.0, max_top_k=300)


def test_bad_filter_parameters_flagged(oracle_mod):
    B = 6
    inp = W.make_accept_inputs(B, 4, 5000, "bf16", 3.0, 1.0, [1.0, 1.0, 1.0, 0.0, 1.0, 1.0],
                               seed=14, draft_top_k=20)
    ks = np.array([20, 0, 20, 0, 65, 20], np.int32)          # 65 > max_top_k = 64
    tps = np.array([0.9, 0.9, 1.5, 0.9, 0.9, np.nan], np.float32)
    ws = binding.new_workspace(1 << 24)
    g = gpu_filtered(inp, ks, tps, max_top_k=64, ws=ws)
    code, flags = binding.read_device_status(ws)
    assert flags & binding.FLAG_BAD_FILTER
    for b in (1, 2, 4, 5):
        assert g["num_accepted"][b] == -1 and g["num_emitted"][b] == 0
        assert np.all(g["out_tokens"][b] == -1)
    # the valid sequences, and the greedy one (whose filter is not read), are unaffected
    o = oracle_filtered(oracle_mod, inp, np.array([20, 20, 20, 20, 20, 20], np.int32),
                        np.full(B, 0.9, np.float32))
    compare_accept(g, o, inp.gamma, skip={1, 2, 4, 5})


def test_bad_logits_flagged(oracle_mod):
    # NaN and +inf in bf16 rows read by the vectorised scan (vocabulary 30,000: a ragged
    # last lane of 48 logits): a NaN in a sampled target row (inside a lane, and the very
    # last logit), +inf in a tempered drafter row, a NaN in a greedy sequence's drafter
    # row (never read) and in its target row (read).
    B, gamma, V = 7, 4, 30000
    T = [1.0, 1.0, 1.0, 1.0, 0.0, 1.0, 0.0]
    inp = W.make_accept_inputs(B, gamma, V, "bf16", 3.0, 1.0, T, seed=16)
    nan, inf = np.uint16(0x7FC0), np.uint16(0x7F80)
    inp.target_logits[1, 3, 17] = nan
    inp.target_logits[2, 0, V - 1] = nan
    inp.drafter_logits[3, 1, 63] = inf
    inp.drafter_logits[4, 2, 5] = nan   # greedy: the drafter row is not read
    inp.target_logits[6, 1, 12345] = nan  # greedy: every target row is read
    ws = binding.new_workspace(1 << 24)
    g = gpu_filtered(inp, 50, 0.95, max_top_k=64, ws=ws)
    code, flags = binding.read_device_status(ws)
    assert flags & binding.FLAG_BAD_LOGITS
    o = oracle_filtered(oracle_mod, inp, np.full(B, 50, np.int32), np.full(B, 0.95, np.float32))
    assert [int(x != 0) for x in o["status"]] == [0, 1, 1, 1, 0, 0, 1]
    for b in (1, 2, 3, 6):
        assert g["num_accepted"][b] == -1 and g["num_emitted"][b] == 0
        assert np.all(g["out_tokens"][b] == -1)
    compare_accept(g, o, inp.gamma, skip={1, 2, 3, 6})


def test_filter_off_matches_unfiltered_entry_point(oracle_mod):
    # k = vocab, top_p = 1: the filtered call must reproduce spec_accept_block
    inp = W.make_accept_inputs(16, 6, 1000, "bf16", 3.0, 1.0, [1.0, 0.0, 0.6], seed=15)
    g = gpu_filtered(inp, 1000, 1.0, max_top_k=1000)
    o = oracle_mod.accept_block(inp.target_logits, inp.drafter_logits, inp.block_tokens,
                                inp.temperature, inp.uniforms)
    compare_accept(g, o, inp.gamma)


def test_deterministic(oracle_mod):
    inp = W.workload("llama8b_topk").accept_inputs(seed=3)
    k, p = W.workload("llama8b_topk").filter_params()
    a = gpu_filtered(inp, k, p)
    b = gpu_filtered(inp, k, p)
    for key in ("num_accepted", "out_tokens", "num_emitted"):
        np.testing.assert_array_equal(a[key], b[key])
