"""GPU tests of the whole verify step and of the support entry points: the fused step
equals its two parts, device Philox equals the generator bit for bit, and the
library loaded is the in-tree sm_103a build."""

import os

import numpy as np
import pytest
import torch

from paper_2609_04010_gb300 import binding, build
from paper_2609_04010_gb300 import workloads as W

from helpers import accept_tensors, attn_tensors, compare_accept, compare_attention, sample_rows

pytestmark = pytest.mark.gpu


def test_loaded_library_is_in_tree():
    binding.lib()
    maps = open("/proc/self/maps").read()
    assert os.path.realpath(build.LIB) in maps


@pytest.mark.parametrize("offset,n", [(0, 1), (0, 1000), (3, 4097), (2 ** 33 + 1, 100)])
def test_philox_matches_generator(offset, n):
    seed = 0x1234_5678_9ABC_DEF0
    dev = binding.philox_uniforms(seed, n, offset).cpu().numpy()
    host = W.philox_uniforms(seed, n, offset)
    np.testing.assert_array_equal(dev.view(np.uint32), host.view(np.uint32))


@pytest.mark.parametrize("temps", [(1.0,), (1.0, 0.0, 0.7)])
def test_large_step(oracle_mod, temps):
    """A step with 381 MB of logits (48 sequences x 31 rows x 128,256 bf16) and 64 query
    rows per KV head, some sequences greedy: the step equals its two parts called
    separately, repeats bit-identically on one workspace (every counter left at zero),
    and agrees with the oracle."""
    B, G, V = 48, 16, 128256
    ai = W.make_attn_inputs(B, G, 32, 8, 128, 16, (100, 600), True, seed=5)
    ci = W.make_accept_inputs(B, G, V, "bf16", 3.0, 1.0, list(temps), seed=6)
    at, ct = attn_tensors(ai), accept_tensors(ci)

    def outputs():
        return (torch.empty_like(at[0]), torch.empty(at[0].shape[:3], dtype=torch.float32, device="cuda"),
                dict(num_accepted=torch.empty(B, dtype=torch.int32, device="cuda"),
                     out_tokens=torch.empty(B, G + 1, dtype=torch.int32, device="cuda"),
                     num_emitted=torch.empty(B, dtype=torch.int32, device="cuda"),
                     diag=torch.empty(B, G, 2, dtype=torch.float32, device="cuda")))

    out, lse, res = outputs()
    a = binding.attn_args(*at, out, lse)
    c = binding.accept_args(*ct, res["num_accepted"], res["out_tokens"], res["num_emitted"],
                            res["diag"])
    ws = binding.new_workspace(binding.workspace_size(a, c))
    binding.verify_step_args(a, c, ws)
    torch.cuda.synchronize()
    assert binding.read_device_status(ws) == (0, 0)
    first = [out.clone(), lse.clone()] + [res[k].clone() for k in res]
    binding.verify_step_args(a, c, ws)
    torch.cuda.synchronize()
    assert binding.read_device_status(ws) == (0, 0)
    again = [out, lse] + [res[k] for k in res]
    for x, y in zip(first, again):
        assert torch.equal(x.nan_to_num(-7), y.nan_to_num(-7))
    part_out, part_lse = binding.verify_attention(*at)
    part_acc = binding.accept_block(*ct)
    assert torch.equal(out, part_out) and torch.equal(lse, part_lse)
    for k in res:
        assert torch.equal(res[k].nan_to_num(-7), part_acc[k].nan_to_num(-7)), k
    n = 8
    o = oracle_mod.accept_block(ci.target_logits[:n], ci.drafter_logits[:n], ci.block_tokens[:n],
                                ci.temperature[:n], ci.uniforms[:n])
    compare_accept({k: v[:n].cpu().numpy() for k, v in res.items()}, o, G)
    rows = sample_rows(ai, 24)
    o_out, o_lse, st = oracle_mod.verify_attention(ai.q, ai.k_cache, ai.v_cache, ai.page_table,
                                                   ai.kv_len, G, rows=rows)
    assert np.all(st == 0)
    compare_attention(out.float().cpu().numpy(), lse.cpu().numpy(), o_out, o_lse, rows)


@pytest.mark.parametrize("name", ["tiny", "llama8b"])
def test_step_equals_parts(oracle_mod, name):
    wl = W.workload(name)
    ai, ci = wl.attn_inputs(seed=0), wl.accept_inputs(seed=0)
    at, ct = attn_tensors(ai), accept_tensors(ci)
    out = torch.empty_like(at[0])
    lse = torch.empty(at[0].shape[:3], dtype=torch.float32, device="cuda")
    B, G = ci.batch, ci.gamma
    res = dict(num_accepted=torch.empty(B, dtype=torch.int32, device="cuda"),
               out_tokens=torch.empty(B, G + 1, dtype=torch.int32, device="cuda"),
               num_emitted=torch.empty(B, dtype=torch.int32, device="cuda"),
               diag=torch.empty(B, G, 2, dtype=torch.float32, device="cuda"))
    a = binding.attn_args(*at, out, lse)
    c = binding.accept_args(*ct, res["num_accepted"], res["out_tokens"], res["num_emitted"],
                            res["diag"])
    ws = binding.new_workspace(binding.workspace_size(a, c))
    binding.verify_step_args(a, c, ws)
    torch.cuda.synchronize()
    assert binding.read_device_status(ws) == (0, 0)
    part_out, part_lse = binding.verify_attention(*at)
    part_acc = binding.accept_block(*ct)
    assert torch.equal(out, part_out) and torch.equal(lse, part_lse)
    for k in res:
        assert torch.equal(res[k].nan_to_num(-7), part_acc[k].nan_to_num(-7)), k
    o = oracle_mod.accept_block(ci.target_logits, ci.drafter_logits, ci.block_tokens,
                                ci.temperature, ci.uniforms)
    compare_accept({k: v.cpu().numpy() for k, v in res.items()}, o, G)
    rows = sample_rows(ai, 16)
    o_out, o_lse, _ = oracle_mod.verify_attention(ai.q, ai.k_cache, ai.v_cache, ai.page_table,
                                                  ai.kv_len, ai.gamma, rows=rows)
    compare_attention(out.float().cpu().numpy(), lse.cpu().numpy(), o_out, o_lse, rows)


def test_workspace_too_small_is_rejected():
    ci = W.make_accept_inputs(2, 4, 1000, "bf16", seed=1)
    ct = accept_tensors(ci)
    r = binding.accept_block(*ct)
    c = binding.accept_args(*ct, r["num_accepted"], r["out_tokens"], r["num_emitted"], r["diag"])
    ws = binding.new_workspace(256)
    with pytest.raises(binding.SpecError) as e:
        binding.accept_block_args(c, ws)
    assert e.value.code == 3


@pytest.mark.parametrize("name,path", [("tiny", binding.ATTN_TENSOR_CORES),
                                       ("llama8b", binding.ATTN_AUTO),
                                       ("tiny", binding.ATTN_CUDA_CORES)])
def test_step_replays_in_a_cuda_graph(name, path):
    """spec_verify_step captured on a stream replays to the eager call's outputs, bit
    for bit, replay after replay (the workspace's tickets reset themselves)."""
    wl = W.workload(name)
    ai, ci = wl.attn_inputs(seed=3), wl.accept_inputs(seed=3)
    at, ct = attn_tensors(ai), accept_tensors(ci)
    B, G = ci.batch, ci.gamma

    def outputs():
        return dict(out=torch.empty_like(at[0]),
                    lse=torch.empty(at[0].shape[:3], dtype=torch.float32, device="cuda"),
                    num_accepted=torch.empty(B, dtype=torch.int32, device="cuda"),
                    out_tokens=torch.empty(B, G + 1, dtype=torch.int32, device="cuda"),
                    num_emitted=torch.empty(B, dtype=torch.int32, device="cuda"),
                    diag=torch.empty(B, G, 2, dtype=torch.float32, device="cuda"))

    def args(r):
        a = binding.attn_args(*at, r["out"], r["lse"], path=path)
        c = binding.accept_args(*ct, r["num_accepted"], r["out_tokens"], r["num_emitted"],
                                r["diag"])
        return a, c

    eager, graphed = outputs(), outputs()
    a0, c0 = args(eager)
    a1, c1 = args(graphed)
    ws0 = binding.new_workspace(binding.workspace_size(a0, c0))
    ws1 = binding.new_workspace(binding.workspace_size(a1, c1))
    binding.verify_step_args(a0, c0, ws0)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        binding.verify_step_args(a1, c1, ws1)
    for _ in range(3):
        for v in graphed.values():
            v.fill_(0)
        g.replay()
        torch.cuda.synchronize()
        assert binding.read_device_status(ws1) == (0, 0)
        for k in eager:
            assert torch.equal(eager[k].nan_to_num(-7), graphed[k].nan_to_num(-7)), k


def test_steps_on_two_streams_are_independent(oracle_mod):
    """Two fused steps issued from one host thread on two streams: each matches the
    oracle, the second finishes while the first stream is still held by a bounded
    spinning kernel (the two steps share no side stream, so neither waits for the
    other), and the calling thread's current device is unchanged."""
    wl = W.workload("tiny")
    ai, ci = wl.attn_inputs(seed=5), wl.accept_inputs(seed=5)
    at, ct = attn_tensors(ai), accept_tensors(ci)
    B, G = ci.batch, ci.gamma

    def outputs():
        return dict(out=torch.empty_like(at[0]),
                    lse=torch.empty(at[0].shape[:3], dtype=torch.float32, device="cuda"),
                    num_accepted=torch.empty(B, dtype=torch.int32, device="cuda"),
                    out_tokens=torch.empty(B, G + 1, dtype=torch.int32, device="cuda"),
                    num_emitted=torch.empty(B, dtype=torch.int32, device="cuda"),
                    diag=torch.empty(B, G, 2, dtype=torch.float32, device="cuda"))

    res = [outputs(), outputs()]
    args = []
    for r in res:
        a = binding.attn_args(*at, r["out"], r["lse"])
        c = binding.accept_args(*ct, r["num_accepted"], r["out_tokens"], r["num_emitted"],
                                r["diag"])
        args.append((a, c, binding.new_workspace(binding.workspace_size(a, c))))
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    dev_before = torch.cuda.current_device()
    for (a, c, ws), s in zip(args, (s1, s2)):  # first calls make each stream's side stream
        binding.verify_step_args(a, c, ws, stream=s)
    torch.cuda.synchronize()
    with torch.cuda.stream(s1):
        torch.cuda._sleep(1_000_000_000)  # about half a second of clock cycles on s1
    binding.verify_step_args(*args[0], stream=s1)
    binding.verify_step_args(*args[1], stream=s2)
    s2.synchronize()
    first_still_busy = not s1.query()
    s1.synchronize()
    assert first_still_busy
    assert torch.cuda.current_device() == dev_before
    o = oracle_mod.accept_block(ci.target_logits, ci.drafter_logits, ci.block_tokens,
                                ci.temperature, ci.uniforms)
    o_out, o_lse, _ = oracle_mod.verify_attention(ai.q, ai.k_cache, ai.v_cache, ai.page_table,
                                                  ai.kv_len, ai.gamma)
    for (a, c, ws), r in zip(args, res):
        assert binding.read_device_status(ws) == (0, 0)
        compare_accept({k: v.cpu().numpy() for k, v in r.items() if k not in ("out", "lse")},
                       o, G)
        compare_attention(r["out"].float().cpu().numpy(), r["lse"].cpu().numpy(), o_out, o_lse)
