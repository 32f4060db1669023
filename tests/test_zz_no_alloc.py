"""spec_accept_block_noalloc, the acceptance entry point for callers that cannot
allocate device memory (its scratch is a fixed device array inside the library).

Collected last on purpose, so that a run stopping at the first failure has already run
every other test. The GPU test calls the entry point twice in a row through the C ABI
and checks each result against spec_accept_block with a caller workspace (the two share
their kernels, so the tokens agree bit for bit) and against the fp64 oracle, within the
acceptance tolerances the other tests use (tokens bit-exact except counted ties)."""

import ctypes

import numpy as np
import pytest
import torch

from paper_2609_04010_gb300 import binding
from paper_2609_04010_gb300 import workloads as W


def test_oversized_batch_is_rejected_without_launch():
    binding.lib()
    # 512 sequences x 127 rows x 32 chunks x 16 bytes is far beyond the fixed 4 MiB array;
    # the size check happens before any device call (none is available here).
    a = binding.AcceptArgs(512, 64, 128256, binding.SPEC_BF16)
    for f in ("target_logits", "drafter_logits", "block_tokens", "temperature", "uniforms",
              "num_accepted", "out_tokens", "num_emitted"):
        setattr(a, f, 4096)
    assert binding.lib().spec_accept_block_noalloc(ctypes.byref(a), None) == 3


def _fake_accept(batch, gamma, vocab, dtype=binding.SPEC_BF16, skip=()):
    a = binding.AcceptArgs(batch, gamma, vocab, dtype)
    for f in ("target_logits", "drafter_logits", "block_tokens", "temperature", "uniforms",
              "num_accepted", "out_tokens", "num_emitted"):
        if f not in skip:
            setattr(a, f, 4096)  # fake aligned addresses: never dereferenced by the checks
    return a


@pytest.mark.parametrize("args,code", [
    ((0, 4, 1000), 1), ((2, 0, 1000), 1), ((2, 4, 0), 1), ((2, 4, 1000, 7), 1),
    ((2, 4, 1000, binding.SPEC_BF16, ("uniforms",)), 1), ((2, 65, 1000), 2),
    ((65536, 1, 1000), 2), ((1, 1, 65536 * 4096 + 1), 2)])
def test_argument_errors_match_the_workspace_entry_point(args, code):
    # the same host check as spec_accept_block, before any device call
    lib = binding.lib()
    a = _fake_accept(*args)
    assert lib.spec_accept_block_noalloc(ctypes.byref(a), None) == code
    assert lib.spec_accept_block(ctypes.byref(a), None, 0, None) == code
    assert lib.spec_accept_block_noalloc(None, None) == 1


@pytest.mark.gpu
def test_matches_workspace_entry_point_twice(oracle_mod):
    from helpers import compare_accept

    def one(inp):
        dev = lambda x: torch.from_numpy(np.ascontiguousarray(x)).cuda()
        bf = lambda x: torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).cuda()
        t = (bf(inp.target_logits), bf(inp.drafter_logits), dev(inp.block_tokens),
             dev(inp.temperature), dev(inp.uniforms))
        ref = binding.accept_block(*t)
        B, G = inp.batch, inp.gamma
        out = dict(num_accepted=torch.full((B,), -5, dtype=torch.int32, device="cuda"),
                   out_tokens=torch.full((B, G + 1), -5, dtype=torch.int32, device="cuda"),
                   num_emitted=torch.full((B,), -5, dtype=torch.int32, device="cuda"),
                   diag=torch.full((B, G, 2), -5.0, dtype=torch.float32, device="cuda"))
        binding.accept_block_noalloc(*t, out["num_accepted"], out["out_tokens"],
                                     out["num_emitted"], out["diag"])
        torch.cuda.synchronize()
        for k in ("num_accepted", "out_tokens", "num_emitted"):
            assert torch.equal(out[k], ref[k]), k
        d_new, d_ref = out["diag"].cpu().numpy(), ref["diag"].cpu().numpy()
        assert np.array_equal(np.isnan(d_new), np.isnan(d_ref))
        ok = ~np.isnan(d_ref)
        np.testing.assert_allclose(d_new[ok], d_ref[ok], rtol=1e-5, atol=0)
        # and against the oracle on the same inputs
        o = oracle_mod.accept_block(inp.target_logits, inp.drafter_logits, inp.block_tokens,
                                    inp.temperature, inp.uniforms)
        g = {k: v.cpu().numpy() for k, v in out.items()}
        ties = compare_accept(g, o, G)
        assert len(ties) <= 1, ties
        assert torch.cuda.current_device() == 0  # the caller's current device is kept

    # two calls in a row on different batches: the second must not see the first's scratch
    one(W.make_accept_inputs(8, 8, 40000, "bf16", 3.0, 1.0, [1.0, 0.0, 0.7], seed=31))
    one(W.make_accept_inputs(5, 16, 128256, "bf16", 3.0, 0.5, [0.0, 1.0], seed=32))
