"""The timeout path of the bounded waits, made to happen without a GPU fault.

The tensor-core kernels wait on asynchronous copies and tensor-core operations through
mbarriers whose waits are bounded (about 1 s of SM clock): a wait that runs out raises the
block's abort flag, sets SPEC_FLAG_TIMEOUT, drains the block's own copies and MMAs, frees
its tensor memory and returns. The test hooks launch the attention kernel (tensor-core
row tiles) and the fused LM head with their copy producers idle, so that the consumers'
first waits can never complete. Each launch must return, report SPEC_ERR_TIMEOUT through
the workspace status word (once: reading clears it), and leave the context and the
workspace usable: the next product call on the same workspace matches the oracle."""

import time

import numpy as np
import pytest
import torch

from paper_2609_04010_gb300 import binding
from paper_2609_04010_gb300 import workloads as W

from helpers import attn_tensors, bf16_dev, compare_attention, dev

pytestmark = pytest.mark.gpu

SPEC_ERR_TIMEOUT = 6


def read_status(ws):
    code, flags = binding.read_device_status(ws)
    return int(code), int(flags)


@pytest.mark.parametrize("group,gamma", [(4, 8), (4, 16), (8, 32)])
def test_attention_wait_runs_out(oracle_mod, group, gamma):
    # 32 rows per KV group (one M tile, 64-row buffers), 64 (two KV heads per block) and
    # 256 (two M tiles)
    hkv = 2
    inp = W.make_attn_inputs(3, gamma, group * hkv, hkv, 128, 16, (100, 700), True, seed=91 + gamma)
    q, k, v, pt, kl = attn_tensors(inp)
    out = torch.full_like(q, float("nan"))
    lse = torch.empty(q.shape[:3], dtype=torch.float32, device=q.device)
    a = binding.attn_args(q, k, v, pt, kl, out, lse, path=binding.ATTN_TENSOR_CORES)
    ws = binding.new_workspace(binding.workspace_size(a, None))
    t0 = time.time()
    binding.test_attention_wait_timeout_args(a, ws)
    torch.cuda.synchronize()
    took = time.time() - t0
    code, flags = read_status(ws)
    assert code == SPEC_ERR_TIMEOUT and flags & binding.FLAG_TIMEOUT, (code, flags)
    assert read_status(ws) == (0, 0)  # reading cleared it
    assert took < 30.0, took  # the blocks returned after their bounded waits
    # the same context and workspace: the product call matches the oracle
    binding.verify_attention_args(a, ws)
    torch.cuda.synchronize()
    assert read_status(ws) == (0, 0)
    o_out, o_lse, st = oracle_mod.verify_attention(inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                                   inp.kv_len, gamma)
    assert np.all(st == 0)
    compare_attention(out.float().cpu().numpy(), lse.cpu().numpy(), o_out, o_lse)


def test_lm_head_wait_runs_out(oracle_mod):
    R, H, V, rps = 40, 256, 3000, 8
    h, w, T, tok = W.make_lm_inputs(R, H, V, rps, seed=93)
    hd, wd, Td, tokd = bf16_dev(h), bf16_dev(w), dev(T), dev(tok)
    out = dict(row_max=torch.empty(R, dtype=torch.float32, device="cuda"),
               row_sum=torch.empty(R, dtype=torch.float32, device="cuda"),
               row_argmax=torch.empty(R, dtype=torch.int32, device="cuda"),
               token_logit=torch.empty(R, dtype=torch.float32, device="cuda"))
    a = binding.lm_head_args(hd, wd, Td, rps, out, tokd)
    ws = binding.new_workspace(binding.lm_head_workspace_size(a))
    t0 = time.time()
    binding.test_lm_head_wait_timeout_args(a, ws)
    torch.cuda.synchronize()
    took = time.time() - t0
    code, flags = read_status(ws)
    assert code == SPEC_ERR_TIMEOUT and flags & binding.FLAG_TIMEOUT, (code, flags)
    assert read_status(ws) == (0, 0)
    assert took < 30.0, took
    binding.lm_head_stats_args(a, ws)
    torch.cuda.synchronize()
    assert read_status(ws) == (0, 0)
    o = oracle_mod.lm_head_stats(h, w, T, rps, tokens=tok)
    err = 2.0 ** -20 * o["abs_bound"]
    np.testing.assert_array_less(np.abs(out["row_max"].cpu().numpy() - o["row_max"]), err + 1e-30)
    Te = np.array([float(T[r // rps]) if T[r // rps] > 0 else 1.0 for r in range(R)])
    np.testing.assert_array_less(np.abs(out["row_sum"].cpu().numpy() - o["row_sum"]),
                                 o["row_sum"] * (1e-4 + 2 * err / Te))
