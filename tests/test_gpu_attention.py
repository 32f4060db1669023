"""GPU parity of block-causal paged GQA verify attention (spec_verify_attention) with
the oracle, through the C ABI: within 1e-2 max-abs on outputs (bf16 inputs, fp32
accumulation, bf16 outputs) and 1e-3 on the log-sum-exp."""

import numpy as np
import pytest
import torch

from paper_2609_04010_gb300 import binding
from paper_2609_04010_gb300 import workloads as W

from helpers import attn_tensors, compare_attention, gpu_attention, sample_rows

pytestmark = pytest.mark.gpu

# the CUDA-core kernel, the row-tile tensor-core kernel (AUTO's choice) and the
# keys-on-lanes tensor-core kernel (where it applies; elsewhere the row-tile one)
PATHS = [binding.ATTN_CUDA_CORES, binding.ATTN_TENSOR_CORES, binding.ATTN_TENSOR_CORES_KEYS_ON_LANES]

SMALL = [
    dict(batch=2, gamma=4, num_q_heads=8, num_kv_heads=8, head_dim=64, page_size=16, ctx=(0, 300)),
    dict(batch=3, gamma=8, num_q_heads=32, num_kv_heads=8, head_dim=128, page_size=16,
         ctx=(1, 700)),
    dict(batch=2, gamma=16, num_q_heads=32, num_kv_heads=8, head_dim=128, page_size=32,
         ctx=(100, 500)),
    dict(batch=2, gamma=32, num_q_heads=64, num_kv_heads=8, head_dim=128, page_size=64,
         ctx=(200, 333)),
    dict(batch=4, gamma=1, num_q_heads=32, num_kv_heads=8, head_dim=128, page_size=16,
         ctx=(0, 1000)),
    dict(batch=1, gamma=3, num_q_heads=6, num_kv_heads=2, head_dim=64, page_size=64, ctx=0),
    dict(batch=2, gamma=64, num_q_heads=8, num_kv_heads=4, head_dim=64, page_size=16,
         ctx=(0, 150)),
    # 512 rows per kv head: two row tiles of two M tiles each
    dict(batch=2, gamma=32, num_q_heads=128, num_kv_heads=8, head_dim=128, page_size=16,
         ctx=(10, 300)),
    # a group that does not divide 128, with two M tiles
    dict(batch=2, gamma=64, num_q_heads=6, num_kv_heads=2, head_dim=128, page_size=32,
         ctx=(5, 200)),
    # keys-on-lanes shapes: group 1 with 64-token pages, 48 rows (not a multiple of 32),
    # group 2 with 64 rows, and contexts shorter than one 128-key tile
    dict(batch=3, gamma=4, num_q_heads=8, num_kv_heads=8, head_dim=128, page_size=64,
         ctx=(0, 700)),
    dict(batch=2, gamma=12, num_q_heads=16, num_kv_heads=4, head_dim=128, page_size=16,
         ctx=(127, 385)),
    dict(batch=5, gamma=32, num_q_heads=16, num_kv_heads=8, head_dim=128, page_size=32,
         ctx=(1, 260)),
    dict(batch=4, gamma=16, num_q_heads=32, num_kv_heads=8, head_dim=128, page_size=16,
         ctx=(0, 100)),
    # two KV heads per block with 64-token pages (32 KB page boxes), head dim 128 and 64
    dict(batch=3, gamma=16, num_q_heads=16, num_kv_heads=4, head_dim=128, page_size=64,
         ctx=(50, 900)),
    dict(batch=2, gamma=10, num_q_heads=32, num_kv_heads=8, head_dim=64, page_size=64,
         ctx=(300, 700)),
]


def oracle_attn(oracle_mod, inp, rows=None):
    return oracle_mod.verify_attention(inp.q, inp.k_cache, inp.v_cache, inp.page_table,
                                       inp.kv_len, inp.gamma, rows=rows)


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("case", range(len(SMALL)))
def test_small_shapes_full(oracle_mod, case, path):
    inp = W.make_attn_inputs(seed=case, **SMALL[case])
    g_out, g_lse = gpu_attention(inp, path)
    o_out, o_lse, st = oracle_attn(oracle_mod, inp)
    assert np.all(st == 0)
    compare_attention(g_out, g_lse, o_out, o_lse)


def random_shape(seed):
    """A seeded random attention problem: GQA group, KV heads, head dim, page size,
    block size and ragged contexts drawn over the ranges the kernels take (up to 512
    query rows per KV head), with spare pages in the pool."""
    rng = np.random.default_rng(1000 + seed)
    group = int(rng.choice([1, 2, 3, 4, 6, 8, 16]))
    hkv = int(rng.choice([1, 2, 4, 8]))
    gamma = int(rng.integers(1, max(2, min(64, 512 // group)) + 1))
    lo = int(rng.integers(0, 900))
    hi = lo + int(rng.integers(0, 700))
    return dict(batch=int(rng.integers(1, 5)), gamma=gamma, num_q_heads=group * hkv,
                num_kv_heads=hkv, head_dim=int(rng.choice([64, 128])),
                page_size=int(rng.choice([16, 32, 64])), ctx=(lo, hi),
                extra_pages=int(rng.integers(0, 8)))


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("seed", range(20))
def test_random_shapes(oracle_mod, seed, path):
    shape = random_shape(seed)
    inp = W.make_attn_inputs(seed=seed, **shape)
    g_out, g_lse = gpu_attention(inp, path)
    o_out, o_lse, st = oracle_attn(oracle_mod, inp)
    assert np.all(st == 0)
    compare_attention(g_out, g_lse, o_out, o_lse)


@pytest.mark.parametrize("name", ["tiny", "llama8b", "serve64", "long70b"])
def test_named_workloads_sampled(oracle_mod, name):
    """Full-size workloads, in the launch configuration the benchmark times (automatic
    kernel choice), on sampled (sequence, position, head) rows."""
    inp = W.workload(name).attn_inputs(seed=0)
    g_out, g_lse = gpu_attention(inp, binding.ATTN_AUTO)
    rows = sample_rows(inp, 48)
    o_out, o_lse, st = oracle_attn(oracle_mod, inp, rows)
    assert np.all(st == 0)
    err, lerr = compare_attention(g_out, g_lse, o_out, o_lse, rows)
    print(f"{name}: max abs err {err:.2e}, lse err {lerr:.2e}")


@pytest.mark.parametrize("name", ["llama8b", "serve64"])
def test_named_workload_every_row(oracle_mod, name):
    """Full-size workloads in the benchmark's launch configuration, every (sequence,
    block position, head) row element-wise against the oracle (2,048 rows at llama8b,
    32,768 at serve64)."""
    inp = W.workload(name).attn_inputs(seed=0)
    g_out, g_lse = gpu_attention(inp, binding.ATTN_AUTO)
    o_out, o_lse, st = oracle_attn(oracle_mod, inp)
    assert np.all(st == 0)
    err, lerr = compare_attention(g_out, g_lse, o_out, o_lse)
    print(f"{name} every row: max abs err {err:.2e}, lse err {lerr:.2e}")


@pytest.mark.parametrize("path", PATHS)
def test_page_order_invariance_bitwise(path):
    inp = W.make_attn_inputs(3, 8, 32, 8, 128, 16, (50, 400), permute_pages=False, seed=11)
    base, base_lse = gpu_attention(inp, path)
    perm = np.random.default_rng(2).permutation(inp.num_pages)
    inv = np.argsort(perm)
    inp.k_cache = inp.k_cache[perm]
    inp.v_cache = inp.v_cache[perm]
    inp.page_table = np.where(inp.page_table >= 0, inv[np.maximum(inp.page_table, 0)],
                              -1).astype(np.int32)
    out, lse = gpu_attention(inp, path)
    np.testing.assert_array_equal(out, base)
    np.testing.assert_array_equal(lse, base_lse)


@pytest.mark.parametrize("head_dim", [64, 128])
@pytest.mark.parametrize("path", PATHS)
def test_bad_pages_and_lengths(oracle_mod, path, head_dim):
    inp = W.make_attn_inputs(4, 4, 8, 2, head_dim, 16, (20, 300), seed=12)
    inp.page_table[1, 2] = inp.num_pages + 5
    inp.kv_len[2] = 2  # shorter than the block
    t = attn_tensors(inp)
    out = torch.empty_like(t[0])
    lse = torch.empty(t[0].shape[:3], dtype=torch.float32, device="cuda")
    a = binding.attn_args(*t, out, lse, path=path)
    ws = binding.new_workspace(binding.workspace_size(attn=a))
    binding.verify_attention_args(a, ws)
    code, flags = binding.read_device_status(ws)
    assert code == 5 and flags == (binding.FLAG_BAD_PAGE | binding.FLAG_BAD_KV_LEN)
    o_out, o_lse, st = oracle_attn(oracle_mod, inp)
    assert list(st) == [0, 1, 1, 0]
    compare_attention(out.float().cpu().numpy(), lse.cpu().numpy(), o_out, o_lse)


@pytest.mark.parametrize("path", PATHS)
def test_garbage_in_unused_slots_is_ignored(oracle_mod, path):
    inp = W.make_attn_inputs(2, 5, 16, 4, 128, 16, (30, 41), seed=13)
    for b in range(2):
        L = int(inp.kv_len[b])
        last = inp.page_table[b, (L - 1) // 16]
        inp.k_cache[last, :, L % 16:] = 0x7FC0  # NaN in the unused tail of the last page
        inp.v_cache[last, :, L % 16:] = 0x7FC0
    g_out, g_lse = gpu_attention(inp, path)
    o_out, o_lse, _ = oracle_attn(oracle_mod, inp)
    compare_attention(g_out, g_lse, o_out, o_lse)


def test_deterministic_repeat():
    inp = W.make_attn_inputs(2, 8, 32, 8, 128, 16, (500, 2000), seed=14)
    t = attn_tensors(inp)
    out1, lse1 = binding.verify_attention(*t)
    out2, lse2 = binding.verify_attention(*t)
    assert torch.equal(out1, out2) and torch.equal(lse1, lse2)
