"""The C ABI library on a machine without a GPU: it builds for sm_103a, loads, exports
every function include/spec_verify.h declares, and rejects bad arguments on the host
before touching the device."""

import ctypes
import subprocess

import pytest
import torch

from paper_2609_04010_gb300 import binding, build


@pytest.fixture(scope="module")
def lib():
    build.build()
    return binding.lib()


def test_exports_every_declared_function(lib):
    names = binding.declared_functions()
    assert len(names) >= 9
    for n in names:
        assert hasattr(lib, n), f"{n} declared in spec_verify.h but not exported"
    out = subprocess.run(["nm", "-D", "--defined-only", build.LIB], capture_output=True,
                         text=True).stdout
    exported = {l.split()[-1] for l in out.splitlines() if " T " in l}
    assert set(names) <= exported


def test_library_targets_sm103a(lib):
    assert build.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]


def test_status_strings(lib):
    for code, name in binding.STATUS_NAMES.items():
        assert lib.spec_status_string(code).decode() == name


def test_host_side_argument_checks(lib):
    # null arguments are rejected before any CUDA call
    assert lib.spec_verify_attention(None, None, 0, None) == 1
    assert lib.spec_accept_block(None, None, 0, None) == 1
    assert lib.spec_verify_step(None, None, None, 0, None) == 1
    a = binding.AttnArgs(2, 4, 32, 8, 128, 16, 10, 20, 0.0, 0)
    assert lib.spec_verify_attention(ctypes.byref(a), None, 0, None) == 1  # null tensors
    acc = binding.AcceptArgs(2, 4, 1000, 1)
    assert lib.spec_accept_block(ctypes.byref(acc), None, 0, None) == 1
    assert lib.spec_philox_uniforms(1, 0, -1, None, None) == 1
    assert lib.spec_read_device_status(None, None, None) == 1
    assert lib.spec_workspace_init(None, 1024, None) == 1


def _attn(**kw):
    base = dict(batch=2, gamma=4, num_q_heads=32, num_kv_heads=8, head_dim=128, page_size=16,
                max_pages_per_seq=10, num_pages=20, softmax_scale=0.0, path=0)
    base.update(kw)
    a = binding.AttnArgs(**base)
    for f in ("q", "k_cache", "v_cache", "page_table", "kv_len", "out"):
        setattr(a, f, 4096)  # fake aligned addresses: never dereferenced by the checks
    return a


@pytest.mark.parametrize("kw,code", [
    (dict(head_dim=96), 2), (dict(page_size=8), 2), (dict(gamma=65), 2),
    (dict(num_q_heads=30), 1), (dict(batch=0), 1), (dict(path=7), 1), (dict(path=4), 1),
    (dict(softmax_scale=-1.0), 1),
])
def test_attention_shape_limits(lib, kw, code):
    a = _attn(**kw)
    assert lib.spec_verify_attention(ctypes.byref(a), ctypes.c_void_p(4096), 1 << 30, None) == code
    assert lib.spec_workspace_size(ctypes.byref(a), None) == 0


def test_workspace_size_is_host_only_and_grows_with_work(lib):
    small = _attn(batch=1, max_pages_per_seq=4)
    big = _attn(batch=8, max_pages_per_seq=300)
    s, b = lib.spec_workspace_size(ctypes.byref(small), None), \
        lib.spec_workspace_size(ctypes.byref(big), None)
    assert 0 < s <= b
    acc = binding.AcceptArgs(8, 8, 128256, 1)
    for f in ("target_logits", "drafter_logits", "block_tokens", "temperature", "uniforms",
              "num_accepted", "out_tokens", "num_emitted"):
        setattr(acc, f, 4096)
    both = lib.spec_workspace_size(ctypes.byref(big), ctypes.byref(acc))
    assert both > b and both % 256 == 0


def test_misaligned_workspace_rejected(lib):
    a = _attn()
    assert lib.spec_verify_attention(ctypes.byref(a), ctypes.c_void_p(4096 + 16), 1 << 30,
                                     None) == 1


def _accept(**kw):
    base = dict(batch=4, gamma=8, vocab=128256, logits_dtype=1)
    base.update(kw)
    acc = binding.AcceptArgs(**base)
    for f in ("target_logits", "drafter_logits", "block_tokens", "temperature", "uniforms",
              "num_accepted", "out_tokens", "num_emitted"):
        setattr(acc, f, 4096)
    return acc


@pytest.mark.parametrize("max_top_k,code", [(0, 1), (-5, 1), (1025, 2), (1 << 20, 2)])
def test_filter_host_checks(lib, max_top_k, code):
    acc = _accept()
    f = binding.FilterArgs(4096, 4096, max_top_k)
    assert lib.spec_accept_block_filtered(ctypes.byref(acc), ctypes.byref(f),
                                          ctypes.c_void_p(4096), 1 << 30, None) == code
    assert lib.spec_filtered_workspace_size(None, ctypes.byref(acc), ctypes.byref(f)) == 0


def test_filter_null_arguments(lib):
    acc = _accept()
    f = binding.FilterArgs(4096, None, 50)
    assert lib.spec_accept_block_filtered(ctypes.byref(acc), None, ctypes.c_void_p(4096),
                                          1 << 30, None) == 1
    assert lib.spec_accept_block_filtered(ctypes.byref(acc), ctypes.byref(f),
                                          ctypes.c_void_p(4096), 1 << 30, None) == 1
    assert lib.spec_verify_step_filtered(None, None, None, None, 0, None) == 1


def test_filtered_workspace_size_and_too_small(lib):
    acc = _accept()
    f50 = binding.FilterArgs(4096, 4096, 50)
    f1k = binding.FilterArgs(4096, 4096, 1024)
    n50 = lib.spec_filtered_workspace_size(None, ctypes.byref(acc), ctypes.byref(f50))
    n1k = lib.spec_filtered_workspace_size(None, ctypes.byref(acc), ctypes.byref(f1k))
    assert 0 < n50 < n1k and n50 % 256 == 0
    # rows x max_top_k x (4-byte id + 4-byte probability) separates the two sizes
    rows = 4 * (2 * 8 - 1)
    assert n1k - n50 >= rows * (1024 - 50) * 8 - 1024
    both = lib.spec_filtered_workspace_size(ctypes.byref(_attn()), ctypes.byref(acc),
                                            ctypes.byref(f50))
    assert both > n50
    assert lib.spec_accept_block_filtered(ctypes.byref(acc), ctypes.byref(f50),
                                          ctypes.c_void_p(4096), 1024, None) == 3


def _draft(**kw):
    base = dict(batch=4, gamma=8, vocab=128256, logits_dtype=1)
    base.update(kw)
    d = binding.DraftArgs(**base)
    for f in ("drafter_logits", "temperature", "uniforms", "block_tokens"):
        setattr(d, f, 4096)
    return d


@pytest.mark.parametrize("kw,code", [(dict(gamma=65), 2), (dict(batch=0), 1), (dict(vocab=0), 1),
                                     (dict(logits_dtype=5), 1)])
def test_draft_host_checks(lib, kw, code):
    d = _draft(**kw)
    assert lib.spec_sample_block(ctypes.byref(d), None, ctypes.c_void_p(4096), 1 << 30, None) == code
    assert lib.spec_draft_workspace_size(ctypes.byref(d), None) == 0


def test_draft_workspace_and_other_checks(lib):
    d = _draft()
    n = lib.spec_draft_workspace_size(ctypes.byref(d), None)
    f = binding.FilterArgs(4096, 4096, 50)
    nf = lib.spec_draft_workspace_size(ctypes.byref(d), ctypes.byref(f))
    assert n > 0 and nf > 0 and n % 256 == 0
    assert lib.spec_sample_block(None, None, ctypes.c_void_p(4096), 1 << 30, None) == 1
    assert lib.spec_sample_block(ctypes.byref(d), None, ctypes.c_void_p(4096), 512, None) == 3
    assert lib.spec_noise_tokens(1, 0, -1, 10, None, None) == 1
    assert lib.spec_noise_tokens(1, 0, 5, 0, ctypes.c_void_p(4096), None) == 1
    assert lib.spec_commit_kv(None, None) == 1
    c = binding.CommitArgs(4, 8, 16, 10, 4096, 4096, 4096, None, 4096, 100, 1, None)
    assert lib.spec_commit_kv(ctypes.byref(c), None) == 1  # no free list
    c = binding.CommitArgs(4, 8, 16, 10, 4096, 4096, 4096, 4096, 4096, 100, 2, None)
    assert lib.spec_commit_kv(ctypes.byref(c), None) == 1  # reserve must be 0 or 1


def _tree_build(**kw):
    a = dict(batch=2, gamma=16, vocab=32000, logits_dtype=binding.SPEC_BF16, top_k=32,
             num_nodes=33, drafter_logits=4096, temperature=4096, root_tokens=4096, tokens=4096,
             parents=4096, depth=None, tree_mask=None)
    a.update(kw)
    return binding.TreeBuildArgs(**a)


@pytest.mark.parametrize("kw,code", [
    (dict(num_nodes=65), 2), (dict(num_nodes=0), 1), (dict(top_k=0), 1), (dict(gamma=0), 1),
    (dict(logits_dtype=7), 1), (dict(parents=None), 1), (dict(batch=70000), 2),
    (dict(gamma=2, top_k=3, num_nodes=5), 1),        # position 1 holds three nodes only
    (dict(gamma=3, top_k=2, vocab=1, num_nodes=4), 1),  # one candidate per position: a chain of 2
    (dict(gamma=1, num_nodes=2), 1),
])
def test_tree_build_host_checks(lib, kw, code):
    t = _tree_build(**kw)
    assert lib.spec_build_tree(ctypes.byref(t), ctypes.c_void_p(4096), 1 << 30, None) == code
    assert lib.spec_tree_build_workspace_size(ctypes.byref(t)) == 0


def test_tree_workspace_sizes_and_checks(lib):
    for kw in (dict(), dict(gamma=2, top_k=3, num_nodes=4), dict(num_nodes=1, gamma=1),
               dict(gamma=3, top_k=2, vocab=1, num_nodes=3)):
        t = _tree_build(**kw)
        n = lib.spec_tree_build_workspace_size(ctypes.byref(t))
        assert n > 0 and n % 256 == 0
        assert lib.spec_build_tree(ctypes.byref(t), ctypes.c_void_p(4096), 256, None) == 3
        assert lib.spec_build_tree(ctypes.byref(t), ctypes.c_void_p(4097), n, None) == 1
    assert lib.spec_build_tree(None, ctypes.c_void_p(4096), 1 << 30, None) == 1
    a = binding.TreeAcceptArgs(2, 33, 32000, binding.SPEC_BF16, *([4096] * 7))
    n = lib.spec_tree_workspace_size(ctypes.byref(a))
    assert n > 0 and n % 256 == 0
    assert lib.spec_accept_tree(ctypes.byref(a), ctypes.c_void_p(4096), 256, None) == 3
    a.num_nodes = 65
    assert lib.spec_accept_tree(ctypes.byref(a), ctypes.c_void_p(4096), 1 << 30, None) == 2
    a.num_nodes, a.path = 33, None
    assert lib.spec_accept_tree(ctypes.byref(a), ctypes.c_void_p(4096), 1 << 30, None) == 1
    assert lib.spec_tree_workspace_size(ctypes.byref(a)) == 0
    c = binding.TreeCommitArgs(2, 33, 8, 96, 16, 10, 100, *([4096] * 6), None)
    assert lib.spec_commit_tree_kv(ctypes.byref(c), None) == 2  # head_dim 64 or 128
    c.head_dim, c.path = 128, None
    assert lib.spec_commit_tree_kv(ctypes.byref(c), None) == 1
    assert lib.spec_commit_tree_kv(None, None) == 1


def _lm(**kw):
    a = dict(rows=64, hidden=4096, vocab=128256, rows_per_seq=8, hidden_states=4096, weight=4096,
             temperature=4096, tokens=None, row_max=4096, row_sum=4096, row_argmax=4096,
             token_logit=None, logits=None)
    a.update(kw)
    return binding.LmHeadArgs(**a)


@pytest.mark.parametrize("kw,code", [
    (dict(rows=0), 1), (dict(hidden=12), 1), (dict(hidden=4), 1), (dict(vocab=0), 1),
    (dict(rows_per_seq=0), 1), (dict(weight=None), 1), (dict(row_argmax=None), 1),
    (dict(hidden_states=4104), 1), (dict(weight=4100), 1), (dict(vocab=224 * 65536), 2),
])
def test_lm_head_host_checks(lib, kw, code):
    a = _lm(**kw)
    assert lib.spec_lm_head_stats(ctypes.byref(a), ctypes.c_void_p(4096), 1 << 30, None) == code
    assert lib.spec_lm_head_workspace_size(ctypes.byref(a)) == 0


def test_lm_head_workspace(lib):
    a = _lm()
    n = lib.spec_lm_head_workspace_size(ctypes.byref(a))
    # a status header and 16 bytes per row and 224-row vocab tile
    assert n >= 256 + 16 * 64 * ((128256 + 223) // 224) and n % 256 == 0
    assert lib.spec_lm_head_stats(ctypes.byref(a), ctypes.c_void_p(4096), n - 256, None) == 3
    assert lib.spec_lm_head_stats(ctypes.byref(a), ctypes.c_void_p(4097), n, None) == 1
    assert lib.spec_lm_head_stats(None, ctypes.c_void_p(4096), n, None) == 1


def test_fused_step_checks_both_parts_before_any_launch(lib):
    # a valid attention half does not hide a bad acceptance half, nor the reverse
    attn = _attn()
    good = _accept()
    bad_gamma = _accept(gamma=65)
    assert lib.spec_verify_step(ctypes.byref(attn), ctypes.byref(bad_gamma), None, 0, None) == 2
    bad_batch = _accept(batch=0)
    assert lib.spec_verify_step(ctypes.byref(attn), ctypes.byref(bad_batch), None, 0, None) == 1
    bad_attn = _attn(num_kv_heads=3)
    assert lib.spec_verify_step(ctypes.byref(bad_attn), ctypes.byref(good), None, 0, None) == 1
    # both halves valid: the missing workspace is the error
    assert lib.spec_verify_step(ctypes.byref(attn), ctypes.byref(good), None, 0, None) == 1


def _cpu_calls():
    """Every tensor-taking binding call, on small CPU tensors of the right dtypes and
    shapes (B = 2 sequences, gamma 4, vocab 64)."""
    B, G, V, Hq, Hkv, D, P = 2, 4, 64, 8, 2, 64, 16
    bf = lambda *s: torch.zeros(*s, dtype=torch.bfloat16)
    i32 = lambda *s: torch.zeros(*s, dtype=torch.int32)
    f32 = lambda *s: torch.ones(*s, dtype=torch.float32)
    tl, dl = bf(B, G, V), bf(B, G, V)
    tok, T, u = i32(B, G), f32(B), f32(B, G)
    q, kc, vc = bf(B, G, Hq, D), bf(4, Hkv, P, D), bf(4, Hkv, P, D)
    table, kv = i32(B, 2), torch.full((B,), 20, dtype=torch.int32)
    return {
        "verify_attention": lambda: binding.verify_attention(q, kc, vc, table, kv),
        "accept_block": lambda: binding.accept_block(tl, dl, tok, T, u),
        "accept_block_noalloc": lambda: binding.accept_block_noalloc(
            tl, dl, tok, T, u, i32(B), i32(B, G + 1), i32(B)),
        "accept_block_filtered": lambda: binding.accept_block_filtered(
            tl, dl, tok, T, i32(B) + 5, f32(B), u, max_top_k=8),
        "sample_block": lambda: binding.sample_block(dl, T, u),
        "build_tree": lambda: binding.build_tree(dl, T, i32(B), 2, 5),
        "accept_tree": lambda: binding.accept_tree(tl, tok, i32(B, G) - 1),
        "lm_head_stats": lambda: binding.lm_head_stats(bf(8, 64), bf(V, 64), f32(2), 4),
        "commit_kv": lambda: binding.commit_kv(kv, i32(B), table, P, G, i32(8), i32(1)),
        "commit_tree_kv": lambda: binding.commit_tree_kv(kc, vc, table, kv, i32(B, G), i32(B)),
    }


HOST_TENSOR_CALLS = ["accept_block", "accept_block_filtered", "accept_block_noalloc", "accept_tree",
                     "build_tree", "commit_kv", "commit_tree_kv", "lm_head_stats", "sample_block",
                     "verify_attention"]


def test_host_tensor_cases_cover_the_table():
    assert sorted(_cpu_calls()) == HOST_TENSOR_CALLS


@pytest.mark.parametrize("name", HOST_TENSOR_CALLS)
def test_binding_rejects_host_tensors(lib, name):
    # a host pointer must never reach a kernel: every call checks its tensors first
    with pytest.raises(ValueError, match="CUDA tensor"):
        _cpu_calls()[name]()
