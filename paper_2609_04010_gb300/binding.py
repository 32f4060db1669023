"""ctypes binding of libspecverify (include/spec_verify.h).

Argument marshalling only: torch tensors (device memory) are checked for dtype, shape
and contiguity, and their pointers go into the C structs; every step of the verify
step runs in the library's CUDA kernels on the current torch stream. The library must
exist (``python -m paper_2609_04010_gb300.build``); there is no fallback.
"""

from __future__ import annotations

import ctypes
import os
import re
import threading
from typing import Dict, Optional

import torch

from . import build as _build

_lock = threading.Lock()
_lib = None

SPEC_OK = 0
STATUS_NAMES = {0: "SPEC_OK", 1: "SPEC_ERR_INVALID_ARGUMENT", 2: "SPEC_ERR_UNSUPPORTED",
                3: "SPEC_ERR_WORKSPACE_TOO_SMALL", 4: "SPEC_ERR_CUDA", 5: "SPEC_ERR_DEVICE_INPUT",
                6: "SPEC_ERR_TIMEOUT"}
SPEC_F32, SPEC_BF16 = 0, 1
ATTN_AUTO, ATTN_CUDA_CORES, ATTN_TENSOR_CORES, ATTN_TENSOR_CORES_KEYS_ON_LANES = 0, 1, 2, 3
FLAG_BAD_TOKEN, FLAG_BAD_LOGITS, FLAG_BAD_PAGE, FLAG_BAD_KV_LEN, FLAG_TIMEOUT = 1, 2, 4, 8, 16
FLAG_BAD_FILTER = 32
FLAG_BAD_TREE = 64
FILTER_MAX_TOP_K = 1024


class SpecError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: {STATUS_NAMES.get(code, code)}")
        self.code = code


class AttnArgs(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("gamma", ctypes.c_int32),
                ("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("page_size", ctypes.c_int32),
                ("max_pages_per_seq", ctypes.c_int32), ("num_pages", ctypes.c_int32),
                ("softmax_scale", ctypes.c_float), ("path", ctypes.c_int32),
                ("q", ctypes.c_void_p), ("k_cache", ctypes.c_void_p),
                ("v_cache", ctypes.c_void_p), ("page_table", ctypes.c_void_p),
                ("kv_len", ctypes.c_void_p), ("out", ctypes.c_void_p), ("lse", ctypes.c_void_p),
                ("tree_mask", ctypes.c_void_p)]


class AcceptArgs(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("gamma", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("logits_dtype", ctypes.c_int32), ("target_logits", ctypes.c_void_p),
                ("drafter_logits", ctypes.c_void_p), ("block_tokens", ctypes.c_void_p),
                ("temperature", ctypes.c_void_p), ("uniforms", ctypes.c_void_p),
                ("num_accepted", ctypes.c_void_p), ("out_tokens", ctypes.c_void_p),
                ("num_emitted", ctypes.c_void_p), ("diag", ctypes.c_void_p)]


class FilterArgs(ctypes.Structure):
    _fields_ = [("top_k", ctypes.c_void_p), ("top_p", ctypes.c_void_p),
                ("max_top_k", ctypes.c_int32)]


class DraftArgs(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("gamma", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("logits_dtype", ctypes.c_int32), ("drafter_logits", ctypes.c_void_p),
                ("temperature", ctypes.c_void_p), ("uniforms", ctypes.c_void_p),
                ("block_tokens", ctypes.c_void_p), ("q_tok", ctypes.c_void_p)]


class CommitArgs(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("gamma", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("max_pages_per_seq", ctypes.c_int32),
                ("kv_len", ctypes.c_void_p), ("num_accepted", ctypes.c_void_p),
                ("page_table", ctypes.c_void_p), ("free_pages", ctypes.c_void_p),
                ("free_count", ctypes.c_void_p), ("free_capacity", ctypes.c_int32),
                ("reserve", ctypes.c_int32), ("flags", ctypes.c_void_p)]


class TreeAcceptArgs(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("num_nodes", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("logits_dtype", ctypes.c_int32),
                ("target_logits", ctypes.c_void_p), ("tokens", ctypes.c_void_p),
                ("parents", ctypes.c_void_p), ("path", ctypes.c_void_p),
                ("num_accepted", ctypes.c_void_p), ("out_tokens", ctypes.c_void_p),
                ("num_emitted", ctypes.c_void_p), ("temperature", ctypes.c_void_p),
                ("uniforms", ctypes.c_void_p)]


class TreeCommitArgs(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("num_nodes", ctypes.c_int32),
                ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("max_pages_per_seq", ctypes.c_int32),
                ("num_pages", ctypes.c_int32), ("k_cache", ctypes.c_void_p),
                ("v_cache", ctypes.c_void_p), ("page_table", ctypes.c_void_p),
                ("kv_len", ctypes.c_void_p), ("path", ctypes.c_void_p),
                ("num_accepted", ctypes.c_void_p), ("status", ctypes.c_void_p)]


class TreeBuildArgs(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("gamma", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("logits_dtype", ctypes.c_int32), ("top_k", ctypes.c_int32),
                ("num_nodes", ctypes.c_int32), ("drafter_logits", ctypes.c_void_p),
                ("temperature", ctypes.c_void_p), ("root_tokens", ctypes.c_void_p),
                ("tokens", ctypes.c_void_p), ("parents", ctypes.c_void_p),
                ("depth", ctypes.c_void_p), ("tree_mask", ctypes.c_void_p)]


class LmHeadArgs(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int32), ("hidden", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("rows_per_seq", ctypes.c_int32), ("hidden_states", ctypes.c_void_p),
                ("weight", ctypes.c_void_p), ("temperature", ctypes.c_void_p),
                ("tokens", ctypes.c_void_p), ("row_max", ctypes.c_void_p),
                ("row_sum", ctypes.c_void_p), ("row_argmax", ctypes.c_void_p),
                ("token_logit", ctypes.c_void_p), ("logits", ctypes.c_void_p)]


HEADER = os.path.join(_build.ROOT, "include", "spec_verify.h")


def declared_functions():
    """Names of the functions include/spec_verify.h declares."""
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(spec_[a-z0-9_]+)\s*\(", text)))


def lib(build_if_missing: bool = True):
    """The loaded library (built first if it is missing and the toolkit is present)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(_build.LIB):
                if not build_if_missing:
                    raise RuntimeError("libspecverify.so is not built")
                _build.build()
            L = ctypes.CDLL(_build.LIB)
            P, i32, i64, u64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64
            L.spec_workspace_size.argtypes = [P, P]
            L.spec_workspace_size.restype = ctypes.c_size_t
            L.spec_workspace_init.argtypes = [P, ctypes.c_size_t, P]
            for f in ("spec_verify_attention", "spec_accept_block"):
                getattr(L, f).argtypes = [P, P, ctypes.c_size_t, P]
            L.spec_verify_step.argtypes = [P, P, P, ctypes.c_size_t, P]
            L.spec_philox_uniforms.argtypes = [u64, u64, i64, P, P]
            L.spec_read_device_status.argtypes = [P, P, ctypes.POINTER(ctypes.c_uint32)]
            L.spec_status_string.argtypes = [ctypes.c_int]
            L.spec_status_string.restype = ctypes.c_char_p
            L.spec_attn_tensor_core_min_rows.restype = i32
            L.spec_accept_block_noalloc.argtypes = [P, P]
            L.spec_accept_block_noalloc.restype = ctypes.c_int
            L.spec_filtered_workspace_size.argtypes = [P, P, P]
            L.spec_filtered_workspace_size.restype = ctypes.c_size_t
            L.spec_accept_block_filtered.argtypes = [P, P, P, ctypes.c_size_t, P]
            L.spec_accept_block_filtered.restype = ctypes.c_int
            L.spec_verify_step_filtered.argtypes = [P, P, P, P, ctypes.c_size_t, P]
            L.spec_verify_step_filtered.restype = ctypes.c_int
            L.spec_draft_workspace_size.argtypes = [P, P]
            L.spec_draft_workspace_size.restype = ctypes.c_size_t
            L.spec_sample_block.argtypes = [P, P, P, ctypes.c_size_t, P]
            L.spec_sample_block.restype = ctypes.c_int
            L.spec_noise_tokens.argtypes = [u64, u64, i64, i32, P, P]
            L.spec_noise_tokens.restype = ctypes.c_int
            L.spec_commit_kv.argtypes = [P, P]
            L.spec_commit_kv.restype = ctypes.c_int
            L.spec_tree_workspace_size.argtypes = [P]
            L.spec_tree_workspace_size.restype = ctypes.c_size_t
            L.spec_accept_tree.argtypes = [P, P, ctypes.c_size_t, P]
            L.spec_accept_tree.restype = ctypes.c_int
            L.spec_commit_tree_kv.argtypes = [P, P]
            L.spec_commit_tree_kv.restype = ctypes.c_int
            L.spec_lm_head_workspace_size.argtypes = [P]
            L.spec_lm_head_workspace_size.restype = ctypes.c_size_t
            L.spec_lm_head_stats.argtypes = [P, P, ctypes.c_size_t, P]
            L.spec_lm_head_stats.restype = ctypes.c_int
            L.spec_tree_build_workspace_size.argtypes = [P]
            L.spec_tree_build_workspace_size.restype = ctypes.c_size_t
            L.spec_build_tree.argtypes = [P, P, ctypes.c_size_t, P]
            L.spec_build_tree.restype = ctypes.c_int
            for f in ("spec_test_attention_wait_timeout", "spec_test_lm_head_wait_timeout"):
                getattr(L, f).argtypes = [P, P, ctypes.c_size_t, P]
                getattr(L, f).restype = ctypes.c_int
            for f in ("spec_workspace_init", "spec_verify_attention", "spec_accept_block",
                      "spec_verify_step", "spec_philox_uniforms", "spec_read_device_status"):
                getattr(L, f).restype = ctypes.c_int
            _lib = L
    return _lib


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _check(t: torch.Tensor, name: str, dtype, shape=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous CUDA tensor")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")


def _raise(code: int, what: str):
    if code != SPEC_OK:
        raise SpecError(code, what)


def attn_args(q, k_cache, v_cache, page_table, kv_len, out, lse=None, softmax_scale=0.0,
              path=ATTN_AUTO, tree_mask=None) -> AttnArgs:
    B, G, Hq, D = q.shape
    num_pages, Hkv, P, D2 = k_cache.shape
    _check(q, "q", torch.bfloat16)
    _check(k_cache, "k_cache", torch.bfloat16)
    _check(v_cache, "v_cache", torch.bfloat16, k_cache.shape)
    _check(page_table, "page_table", torch.int32)
    _check(kv_len, "kv_len", torch.int32, (B,))
    _check(out, "out", torch.bfloat16, q.shape)
    if lse is not None:
        _check(lse, "lse", torch.float32, (B, G, Hq))
    if tree_mask is not None:
        _check(tree_mask, "tree_mask", torch.int64, (B, G))
    if D2 != D or page_table.dim() != 2 or page_table.shape[0] != B:
        raise ValueError("inconsistent attention shapes")
    return AttnArgs(B, G, Hq, Hkv, D, P, page_table.shape[1], num_pages, float(softmax_scale),
                    int(path), q.data_ptr(), k_cache.data_ptr(), v_cache.data_ptr(),
                    page_table.data_ptr(), kv_len.data_ptr(), out.data_ptr(),
                    None if lse is None else lse.data_ptr(),
                    None if tree_mask is None else tree_mask.data_ptr())


def accept_args(target_logits, drafter_logits, block_tokens, temperature, uniforms, num_accepted,
                out_tokens, num_emitted, diag=None) -> AcceptArgs:
    B, G, V = target_logits.shape
    if target_logits.dtype == torch.bfloat16:
        dt = SPEC_BF16
    elif target_logits.dtype == torch.float32:
        dt = SPEC_F32
    else:
        raise TypeError("logits must be bfloat16 or float32")
    _check(target_logits, "target_logits", target_logits.dtype)
    _check(drafter_logits, "drafter_logits", target_logits.dtype, target_logits.shape)
    _check(block_tokens, "block_tokens", torch.int32, (B, G))
    _check(temperature, "temperature", torch.float32, (B,))
    _check(uniforms, "uniforms", torch.float32, (B, G))
    _check(num_accepted, "num_accepted", torch.int32, (B,))
    _check(out_tokens, "out_tokens", torch.int32, (B, G + 1))
    _check(num_emitted, "num_emitted", torch.int32, (B,))
    if diag is not None:
        _check(diag, "diag", torch.float32, (B, G, 2))
    return AcceptArgs(B, G, V, dt, target_logits.data_ptr(), drafter_logits.data_ptr(),
                      block_tokens.data_ptr(), temperature.data_ptr(), uniforms.data_ptr(),
                      num_accepted.data_ptr(), out_tokens.data_ptr(), num_emitted.data_ptr(),
                      None if diag is None else diag.data_ptr())


def workspace_size(attn: Optional[AttnArgs] = None, accept: Optional[AcceptArgs] = None) -> int:
    n = lib().spec_workspace_size(None if attn is None else ctypes.byref(attn),
                                  None if accept is None else ctypes.byref(accept))
    if n == 0:
        raise SpecError(1, "spec_workspace_size")
    return int(n)


def new_workspace(nbytes: int, device=None) -> torch.Tensor:
    """A zero-filled workspace tensor (torch's allocator is 512-byte aligned)."""
    return torch.zeros(int(nbytes), dtype=torch.uint8, device=device or "cuda")


def verify_attention_args(attn: AttnArgs, ws: torch.Tensor, stream=None):
    _raise(lib().spec_verify_attention(ctypes.byref(attn), _ptr(ws), ws.numel(), _stream(stream)),
           "spec_verify_attention")


def test_attention_wait_timeout_args(attn: AttnArgs, ws: torch.Tensor, stream=None):
    """Test hook: spec_verify_attention on the tensor-core row-tile path with its copy
    producers idle, so that the kernel's bounded waits run out (about 1 s) and it returns
    with SPEC_FLAG_TIMEOUT set."""
    _raise(lib().spec_test_attention_wait_timeout(ctypes.byref(attn), _ptr(ws), ws.numel(),
                                                  _stream(stream)), "spec_test_attention_wait_timeout")


def accept_block_args(acc: AcceptArgs, ws: torch.Tensor, stream=None):
    _raise(lib().spec_accept_block(ctypes.byref(acc), _ptr(ws), ws.numel(), _stream(stream)),
           "spec_accept_block")


def verify_step_args(attn: Optional[AttnArgs], acc: Optional[AcceptArgs], ws: torch.Tensor,
                     stream=None):
    _raise(lib().spec_verify_step(None if attn is None else ctypes.byref(attn),
                                  None if acc is None else ctypes.byref(acc), _ptr(ws),
                                  ws.numel(), _stream(stream)), "spec_verify_step")


def verify_attention(q, k_cache, v_cache, page_table, kv_len, softmax_scale=0.0, path=ATTN_AUTO,
                     want_lse=True, ws=None, stream=None, tree_mask=None):
    """Block-causal (or, with tree_mask, tree) paged GQA verify attention. Returns
    (out bf16, lse fp32 or None). tree_mask: int64 [batch][gamma] bit sets."""
    out = torch.empty_like(q)
    lse = torch.empty(q.shape[:3], dtype=torch.float32, device=q.device) if want_lse else None
    a = attn_args(q, k_cache, v_cache, page_table, kv_len, out, lse, softmax_scale, path, tree_mask)
    if ws is None:
        ws = new_workspace(workspace_size(attn=a), q.device)
    verify_attention_args(a, ws, stream)
    return out, lse


def accept_block(target_logits, drafter_logits, block_tokens, temperature, uniforms,
                 want_diag=True, ws=None, stream=None) -> Dict[str, torch.Tensor]:
    """Lossless acceptance over a batch. Returns num_accepted, out_tokens, num_emitted, diag."""
    B, G, _ = target_logits.shape
    dev = target_logits.device
    res = dict(num_accepted=torch.empty(B, dtype=torch.int32, device=dev),
               out_tokens=torch.empty(B, G + 1, dtype=torch.int32, device=dev),
               num_emitted=torch.empty(B, dtype=torch.int32, device=dev),
               diag=torch.empty(B, G, 2, dtype=torch.float32, device=dev) if want_diag else None)
    a = accept_args(target_logits, drafter_logits, block_tokens, temperature, uniforms,
                    res["num_accepted"], res["out_tokens"], res["num_emitted"], res["diag"])
    if ws is None:
        ws = new_workspace(workspace_size(accept=a), dev)
    accept_block_args(a, ws, stream)
    return res


def accept_block_noalloc(target_logits, drafter_logits, block_tokens, temperature, uniforms,
                         num_accepted, out_tokens, num_emitted, diag=None, stream=None):
    """spec_accept_block_noalloc: the acceptance step with the library's fixed scratch
    array instead of a caller workspace (for callers that cannot allocate device memory;
    the outputs are the caller's tensors). Calls that overlap on the GPU race."""
    a = accept_args(target_logits, drafter_logits, block_tokens, temperature, uniforms,
                    num_accepted, out_tokens, num_emitted, diag)
    _raise(lib().spec_accept_block_noalloc(ctypes.byref(a), _stream(stream)),
           "spec_accept_block_noalloc")


def filter_args(top_k, top_p, batch: int, max_top_k: Optional[int] = None) -> FilterArgs:
    """spec_filter_args_t over int32 top_k [batch] and fp32 top_p [batch] device tensors.

    max_top_k defaults to FILTER_MAX_TOP_K (it sizes the workspace)."""
    _check(top_k, "top_k", torch.int32, (batch,))
    _check(top_p, "top_p", torch.float32, (batch,))
    return FilterArgs(top_k.data_ptr(), top_p.data_ptr(),
                      int(FILTER_MAX_TOP_K if max_top_k is None else max_top_k))


def filtered_workspace_size(accept: AcceptArgs, filt: FilterArgs,
                            attn: Optional[AttnArgs] = None) -> int:
    n = lib().spec_filtered_workspace_size(None if attn is None else ctypes.byref(attn),
                                           ctypes.byref(accept), ctypes.byref(filt))
    if n == 0:
        raise SpecError(1, "spec_filtered_workspace_size")
    return int(n)


def verify_step_filtered_args(attn: Optional[AttnArgs], acc: AcceptArgs, filt: FilterArgs,
                              ws: torch.Tensor, stream=None):
    _raise(lib().spec_verify_step_filtered(None if attn is None else ctypes.byref(attn),
                                           ctypes.byref(acc), ctypes.byref(filt), _ptr(ws),
                                           ws.numel(), _stream(stream)),
           "spec_verify_step_filtered")


def accept_block_filtered_args(acc: AcceptArgs, filt: FilterArgs, ws: torch.Tensor, stream=None):
    _raise(lib().spec_accept_block_filtered(ctypes.byref(acc), ctypes.byref(filt), _ptr(ws),
                                            ws.numel(), _stream(stream)),
           "spec_accept_block_filtered")


def accept_block_filtered(target_logits, drafter_logits, block_tokens, temperature, top_k, top_p,
                          uniforms, max_top_k: Optional[int] = None, want_diag=True, ws=None,
                          stream=None) -> Dict[str, torch.Tensor]:
    """Top-k / top-p filtered lossless acceptance over a batch (spec_accept_block_filtered).

    top_k: int32 [batch], top_p: fp32 [batch] device tensors. Returns num_accepted,
    out_tokens, num_emitted, diag."""
    B, G, _ = target_logits.shape
    dev = target_logits.device
    res = dict(num_accepted=torch.empty(B, dtype=torch.int32, device=dev),
               out_tokens=torch.empty(B, G + 1, dtype=torch.int32, device=dev),
               num_emitted=torch.empty(B, dtype=torch.int32, device=dev),
               diag=torch.empty(B, G, 2, dtype=torch.float32, device=dev) if want_diag else None)
    a = accept_args(target_logits, drafter_logits, block_tokens, temperature, uniforms,
                    res["num_accepted"], res["out_tokens"], res["num_emitted"], res["diag"])
    f = filter_args(top_k, top_p, B, max_top_k)
    if ws is None:
        ws = new_workspace(filtered_workspace_size(a, f), dev)
    accept_block_filtered_args(a, f, ws, stream)
    return res


def draft_args(drafter_logits, temperature, uniforms, block_tokens, q_tok=None) -> DraftArgs:
    B, G, V = drafter_logits.shape
    if drafter_logits.dtype == torch.bfloat16:
        dt = SPEC_BF16
    elif drafter_logits.dtype == torch.float32:
        dt = SPEC_F32
    else:
        raise TypeError("logits must be bfloat16 or float32")
    _check(drafter_logits, "drafter_logits", drafter_logits.dtype)
    _check(temperature, "temperature", torch.float32, (B,))
    _check(uniforms, "uniforms", torch.float32, (B, G))
    _check(block_tokens, "block_tokens", torch.int32, (B, G))
    if q_tok is not None:
        _check(q_tok, "q_tok", torch.float32, (B, G))
    return DraftArgs(B, G, V, dt, drafter_logits.data_ptr(), temperature.data_ptr(),
                     uniforms.data_ptr(), block_tokens.data_ptr(),
                     None if q_tok is None else q_tok.data_ptr())


def draft_workspace_size(d: DraftArgs, filt: Optional[FilterArgs] = None) -> int:
    n = lib().spec_draft_workspace_size(ctypes.byref(d), None if filt is None else ctypes.byref(filt))
    if n == 0:
        raise SpecError(1, "spec_draft_workspace_size")
    return int(n)


def sample_block_args(d: DraftArgs, filt: Optional[FilterArgs], ws: torch.Tensor, stream=None):
    _raise(lib().spec_sample_block(ctypes.byref(d), None if filt is None else ctypes.byref(filt),
                                   _ptr(ws), ws.numel(), _stream(stream)), "spec_sample_block")


def sample_block(drafter_logits, temperature, uniforms, top_k=None, top_p=None, max_top_k=None,
                 ws=None, stream=None) -> Dict[str, torch.Tensor]:
    """Draft-side sampling of every block token from its drafter row (x^{L+1} ~ q_0,
    drafts ~ q), optionally top-k / top-p filtered. Returns block_tokens and q_tok."""
    B, G, _ = drafter_logits.shape
    dev = drafter_logits.device
    res = dict(block_tokens=torch.empty(B, G, dtype=torch.int32, device=dev),
               q_tok=torch.empty(B, G, dtype=torch.float32, device=dev))
    d = draft_args(drafter_logits, temperature, uniforms, res["block_tokens"], res["q_tok"])
    f = None if top_k is None else filter_args(top_k, top_p, B, max_top_k)
    if ws is None:
        ws = new_workspace(draft_workspace_size(d, f), dev)
    sample_block_args(d, f, ws, stream)
    return res


def noise_tokens(seed: int, n: int, vocab: int, offset: int = 0, device=None,
                 stream=None) -> torch.Tensor:
    """The uniform noise tokens z ~ U[V] that start a draft pass (Alg. line 1)."""
    out = torch.empty(n, dtype=torch.int32, device=device or "cuda")
    _raise(lib().spec_noise_tokens(ctypes.c_uint64(seed), ctypes.c_uint64(offset), n, int(vocab),
                                   _ptr(out), _stream(stream)), "spec_noise_tokens")
    return out


def commit_kv(kv_len, num_accepted, page_table, page_size: int, gamma: int, free_pages, free_count,
              reserve: bool = True, flags=None, stream=None):
    """spec_commit_kv on device tensors (kv_len, page_table, free_pages, free_count are
    updated in place; free_count is an int32 tensor of one element)."""
    B, MP = page_table.shape
    _check(kv_len, "kv_len", torch.int32, (B,))
    _check(num_accepted, "num_accepted", torch.int32, (B,))
    _check(page_table, "page_table", torch.int32)
    _check(free_pages, "free_pages", torch.int32)
    _check(free_count, "free_count", torch.int32, (1,))
    if flags is not None:
        _check(flags, "flags", torch.int32, (B,))
    a = CommitArgs(B, int(gamma), int(page_size), MP, kv_len.data_ptr(), num_accepted.data_ptr(),
                   page_table.data_ptr(), free_pages.data_ptr(), free_count.data_ptr(),
                   free_pages.numel(), 1 if reserve else 0,
                   None if flags is None else flags.data_ptr())
    _raise(lib().spec_commit_kv(ctypes.byref(a), _stream(stream)), "spec_commit_kv")


def tree_accept_args(target_logits, tokens, parents, path, num_accepted, out_tokens,
                     num_emitted, temperature=None, uniforms=None) -> TreeAcceptArgs:
    B, N, V = target_logits.shape
    if target_logits.dtype == torch.bfloat16:
        dt = SPEC_BF16
    elif target_logits.dtype == torch.float32:
        dt = SPEC_F32
    else:
        raise TypeError("logits must be bfloat16 or float32")
    _check(target_logits, "target_logits", target_logits.dtype)
    for t, name, shape in ((tokens, "tokens", (B, N)), (parents, "parents", (B, N)),
                           (path, "path", (B, N)), (num_accepted, "num_accepted", (B,)),
                           (out_tokens, "out_tokens", (B, N + 1)), (num_emitted, "num_emitted", (B,))):
        _check(t, name, torch.int32, shape)
    if (temperature is None) != (uniforms is None):
        raise ValueError("temperature and uniforms go together")
    if temperature is not None:
        _check(temperature, "temperature", torch.float32, (B,))
        _check(uniforms, "uniforms", torch.float32, (B, N))
    return TreeAcceptArgs(B, N, V, dt, target_logits.data_ptr(), tokens.data_ptr(),
                          parents.data_ptr(), path.data_ptr(), num_accepted.data_ptr(),
                          out_tokens.data_ptr(), num_emitted.data_ptr(),
                          None if temperature is None else temperature.data_ptr(),
                          None if uniforms is None else uniforms.data_ptr())


def tree_workspace_size(t: TreeAcceptArgs) -> int:
    n = lib().spec_tree_workspace_size(ctypes.byref(t))
    if n == 0:
        raise SpecError(1, "spec_tree_workspace_size")
    return int(n)


def accept_tree_args(t: TreeAcceptArgs, ws: torch.Tensor, stream=None):
    _raise(lib().spec_accept_tree(ctypes.byref(t), _ptr(ws), ws.numel(), _stream(stream)),
           "spec_accept_tree")


def accept_tree(target_logits, tokens, parents, ws=None, stream=None, temperature=None,
                uniforms=None) -> Dict[str, torch.Tensor]:
    """Verification of a candidate tree (spec_accept_tree): greedy, or sampled for the
    sequences with temperature > 0 (temperature float32 [batch] and uniforms float32
    [batch][num_nodes] together). Returns path, num_accepted, out_tokens, num_emitted."""
    B, N, _ = target_logits.shape
    dev = target_logits.device
    res = dict(path=torch.empty(B, N, dtype=torch.int32, device=dev),
               num_accepted=torch.empty(B, dtype=torch.int32, device=dev),
               out_tokens=torch.empty(B, N + 1, dtype=torch.int32, device=dev),
               num_emitted=torch.empty(B, dtype=torch.int32, device=dev))
    t = tree_accept_args(target_logits, tokens, parents, res["path"], res["num_accepted"],
                         res["out_tokens"], res["num_emitted"], temperature, uniforms)
    if ws is None:
        ws = new_workspace(tree_workspace_size(t), dev)
    accept_tree_args(t, ws, stream)
    return res


def commit_tree_kv(k_cache, v_cache, page_table, kv_len, path, num_accepted, status_ws=None,
                   stream=None):
    """spec_commit_tree_kv: move the accepted path's keys and values into place and
    shorten kv_len (k_cache, v_cache and kv_len are updated in place)."""
    num_pages, Hkv, P, D = k_cache.shape
    B, N = path.shape
    _check(k_cache, "k_cache", torch.bfloat16)
    _check(v_cache, "v_cache", torch.bfloat16, k_cache.shape)
    _check(page_table, "page_table", torch.int32)
    _check(kv_len, "kv_len", torch.int32, (B,))
    _check(path, "path", torch.int32)
    _check(num_accepted, "num_accepted", torch.int32, (B,))
    a = TreeCommitArgs(B, N, Hkv, D, P, page_table.shape[1], num_pages, k_cache.data_ptr(),
                       v_cache.data_ptr(), page_table.data_ptr(), kv_len.data_ptr(),
                       path.data_ptr(), num_accepted.data_ptr(),
                       None if status_ws is None else status_ws.data_ptr())
    _raise(lib().spec_commit_tree_kv(ctypes.byref(a), _stream(stream)), "spec_commit_tree_kv")


def tree_build_args(drafter_logits, temperature, root_tokens, top_k: int, tokens, parents,
                    depth=None, tree_mask=None) -> TreeBuildArgs:
    B, G, V = drafter_logits.shape
    N = tokens.shape[1]
    if drafter_logits.dtype == torch.bfloat16:
        dt = SPEC_BF16
    elif drafter_logits.dtype == torch.float32:
        dt = SPEC_F32
    else:
        raise TypeError("logits must be bfloat16 or float32")
    _check(drafter_logits, "drafter_logits", drafter_logits.dtype)
    _check(temperature, "temperature", torch.float32, (B,))
    _check(root_tokens, "root_tokens", torch.int32, (B,))
    _check(tokens, "tokens", torch.int32, (B, N))
    _check(parents, "parents", torch.int32, (B, N))
    if depth is not None:
        _check(depth, "depth", torch.int32, (B, N))
    if tree_mask is not None:
        _check(tree_mask, "tree_mask", torch.int64, (B, N))
    return TreeBuildArgs(B, G, V, dt, int(top_k), N, drafter_logits.data_ptr(),
                         temperature.data_ptr(), root_tokens.data_ptr(), tokens.data_ptr(),
                         parents.data_ptr(), None if depth is None else depth.data_ptr(),
                         None if tree_mask is None else tree_mask.data_ptr())


def tree_build_workspace_size(t: TreeBuildArgs) -> int:
    n = lib().spec_tree_build_workspace_size(ctypes.byref(t))
    if n == 0:
        raise SpecError(1, "spec_tree_build_workspace_size")
    return int(n)


def build_tree_args(t: TreeBuildArgs, ws: torch.Tensor, stream=None):
    _raise(lib().spec_build_tree(ctypes.byref(t), _ptr(ws), ws.numel(), _stream(stream)),
           "spec_build_tree")


def build_tree(drafter_logits, temperature, root_tokens, top_k: int, num_nodes: int, ws=None,
               stream=None) -> Dict[str, torch.Tensor]:
    """The tree sampler (spec_build_tree). Returns tokens, parents, depth and mask
    (int64 bit sets, the tree_mask input of verify_attention), each [batch][num_nodes]."""
    B = drafter_logits.shape[0]
    dev = drafter_logits.device
    res = {k: torch.empty(B, num_nodes, dtype=torch.int32, device=dev)
           for k in ("tokens", "parents", "depth")}
    res["mask"] = torch.empty(B, num_nodes, dtype=torch.int64, device=dev)
    t = tree_build_args(drafter_logits, temperature, root_tokens, top_k, res["tokens"],
                        res["parents"], res["depth"], res["mask"])
    if ws is None:
        ws = new_workspace(tree_build_workspace_size(t), dev)
    build_tree_args(t, ws, stream)
    return res


def lm_head_args(hidden_states, weight, temperature, rows_per_seq: int, out: Dict[str, torch.Tensor],
                 tokens=None) -> LmHeadArgs:
    R, H = hidden_states.shape
    V, H2 = weight.shape
    if H2 != H:
        raise ValueError("weight and hidden states disagree on the hidden size")
    _check(hidden_states, "hidden_states", torch.bfloat16)
    _check(weight, "weight", torch.bfloat16)
    _check(temperature, "temperature", torch.float32, ((R + rows_per_seq - 1) // rows_per_seq,))
    if tokens is not None:
        _check(tokens, "tokens", torch.int32, (R,))
    for k in ("row_max", "row_sum"):
        _check(out[k], k, torch.float32, (R,))
    _check(out["row_argmax"], "row_argmax", torch.int32, (R,))
    if out.get("token_logit") is not None:
        _check(out["token_logit"], "token_logit", torch.float32, (R,))
    if out.get("logits") is not None:
        _check(out["logits"], "logits", torch.bfloat16, (R, V))
    return LmHeadArgs(R, H, V, int(rows_per_seq), hidden_states.data_ptr(), weight.data_ptr(),
                      temperature.data_ptr(), _ptr(tokens), out["row_max"].data_ptr(),
                      out["row_sum"].data_ptr(), out["row_argmax"].data_ptr(),
                      _ptr(out.get("token_logit")), _ptr(out.get("logits")))


def lm_head_workspace_size(a: LmHeadArgs) -> int:
    n = lib().spec_lm_head_workspace_size(ctypes.byref(a))
    if n == 0:
        raise SpecError(1, "spec_lm_head_workspace_size")
    return int(n)


def lm_head_stats_args(a: LmHeadArgs, ws: torch.Tensor, stream=None):
    _raise(lib().spec_lm_head_stats(ctypes.byref(a), _ptr(ws), ws.numel(), _stream(stream)),
           "spec_lm_head_stats")


def test_lm_head_wait_timeout_args(a: LmHeadArgs, ws: torch.Tensor, stream=None):
    """Test hook: spec_lm_head_stats with its copy producer idle, so that the kernel's
    bounded waits run out (about 1 s) and it returns with SPEC_FLAG_TIMEOUT set."""
    _raise(lib().spec_test_lm_head_wait_timeout(ctypes.byref(a), _ptr(ws), ws.numel(),
                                                _stream(stream)), "spec_test_lm_head_wait_timeout")


def lm_head_stats(hidden_states, weight, temperature, rows_per_seq: int, tokens=None,
                  want_logits: bool = False, ws=None, stream=None) -> Dict[str, torch.Tensor]:
    """spec_lm_head_stats: the LM head's logits reduced per row (max, sum of
    exp((l - max) / T), lowest-index argmax, the token's logit); the logits themselves
    (bf16) only if want_logits."""
    R = hidden_states.shape[0]
    V = weight.shape[0]
    dev = hidden_states.device
    out = dict(row_max=torch.empty(R, dtype=torch.float32, device=dev),
               row_sum=torch.empty(R, dtype=torch.float32, device=dev),
               row_argmax=torch.empty(R, dtype=torch.int32, device=dev),
               token_logit=torch.empty(R, dtype=torch.float32, device=dev) if tokens is not None else None,
               logits=torch.empty(R, V, dtype=torch.bfloat16, device=dev) if want_logits else None)
    a = lm_head_args(hidden_states, weight, temperature, rows_per_seq, out, tokens)
    if ws is None:
        ws = new_workspace(lm_head_workspace_size(a), dev)
    lm_head_stats_args(a, ws, stream)
    return {k: v for k, v in out.items() if v is not None}


def philox_uniforms(seed: int, n: int, offset: int = 0, device=None, stream=None) -> torch.Tensor:
    out = torch.empty(n, dtype=torch.float32, device=device or "cuda")
    _raise(lib().spec_philox_uniforms(ctypes.c_uint64(seed), ctypes.c_uint64(offset), n,
                                      _ptr(out), _stream(stream)), "spec_philox_uniforms")
    return out


def read_device_status(ws: torch.Tensor, stream=None):
    """(status code, flags) of the workspace status word; reading clears it."""
    flags = ctypes.c_uint32(0)
    code = lib().spec_read_device_status(_ptr(ws), _stream(stream), ctypes.byref(flags))
    return int(code), int(flags.value)


def tensor_core_min_rows() -> int:
    return int(lib().spec_attn_tensor_core_min_rows())
