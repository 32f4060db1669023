"""Seeded synthetic inputs for the verify step.

This module is shared by the tests, the benchmark, the CUDA path and the oracle, and
holds none of the verify step's arithmetic: it only draws random inputs.  The paper's
throughput methodology drives its models with random input tokens (Sec. 5, "Throughput
Analysis"); without trained weights, the logits and the KV cache here are random too,
with the shapes and distributions of five named workloads.

Random streams
--------------
* Acceptance uniforms come from Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel
  random numbers: as easy as 1, 2, 3", SC'11), written here from that paper's
  definition.  Element i of a stream with 64-bit key k uses the counter
  (i >> 2 low word, i >> 2 high word, 0, 0), the key (k low word, k high word) and
  output word i & 3; the uniform is ((x >> 8) + 1) * 2^-24, which lies in (0, 1] and
  is exact in fp32.  The CUDA library's ``spec_philox_uniforms`` produces the same
  bits.
* Everything else (logits, KV, Q, contexts, page permutations, draft sampling) comes
  from numpy's PCG64 seeded by ``SeedSequence([seed, stream])``.

Draft tokens are drawn from the drafter's tempered distribution with the Gumbel-max
construction (argmax of l / T + Gumbel noise), and as the argmax of the drafter row at
T = 0, so that the drafts follow the proposal without this module evaluating a softmax.
"""

from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

# ---------------------------------------------------------------------------------
# Philox4x32-10 (Salmon et al., SC'11)
# ---------------------------------------------------------------------------------
PHILOX_M0 = np.uint64(0xD2511F53)
PHILOX_M1 = np.uint64(0xCD9E8D57)
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
_MASK32 = np.uint64(0xFFFFFFFF)


def philox4x32_10(counter: np.ndarray, key: Tuple[int, int]) -> np.ndarray:
    """Philox4x32 with 10 rounds.  counter: uint32 [..., 4]; key: two 32-bit words.

    Each round multiplies words 0 and 2 by the two Philox multipliers (64-bit
    products split into high and low halves), mixes the high halves with words 1
    and 3 and the round key, and permutes; the key advances by the two Weyl
    constants between rounds.
    """
    c = np.asarray(counter, dtype=np.uint32).astype(np.uint64)
    c0, c1, c2, c3 = c[..., 0], c[..., 1], c[..., 2], c[..., 3]
    k0 = int(key[0]) & 0xFFFFFFFF
    k1 = int(key[1]) & 0xFFFFFFFF
    for r in range(10):
        if r:
            k0 = (k0 + PHILOX_W0) & 0xFFFFFFFF
            k1 = (k1 + PHILOX_W1) & 0xFFFFFFFF
        p0 = PHILOX_M0 * c0
        p1 = PHILOX_M1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        c0, c1, c2, c3 = (hi1 ^ c1 ^ np.uint64(k0), lo1, hi0 ^ c3 ^ np.uint64(k1), lo0)
    return np.stack([c0, c1, c2, c3], axis=-1).astype(np.uint32)


def philox_words(seed: int, n: int, offset: int = 0) -> np.ndarray:
    """Words offset .. offset+n-1 of the Philox stream keyed by the 64-bit ``seed``."""
    idx = np.arange(offset, offset + n, dtype=np.uint64)
    blk = idx >> np.uint64(2)
    ctr = np.zeros((n, 4), dtype=np.uint32)
    ctr[:, 0] = (blk & _MASK32).astype(np.uint32)
    ctr[:, 1] = (blk >> np.uint64(32)).astype(np.uint32)
    out = philox4x32_10(ctr, (seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF))
    lane = (idx & np.uint64(3)).astype(np.int64)
    return out[np.arange(n), lane]


def philox_uniforms(seed: int, n: int, offset: int = 0) -> np.ndarray:
    """Uniforms in (0, 1] from the Philox stream: ((x >> 8) + 1) * 2^-24, as fp32."""
    x = philox_words(seed, n, offset)
    return (((x >> np.uint32(8)).astype(np.float64) + 1.0) * 2.0 ** -24).astype(np.float32)


# ---------------------------------------------------------------------------------
# bf16 helpers (bf16 tensors travel as uint16 bit patterns on the host)
# ---------------------------------------------------------------------------------
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (round to nearest, ties to even); returns uint16 bits."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounding = ((b >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((b + rounding) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(h: np.ndarray) -> np.ndarray:
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# ---------------------------------------------------------------------------------
# Streams
# ---------------------------------------------------------------------------------
STREAM_TARGET, STREAM_DRAFT_NOISE, STREAM_DRAFT_SAMPLE = 1, 2, 3
STREAM_UNIFORMS = 4
STREAM_Q, STREAM_K, STREAM_V, STREAM_PAGES, STREAM_CTX = 5, 6, 7, 8, 9


def _rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(seed), int(stream)])))


def uniform_seed(seed: int) -> int:
    """64-bit Philox key of the acceptance uniforms of workload seed ``seed``."""
    return (int(seed) & 0xFFFFFFFF) | (STREAM_UNIFORMS << 32)


# ---------------------------------------------------------------------------------
# Acceptance inputs
# ---------------------------------------------------------------------------------
@dataclasses.dataclass
class AcceptInputs:
    target_logits: np.ndarray   # [batch][gamma][vocab] float32 or uint16 (bf16 bits)
    drafter_logits: np.ndarray  # same
    block_tokens: np.ndarray    # int32 [batch][gamma]
    temperature: np.ndarray     # float32 [batch]
    uniforms: np.ndarray        # float32 [batch][gamma], in (0, 1]

    @property
    def batch(self) -> int:
        return self.target_logits.shape[0]

    @property
    def gamma(self) -> int:
        return self.target_logits.shape[1]

    @property
    def vocab(self) -> int:
        return self.target_logits.shape[2]

    @property
    def is_bf16(self) -> bool:
        return self.target_logits.dtype == np.uint16


def _gumbel_argmax(rng: np.random.Generator, logits_f32: np.ndarray, T: float,
                   top_k: int = 0) -> int:
    if not T > 0.0:
        return int(np.argmax(logits_f32))
    u = rng.random(logits_f32.shape[0])
    g = -np.log(-np.log(np.maximum(u, 1e-300)))
    score = logits_f32.astype(np.float64) / T + g
    if top_k > 0 and top_k < logits_f32.shape[0]:
        # only the top_k largest logits (equal logits by lower id) can be drawn
        order = np.argsort(-logits_f32, kind="stable")
        score[order[top_k:]] = -np.inf
    return int(np.argmax(score))


def make_accept_inputs(batch: int, gamma: int, vocab: int, logits_dtype: str = "bf16",
                       target_sigma: float = 3.0, drafter_sigma: float = 1.0,
                       temperature=1.0, seed: int = 0, draft_top_k: int = 0) -> AcceptInputs:
    """Synthetic logits for the acceptance rule.

    Target row j ~ N(0, target_sigma^2) per element.  Drafter row j (j >= 1) is target
    row j-1 plus N(0, drafter_sigma^2) noise (drafter row j proposes block token j,
    whose verifier distribution is target row j-1); drafter row 0 is independent.
    Rows are rounded to bf16 when ``logits_dtype == "bf16"``.  Block token j is drawn
    from drafter row j at the sequence's temperature (argmax at T = 0); with
    ``draft_top_k`` > 0, only among that row's draft_top_k largest logits (the support
    of a top-k filtered proposal).
    ``temperature`` is a scalar or a sequence cycled over the batch.
    """
    temps = np.resize(np.asarray(temperature, dtype=np.float32).ravel(), batch)
    rng_t = _rng(seed, STREAM_TARGET)
    rng_n = _rng(seed, STREAM_DRAFT_NOISE)
    rng_s = _rng(seed, STREAM_DRAFT_SAMPLE)
    bf16 = logits_dtype == "bf16"
    store = np.uint16 if bf16 else np.float32
    tl = np.empty((batch, gamma, vocab), dtype=store)
    dl = np.empty((batch, gamma, vocab), dtype=store)
    tokens = np.empty((batch, gamma), dtype=np.int32)
    for b in range(batch):
        t32 = rng_t.standard_normal((gamma, vocab), dtype=np.float32) * np.float32(target_sigma)
        d32 = np.empty_like(t32)
        d32[0] = rng_t.standard_normal(vocab, dtype=np.float32) * np.float32(target_sigma)
        if gamma > 1:
            d32[1:] = t32[:-1] + rng_n.standard_normal((gamma - 1, vocab), dtype=np.float32) \
                * np.float32(drafter_sigma)
        if bf16:
            tl[b] = f32_to_bf16_bits(t32)
            dl[b] = f32_to_bf16_bits(d32)
            dseen = bf16_bits_to_f32(dl[b])
        else:
            tl[b] = t32
            dl[b] = d32
            dseen = d32
        for j in range(gamma):
            tokens[b, j] = _gumbel_argmax(rng_s, dseen[j], float(temps[b]), draft_top_k)
    u = philox_uniforms(uniform_seed(seed), batch * gamma).reshape(batch, gamma)
    return AcceptInputs(tl, dl, tokens, temps, u)


# ---------------------------------------------------------------------------------
# Attention inputs
# ---------------------------------------------------------------------------------
@dataclasses.dataclass
class AttnInputs:
    q: np.ndarray           # uint16 bf16 bits [batch][gamma][Hq][D]
    k_cache: np.ndarray     # uint16 bf16 bits [num_pages][Hkv][page_size][D]
    v_cache: np.ndarray     # same
    page_table: np.ndarray  # int32 [batch][max_pages_per_seq], unused entries -1
    kv_len: np.ndarray      # int32 [batch] = context + gamma

    @property
    def batch(self) -> int:
        return self.q.shape[0]

    @property
    def gamma(self) -> int:
        return self.q.shape[1]

    @property
    def num_q_heads(self) -> int:
        return self.q.shape[2]

    @property
    def head_dim(self) -> int:
        return self.q.shape[3]

    @property
    def num_pages(self) -> int:
        return self.k_cache.shape[0]

    @property
    def num_kv_heads(self) -> int:
        return self.k_cache.shape[1]

    @property
    def page_size(self) -> int:
        return self.k_cache.shape[2]

    def kv_bytes(self) -> int:
        """Bytes of K and V the block-causal attention must read (bf16)."""
        return int(self.kv_len.astype(np.int64).sum()) * self.num_kv_heads * self.head_dim * 2 * 2


def _bf16_normals(rng: np.random.Generator, shape, chunk: int = 1 << 24) -> np.ndarray:
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.uint16)
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        out[s:e] = f32_to_bf16_bits(rng.standard_normal(e - s, dtype=np.float32))
    return out.reshape(shape)


def make_lm_inputs(rows: int, hidden: int, vocab: int, rows_per_seq: int, sigma: float = 3.0,
                   temperature=1.0, seed: int = 0, chunk: int = 1 << 14):
    """Synthetic LM-head operands: hidden states ~ N(0, 1) rounded to bf16, and weight
    entries uniform with variance sigma^2 / hidden, cut to bf16 by dropping the low 16
    bits of the fp32 value (one cheap pass over the 10^8..10^9 entries of a real head),
    so that logits are about N(0, sigma^2); per-sequence temperatures (cycled from
    `temperature`) and one token per row. Returns (hidden uint16 [rows][hidden], weight
    uint16 [vocab][hidden], temperature float32 [rows // rows_per_seq], tokens int32
    [rows])."""
    ss = np.random.SeedSequence([seed, 41])
    g_h, g_w, g_t = (np.random.Generator(np.random.PCG64(c)) for c in ss.spawn(3))
    h = f32_to_bf16_bits(g_h.standard_normal((rows, hidden), dtype=np.float32)).reshape(rows, hidden)
    w = np.empty((vocab, hidden), np.uint16)
    half = np.float32(np.sqrt(3.0) * sigma / np.sqrt(hidden))  # U(-a, a) has variance a^2 / 3
    for v0 in range(0, vocab, chunk):
        n = min(chunk, vocab - v0)
        x = g_w.random((n, hidden), dtype=np.float32)
        x *= np.float32(2) * half
        x -= half
        w[v0:v0 + n] = (x.view(np.uint32) >> np.uint32(16)).astype(np.uint16)
    nseq = (rows + rows_per_seq - 1) // rows_per_seq
    temps = np.resize(np.asarray(temperature, np.float32), nseq).astype(np.float32)
    tokens = g_t.integers(0, vocab, rows).astype(np.int32)
    return h, w, temps, tokens


def make_attn_inputs(batch: int, gamma: int, num_q_heads: int, num_kv_heads: int, head_dim: int,
                     page_size: int, ctx, permute_pages: bool = True, seed: int = 0,
                     extra_pages: int = 0) -> AttnInputs:
    """Synthetic Q and paged KV cache.

    ``ctx`` is an int (every sequence has that many prefix tokens) or a (lo, hi) pair
    (context lengths uniform on the integers lo..hi).  kv_len = ctx + gamma: the
    block's own keys are already in the cache.  Sequence b owns ceil(kv_len/page_size)
    pages; physical page ids are a seeded permutation of all pages when
    ``permute_pages`` (else sequences own consecutive pages).  Q, K, V ~ N(0, 1) in
    bf16, including the unused slots of the last page of each sequence.
    """
    if isinstance(ctx, (tuple, list)):
        lo, hi = int(ctx[0]), int(ctx[1])
        ctxs = _rng(seed, STREAM_CTX).integers(lo, hi + 1, size=batch).astype(np.int32)
    else:
        ctxs = np.full(batch, int(ctx), dtype=np.int32)
    kv_len = (ctxs + gamma).astype(np.int32)
    pages = (kv_len + page_size - 1) // page_size
    total = int(pages.sum()) + int(extra_pages)
    max_pages = int(pages.max())
    phys = np.arange(total, dtype=np.int32)
    if permute_pages:
        phys = _rng(seed, STREAM_PAGES).permutation(total).astype(np.int32)
    pt = np.full((batch, max_pages), -1, dtype=np.int32)
    cur = 0
    for b in range(batch):
        pt[b, :pages[b]] = phys[cur:cur + pages[b]]
        cur += int(pages[b])
    q = _bf16_normals(_rng(seed, STREAM_Q), (batch, gamma, num_q_heads, head_dim))
    k = _bf16_normals(_rng(seed, STREAM_K), (total, num_kv_heads, page_size, head_dim))
    v = _bf16_normals(_rng(seed, STREAM_V), (total, num_kv_heads, page_size, head_dim))
    return AttnInputs(q, k, v, pt, kv_len)


# ---------------------------------------------------------------------------------
# Named workloads
# ---------------------------------------------------------------------------------
@dataclasses.dataclass
class Workload:
    name: str
    batch: int
    gamma: int
    vocab: int
    logits_dtype: str
    target_sigma: float
    drafter_sigma: float
    temperatures: Tuple[float, ...]  # cycled over the batch
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    page_size: int
    ctx: object                      # int or (lo, hi)
    permute_pages: bool = True
    note: str = ""
    top_k: int = 0        # > 0: top-k / top-p filtered verification (drafts from the top-k)
    top_p: float = 1.0

    def temps(self) -> np.ndarray:
        t = np.asarray(self.temperatures, dtype=np.float32)
        return np.resize(t, self.batch).astype(np.float32)

    def accept_inputs(self, seed: int = 0) -> AcceptInputs:
        return make_accept_inputs(self.batch, self.gamma, self.vocab, self.logits_dtype,
                                  self.target_sigma, self.drafter_sigma, self.temps(), seed,
                                  draft_top_k=self.top_k)

    def filter_params(self):
        """(top_k [batch] int32, top_p [batch] float32) of a filtered workload."""
        return (np.full(self.batch, self.top_k, np.int32),
                np.full(self.batch, self.top_p, np.float32))

    def attn_inputs(self, seed: int = 0) -> AttnInputs:
        return make_attn_inputs(self.batch, self.gamma, self.num_q_heads, self.num_kv_heads,
                                self.head_dim, self.page_size, self.ctx, self.permute_pages, seed)

    def describe(self) -> Dict[str, object]:
        d = dict(workload=self.name, batch=self.batch, gamma=self.gamma, vocab=self.vocab,
                 logits_dtype=self.logits_dtype, num_q_heads=self.num_q_heads,
                 num_kv_heads=self.num_kv_heads, head_dim=self.head_dim,
                 page_size=self.page_size, ctx=self.ctx)
        if self.top_k > 0:
            d.update(top_k=self.top_k, top_p=self.top_p)
        return d


WORKLOADS: Dict[str, Workload] = {
    # batch 1, gamma 4, vocab 32,000 fp32 logits; 8/8 heads, head_dim 64, context 512
    # stored contiguously (identity page table of 16-token pages).
    "tiny": Workload("tiny", 1, 4, 32000, "f32", 2.0, 0.5, (1.0,), 8, 8, 64, 16, 512,
                     permute_pages=False),
    # Llama-3-8B-shaped: batch 8, gamma 8, 32/8 heads, head_dim 128, context 4,096 in
    # 16-token pages (permuted), vocab 128,256 bf16, drafter noise 1, T = 1.
    "llama8b": Workload("llama8b", 8, 8, 128256, "bf16", 3.0, 1.0, (1.0,), 32, 8, 128, 16, 4096),
    # high-batch serving: batch 64, gamma 16, ragged contexts 512..4,096; half greedy.
    "serve64": Workload("serve64", 64, 16, 128256, "bf16", 3.0, 0.5, (0.0, 1.0), 32, 8, 128, 16,
                        (512, 4096)),
    # 70B-shaped long context: batch 4, gamma 32, 64/8 heads, context 32,768 in 64-token
    # pages, T = 0.7.
    "long70b": Workload("long70b", 4, 32, 128256, "bf16", 3.0, 1.0, (0.7,), 64, 8, 128, 64, 32768),
    # the paper's evaluation sampling (T = 1, top-k 50, top-p 0.95) on the Llama-3-8B
    # shape and on the high-batch serving shape (all sequences tempered)
    "llama8b_topk": Workload("llama8b_topk", 8, 8, 128256, "bf16", 3.0, 1.0, (1.0,), 32, 8, 128,
                             16, 4096, top_k=50, top_p=0.95),
    "serve64_topk": Workload("serve64_topk", 64, 16, 128256, "bf16", 3.0, 0.5, (1.0,), 32, 8, 128,
                             16, (512, 4096), top_k=50, top_p=0.95),
}

SWEEP_GAMMAS = (1, 2, 4, 8, 16, 32)
SWEEP_BATCHES = (1, 8, 32, 128)
SWEEP_SIGMAS = (0.1, 1.0, 3.0)
SWEEP_TEMPS = (0.0, 1.0)


def sweep_workload(gamma: int, batch: int, drafter_sigma: float = 1.0,
                   temperature: float = 1.0) -> Workload:
    """One point of the sweep: 32/8 heads, head_dim 128, contexts 256..16,384 in 16-token
    pages, vocab 151,936 bf16, target sigma 3."""
    name = f"sweep_g{gamma}_b{batch}_s{drafter_sigma:g}_t{temperature:g}"
    return Workload(name, batch, gamma, 151936, "bf16", 3.0, float(drafter_sigma),
                    (float(temperature),), 32, 8, 128, 16, (256, 16384))


def workload(name: str) -> Workload:
    if name in WORKLOADS:
        return WORKLOADS[name]
    if name.startswith("sweep_"):
        parts = dict((p[0], p[1:]) for p in name.split("_")[1:])
        return sweep_workload(int(parts["g"]), int(parts["b"]), float(parts.get("s", 1.0)),
                              float(parts.get("t", 1.0)))
    raise KeyError(name)


def logits_bytes_baseline(batch: int, gamma: int, vocab: int, elem_bytes: int) -> int:
    """Logits bytes in the headline roofline count: 2 * vocab * gamma per sequence."""
    return 2 * vocab * gamma * elem_bytes * batch


def logits_bytes_strict(temps: np.ndarray, gamma: int, vocab: int, elem_bytes: int) -> int:
    """Logits bytes the step must read: gamma target rows, plus gamma-1 drafter rows for
    sequences with T > 0."""
    t = np.asarray(temps)
    rows = gamma * len(t) + (gamma - 1) * int((t > 0).sum())
    return rows * vocab * elem_bytes


# ---------------------------------------------------------------------------------
# Device-side generators for sizes the host generator cannot fill quickly
# ---------------------------------------------------------------------------------
# The sweep's largest points hold billions of random values (batch 128 with contexts up
# to 16,384, or 128 x 32 x 151,936 logits per side). These generators draw the same
# distributions on the GPU with torch's seeded generator; the tests copy to the host
# only what the oracle needs. Like the rest of this module they draw inputs and compute
# nothing of the verify step.
def _torch_gen(seed: int, stream: int, device):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1_000_003 + int(stream) * 7_919) & 0x7FFF_FFFF_FFFF_FFFF)
    return g


@dataclasses.dataclass
class DeviceAttnInputs:
    q: object            # torch bf16 [batch][gamma][Hq][D] on the device
    k_cache: object      # torch bf16 [num_pages][Hkv][page_size][D]
    v_cache: object
    page_table: object   # torch int32 [batch][max_pages]
    kv_len: object       # torch int32 [batch]
    page_table_host: np.ndarray
    kv_len_host: np.ndarray
    gamma: int

    def host(self) -> AttnInputs:
        """The same inputs as host arrays (bf16 as uint16 bits), for the oracle."""
        import torch

        def bits(t):
            return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        return AttnInputs(bits(self.q), bits(self.k_cache), bits(self.v_cache),
                          self.page_table_host.copy(), self.kv_len_host.copy())


def make_attn_inputs_device(batch: int, gamma: int, num_q_heads: int, num_kv_heads: int,
                            head_dim: int, page_size: int, ctx, seed: int = 0,
                            device="cuda") -> DeviceAttnInputs:
    """make_attn_inputs' shapes and distributions (contexts uniform on lo..hi, a seeded
    permutation of physical pages, Q, K, V ~ N(0, 1) rounded to bf16), with Q, K and V
    drawn on the device. Contexts and the page table come from the host streams of
    make_attn_inputs, so they equal its own for the same arguments."""
    import torch
    if isinstance(ctx, (tuple, list)):
        lo, hi = int(ctx[0]), int(ctx[1])
        ctxs = _rng(seed, STREAM_CTX).integers(lo, hi + 1, size=batch).astype(np.int32)
    else:
        ctxs = np.full(batch, int(ctx), dtype=np.int32)
    kv_len = (ctxs + gamma).astype(np.int32)
    pages = (kv_len + page_size - 1) // page_size
    total = int(pages.sum())
    phys = _rng(seed, STREAM_PAGES).permutation(total).astype(np.int32)
    pt = np.full((batch, int(pages.max())), -1, dtype=np.int32)
    cur = 0
    for b in range(batch):
        pt[b, :pages[b]] = phys[cur:cur + pages[b]]
        cur += int(pages[b])

    def normals(stream, shape):
        g = _torch_gen(seed, stream, device)
        return torch.randn(*shape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)

    q = normals(STREAM_Q, (batch, gamma, num_q_heads, head_dim))
    k = normals(STREAM_K, (total, num_kv_heads, page_size, head_dim))
    v = normals(STREAM_V, (total, num_kv_heads, page_size, head_dim))
    return DeviceAttnInputs(q, k, v, torch.from_numpy(pt).to(device),
                            torch.from_numpy(kv_len).to(device), pt, kv_len, gamma)


@dataclasses.dataclass
class DeviceAcceptInputs:
    target_logits: object   # torch bf16 [batch][gamma][vocab] on the device
    drafter_logits: object
    block_tokens: object    # torch int32 [batch][gamma]
    temperature: object     # torch float32 [batch]
    uniforms: object        # torch float32 [batch][gamma]

    def host(self, nseq: int) -> AcceptInputs:
        """The first nseq sequences as host arrays (bf16 as uint16 bits), for the oracle."""
        import torch

        def bits(t):
            return t[:nseq].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        return AcceptInputs(bits(self.target_logits), bits(self.drafter_logits),
                            self.block_tokens[:nseq].cpu().numpy(),
                            self.temperature[:nseq].cpu().numpy(),
                            self.uniforms[:nseq].cpu().numpy())


def make_accept_inputs_device(batch: int, gamma: int, vocab: int, target_sigma: float = 3.0,
                              drafter_sigma: float = 1.0, temperature=1.0, seed: int = 0,
                              device="cuda", chunk: int = 8) -> DeviceAcceptInputs:
    """make_accept_inputs' distributions with bf16 logits drawn on the device: target rows
    ~ N(0, target_sigma^2), drafter row j >= 1 = target row j-1 + N(0, drafter_sigma^2),
    drafter row 0 independent, both rounded to bf16; block token j drawn from drafter
    row j at the sequence's temperature by Gumbel-max (argmax at T = 0, lowest index on
    ties). The uniforms are the host Philox stream of make_accept_inputs, bit for bit."""
    import torch
    temps = np.resize(np.asarray(temperature, dtype=np.float32).ravel(), batch)
    g = _torch_gen(seed, STREAM_TARGET, device)
    tl = torch.empty(batch, gamma, vocab, dtype=torch.bfloat16, device=device)
    dl = torch.empty_like(tl)
    tok = torch.empty(batch, gamma, dtype=torch.int32, device=device)
    for b0 in range(0, batch, chunk):
        n = min(chunk, batch - b0)
        t32 = torch.randn(n, gamma, vocab, generator=g, device=device) * target_sigma
        d32 = torch.empty_like(t32)
        d32[:, 0] = torch.randn(n, vocab, generator=g, device=device) * target_sigma
        if gamma > 1:
            d32[:, 1:] = t32[:, :-1] + torch.randn(n, gamma - 1, vocab, generator=g,
                                                   device=device) * drafter_sigma
        tl[b0:b0 + n] = t32.to(torch.bfloat16)
        dl[b0:b0 + n] = d32.to(torch.bfloat16)
        dseen = dl[b0:b0 + n].float()
        T = torch.from_numpy(temps[b0:b0 + n]).to(device).view(n, 1, 1)
        u = torch.rand(n, gamma, vocab, generator=g, device=device).clamp_min(1e-30)
        gumbel = -torch.log(-torch.log(u))
        score = torch.where(T > 0, dseen / torch.where(T > 0, T, torch.ones_like(T)) + gumbel, dseen)
        tok[b0:b0 + n] = torch.argmax(score, dim=-1).to(torch.int32)
        del t32, d32, dseen, u, gumbel, score
    uni = philox_uniforms(uniform_seed(seed), batch * gamma).reshape(batch, gamma)
    return DeviceAcceptInputs(tl, dl, tok, torch.from_numpy(temps).to(device),
                              torch.from_numpy(uni).to(device))
