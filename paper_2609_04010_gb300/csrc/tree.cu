// Tree verification (Sec. 4.2: more than one candidate is verified at once as a prefix
// tree under tree attention; Sec. 3.3, "Tree Sampler"): the tree sampler that builds the
// candidate tree from the drafter's rows, greedy acceptance along it, and the
// compaction of the accepted path's keys and values.
//
// tree_greedy_kernel: grid (splits, nodes, sequences) of 128-thread blocks. Each block
// finds the lowest-index argmax of its part of a node's target row; the row's last block
// (ticket) merges the parts, and the sequence's last block walks the tree from the root,
// moving to the child whose token is the current node's argmax.
//
// tree_compact_kernel: one block per (cache, KV head, sequence) moves the accepted
// path's key or value rows into consecutive positions after the context.
#include <cuda_bf16.h>

#include <algorithm>
#include <cfloat>
#include <climits>
#include <cmath>

#include "common.cuh"

namespace specv {

TreeLayout tree_layout(int batch, int nodes, int vocab, size_t base, int sms, bool vec) {
  TreeLayout L;
  const int lane = vec ? 64 : 32;
  const int nlanes = (vocab + lane - 1) / lane;
  const int64_t rows = static_cast<int64_t>(batch) * nodes;
  int64_t splits = (static_cast<int64_t>(kFiltBlocksPerSm) * sms + rows - 1) / rows;
  splits = splits < 1 ? 1 : (splits > kFiltMaxSplits ? kFiltMaxSplits : splits);
  if (splits > nlanes) splits = nlanes;
  L.elems_per_split = static_cast<int>((nlanes + splits - 1) / splits) * lane;
  L.splits = (vocab + L.elems_per_split - 1) / L.elems_per_split;
  L.tickets = base;
  L.row_tickets = ws_round(L.tickets + sizeof(uint32_t) * batch);
  L.parts = ws_round(L.row_tickets + sizeof(uint32_t) * rows);
  L.argmax = ws_round(L.parts + 16 * rows * L.splits);
  L.end = ws_round(L.argmax + sizeof(int32_t) * rows);
  return L;
}

namespace {

constexpr int kThreads = 128;
constexpr int kUnroll = 8;

struct TreeParams {
  int batch, nodes, vocab, splits, elems_per_split;
  const void* target;
  const int32_t* tokens;   // [batch][nodes]
  const int32_t* parents;  // [batch][nodes]
  int32_t* path;           // [batch][nodes]
  int32_t* num_accepted;   // [batch]
  int32_t* out_tokens;     // [batch][nodes + 1]
  int32_t* num_emitted;    // [batch]
  uint32_t* status;
  uint32_t* tickets;
  uint32_t* row_tickets;
  uint4* parts;
  int32_t* argmax;         // [batch][nodes]; -1 marks a row with NaN
};

template <bool BF16>
__device__ __forceinline__ float load_elem(const void* base, int64_t i) {
  if (BF16) return bf16_bits_to_f32(static_cast<const uint16_t*>(base)[i]);
  return static_cast<const float*>(base)[i];
}

__device__ __forceinline__ uint32_t order_key(float x) {
  uint32_t f = __float_as_uint(x);
  if (f == 0x80000000u) f = 0u;
  return (f & 0x80000000u) ? ~f : (f | 0x80000000u);
}

template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kThreads, 8) tree_greedy_kernel(TreeParams p) {
  __shared__ unsigned long long s_red[kThreads / 32];
  __shared__ int s_bad, s_last;
  __shared__ int s_arg[64];
  const int split = blockIdx.x, j = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int N = p.nodes, V = p.vocab;
  const int64_t rid = static_cast<int64_t>(b) * N + j;
  const char* rowp = static_cast<const char*>(p.target) + rid * V * (BF16 ? 2 : 4);
  const int e_begin = split * p.elems_per_split, e_end = min(V, e_begin + p.elems_per_split);
  if (tid == 0) s_bad = 0;
  __syncthreads();

  // the lowest-index maximum of this part of the row
  float m = -INFINITY;
  int a = INT_MAX;
  bool bad = false;
  if (VEC) {
    constexpr int kEpv = BF16 ? 8 : 4;
    const uint32_t ninf = BF16 ? 0xFF80FF80u : 0xFF800000u;
    const int vbeg = e_begin / kEpv, vend = e_end / kEpv;
    const uint4* rv = reinterpret_cast<const uint4*>(rowp);
    if (vbeg + tid < vend) a = (vbeg + tid) * kEpv;
    for (int v0 = vbeg; v0 < vend; v0 += kThreads * kUnroll) {
      uint4 dv[kUnroll];
#pragma unroll
      for (int k = 0; k < kUnroll; ++k) {
        const int vi = v0 + k * kThreads + tid;
        dv[k] = vi < vend ? __ldg(rv + vi) : make_uint4(ninf, ninf, ninf, ninf);
      }
#pragma unroll
      for (int k = 0; k < kUnroll; ++k) {
        const int vi = v0 + k * kThreads + tid;
        const uint32_t wv[4] = {dv[k].x, dv[k].y, dv[k].z, dv[k].w};
#pragma unroll
        for (int q = 0; q < kEpv; ++q) {
          const float x = BF16 ? __uint_as_float((q & 1) ? (wv[q >> 1] & 0xffff0000u) : (wv[q >> 1] << 16))
                               : __uint_as_float(wv[q]);
          bad |= x != x;
          if (x > m) { m = x; a = vi * kEpv + q; }
        }
      }
    }
  } else {
    if (e_begin + tid < e_end) a = e_begin + tid;
    for (int e0 = e_begin; e0 < e_end; e0 += kThreads * kUnroll) {
      float x[kUnroll];
#pragma unroll
      for (int k = 0; k < kUnroll; ++k) {
        const int ei = e0 + k * kThreads + tid;
        x[k] = ei < e_end ? load_elem<BF16>(rowp, ei) : -INFINITY;
      }
#pragma unroll
      for (int k = 0; k < kUnroll; ++k) {
        bad |= x[k] != x[k];
        if (x[k] > m) { m = x[k]; a = e0 + k * kThreads + tid; }
      }
    }
  }
  unsigned long long best = (static_cast<unsigned long long>(order_key(m)) << 32) |
                            (0xffffffffu - static_cast<uint32_t>(a));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long y = __shfl_xor_sync(0xffffffffu, best, o);
    best = y > best ? y : best;
  }
  if (bad) s_bad = 1;
  if ((tid & 31) == 0) s_red[tid >> 5] = best;
  __syncthreads();
  best = s_red[0];
#pragma unroll
  for (int k = 1; k < kThreads / 32; ++k) best = s_red[k] > best ? s_red[k] : best;

  if (p.splits > 1) {
    if (tid == 0)
      p.parts[rid * p.splits + split] = make_uint4(static_cast<uint32_t>(best), static_cast<uint32_t>(best >> 32),
                                                   static_cast<uint32_t>(s_bad), 0u);
    __threadfence();
    __syncthreads();
    if (tid == 0) {
      const uint32_t prev = atomicAdd(&p.row_tickets[rid], 1u);
      s_last = prev == static_cast<uint32_t>(p.splits - 1);
      if (s_last) p.row_tickets[rid] = 0;
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    if (tid < 32) {
      unsigned long long bb = 0ull;
      uint32_t anybad = 0;
      for (int k = tid; k < p.splits; k += 32) {
        const uint4 q = __ldcg(p.parts + rid * p.splits + k);
        const unsigned long long c = (static_cast<unsigned long long>(q.y) << 32) | q.x;
        bb = c > bb ? c : bb;
        anybad |= q.z;
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long y = __shfl_xor_sync(0xffffffffu, bb, o);
        bb = y > bb ? y : bb;
      }
      anybad = __reduce_or_sync(0xffffffffu, anybad);
      if (tid == 0) {
        s_red[0] = bb;
        s_bad = anybad ? 1 : 0;
      }
    }
    __syncthreads();
    best = s_red[0];
  }
  if (tid == 0) p.argmax[rid] = s_bad ? -1 : static_cast<int>(0xffffffffu - static_cast<uint32_t>(best));

  // the sequence's last row block walks the tree
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const uint32_t prev = atomicAdd(&p.tickets[b], 1u);
    s_last = prev == static_cast<uint32_t>(N - 1);
    if (s_last) p.tickets[b] = 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid < N) s_arg[tid] = __ldcg(p.argmax + static_cast<int64_t>(b) * N + tid);
  __syncthreads();
  if (tid >= 32) return;
  // one warp: lane c holds node c (N <= 64: two nodes per lane)
  const int lane = tid;
  const int64_t brow = static_cast<int64_t>(b) * N;
  int tok[2], par[2];
  uint32_t bad_in = 0;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int c = lane + 32 * h;
    tok[h] = c < N ? p.tokens[brow + c] : -1;
    par[h] = c < N ? p.parents[brow + c] : -2;
    if (c < N) {
      if (tok[h] < 0 || tok[h] >= V) bad_in |= SPEC_FLAG_BAD_TOKEN;
      if (c == 0 ? par[h] != -1 : (par[h] < 0 || par[h] >= c)) bad_in |= SPEC_FLAG_BAD_TREE;
      if (s_arg[c] < 0) bad_in |= SPEC_FLAG_BAD_LOGITS;
    }
  }
  bad_in = __reduce_or_sync(0xffffffffu, bad_in);
  int32_t* path = p.path + brow;
  int32_t* out = p.out_tokens + static_cast<int64_t>(b) * (N + 1);
  if (bad_in) {
    for (int c = lane; c < N; c += 32) path[c] = -1;
    for (int c = lane; c <= N; c += 32) out[c] = -1;
    if (lane == 0) {
      p.num_accepted[b] = -1;
      p.num_emitted[b] = 0;
      set_status(p.status, bad_in);
    }
    return;
  }
  int cur = 0, len = 1;
  if (lane == 0) {
    path[0] = 0;
    out[0] = tok[0];  // the root: lane 0 holds node 0
  }
  for (int step = 1; step < N; ++step) {
    const int want = s_arg[cur];
    const unsigned m0 = __ballot_sync(0xffffffffu, par[0] == cur && tok[0] == want);
    const unsigned m1 = __ballot_sync(0xffffffffu, par[1] == cur && tok[1] == want);
    int nxt = -1;
    if (m0) nxt = __ffs(m0) - 1;
    else if (m1) nxt = 32 + __ffs(m1) - 1;
    if (nxt < 0) break;
    const int t = __shfl_sync(0xffffffffu, nxt < 32 ? tok[0] : tok[1], nxt & 31);
    if (lane == 0) {
      path[len] = nxt;
      out[len] = t;
    }
    cur = nxt;
    ++len;
  }
  for (int c = len + lane; c < N; c += 32) path[c] = -1;
  if (lane == 0) out[len] = s_arg[cur];
  for (int c = len + 1 + lane; c <= N; c += 32) out[c] = -1;
  if (lane == 0) {
    p.num_accepted[b] = len - 1;
    p.num_emitted[b] = len + 1;
  }
}

// Flags of sequence b's commit inputs (0 = valid), evaluated by one full warp: kv_len
// within the table and at least num_nodes, num_accepted in [-1, num_nodes), a path that
// starts at the root and rises strictly inside the tree, and the pages of every moved row.
__device__ uint32_t tree_commit_check(const spec_tree_commit_args_t& a, int b, int lane) {
  const int N = a.num_nodes, P = a.page_size;
  const int kv = a.kv_len[b], na = a.num_accepted[b];
  if (kv < N || static_cast<int64_t>(kv) > static_cast<int64_t>(a.max_pages_per_seq) * P)
    return SPEC_FLAG_BAD_KV_LEN;
  if (na < -1 || na >= N) return SPEC_FLAG_BAD_TREE;
  const int ctx = kv - N;
  const int32_t* path = a.path + static_cast<int64_t>(b) * N;
  const int32_t* table = a.page_table + static_cast<int64_t>(b) * a.max_pages_per_seq;
  uint32_t f = 0;
  for (int d = lane; d <= na; d += 32) {
    const int s = path[d];
    if (d == 0 ? s != 0 : (s <= path[d - 1] || s >= N)) {
      f |= SPEC_FLAG_BAD_TREE;
    } else if (s != d) {
      const int ps = table[(ctx + s) / P], pd = table[(ctx + d) / P];
      if (ps < 0 || ps >= a.num_pages || pd < 0 || pd >= a.num_pages) f |= SPEC_FLAG_BAD_PAGE;
    }
  }
  return __reduce_or_sync(0xffffffffu, f);
}

// One block per (cache, KV head, sequence) moves that head's rows of the accepted path:
// row path[d] to block position d for d = 1 .. num_accepted. A source path[d] >= d may be
// another position's destination (path 0, 2, 3: position 1 reads slot 2, which position 2
// writes), so every source piece is loaded into registers before any is stored; that is
// the result of moving the rows one after another in increasing d, as no row is read
// after a lower position was written over it.
template <int D>
__global__ void __launch_bounds__(128) tree_compact_kernel(spec_tree_commit_args_t a) {
  constexpr int kPieces = D / 8;                          // 16-byte pieces of a row
  constexpr int kIter = (63 * kPieces + 127) / 128;       // num_accepted <= 63
  __shared__ uint32_t s_flags;
  const int which = blockIdx.x & 1, h = blockIdx.x >> 1, b = blockIdx.y, tid = threadIdx.x;
  if (tid < 32) {
    const uint32_t f = tree_commit_check(a, b, tid);
    if (tid == 0) s_flags = f;
  }
  __syncthreads();
  if (s_flags) {
    if (tid == 0 && blockIdx.x == 0 && a.status) set_status(a.status, s_flags);
    return;
  }
  const int N = a.num_nodes, P = a.page_size, H = a.num_kv_heads;
  const int na = a.num_accepted[b];
  if (na <= 0) return;
  const int ctx = a.kv_len[b] - N;
  const int32_t* path = a.path + static_cast<int64_t>(b) * N;
  const int32_t* table = a.page_table + static_cast<int64_t>(b) * a.max_pages_per_seq;
  uint4* cache = static_cast<uint4*>(which ? a.v_cache : a.k_cache);
  const int n = na * kPieces;
  // the piece's offset in uint4 units, or -1 where the row stays in place
  auto offset = [&](int i, bool src) -> int64_t {
    const int d = 1 + i / kPieces, c = i % kPieces, s = path[d];
    if (s == d) return -1;
    const int pos = ctx + (src ? s : d);
    return ((static_cast<int64_t>(table[pos / P]) * H + h) * P + pos % P) * kPieces + c;
  };
  uint4 r[kIter];
#pragma unroll
  for (int k = 0; k < kIter; ++k) {
    const int i = tid + k * 128;
    if (i < n) {
      const int64_t o = offset(i, true);
      if (o >= 0) r[k] = cache[o];
    }
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < kIter; ++k) {
    const int i = tid + k * 128;
    if (i < n) {
      const int64_t o = offset(i, false);
      if (o >= 0) cache[o] = r[k];
    }
  }
}

// One warp per sequence: kv_len = ctx + num_accepted + 1 where the inputs are valid.
__global__ void tree_commit_len_kernel(spec_tree_commit_args_t a) {
  const int b = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (b >= a.batch) return;
  const uint32_t f = tree_commit_check(a, b, lane);
  if (lane == 0 && f == 0) {
    const int na = a.num_accepted[b];
    a.kv_len[b] = a.kv_len[b] - a.num_nodes + (na >= 0 ? na + 1 : 0);
  }
}

// ---------------------------------------------------------------------------------
// The tree sampler. tree_build_kernel: grid (splits, positions, sequences) of 128-thread
// blocks. A block ranks the candidates of its part of a drafter row: composite keys
// (order of the logit, then the lower token id) are unique, so the top-K of the part
// lie among the keys at or above the K-th largest per-thread maximum; those few are
// ranked by counting. The row's last part block merges the parts' sorted lists and
// the parts' (max, sum of exponentials) into the row's log-normaliser and writes the
// position's ranked (token, log q) table; the sequence's last row block selects the
// tree's nodes best first, one warp holding the offers of two nodes per lane (path
// scores are fp64 sums of the fp32 log q).
// ---------------------------------------------------------------------------------
struct BuildParams {
  int batch, gamma, vocab, rows, keff, nodes, splits, eps;
  const void* logits;
  const float* temperature;
  const int32_t* root;
  int32_t* tokens;
  int32_t* parents;
  int32_t* depth;
  uint64_t* mask;
  uint32_t* status;
  uint32_t* tickets;
  uint32_t* seq_flags;
  uint32_t* row_tickets;
  unsigned long long* keys;
  float4* stats;
  int2* table;
};

constexpr int kPartUnroll = 4;

__device__ __forceinline__ unsigned long long cand_key(float x, int idx) {
  return (static_cast<unsigned long long>(order_key(x)) << 32) | (0xffffffffu - static_cast<uint32_t>(idx));
}
__device__ __forceinline__ float key_value(unsigned long long k) {
  const uint32_t h = static_cast<uint32_t>(k >> 32);
  return __uint_as_float((h & 0x80000000u) ? (h & 0x7fffffffu) : ~h);
}
__device__ __forceinline__ int key_index(unsigned long long k) {
  return static_cast<int>(0xffffffffu - static_cast<uint32_t>(k));
}

// (max, sum of 2^((x - max) c2)) pairs combined; a -inf max carries no mass
__device__ __forceinline__ void merge_ms(float& m, float& s, float m2, float s2, float c2) {
  const float M = fmaxf(m, m2);
  float t = 0.f;
  if (m > -INFINITY) t += s * ex2((m - M) * c2);
  if (m2 > -INFINITY) t += s2 * ex2((m2 - M) * c2);
  m = M;
  s = t;
}

// Calls f(x, index) on each of this thread's logits of [e_begin, e_end) of the row.
template <bool BF16, bool VEC, class F>
__device__ __forceinline__ void for_part(const char* rowp, int e_begin, int e_end, int tid, F&& f) {
  if (VEC) {
    constexpr int kEpv = BF16 ? 8 : 4;
    const uint4* rv = reinterpret_cast<const uint4*>(rowp);
    const int vbeg = e_begin / kEpv, vend = e_end / kEpv;
    for (int v0 = vbeg + tid; v0 < vend; v0 += kThreads * kPartUnroll) {
      uint4 dv[kPartUnroll];
#pragma unroll
      for (int k = 0; k < kPartUnroll; ++k) {
        const int vi = v0 + k * kThreads;
        if (vi < vend) dv[k] = __ldg(rv + vi);
      }
#pragma unroll
      for (int k = 0; k < kPartUnroll; ++k) {
        const int vi = v0 + k * kThreads;
        if (vi < vend) {
          const uint32_t wv[4] = {dv[k].x, dv[k].y, dv[k].z, dv[k].w};
#pragma unroll
          for (int q = 0; q < kEpv; ++q) {
            const float x = BF16 ? __uint_as_float((q & 1) ? (wv[q >> 1] & 0xffff0000u) : (wv[q >> 1] << 16))
                                 : __uint_as_float(wv[q]);
            f(x, vi * kEpv + q);
          }
        }
      }
    }
  } else {
    for (int e0 = e_begin + tid; e0 < e_end; e0 += kThreads * kPartUnroll) {
      float x[kPartUnroll];
#pragma unroll
      for (int k = 0; k < kPartUnroll; ++k) {
        const int ei = e0 + k * kThreads;
        x[k] = ei < e_end ? load_elem<BF16>(rowp, ei) : 0.f;
      }
#pragma unroll
      for (int k = 0; k < kPartUnroll; ++k)
        if (e0 + k * kThreads < e_end) f(x[k], e0 + k * kThreads);
    }
  }
}

__device__ __forceinline__ unsigned long long block_max_u64(unsigned long long v, unsigned long long* s_red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long y = __shfl_xor_sync(0xffffffffu, v, o);
    v = y > v ? y : v;
  }
  __syncthreads();
  if ((threadIdx.x & 31) == 0) s_red[threadIdx.x >> 5] = v;
  __syncthreads();
  v = s_red[0];
#pragma unroll
  for (int k = 1; k < kThreads / 32; ++k) v = s_red[k] > v ? s_red[k] : v;
  return v;
}

struct TreeNode {
  int dep, nx, tok, par;   // dep < 0: no node in this slot
  double sc, osc;          // path score; score of the current offer (sums of fp32 log q)
  int otk;                 // token of the current offer
  unsigned long long key;  // order key of the offer's score, 0 if none
  unsigned long long msk;  // ancestor bits
};

__device__ __forceinline__ unsigned long long order_key64(double x) {
  unsigned long long f = static_cast<unsigned long long>(__double_as_longlong(x));
  if (f == 0x8000000000000000ull) f = 0ull;
  return (f >> 63) ? ~f : (f | 0x8000000000000000ull);
}

// The node's next offer: its candidate nx of position dep + 1 (table row dep).
__device__ __forceinline__ void refresh_offer(TreeNode& n, const int2* tab, int rows, int K) {
  n.key = 0ull;
  if (n.dep >= 0 && n.dep < rows && n.nx < K) {
    const int2 e = tab[n.dep * K + n.nx];
    n.osc = n.sc + static_cast<double>(__int_as_float(e.y));
    n.otk = e.x;
    n.key = order_key64(n.osc);
  }
}

template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kThreads) tree_build_kernel(BuildParams p) {
  extern __shared__ unsigned long long s_dyn[];
  __shared__ unsigned long long s_tmax[kThreads];
  __shared__ unsigned long long s_tau;
  __shared__ float s_wm[kThreads / 32], s_ws[kThreads / 32];
  __shared__ int s_count, s_bad, s_last;
  __shared__ uint32_t s_flags;
  const int split = blockIdx.x, r = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int K = p.keff, S = p.splits;
  const int64_t rid = static_cast<int64_t>(b) * p.rows + r;
  const char* rowp = static_cast<const char*>(p.logits) +
                     (static_cast<int64_t>(b) * p.gamma + r + 1) * p.vocab * (BF16 ? 2 : 4);
  const int e_begin = split * p.eps, e_end = min(p.vocab, e_begin + p.eps);
  const float T = p.temperature[b];
  const float invT = 1.f / (T > 0.f ? T : 1.f);
  const float c2 = invT * kLog2e;
  if (tid == 0) {
    s_tau = 0ull;
    s_count = 0;
    s_bad = 0;
  }
  __syncthreads();

  // pass 1: the thread's largest key, its (max, sum), NaN or +inf seen
  unsigned long long kmax = 0ull;
  float m = -INFINITY, s = 0.f;
  bool bad = false;
  for_part<BF16, VEC>(rowp, e_begin, e_end, tid, [&](float x, int i) {
    bad |= !(x < INFINITY);
    const unsigned long long k = cand_key(x, i);
    kmax = k > kmax ? k : kmax;
    if (x > m) {
      s = s * ex2((m - x) * c2) + 1.f;
      m = x;
    } else if (x > -INFINITY) {
      s += ex2((x - m) * c2);
    }
  });
  s_tmax[tid] = kmax;
  if (bad) s_bad = 1;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
    merge_ms(m, s, m2, s2, c2);
  }
  if ((tid & 31) == 0) {
    s_wm[tid >> 5] = m;
    s_ws[tid >> 5] = s;
  }
  __syncthreads();
  // tau: the K-th largest thread maximum (0 where fewer threads hold logits); the part's
  // top K keys are among the keys >= tau, which lie in the K threads at or above it
  {
    int rank = 0;
    for (int j = 0; j < kThreads; ++j) rank += s_tmax[j] > kmax;
    if (rank == K - 1) s_tau = kmax;
  }
  __syncthreads();
  const unsigned long long tau = s_tau;
  for_part<BF16, VEC>(rowp, e_begin, e_end, tid, [&](float x, int i) {
    const unsigned long long k = cand_key(x, i);
    if (k >= tau) {
      const int slot = atomicAdd(&s_count, 1);
      if (slot < kTreeCandCap) s_dyn[slot] = k;
    }
  });
  __syncthreads();
  const int C = s_count;
  unsigned long long* out = p.keys + (rid * S + split) * 64;
  if (C <= kTreeCandCap) {
    for (int i = tid; i < C; i += kThreads) {
      const unsigned long long k = s_dyn[i];
      int rk = 0;
      for (int j = 0; j < C; ++j) rk += s_dyn[j] > k;
      if (rk < K) out[rk] = k;
    }
    for (int i = C + tid; i < K; i += kThreads) out[i] = 0ull;
  } else {
    // many keys at the threshold (an adversarial order): K exact rounds instead
    unsigned long long prev = ~0ull;
    for (int rk = 0; rk < K; ++rk) {
      unsigned long long best = 0ull;
      for_part<BF16, VEC>(rowp, e_begin, e_end, tid, [&](float x, int i) {
        const unsigned long long k = cand_key(x, i);
        if (k < prev && k > best) best = k;
      });
      best = block_max_u64(best, s_tmax);
      if (tid == 0) out[rk] = best;
      prev = best;
    }
  }
  if (tid == 0) {
    float M = s_wm[0], Sum = s_ws[0];
    for (int w = 1; w < kThreads / 32; ++w) merge_ms(M, Sum, s_wm[w], s_ws[w], c2);
    p.stats[rid * S + split] = make_float4(M, Sum, __uint_as_float(static_cast<uint32_t>(s_bad)), 0.f);
  }

  // the row's last part block: merge the parts' lists and normalisers
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const uint32_t prev = atomicAdd(&p.row_tickets[rid], 1u);
    s_last = prev == static_cast<uint32_t>(S - 1);
    if (s_last) p.row_tickets[rid] = 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  unsigned long long* in = s_dyn;
  unsigned long long* nxt = s_dyn + S * K;
  for (int i = tid; i < S * K; i += kThreads)
    in[i] = __ldcg(p.keys + (rid * S + i / K) * 64 + i % K);
  __syncthreads();
  // pairwise merges of sorted (descending) lists, each kept to its top K: a key's place
  // is its place in its list plus the keys of the partner list above it (ties, only
  // the zero padding, go to the even list)
  for (int n = S; n > 1; n = (n + 1) / 2) {
    for (int t = tid; t < n * K; t += kThreads) {
      const int l = t / K, i = t % K, partner = l ^ 1;
      const unsigned long long key = in[t];
      if (partner >= n) {
        nxt[(l >> 1) * K + i] = key;
        continue;
      }
      const unsigned long long* P = in + partner * K;
      int lo = 0, hi = K;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if ((l & 1) ? P[mid] >= key : P[mid] > key) lo = mid + 1;
        else hi = mid;
      }
      if (i + lo < K) nxt[(l >> 1) * K + i + lo] = key;
    }
    __syncthreads();
    unsigned long long* t2 = in;
    in = nxt;
    nxt = t2;
  }
  if (tid < 32) {
    float M = -INFINITY, Sum = 0.f;
    uint32_t anybad = 0;
    for (int l = tid; l < S; l += 32) {
      const float4 st = __ldcg(p.stats + rid * S + l);
      merge_ms(M, Sum, st.x, st.y, c2);
      anybad |= __float_as_uint(st.z);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, M, o), s2 = __shfl_xor_sync(0xffffffffu, Sum, o);
      merge_ms(M, Sum, m2, s2, c2);
    }
    anybad = __reduce_or_sync(0xffffffffu, anybad);
    if (tid == 0) {
      s_wm[0] = M;
      s_ws[0] = Sum;
      s_bad = (anybad || !(M > -INFINITY)) ? 1 : 0;
    }
  }
  __syncthreads();
  {
    const float M = s_wm[0], lnS = logf(s_ws[0]);
    // log q = (x - max) / T - log sum exp((x_j - max) / T)
    if (tid < K) {
      const unsigned long long k = in[tid];
      p.table[rid * 64 + tid] = make_int2(key_index(k), __float_as_int((key_value(k) - M) * invT - lnS));
    }
    if (tid == 0 && s_bad) atomicOr(&p.seq_flags[b], SPEC_FLAG_BAD_LOGITS);
  }

  // the sequence's last row block selects the nodes
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const uint32_t prev = atomicAdd(&p.tickets[b], 1u);
    s_last = prev == static_cast<uint32_t>(p.rows - 1);
    if (s_last) p.tickets[b] = 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  int2* tab = reinterpret_cast<int2*>(s_dyn);
  for (int i = tid; i < p.rows * K; i += kThreads)
    tab[i] = __ldcg(p.table + (static_cast<int64_t>(b) * p.rows + i / K) * 64 + i % K);
  if (tid == 0) {
    uint32_t f = __ldcg(p.seq_flags + b);
    p.seq_flags[b] = 0;
    const int rt = p.root[b];
    if (rt < 0 || rt >= p.vocab) f |= SPEC_FLAG_BAD_TOKEN;
    s_flags = f;
  }
  __syncthreads();
  if (tid >= 32) return;
  const int lane = tid, N = p.nodes;
  const int64_t base = static_cast<int64_t>(b) * N;
  uint32_t flags = s_flags;
  TreeNode n0, n1;
  n0.dep = n1.dep = -1;
  n0.key = n1.key = 0ull;
  n0.nx = n1.nx = 0;
  n0.tok = n1.tok = -1;
  n0.par = n1.par = -1;
  n0.msk = n1.msk = 0ull;
  n0.sc = n1.sc = 0.0;
  if (!flags) {
    if (lane == 0) {
      n0.dep = 0;
      n0.tok = p.root[b];
      n0.msk = 1ull;
      refresh_offer(n0, tab, p.rows, K);
    }
    for (int i = 1; i < N; ++i) {
      // the best offer: the largest key, then the lowest node index
      const unsigned long long kl = n0.key > n1.key ? n0.key : n1.key;
      const uint32_t Mh = __reduce_max_sync(0xffffffffu, static_cast<uint32_t>(kl >> 32));
      const uint32_t Ml = __reduce_max_sync(
          0xffffffffu, static_cast<uint32_t>(kl >> 32) == Mh ? static_cast<uint32_t>(kl) : 0u);
      const unsigned long long M = (static_cast<unsigned long long>(Mh) << 32) | Ml;
      if (M == 0ull) {  // no offer left: excluded by the host's capacity check
        flags |= SPEC_FLAG_BAD_TREE;
        break;
      }
      const unsigned b0 = __ballot_sync(0xffffffffu, n0.key == M);
      const int u = b0 ? __ffs(b0) - 1 : 32 + __ffs(__ballot_sync(0xffffffffu, n1.key == M)) - 1;
      const int src = u & 31;
      const bool hs = u >= 32;
      const double osc = __shfl_sync(0xffffffffu, hs ? n1.osc : n0.osc, src);
      const int otk = __shfl_sync(0xffffffffu, hs ? n1.otk : n0.otk, src);
      const int pdep = __shfl_sync(0xffffffffu, hs ? n1.dep : n0.dep, src);
      const unsigned long long pm = __shfl_sync(0xffffffffu, hs ? n1.msk : n0.msk, src);
      if (lane == src) {
        if (hs) {
          ++n1.nx;
          refresh_offer(n1, tab, p.rows, K);
        } else {
          ++n0.nx;
          refresh_offer(n0, tab, p.rows, K);
        }
      }
      if (lane == (i & 31)) {
        TreeNode c;
        c.dep = pdep + 1;
        c.nx = 0;
        c.tok = otk;
        c.par = u;
        c.sc = osc;
        c.msk = pm | (1ull << i);
        refresh_offer(c, tab, p.rows, K);
        if (i >= 32) n1 = c;
        else n0 = c;
      }
    }
  }
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int c = lane + 32 * h;
    if (c >= N) continue;
    const TreeNode& n = h ? n1 : n0;
    p.tokens[base + c] = flags ? -1 : n.tok;
    p.parents[base + c] = flags ? -1 : n.par;
    if (p.depth) p.depth[base + c] = flags ? -1 : n.dep;
    if (p.mask) p.mask[base + c] = flags ? 0ull : n.msk;
  }
  if (lane == 0 && flags) set_status(p.status, flags);
}

// num_nodes = 1: the tree is its root
__global__ void tree_root_kernel(BuildParams p) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= p.batch) return;
  const int rt = p.root[b];
  const bool ok = rt >= 0 && rt < p.vocab;
  p.tokens[b] = ok ? rt : -1;
  p.parents[b] = -1;
  if (p.depth) p.depth[b] = ok ? 0 : -1;
  if (p.mask) p.mask[b] = ok ? 1ull : 0ull;
  if (!ok) set_status(p.status, SPEC_FLAG_BAD_TOKEN);
}

template <bool BF16, bool VEC>
cudaError_t launch_build_typed(const BuildParams& p, int smem, cudaStream_t s) {
  tree_build_kernel<BF16, VEC><<<dim3(p.splits, p.rows, p.batch), kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

template <bool BF16, bool VEC>
cudaError_t launch_tree_typed(const TreeParams& p, cudaStream_t s) {
  tree_greedy_kernel<BF16, VEC><<<dim3(p.splits, p.nodes, p.batch), kThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_tree_greedy(const spec_tree_accept_args_t& a, const TreeLayout& L, char* ws,
                               cudaStream_t stream, bool vec) {
  TreeParams p;
  p.batch = a.batch;
  p.nodes = a.num_nodes;
  p.vocab = a.vocab;
  p.splits = L.splits;
  p.elems_per_split = L.elems_per_split;
  p.target = a.target_logits;
  p.tokens = a.tokens;
  p.parents = a.parents;
  p.path = a.path;
  p.num_accepted = a.num_accepted;
  p.out_tokens = a.out_tokens;
  p.num_emitted = a.num_emitted;
  p.status = reinterpret_cast<uint32_t*>(ws);
  p.tickets = reinterpret_cast<uint32_t*>(ws + L.tickets);
  p.row_tickets = reinterpret_cast<uint32_t*>(ws + L.row_tickets);
  p.parts = reinterpret_cast<uint4*>(ws + L.parts);
  p.argmax = reinterpret_cast<int32_t*>(ws + L.argmax);
  (void)cudaGetLastError();
  if (a.logits_dtype == SPEC_BF16)
    return vec ? launch_tree_typed<true, true>(p, stream) : launch_tree_typed<true, false>(p, stream);
  return vec ? launch_tree_typed<false, true>(p, stream) : launch_tree_typed<false, false>(p, stream);
}

cudaError_t launch_tree_commit(const spec_tree_commit_args_t& a, cudaStream_t stream) {
  (void)cudaGetLastError();
  const dim3 grid(2 * a.num_kv_heads, a.batch);
  if (a.head_dim == 64)
    tree_compact_kernel<64><<<grid, 128, 0, stream>>>(a);
  else
    tree_compact_kernel<128><<<grid, 128, 0, stream>>>(a);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  tree_commit_len_kernel<<<(a.batch + 7) / 8, 256, 0, stream>>>(a);
  return cudaGetLastError();
}

TreeBuildLayout tree_build_layout(const spec_tree_build_args_t& t, size_t base, int sms) {
  TreeBuildLayout L;
  const int budget = t.num_nodes - 1;
  L.rows = std::min(t.gamma - 1, budget);
  L.keff = std::min(std::min(t.top_k, t.vocab), std::max(budget, 1));
  const int lane = 64;  // split boundaries on 64 logits keep vector loads aligned
  const int nl = (t.vocab + lane - 1) / lane;
  const int64_t rows = static_cast<int64_t>(t.batch) * std::max(L.rows, 1);
  int64_t splits = (static_cast<int64_t>(kFiltBlocksPerSm) * sms + rows - 1) / rows;
  splits = std::max<int64_t>(1, std::min<int64_t>(splits, kFiltMaxSplits));
  if (splits > nl) splits = nl;
  L.elems_per_split = static_cast<int>((nl + splits - 1) / splits) * lane;
  L.splits = (t.vocab + L.elems_per_split - 1) / L.elems_per_split;
  const size_t nrows = static_cast<size_t>(t.batch) * std::max(L.rows, 1);
  L.tickets = base;
  L.seq_flags = ws_round(L.tickets + sizeof(uint32_t) * t.batch);
  L.row_tickets = ws_round(L.seq_flags + sizeof(uint32_t) * t.batch);
  L.keys = ws_round(L.row_tickets + sizeof(uint32_t) * nrows);
  L.stats = ws_round(L.keys + 64 * sizeof(uint64_t) * nrows * L.splits);
  L.table = ws_round(L.stats + 16 * nrows * L.splits);
  L.end = ws_round(L.table + 64 * 8 * nrows);
  const int k = L.keff;
  L.smem = static_cast<int>(8 * std::max(std::max(kTreeCandCap, 2 * L.splits * k), L.rows * k));
  return L;
}

cudaError_t launch_tree_build(const spec_tree_build_args_t& t, const TreeBuildLayout& L, char* ws,
                              cudaStream_t stream, bool vec) {
  BuildParams p;
  p.batch = t.batch;
  p.gamma = t.gamma;
  p.vocab = t.vocab;
  p.rows = L.rows;
  p.keff = L.keff;
  p.nodes = t.num_nodes;
  p.splits = L.splits;
  p.eps = L.elems_per_split;
  p.logits = t.drafter_logits;
  p.temperature = t.temperature;
  p.root = t.root_tokens;
  p.tokens = t.tokens;
  p.parents = t.parents;
  p.depth = t.depth;
  p.mask = t.tree_mask;
  p.status = reinterpret_cast<uint32_t*>(ws);
  p.tickets = reinterpret_cast<uint32_t*>(ws + L.tickets);
  p.seq_flags = reinterpret_cast<uint32_t*>(ws + L.seq_flags);
  p.row_tickets = reinterpret_cast<uint32_t*>(ws + L.row_tickets);
  p.keys = reinterpret_cast<unsigned long long*>(ws + L.keys);
  p.stats = reinterpret_cast<float4*>(ws + L.stats);
  p.table = reinterpret_cast<int2*>(ws + L.table);
  (void)cudaGetLastError();
  if (L.rows < 1) {
    tree_root_kernel<<<(t.batch + 127) / 128, 128, 0, stream>>>(p);
    return cudaGetLastError();
  }
  if (t.logits_dtype == SPEC_BF16)
    return vec ? launch_build_typed<true, true>(p, L.smem, stream) : launch_build_typed<true, false>(p, L.smem, stream);
  return vec ? launch_build_typed<false, true>(p, L.smem, stream) : launch_build_typed<false, false>(p, L.smem, stream);
}

}  // namespace specv
