// Tree verification (Sec. 4.2: more than one candidate is verified at once as a prefix
// tree under tree attention; Sec. 3.3, "Tree Sampler"): greedy acceptance along a
// candidate tree and the compaction of the accepted path's keys and values.
//
// tree_greedy_kernel: grid (splits, nodes, sequences) of 128-thread blocks. Each block
// finds the lowest-index argmax of its part of a node's target row; the row's last block
// (ticket) merges the parts, and the sequence's last block walks the tree from the root,
// moving to the child whose token is the current node's argmax.
//
// tree_compact_kernel: one block per (cache, KV head, sequence) moves the accepted
// path's key or value rows into consecutive positions after the context.
#include <cuda_bf16.h>

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

}  // namespace specv
