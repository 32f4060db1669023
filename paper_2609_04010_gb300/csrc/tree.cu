// Tree verification (Sec. 4.2: more than one candidate is verified at once as a prefix
// tree under tree attention; Sec. 3.3, "Tree Sampler"): the tree sampler that builds the
// candidate tree from the drafter's rows, greedy acceptance along it, and the
// compaction of the accepted path's keys and values.
//
// tree_greedy_kernel (tree acceptance): grid (splits, nodes, sequences) of 128-thread
// blocks. Each block finds the lowest-index argmax of its part of a node's target row
// and, for a tempered sequence, the part's sum of 2^((l - max) log2e / T); the row's
// last block (ticket) merges the parts, and the sequence's last block walks the tree
// from the root. Greedy: to the child whose token is the current node's argmax.
// Sampled: the children are tried in node order as point-mass proposals (accepted iff
// u <= p'(token), p' without the siblings rejected before), decided in fp64 from the
// gathered logits (every node's weight under its parent's row and its earlier siblings'
// weight are taken once, before the walk, so a step is a shuffle, a division and two
// ballots); after the last rejection the block draws the final token from p' by
// inverse CDF: the part where the remaining mass crosses u x total, from the stored part
// sums minus the rejected tokens' weights, then one pass over that part.
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

// Row blocks of the tree acceptance kernel resident per SM (80 registers a thread).
constexpr int kTreeBlocksPerSm = 6;

TreeLayout tree_layout(int batch, int nodes, int vocab, size_t base, int sms, bool vec) {
  TreeLayout L;
  const int lane = vec ? 64 : 32;
  const int nlanes = (vocab + lane - 1) / lane;
  const int64_t rows = static_cast<int64_t>(batch) * nodes;
  int64_t splits = (static_cast<int64_t>(kTreeBlocksPerSm) * sms + rows - 1) / rows;
  splits = splits < 1 ? 1 : (splits > kFiltMaxSplits ? kFiltMaxSplits : splits);
  if (splits > nlanes) splits = nlanes;
  L.elems_per_split = static_cast<int>((nlanes + splits - 1) / splits) * lane;
  L.splits = (vocab + L.elems_per_split - 1) / L.elems_per_split;
  L.tickets = base;
  L.row_tickets = ws_round(L.tickets + sizeof(uint32_t) * batch);
  L.parts = ws_round(L.row_tickets + sizeof(uint32_t) * rows);
  L.argmax = ws_round(L.parts + 16 * rows * L.splits);
  L.rowstat = ws_round(L.argmax + sizeof(int32_t) * rows);
  L.end = ws_round(L.rowstat + sizeof(float) * 2 * rows);
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
  int32_t* argmax;         // [batch][nodes]; -1 marks an unusable row
  float2* rowstat;         // [batch][nodes]: (max logit, sum of 2^((l - max) log2e / T))
  const float* temperature;  // [batch] or NULL (greedy)
  const float* uniforms;     // [batch][nodes]
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
// The float whose order_key is k.
__device__ __forceinline__ float key_to_float(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}
// 2^((x - m) * c) for a running reference m (an all -inf prefix has m = -inf and weight 0).
__device__ __forceinline__ float rel_weight(float x, float m, float c) {
  return m == -INFINITY ? 0.f : ex2((x - m) * c);
}

template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kThreads, kTreeBlocksPerSm) tree_greedy_kernel(TreeParams p) {
  __shared__ unsigned long long s_red[kThreads / 32];
  __shared__ float s_fsum[kThreads / 32];
  __shared__ int s_bad, s_last;
  __shared__ int s_arg[64];
  // hand-off from the walking warp to the sampled final draw
  __shared__ int s_final, s_len, s_nrm, s_kcross, s_tok;
  __shared__ int s_rm[64];                 // tokens rejected at the final node, ascending
  __shared__ float s_rmw[64];              // their weights 2^((l - M) log2e / T)
  __shared__ int s_rmk[64];                // their parts of the row
  __shared__ double s_target, s_dsum[kThreads / 32];
  const int split = blockIdx.x, j = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int N = p.nodes, V = p.vocab;
  const int64_t rid = static_cast<int64_t>(b) * N + j;
  const char* rowp = static_cast<const char*>(p.target) + rid * V * (BF16 ? 2 : 4);
  const int e_begin = split * p.elems_per_split, e_end = min(V, e_begin + p.elems_per_split);
  const float T = p.temperature ? p.temperature[b] : 0.f;
  const bool tempered = T > 0.f;
  const float cs = tempered ? kLog2e / T : 0.f;
  if (tid == 0) s_bad = 0;
  __syncthreads();

  // the lowest-index maximum of this part of the row and, for a tempered sequence, the
  // sum of 2^((l - max) log2e / T) over it (rescaled whenever the running maximum grows)
  float m = -INFINITY, sum = 0.f;
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
      auto val = [&](int k, int q) {
        const uint32_t wv[4] = {dv[k].x, dv[k].y, dv[k].z, dv[k].w};
        return BF16 ? __uint_as_float((q & 1) ? (wv[q >> 1] & 0xffff0000u) : (wv[q >> 1] << 16))
                    : __uint_as_float(wv[q]);
      };
      const float m_old = m;
#pragma unroll
      for (int k = 0; k < kUnroll; ++k) {
        const int vi = v0 + k * kThreads + tid;
#pragma unroll
        for (int q = 0; q < kEpv; ++q) {
          const float x = val(k, q);
          bad |= x != x || (tempered && x == INFINITY);
          if (x > m) { m = x; a = vi * kEpv + q; }
        }
      }
      if (tempered) {
        sum = m_old == -INFINITY ? 0.f : sum * ex2((m_old - m) * cs);
#pragma unroll
        for (int k = 0; k < kUnroll; ++k)
#pragma unroll
          for (int q = 0; q < kEpv; ++q) sum += rel_weight(val(k, q), m, cs);
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
      const float m_old = m;
#pragma unroll
      for (int k = 0; k < kUnroll; ++k) {
        bad |= x[k] != x[k] || (tempered && x[k] == INFINITY);
        if (x[k] > m) { m = x[k]; a = e0 + k * kThreads + tid; }
      }
      if (tempered) {
        sum = m_old == -INFINITY ? 0.f : sum * ex2((m_old - m) * cs);
#pragma unroll
        for (int k = 0; k < kUnroll; ++k) sum += rel_weight(x[k], m, cs);
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
  float part_sum = 0.f;
  if (tempered) {
    // the part's sum relative to its maximum
    const float pm = key_to_float(static_cast<uint32_t>(best >> 32));
    float v = (pm == -INFINITY || !(pm < INFINITY)) ? 0.f : sum * rel_weight(m, pm, cs) * (m == -INFINITY ? 0.f : 1.f);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();  // s_red is read above by every thread
    if ((tid & 31) == 0) s_fsum[tid >> 5] = v;
    __syncthreads();
    for (int k = 0; k < kThreads / 32; ++k) part_sum += s_fsum[k];
  }

  float2 stat = make_float2(key_to_float(static_cast<uint32_t>(best >> 32)), part_sum);
  if (p.splits > 1 || tempered) {
    if (tid == 0)
      p.parts[rid * p.splits + split] = make_uint4(static_cast<uint32_t>(best), static_cast<uint32_t>(best >> 32),
                                                   static_cast<uint32_t>(s_bad), __float_as_uint(part_sum));
  }
  if (p.splits > 1) {
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
      // the row's sum relative to its maximum
      const float M = key_to_float(static_cast<uint32_t>(bb >> 32));
      float z = 0.f;
      if (tempered && M > -INFINITY && M < INFINITY) {
        for (int k = tid; k < p.splits; k += 32) {
          const uint4 q = __ldcg(p.parts + rid * p.splits + k);
          z += __uint_as_float(q.w) * rel_weight(key_to_float(q.y), M, cs);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
      }
      if (tid == 0) {
        s_red[0] = bb;
        s_bad = anybad ? 1 : 0;
        s_fsum[0] = z;
      }
    }
    __syncthreads();
    best = s_red[0];
    stat = make_float2(key_to_float(static_cast<uint32_t>(best >> 32)), s_fsum[0]);
  }
  if (tid == 0) {
    // a tempered row needs a finite maximum (NaN and +inf are flagged above)
    const bool unusable = s_bad || (tempered && !(stat.x > -INFINITY));
    p.argmax[rid] = unusable ? -1 : static_cast<int>(0xffffffffu - static_cast<uint32_t>(best));
    if (tempered) p.rowstat[rid] = stat;
  }

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
  if (tid == 0) s_final = -1;
  __syncthreads();
  const int64_t brow = static_cast<int64_t>(b) * N;
  int32_t* path = p.path + brow;
  int32_t* out = p.out_tokens + static_cast<int64_t>(b) * (N + 1);
  if (tid < 32) {
    // one warp: lane c holds node c (N <= 64: two nodes per lane)
    const int lane = tid;
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
    if (bad_in) {
      for (int c = lane; c < N; c += 32) path[c] = -1;
      for (int c = lane; c <= N; c += 32) out[c] = -1;
      if (lane == 0) {
        p.num_accepted[b] = -1;
        p.num_emitted[b] = 0;
        set_status(p.status, bad_in);
      }
    } else {
      int cur = 0, len = 1;
      if (lane == 0) {
        path[0] = 0;
        out[0] = tok[0];  // the root: lane 0 holds node 0
      }
      if (!tempered) {
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
      } else {
        // sampled walk: the children of the current node, in node order, are point-mass
        // proposals; child c is accepted iff u[c] <= p'(token), p' the node's target
        // distribution without the tokens of the siblings rejected before it.
        // Everything a step reads is fixed by the tree, so it is gathered once, for all
        // nodes at the same time: each node's weight e_c = exp((l(t_c) - M) / T) in fp64
        // under its parent's row (M that row's maximum; 0 for a repeated sibling token,
        // removed with its first occurrence), the weight of its earlier siblings in node
        // order, its own row's (maximum, sum) and its uniform.
        const char* tbase = static_cast<const char*>(p.target);
        const size_t rbytes = static_cast<size_t>(V) * (BF16 ? 2 : 4);
        double e[2];
        float2 own[2];
        float uu[2];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int c = lane + 32 * h;
          own[h] = c < N ? __ldcg(p.rowstat + brow + c) : make_float2(0.f, 0.f);
          uu[h] = c < N ? p.uniforms[brow + c] : 1.f;
          e[h] = 0.0;
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int c = lane + 32 * h;
          if (c >= 1 && c < N) {
            const float2 prs = __ldcg(p.rowstat + brow + par[h]);
            const float x = load_elem<BF16>(tbase + (brow + par[h]) * rbytes, tok[h]);
            e[h] = exp((static_cast<double>(x) - prs.x) / static_cast<double>(T));
          }
        }
        bool dup[2] = {false, false};
        for (int o = 0; o < 64; ++o) {
          const int t_o = __shfl_sync(0xffffffffu, o < 32 ? tok[0] : tok[1], o & 31);
          const int p_o = __shfl_sync(0xffffffffu, o < 32 ? par[0] : par[1], o & 31);
#pragma unroll
          for (int h = 0; h < 2; ++h) dup[h] |= o < lane + 32 * h && p_o == par[h] && t_o == tok[h];
        }
        int live[2];  // a proposal with weight (not a repeat)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          if (dup[h]) e[h] = 0.0;
          live[h] = e[h] > 0.0 ? 1 : 0;
        }
        for (int step = 1; step <= N; ++step) {
          const float s_cur = __shfl_sync(0xffffffffu, cur < 32 ? own[0].y : own[1].y, cur & 31);
          bool ch[2], acc[2];
          double w[2];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            ch[h] = par[h] == cur;
            w[h] = ch[h] ? e[h] : 0.0;
          }
          // mass removed before each child: exclusive prefix over node order
          double inc0 = w[0], inc1 = w[1];
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const double y0 = __shfl_up_sync(0xffffffffu, inc0, o);
            const double y1 = __shfl_up_sync(0xffffffffu, inc1, o);
            if (lane >= o) { inc0 += y0; inc1 += y1; }
          }
          const double tot0 = __shfl_sync(0xffffffffu, inc0, 31);
          const double ex0 = inc0 - w[0], ex1 = tot0 + inc1 - w[1];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const double S = static_cast<double>(s_cur) - (h == 0 ? ex0 : ex1);
            acc[h] = ch[h] && live[h] &&
                     (S <= w[h] || static_cast<double>(uu[h]) <= w[h] / S);
          }
          const unsigned m0 = __ballot_sync(0xffffffffu, acc[0]);
          const unsigned m1 = __ballot_sync(0xffffffffu, acc[1]);
          int nxt = -1;
          if (m0) nxt = __ffs(m0) - 1;
          else if (m1) nxt = 32 + __ffs(m1) - 1;
          if (nxt >= 0) {
            const int t = __shfl_sync(0xffffffffu, nxt < 32 ? tok[0] : tok[1], nxt & 31);
            if (lane == 0) {
              path[len] = nxt;
              out[len] = t;
            }
            cur = nxt;
            ++len;
            continue;
          }
          const float m_cur = __shfl_sync(0xffffffffu, cur < 32 ? own[0].x : own[1].x, cur & 31);
          const char* crow = tbase + (brow + cur) * rbytes;
          // every child rejected: hand the final node and its rejected tokens (ascending,
          // with their weights relative to the row maximum) to the whole block
          float wrm[2];
#pragma unroll
          for (int h = 0; h < 2; ++h)
            wrm[h] = ch[h] && live[h] ? rel_weight(load_elem<BF16>(crow, tok[h]), m_cur, cs) : 0.f;
          int rank[2] = {0, 0};
          for (int o = 0; o < 64; ++o) {
            const int t_o = __shfl_sync(0xffffffffu, o < 32 ? tok[0] : tok[1], o & 31);
            const int p_o = __shfl_sync(0xffffffffu, o < 32 ? par[0] : par[1], o & 31);
            const int l_o = __shfl_sync(0xffffffffu, o < 32 ? live[0] : live[1], o & 31);
            const bool in = p_o == cur && l_o;
#pragma unroll
            for (int h = 0; h < 2; ++h)
              rank[h] += in && (t_o < tok[h] || (t_o == tok[h] && o < lane + 32 * h));
          }
#pragma unroll
          for (int h = 0; h < 2; ++h)
            if (ch[h] && live[h]) {
              s_rm[rank[h]] = tok[h];
              s_rmw[rank[h]] = wrm[h];
              s_rmk[rank[h]] = tok[h] / p.elems_per_split;
            }
          const int nrm = __popc(__ballot_sync(0xffffffffu, ch[0] && live[0])) +
                          __popc(__ballot_sync(0xffffffffu, ch[1] && live[1]));
          if (lane == 0) {
            s_final = cur;
            s_len = len;
            s_nrm = nrm;
          }
          break;
        }
        for (int c = len + lane; c < N; c += 32) path[c] = -1;
      }
    }
  }
  __syncthreads();
  if (s_final < 0) return;  // greedy, bad input: done

  // ---- the final draw from p' of node s_final: inverse CDF in ascending token order ----
  const int fin = s_final, len = s_len, nrm = s_nrm;
  const int64_t frid = brow + fin;
  const float M = __ldcg(p.rowstat + frid).x;
  const int eps = p.elems_per_split;
  if (tid < 32) {
    // remaining mass of each part (its sum minus its rejected tokens' weights), the total,
    // and the part where the cumulative mass reaches u[0] x total: one part per lane
    // (at most kFiltMaxSplits parts)
    const int k = tid;
    double base = 0.0;
    if (k < p.splits) {
      const uint4 q = __ldcg(p.parts + frid * p.splits + k);
      base = static_cast<double>(__uint_as_float(q.w)) * rel_weight(key_to_float(q.y), M, cs);
    }
    double removed = 0.0;
    for (int r = 0; r < nrm; ++r)
      if (s_rmk[r] == k) removed += static_cast<double>(s_rmw[r]);
    double mass = base - removed;
    if (mass < 0.0) mass = 0.0;
    double S = mass;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) S += __shfl_xor_sync(0xffffffffu, S, o);
    if (!(S > 0.0)) {
      // nothing left after the removals (rounding only): draw from p itself
      mass = base;
      S = mass;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) S += __shfl_xor_sync(0xffffffffu, S, o);
      if (k == 0) s_nrm = 0;
    }
    const double target = static_cast<double>(p.uniforms[brow]) * S;
    double incl = mass;  // inclusive prefix over parts
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const double y = __shfl_up_sync(0xffffffffu, incl, o);
      if (k >= o) incl += y;
    }
    const double excl = incl - mass;
    const unsigned hit = __ballot_sync(0xffffffffu, mass > 0.0 && incl >= target);
    // rounding may leave the target above the total: then the last part with mass
    const unsigned pos = __ballot_sync(0xffffffffu, mass > 0.0);
    const int kc = hit ? __ffs(hit) - 1 : (pos ? 31 - __clz(pos) : -1);
    const double before = __shfl_sync(0xffffffffu, excl, kc < 0 ? 0 : kc);
    if (k == 0) {
      s_kcross = kc < 0 ? 0 : kc;  // the part of the row maximum always has mass
      s_target = target - before;
    }
  }
  __syncthreads();
  const int kc = s_kcross, nrm_scan = s_nrm;
  const double tin = s_target;
  // each thread a contiguous run of the crossing part (multiples of 8 elements)
  const int pb = kc * eps, pe = min(V, pb + eps);
  const int per = ((pe - pb + kThreads - 1) / kThreads + 7) / 8 * 8;
  const int lo = min(pe, pb + tid * per), hi = min(pe, lo + per);
  const char* frow = static_cast<const char*>(p.target) + frid * V * (BF16 ? 2 : 4);
  int ptr = 0;
  while (ptr < nrm_scan && s_rm[ptr] < lo) ++ptr;
  // The run is read kChunk elements at a time, all of a chunk's loads issued before any
  // is used (16-byte vectors when the rows allow: a run starts on a multiple of 8
  // elements, and hi is a multiple of the vector's elements).
  constexpr int kChunk = 16;
  auto load_chunk = [&](int x0, float* lv) {
    if (VEC) {
      constexpr int kEpv = BF16 ? 8 : 4;
#pragma unroll
      for (int v = 0; v < kChunk / kEpv; ++v) {
        const int x = x0 + v * kEpv;
        uint4 raw = make_uint4(0u, 0u, 0u, 0u);
        if (x < hi) raw = __ldg(reinterpret_cast<const uint4*>(frow + static_cast<int64_t>(x) * (BF16 ? 2 : 4)));
        const uint32_t wv[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
        for (int q = 0; q < kEpv; ++q)
          lv[v * kEpv + q] = BF16 ? __uint_as_float((q & 1) ? (wv[q >> 1] & 0xffff0000u) : (wv[q >> 1] << 16))
                                  : __uint_as_float(wv[q]);
      }
    } else {
#pragma unroll
      for (int i = 0; i < kChunk; ++i) lv[i] = x0 + i < hi ? load_elem<BF16>(frow, x0 + i) : 0.f;
    }
  };
  // The weight of element x from its logit l, 0 for a removed token. Elements come in
  // ascending order and the removed tokens are distinct and ascending, so the next one is
  // kept in a register.
  auto weight_of = [&](int x, float l, int& q, int& next_rm) {
    if (x == next_rm) {
      ++q;
      next_rm = q < nrm_scan ? s_rm[q] : INT_MAX;
      return 0.f;
    }
    return rel_weight(l, M, cs);
  };
  float run = 0.f;
  {
    int q = ptr, next_rm = ptr < nrm_scan ? s_rm[ptr] : INT_MAX;
    for (int x0 = lo; x0 < hi; x0 += kChunk) {
      float lv[kChunk];
      load_chunk(x0, lv);
#pragma unroll
      for (int i = 0; i < kChunk; ++i)
        if (x0 + i < hi) run += weight_of(x0 + i, lv[i], q, next_rm);
    }
  }
  // block exclusive scan of the runs' sums; the run that holds the crossing is the last
  // one with weight whose exclusive prefix is below the target
  double incl = static_cast<double>(run);
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const double y = __shfl_up_sync(0xffffffffu, incl, o);
    if ((tid & 31) >= o) incl += y;
  }
  double prev = __shfl_up_sync(0xffffffffu, incl, 1);
  if ((tid & 31) == 0) prev = 0.0;
  if ((tid & 31) == 31) s_dsum[tid >> 5] = incl;
  __syncthreads();
  double wbase = 0.0;
  for (int k = 0; k < (tid >> 5); ++k) wbase += s_dsum[k];
  const double excl = wbase + prev;
  int owner = (run > 0.f && excl < tin) ? tid : -1;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) owner = max(owner, __shfl_xor_sync(0xffffffffu, owner, o));
  __syncthreads();  // every thread has read s_dsum
  if ((tid & 31) == 0) s_fsum[tid >> 5] = __int_as_float(owner);
  __syncthreads();
  owner = -1;
  for (int k = 0; k < kThreads / 32; ++k) owner = max(owner, __float_as_int(s_fsum[k]));
  if (tid == owner) {
    // walk the run: the first token whose cumulative weight reaches the target, else (if
    // rounding leaves the target above the run) its last positive-weight token
    double C = excl;
    int q = ptr, next_rm = ptr < nrm_scan ? s_rm[ptr] : INT_MAX, pick = -1;
    bool done = false;
    for (int x0 = lo; x0 < hi && !done; x0 += kChunk) {
      float lv[kChunk];
      load_chunk(x0, lv);
      for (int i = 0; i < kChunk && !done && x0 + i < hi; ++i) {
        const float w = weight_of(x0 + i, lv[i], q, next_rm);
        C += static_cast<double>(w);
        if (w > 0.f) {
          pick = x0 + i;
          done = C >= tin;
        }
      }
    }
    s_tok = pick;
  }
  if (owner < 0 && tid == 0) s_tok = s_arg[fin];  // no weight left in fp32: the row maximum
  __syncthreads();
  if (tid == 0) {
    out[len] = s_tok;
    p.num_accepted[b] = len - 1;
    p.num_emitted[b] = len + 1;
  }
  for (int c = len + 1 + tid; c <= N; c += kThreads) out[c] = -1;
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
// scores are double-float sums of the fp32 log q).
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

// Calls f(x, base) on this thread's logits of [e_begin, e_end) of the row, a 16-byte
// group at a time (x[q] is logit base + q; groups of one where rows are not aligned).
template <bool BF16, bool VEC, class F>
__device__ __forceinline__ void for_groups(const char* rowp, int e_begin, int e_end, int tid, F&& f) {
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
          float x[kEpv];
#pragma unroll
          for (int q = 0; q < kEpv; ++q)
            x[q] = BF16 ? __uint_as_float((q & 1) ? (wv[q >> 1] & 0xffff0000u) : (wv[q >> 1] << 16))
                        : __uint_as_float(wv[q]);
          f(x, vi * kEpv);
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
      for (int k = 0; k < kPartUnroll; ++k) {
        const float one[1] = {x[k]};
        if (e0 + k * kThreads < e_end) f(one, e0 + k * kThreads);
      }
    }
  }
}

// Sorts one key per lane of the warp into descending order (bitonic network).
__device__ __forceinline__ unsigned long long warp_sort_desc(unsigned long long v, int lane) {
#pragma unroll
  for (int k = 2; k <= 32; k <<= 1) {
#pragma unroll
    for (int j = k >> 1; j > 0; j >>= 1) {
      const unsigned long long o = __shfl_xor_sync(0xffffffffu, v, j);
      const bool keep_max = ((lane & j) == 0) == ((lane & k) == 0);
      v = keep_max ? (o > v ? o : v) : (o < v ? o : v);
    }
  }
  return v;
}

// The 64 largest of two descending lists of 64 keys (a0, a1 and b0, b1: the lane's
// entries lane and lane + 32 of each), descending, as the lane's two entries. The elementwise
// maximum of one list and the other reversed is bitonic and holds the 64 largest; a
// bitonic merge (half-cleaners of 32, 16, .., 1) sorts it.
__device__ __noinline__ ulonglong2 merge_top64(unsigned long long a0, unsigned long long a1,
                                               unsigned long long b0, unsigned long long b1, int lane) {
  const unsigned long long rb0 = __shfl_sync(0xffffffffu, b1, 31 - lane);
  const unsigned long long rb1 = __shfl_sync(0xffffffffu, b0, 31 - lane);
  unsigned long long c0 = a0 > rb0 ? a0 : rb0;
  unsigned long long c1 = a1 > rb1 ? a1 : rb1;
  {
    const unsigned long long hi = c0 > c1 ? c0 : c1, lo = c0 > c1 ? c1 : c0;
    c0 = hi;
    c1 = lo;
  }
#pragma unroll
  for (int j = 16; j > 0; j >>= 1) {
    const unsigned long long o0 = __shfl_xor_sync(0xffffffffu, c0, j);
    const unsigned long long o1 = __shfl_xor_sync(0xffffffffu, c1, j);
    const bool lower = (lane & j) == 0;
    c0 = lower ? (c0 > o0 ? c0 : o0) : (c0 < o0 ? c0 : o0);
    c1 = lower ? (c1 > o1 ? c1 : o1) : (c1 < o1 ? c1 : o1);
  }
  return make_ulonglong2(c0, c1);
}

// x[q] for a q known only at run time, by selects (no local-memory copy of x).
template <int E>
__device__ __forceinline__ float pick(const float (&x)[E], int q) {
  float v = x[0];
#pragma unroll
  for (int j = 1; j < E; ++j) v = j == q ? x[j] : v;
  return v;
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

// (ah + al) + b as a normalised double-float (rh + rl): the exact sum of ah and b by
// Knuth's two-sum, then the low parts folded in (a fast two-sum). Path scores keep
// about 48 bits this way without fp64 arithmetic, whose latency is high on this part.
__device__ __forceinline__ void df_add(float ah, float al, float b, float& rh, float& rl) {
  const float s = __fadd_rn(ah, b);
  if (!(s > -INFINITY)) {  // a -inf term
    rh = s;
    rl = 0.f;
    return;
  }
  const float bb = __fsub_rn(s, ah);
  const float e = __fadd_rn(__fsub_rn(ah, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  const float t = __fadd_rn(e, al);
  rh = __fadd_rn(s, t);
  rl = __fsub_rn(t, __fsub_rn(rh, s));
}

struct TreeNode {
  int dep, nx, tok, par;   // dep < 0: no node in this slot
  float sh, sl;            // path score as an unevaluated sum sh + sl (double-float)
  float oh, ol;            // score of the current offer, the same way
  int otk;                 // token of the current offer
  unsigned long long key;  // order key of the offer's score, 0 if none
  unsigned long long msk;  // ancestor bits
};

// The node's next offer, its candidate nx of position dep + 1 (table row dep): its score
// (oh + ol) and token, and the key (0 if there is none) that orders normalised
// double-floats: high parts first, then low parts.
__device__ __forceinline__ unsigned long long offer_of(const TreeNode& n, const int2* tab, int rows, int K,
                                                       float& oh, float& ol, int& otk) {
  if (n.dep < 0 || n.dep >= rows || n.nx >= K) return 0ull;
  const int2 e = tab[n.dep * K + n.nx];
  df_add(n.sh, n.sl, __int_as_float(e.y), oh, ol);
  otk = e.x;
  return (static_cast<unsigned long long>(order_key(oh)) << 32) | order_key(ol);
}

// Best-first selection of the tree's nodes by one warp. The root (node 0) is kept in
// every lane; node c >= 1 is slot (c - 1) / 32 of lane (c - 1) % 32. Each step takes the
// best offer (largest high word of its key; on a tie the largest low word, then the
// lowest node index, the root first), makes it node i, and moves its parent to its next
// candidate.
template <int SLOTS>
__device__ __forceinline__ void select_nodes(const BuildParams& p, const int2* tab, int K, int b,
                                             uint32_t flags, int lane) {
  const int N = p.nodes;
  const int64_t base = static_cast<int64_t>(b) * N;
  TreeNode root, n[SLOTS];
  root.dep = 0;
  root.nx = 0;
  root.tok = flags ? -1 : p.root[b];
  root.par = -1;
  root.msk = 1ull;
  root.sh = root.sl = 0.f;
  root.oh = root.ol = 0.f;
  root.otk = -1;
  root.key = 0ull;
#pragma unroll
  for (int h = 0; h < SLOTS; ++h) {
    n[h].dep = -1;
    n[h].nx = 0;
    n[h].tok = -1;
    n[h].par = -1;
    n[h].msk = 0ull;
    n[h].sh = n[h].sl = 0.f;
    n[h].oh = n[h].ol = 0.f;
    n[h].otk = -1;
    n[h].key = 0ull;
  }
  if (!flags) {
    root.key = offer_of(root, tab, p.rows, K, root.oh, root.ol, root.otk);
    for (int i = 1; i < N; ++i) {
      const uint32_t rh = static_cast<uint32_t>(root.key >> 32);
      uint32_t hl = 0u;
#pragma unroll
      for (int h = 0; h < SLOTS; ++h) hl = max(hl, static_cast<uint32_t>(n[h].key >> 32));
      const uint32_t Mh = max(__reduce_max_sync(0xffffffffu, hl), rh);
      if (Mh == 0u) {  // no offer left: excluded by the host's capacity check
        flags |= SPEC_FLAG_BAD_TREE;
        break;
      }
      unsigned bal[SLOTS];
      int ties = rh == Mh;
#pragma unroll
      for (int h = 0; h < SLOTS; ++h) {
        bal[h] = __ballot_sync(0xffffffffu, static_cast<uint32_t>(n[h].key >> 32) == Mh);
        ties += __popc(bal[h]);
      }
      bool root_wins = rh == Mh;
      if (ties > 1) {
        const uint32_t rl = rh == Mh ? static_cast<uint32_t>(root.key) : 0u;
        uint32_t ll = 0u;
#pragma unroll
        for (int h = 0; h < SLOTS; ++h)
          if (static_cast<uint32_t>(n[h].key >> 32) == Mh) ll = max(ll, static_cast<uint32_t>(n[h].key));
        const uint32_t Ml = max(__reduce_max_sync(0xffffffffu, ll), rl);
        root_wins = rh == Mh && rl == Ml;
#pragma unroll
        for (int h = 0; h < SLOTS; ++h)
          bal[h] = __ballot_sync(0xffffffffu, static_cast<uint32_t>(n[h].key >> 32) == Mh &&
                                                  static_cast<uint32_t>(n[h].key) == Ml);
      }
      // the winner u and its offer (score, token), depth and ancestor bits
      int u = 0, hs = 0;
      if (!root_wins) {
#pragma unroll
        for (int h = SLOTS - 1; h >= 0; --h)
          if (bal[h]) {
            u = 1 + 32 * h + __ffs(bal[h]) - 1;
            hs = h;
          }
      }
      const int src = (u - 1) & 31;
      float oh = root.oh, ol = root.ol;
      int otk = root.otk, pdep = 0;
      unsigned long long pm = 1ull;
      {
        float soh = n[0].oh, sol = n[0].ol;
        int sotk = n[0].otk, sdep = n[0].dep;
        unsigned long long smsk = n[0].msk;
#pragma unroll
        for (int h = 1; h < SLOTS; ++h)
          if (hs == h) {
            soh = n[h].oh;
            sol = n[h].ol;
            sotk = n[h].otk;
            sdep = n[h].dep;
            smsk = n[h].msk;
          }
        soh = __shfl_sync(0xffffffffu, soh, src);
        sol = __shfl_sync(0xffffffffu, sol, src);
        sotk = __shfl_sync(0xffffffffu, sotk, src);
        sdep = __shfl_sync(0xffffffffu, sdep, src);
        smsk = __shfl_sync(0xffffffffu, smsk, src);
        if (u != 0) {
          oh = soh;
          ol = sol;
          otk = sotk;
          pdep = sdep;
          pm = smsk;
        }
      }
      // node i takes the offer; its parent moves to its next candidate
      const int ci = (i - 1) & 31, ch = (i - 1) >> 5;
#pragma unroll
      for (int h = 0; h < SLOTS; ++h) {
        const bool is_new = lane == ci && ch == h;
        const bool adv = u != 0 && lane == src && hs == h;
        if (is_new) {
          n[h].dep = pdep + 1;
          n[h].nx = 0;
          n[h].tok = otk;
          n[h].par = u;
          n[h].sh = oh;
          n[h].sl = ol;
          n[h].msk = pm | (1ull << i);
        }
        if (adv) ++n[h].nx;
        float ph = 0.f, pl = 0.f;
        int pt = -1;
        const unsigned long long k = offer_of(n[h], tab, p.rows, K, ph, pl, pt);
        if (is_new || adv) {
          n[h].key = k;
          n[h].oh = ph;
          n[h].ol = pl;
          n[h].otk = pt;
        }
      }
      if (u == 0) {
        ++root.nx;
        root.key = offer_of(root, tab, p.rows, K, root.oh, root.ol, root.otk);
      }
    }
  }
  if (lane == 0) {
    p.tokens[base] = flags ? -1 : root.tok;
    p.parents[base] = -1;
    if (p.depth) p.depth[base] = flags ? -1 : 0;
    if (p.mask) p.mask[base] = flags ? 0ull : 1ull;
  }
#pragma unroll
  for (int h = 0; h < SLOTS; ++h) {
    const int c = 1 + lane + 32 * h;
    if (c >= N) continue;
    p.tokens[base + c] = flags ? -1 : n[h].tok;
    p.parents[base + c] = flags ? -1 : n[h].par;
    if (p.depth) p.depth[base + c] = flags ? -1 : n[h].dep;
    if (p.mask) p.mask[base + c] = flags ? 0ull : n[h].msk;
  }
  if (lane == 0 && flags) set_status(p.status, flags);
}

template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kThreads) tree_build_kernel(BuildParams p) {
  extern __shared__ unsigned long long s_dyn[];
  __shared__ unsigned long long s_tmax[kThreads];
  __shared__ unsigned long long s_tau;
  __shared__ float s_wm[kThreads / 32], s_ws[kThreads / 32];
  __shared__ int s_wcnt[kThreads / 32];
  __shared__ int s_count, s_bad, s_last;
  __shared__ uint32_t s_flags;
  const int split = blockIdx.x, r = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int lane = tid & 31, w = tid >> 5;
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

  // pass 1, a 16-byte group at a time: the thread's maximum and its lowest index, the
  // sum of 2^((x - max) c2) (rescaled when the maximum rises), NaN or +inf seen (a NaN
  // sum, or a NaN among logits that are all -inf so far)
  float m = -INFINITY, s = 0.f;
  int mi = -1;
  bool nan_seen = false;
  for_groups<BF16, VEC>(rowp, e_begin, e_end, tid, [&](const auto& x, int base) {
    constexpr int E = sizeof(x) / sizeof(float);
    float vmax = x[0];
#pragma unroll
    for (int q = 1; q < E; ++q) vmax = fmaxf(vmax, x[q]);
    if (mi < 0) mi = base;  // the first logit: the maximum of a part of -inf
    if (vmax > m) {
      unsigned eq = 0u;
#pragma unroll
      for (int q = 0; q < E; ++q) eq |= (x[q] == vmax ? 1u : 0u) << q;
      const int q0 = __ffs(eq) - 1;
      s *= ex2((m - vmax) * c2);
      m = vmax;
      mi = base + q0;
    }
    if (m > -INFINITY) {
      const float mc = m * c2;
#pragma unroll
      for (int q = 0; q < E; ++q) s += ex2(fmaf(x[q], c2, -mc));
    } else {
#pragma unroll
      for (int q = 0; q < E; ++q) nan_seen |= x[q] != x[q];
    }
  });
  if (nan_seen || s != s) s_bad = 1;
  const unsigned long long L0 = mi >= 0 ? cand_key(m, mi) : 0ull;
  // tau: the K-th largest of the threads' maximum keys (0 if fewer threads hold
  // logits); the part's top K keys are among the keys >= tau. Each warp sorts its 32
  // keys; a key's rank is its place in its warp plus the keys above it in the others.
  {
    const unsigned long long v = warp_sort_desc(L0, lane);
    s_tmax[tid] = v;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
      merge_ms(m, s, m2, s2, c2);
    }
    if (lane == 0) {
      s_wm[w] = m;
      s_ws[w] = s;
    }
    __syncthreads();
    int rank = lane;
#pragma unroll
    for (int w2 = 0; w2 < kThreads / 32; ++w2) {
      if (w2 == w) continue;
      const unsigned long long* run = s_tmax + w2 * 32;
      int lo = 0, hi = 32;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (run[mid] > v) lo = mid + 1;
        else hi = mid;
      }
      rank += lo;
    }
    if (rank == K - 1) s_tau = v;
  }
  __syncthreads();
  const unsigned long long tau = s_tau;
  // pass 2: the keys >= tau (logit above tv, or equal with index at most ti), kept in
  // four registers per thread and placed by a block scan; a thread with more (or tau =
  // 0: every logit is one) sends the block to shared-memory atomics instead
  const float tv = tau ? key_value(tau) : -INFINITY;
  const int ti = tau ? key_index(tau) : INT_MAX;
  unsigned long long c0 = 0ull, c1 = 0ull, c2k = 0ull, c3 = 0ull;
  int cnt = 0;
  if (tau != 0ull) {
    for_groups<BF16, VEC>(rowp, e_begin, e_end, tid, [&](const auto& x, int base) {
      constexpr int E = sizeof(x) / sizeof(float);
      float vmax = x[0];
#pragma unroll
      for (int q = 1; q < E; ++q) vmax = fmaxf(vmax, x[q]);
      if (vmax >= tv) {
        unsigned cm = 0u;
#pragma unroll
        for (int q = 0; q < E; ++q)
          cm |= ((x[q] > tv || (x[q] == tv && base + q <= ti)) ? 1u : 0u) << q;
        while (cm) {
          const int q = __ffs(cm) - 1;
          cm &= cm - 1;
          const unsigned long long k = cand_key(pick(x, q), base + q);
          if (cnt == 0) c0 = k;
          else if (cnt == 1) c1 = k;
          else if (cnt == 2) c2k = k;
          else if (cnt == 3) c3 = k;
          ++cnt;
        }
      }
    });
  }
  if (!__syncthreads_or(tau == 0ull || cnt > 4)) {
    int incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) s_wcnt[w] = incl;
    __syncthreads();
    int off = incl - cnt;
    for (int w2 = 0; w2 < w; ++w2) off += s_wcnt[w2];
    if (cnt > 0) s_dyn[off] = c0;
    if (cnt > 1) s_dyn[off + 1] = c1;
    if (cnt > 2) s_dyn[off + 2] = c2k;
    if (cnt > 3) s_dyn[off + 3] = c3;
    if (tid == kThreads - 1) s_count = off + cnt;
  } else {
    for_groups<BF16, VEC>(rowp, e_begin, e_end, tid, [&](const auto& x, int base) {
      constexpr int E = sizeof(x) / sizeof(float);
      float vmax = x[0];
#pragma unroll
      for (int q = 1; q < E; ++q) vmax = fmaxf(vmax, x[q]);
      if (vmax >= tv) {
        unsigned cm = 0u;
#pragma unroll
        for (int q = 0; q < E; ++q)
          cm |= ((x[q] > tv || (x[q] == tv && base + q <= ti)) ? 1u : 0u) << q;
        while (cm) {
          const int q = __ffs(cm) - 1;
          cm &= cm - 1;
          const int slot = atomicAdd(&s_count, 1);
          if (slot < kTreeCandCap) s_dyn[slot] = cand_key(pick(x, q), base + q);
        }
      }
    });
  }
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
      for_groups<BF16, VEC>(rowp, e_begin, e_end, tid, [&](const auto& x, int base) {
        constexpr int E = sizeof(x) / sizeof(float);
#pragma unroll
        for (int q = 0; q < E; ++q) {
          const unsigned long long k = cand_key(x[q], base + q);
          if (k < prev && k > best) best = k;
        }
      });
      best = block_max_u64(best, s_tmax);
      if (tid == 0) out[rk] = best;
      prev = best;
    }
  }
  if (tid == 0) {
    float M = s_wm[0], Sum = s_ws[0];
    for (int w2 = 1; w2 < kThreads / 32; ++w2) merge_ms(M, Sum, s_wm[w2], s_ws[w2], c2);
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
  // warp w merges parts w, w + 4, w + 8, w + 12 (entries K..63 read as 0), then warp 0
  // merges the four results; warp 1 merges the normalisers meanwhile
  unsigned long long a0, a1;
  {
    const unsigned long long* kb = p.keys + rid * S * 64;
    unsigned long long x0[4], x1[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int l = w + 4 * j;
      x0[j] = (l < S && lane < K) ? __ldcg(kb + l * 64 + lane) : 0ull;
      x1[j] = (l < S && lane + 32 < K) ? __ldcg(kb + l * 64 + 32 + lane) : 0ull;
    }
    a0 = x0[0];
    a1 = x1[0];
#pragma unroll
    for (int j = 1; j < 4; ++j)
      if (w + 4 * j < S) {
        const ulonglong2 m2 = merge_top64(a0, a1, x0[j], x1[j], lane);
        a0 = m2.x;
        a1 = m2.y;
      }
  }
  s_dyn[w * 64 + lane] = a0;
  s_dyn[w * 64 + 32 + lane] = a1;
  __syncthreads();
  if (w == 0) {
#pragma unroll
    for (int w2 = 1; w2 < kThreads / 32; ++w2)
      if (w2 < S) {
        const ulonglong2 m2 = merge_top64(a0, a1, s_dyn[w2 * 64 + lane], s_dyn[w2 * 64 + 32 + lane], lane);
        a0 = m2.x;
        a1 = m2.y;
      }
  } else if (w == 1) {
    float M = -INFINITY, Sum = 0.f;
    uint32_t anybad = 0;
    for (int l = lane; l < S; l += 32) {
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
    if (lane == 0) {
      s_wm[0] = M;
      s_ws[0] = Sum;
      s_bad = (anybad || !(M > -INFINITY)) ? 1 : 0;
    }
  }
  __syncthreads();
  if (w == 0) {
    // log q = (x - max) / T - log sum exp((x_j - max) / T)
    const float M = s_wm[0], lnS = logf(s_ws[0]);
    int2* trow = p.table + rid * 64;
    if (lane < K) trow[lane] = make_int2(key_index(a0), __float_as_int((key_value(a0) - M) * invT - lnS));
    if (lane + 32 < K)
      trow[lane + 32] = make_int2(key_index(a1), __float_as_int((key_value(a1) - M) * invT - lnS));
    if (lane == 0 && s_bad) atomicOr(&p.seq_flags[b], SPEC_FLAG_BAD_LOGITS);
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
  if (p.nodes <= 33) select_nodes<1>(p, tab, K, b, s_flags, lane);
  else select_nodes<2>(p, tab, K, b, s_flags, lane);
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
  p.rowstat = reinterpret_cast<float2*>(ws + L.rowstat);
  p.temperature = a.temperature;
  p.uniforms = a.uniforms;
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
  L.smem = static_cast<int>(8 * std::max(std::max(kTreeCandCap, 4 * 64), L.rows * k));
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
