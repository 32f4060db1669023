// Top-k / top-p filtered acceptance: the sampling of the paper's evaluations (top-k 50
// and top-p 0.95 for drafting and verification, Sec. 5.1, Sec. 5.2, Appendix C.1)
// applied to the lossless rule of Alg. "Lossless Psi-Spec decoding (Linear Sampler)"
// (Appendix B.3). Each used row's distribution is replaced by its filtered form: the
// top_k tokens by logit (ties to the lower token id), then the shortest prefix of them,
// in rank order, whose renormalised mass reaches top_p, renormalised. The rule then
// runs on the filtered p' and q'.
//
// The filtered distribution needs no vocabulary-wide normaliser: p'(x) is
// exp((l_x - l_max)/T) over the same sum restricted to the kept tokens. So a row is
// read once, for the maxima of 128-element lanes, and the top-k is then found among
// the few lanes that can hold it. Three launches, each a programmatic dependent of the
// one before:
//   1. filter_scan_kernel: one warp per (sequence, row, 4096-entry chunk) writes each
//      lane's maximum as an order-preserving key (and, for greedy rows, the lowest
//      index holding it). The k-th largest lane maximum bounds the k-th largest logit
//      from below: k distinct lanes each hold an element at least that large.
//   2. filter_select_kernel: one block per (sequence, row) finds that bound by a
//      two-digit radix select over the lane keys, rescans only the lanes whose maximum
//      reaches it, sorts the candidates, and takes the top-k, the top-p cut and the
//      renormalised probabilities in fp64. If the candidates overflow shared memory
//      (many equal logits), an exact radix select over the whole row replaces the bound.
//   3. filter_decide_kernel: one block per sequence takes the gamma-1 decisions on
//      p'(t_i) / q'(t_i) and draws the final token by inverse CDF, in ascending token
//      order, over the kept tokens of p'_n (weights [p'_n - q'_n]_+, or p'_B).
#include <cuda_bf16.h>

#include <cfloat>
#include <climits>
#include <cmath>

#include "common.cuh"

namespace specv {

FilterLayout filter_layout(const spec_accept_args_t& a, int max_top_k, size_t base) {
  FilterLayout L;
  L.nchunk = (a.vocab + kStatsChunk - 1) / kStatsChunk;
  L.nlanes = L.nchunk * 32;
  const size_t rows = static_cast<size_t>(a.batch) * (2 * static_cast<size_t>(a.gamma) - 1);
  L.lanes = base;
  L.rows = ws_round(L.lanes + sizeof(uint64_t) * rows * L.nlanes);
  L.ids = ws_round(L.rows + sizeof(FiltRow) * rows);
  L.probs = ws_round(L.ids + sizeof(int32_t) * rows * max_top_k);
  L.end = ws_round(L.probs + sizeof(double) * rows * max_top_k);
  return L;
}

namespace {

constexpr int kSelectThreads = 256;
constexpr int kFiltCap = 4096;      // candidates one select block holds
constexpr int kFiltLaneCap = 2048;  // lanes one select block rescans
constexpr int kFiltDecideThreads = 256;
constexpr uint32_t kRowBadLogits = 1u, kRowBadFilter = 2u;

struct FiltParams {
  int batch, gamma, vocab, nchunk, nlanes, max_top_k;
  const void* target;
  const void* drafter;
  const int32_t* tokens;
  const float* temperature;
  const float* uniforms;
  const int32_t* top_k;
  const float* top_p;
  int32_t* num_accepted;
  int32_t* out_tokens;
  int32_t* num_emitted;
  float* diag;
  uint32_t* status;
  unsigned long long* lanes;  // [batch][2*gamma-1][nlanes]
  FiltRow* rows;              // [batch][2*gamma-1]
  int32_t* ids;               // [batch][2*gamma-1][max_top_k], kept tokens in rank order
  double* probs;              // same layout, their filtered probabilities
};

template <bool BF16>
__device__ __forceinline__ float load_elem(const void* base, int64_t i) {
  if (BF16) return bf16_bits_to_f32(static_cast<const uint16_t*>(base)[i]);
  return static_cast<const float*>(base)[i];
}

// Order-preserving key of a float: a larger value has a larger key; -0 shares +0's key
// so that equal values tie. Keys above order_key(+inf) are NaNs.
__device__ __forceinline__ uint32_t order_key(float x) {
  uint32_t f = __float_as_uint(x);
  if (f == 0x80000000u) f = 0u;
  return (f & 0x80000000u) ? ~f : (f | 0x80000000u);
}
__device__ __forceinline__ float key_value(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}
// A candidate: key in the high word, 0xffffffff - token in the low word, so that the
// larger of two candidates is the higher logit, then the lower token id.
__device__ __forceinline__ unsigned long long cand_of(uint32_t key, uint32_t tok) {
  return (static_cast<unsigned long long>(key) << 32) | (0xffffffffu - tok);
}
__device__ __forceinline__ int cand_tok(unsigned long long c) {
  return static_cast<int>(0xffffffffu - static_cast<uint32_t>(c));
}
constexpr unsigned long long kBadLane = ~0ull;  // a lane that saw NaN (or +inf, tempered)

// Row r of sequence b: target row r for r < gamma, else drafter row r - gamma + 1.
__device__ __forceinline__ const char* row_ptr(const FiltParams& p, int b, int r, int esz) {
  const int64_t row = static_cast<int64_t>(b) * p.gamma + (r < p.gamma ? r : r - p.gamma + 1);
  const void* base = r < p.gamma ? p.target : p.drafter;
  return static_cast<const char*>(base) + row * p.vocab * esz;
}

// 1. Lane maxima: one warp per (chunk, row, sequence). Lane l of a chunk owns 128 of its
// elements: with 16-byte loads, the 8 (bf16) or 4 (fp32) elements of groups g*32 + l;
// with element loads, elements j*32 + l.
template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kStatsThreads, 5) filter_scan_kernel(FiltParams p) {
  pdl_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int c = blockIdx.x * (kStatsThreads / 32) + (threadIdx.x >> 5);
  const int r = blockIdx.y, b = blockIdx.z;
  if (c >= p.nchunk) return;
  const int nrows = 2 * p.gamma - 1;
  const float T = p.temperature[b];
  const bool greedy = !(T > 0.f);
  if (greedy && r >= p.gamma) return;  // greedy sequences never read drafter rows
  const char* rowp = row_ptr(p, b, r, BF16 ? 2 : 4);
  const int start = c * kStatsChunk;
  const int len = min(kStatsChunk, p.vocab - start);

  bool bad = false;
  float m = -INFINITY;
  int a = INT_MAX;
  bool any;
  if (VEC) {
    constexpr int kEpv = BF16 ? 8 : 4;
    constexpr int kGroups = 16;
    constexpr int kRounds = kStatsChunk / (32 * kGroups * kEpv);
    const uint32_t ninf = BF16 ? 0xFF80FF80u : 0xFF800000u;
    // NaN test on packed words: a magnitude above +inf's carries into the top bit
    const uint32_t nan_mask = BF16 ? 0x7FFF7FFFu : 0x7FFFFFFFu;
    const uint32_t nan_add = BF16 ? 0x007F007Fu : 0x007FFFFFu;
    const uint32_t nan_top = BF16 ? 0x80008000u : 0x80000000u;
    any = lane * kEpv < len;
    a = any ? start + lane * kEpv : INT_MAX;
    uint32_t nacc = 0;
#pragma unroll
    for (int rd = 0; rd < kRounds; ++rd) {
      uint32_t w[kGroups * 4];
#pragma unroll
      for (int k = 0; k < kGroups; ++k) {
        const int e = ((rd * kGroups + k) * 32 + lane) * kEpv;
        const uint4 v = e < len ? __ldg(reinterpret_cast<const uint4*>(rowp + static_cast<int64_t>(start + e) * (BF16 ? 2 : 4)))
                                : make_uint4(ninf, ninf, ninf, ninf);
        w[4 * k] = v.x; w[4 * k + 1] = v.y; w[4 * k + 2] = v.z; w[4 * k + 3] = v.w;
      }
#pragma unroll
      for (int i = 0; i < kGroups * 4; ++i) nacc |= (w[i] & nan_mask) + nan_add;
      if (greedy) {
        // elements in increasing index order: a strict > keeps the lowest index
#pragma unroll
        for (int k = 0; k < kGroups; ++k) {
          const int e = ((rd * kGroups + k) * 32 + lane) * kEpv;
#pragma unroll
          for (int q = 0; q < kEpv; ++q) {
            float x;
            if (BF16) {
              const uint32_t word = w[4 * k + (q >> 1)];
              x = __uint_as_float((q & 1) ? (word & 0xffff0000u) : (word << 16));
            } else {
              x = __uint_as_float(w[4 * k + q]);
            }
            if (x > m) { m = x; a = start + e + q; }
          }
        }
      } else {
        float mr;
        if (BF16) {
          __nv_bfloat162 mx = *reinterpret_cast<const __nv_bfloat162*>(&w[0]);
#pragma unroll
          for (int i = 1; i < kGroups * 4; ++i) mx = __hmax2(mx, *reinterpret_cast<const __nv_bfloat162*>(&w[i]));
          mr = fmaxf(__bfloat162float(mx.x), __bfloat162float(mx.y));
        } else {
          mr = -INFINITY;
#pragma unroll
          for (int i = 0; i < kGroups * 4; ++i) mr = fmaxf(mr, __uint_as_float(w[i]));
        }
        m = fmaxf(m, mr);
      }
    }
    bad = (nacc & nan_top) != 0;
  } else {
    any = lane < len;
    a = any ? start + lane : INT_MAX;
    for (int j = 0; j < kStatsChunk / 32; ++j) {
      const int e = j * 32 + lane;
      if (e >= len) break;
      const float x = load_elem<BF16>(rowp, start + e);
      bad |= x != x;
      if (x > m) { m = x; a = start + e; }
    }
  }
  if (!greedy && m == INFINITY) bad = true;  // +inf leaves a tempered softmax undefined
  unsigned long long out;
  if (bad) out = kBadLane;
  else if (!any) out = 0ull;  // no element: below every real key
  else out = cand_of(order_key(m), greedy ? static_cast<uint32_t>(a) : 0xffffffffu);
  p.lanes[(static_cast<int64_t>(b) * nrows + r) * p.nlanes + c * 32 + lane] = out;
}

// Block-wide maximum of one value per thread (every thread gets it).
template <int kThreads>
__device__ __forceinline__ unsigned long long block_max(unsigned long long v, unsigned long long* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long y = __shfl_xor_sync(0xffffffffu, v, o);
    v = y > v ? y : v;
  }
  if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = v;
  __syncthreads();
  v = sh[0];
#pragma unroll
  for (int k = 1; k < kThreads / 32; ++k) v = sh[k] > v ? sh[k] : v;
  __syncthreads();
  return v;
}

// Block-wide exclusive scan of one value per thread, in thread order; *total gets the sum.
template <int kThreads, class Tv>
__device__ __forceinline__ Tv block_excl_scan(Tv x, Tv* sh, Tv* total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  Tv in = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const Tv y = __shfl_up_sync(0xffffffffu, in, o);
    if (lane >= o) in += y;
  }
  if (lane == 31) sh[w] = in;
  __syncthreads();
  if (threadIdx.x == 0) {
    Tv run = 0;
    for (int k = 0; k < kThreads / 32; ++k) {
      const Tv t = sh[k];
      sh[k] = run;
      run += t;
    }
    sh[kThreads / 32] = run;
  }
  __syncthreads();
  const Tv ex = sh[w] + in - x;
  *total = sh[kThreads / 32];
  __syncthreads();
  return ex;
}

// Warp 0 of the block: the bin of a 256-bin histogram that holds the need-th largest
// item, counting from the top bin down; *above receives the items in higher bins.
// Returns -1 when the histogram holds fewer than need items.
__device__ int find_bin_desc(const uint32_t* hist, uint32_t need, uint32_t* above) {
  const int lane = threadIdx.x & 31;
  uint32_t cnt[8], sum = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    cnt[j] = hist[255 - (lane * 8 + j)];
    sum += cnt[j];
  }
  uint32_t incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  const uint32_t total = __shfl_sync(0xffffffffu, incl, 31);
  if (total < need) return -1;
  const unsigned hit = __ballot_sync(0xffffffffu, incl >= need);
  const int src = __ffs(hit) - 1;
  int bin = -1;
  uint32_t ab = 0;
  if (lane == src) {
    uint32_t run = incl - sum;
    for (int j = 0; j < 8; ++j) {
      if (run + cnt[j] >= need) {
        bin = 255 - (lane * 8 + j);
        ab = run;
        break;
      }
      run += cnt[j];
    }
  }
  bin = __shfl_sync(0xffffffffu, bin, src);
  *above = __shfl_sync(0xffffffffu, ab, src);
  return bin;
}

// In-place bitonic sort of n2 (a power of two) candidates, descending.
template <int kThreads>
__device__ void bitonic_desc(unsigned long long* s, int n2) {
  for (int k = 2; k <= n2; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n2; i += kThreads) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const unsigned long long x = s[i], y = s[ixj];
          const bool desc = (i & k) == 0;
          if (desc ? x < y : x > y) {
            s[i] = y;
            s[ixj] = x;
          }
        }
      }
      __syncthreads();
    }
  }
}

// In-place bitonic sort of n2 (id, value) pairs by ascending id.
template <int kThreads>
__device__ void bitonic_pairs_asc(int* id, double* val, int n2) {
  for (int k = 2; k <= n2; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n2; i += kThreads) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const int x = id[i], y = id[ixj];
          const bool asc = (i & k) == 0;
          if (asc ? x > y : x < y) {
            id[i] = y;
            id[ixj] = x;
            const double t = val[i];
            val[i] = val[ixj];
            val[ixj] = t;
          }
        }
      }
      __syncthreads();
    }
  }
}

__device__ __forceinline__ int pow2_at_least(int n) {
  int m = 1;
  while (m < n) m <<= 1;
  return m;
}

// Exact fallback of the select kernel: the K largest candidates of the whole row by a
// four-digit radix select on the keys, then one pass in token order that keeps every
// element above the K-th key and the lowest-id elements equal to it.
template <bool BF16>
__device__ void exact_topk(const char* rowp, int V, int K, unsigned long long* s_cand,
                           uint32_t* s_hist, int* s_ncand, int* s_scan, int* s_misc) {
  const int tid = threadIdx.x;
  uint32_t prefix = 0, pmask = 0, need = static_cast<uint32_t>(K);
  for (int d = 3; d >= 0; --d) {
    for (int i = tid; i < 256; i += kSelectThreads) s_hist[i] = 0;
    __syncthreads();
    for (int i = tid; i < V; i += kSelectThreads) {
      const uint32_t k = order_key(load_elem<BF16>(rowp, i));
      if ((k & pmask) == prefix) atomicAdd(&s_hist[(k >> (8 * d)) & 0xffu], 1u);
    }
    __syncthreads();
    if (tid < 32) {
      uint32_t above = 0;
      const int bin = find_bin_desc(s_hist, need, &above);
      if (tid == 0) {
        s_misc[0] = bin;
        s_misc[1] = static_cast<int>(above);
      }
    }
    __syncthreads();
    const int bin = s_misc[0];  // exists: the row holds at least K elements
    need -= static_cast<uint32_t>(s_misc[1]);
    prefix |= static_cast<uint32_t>(bin) << (8 * d);
    pmask |= 0xffu << (8 * d);
    __syncthreads();
  }
  const uint32_t kappa = prefix;
  const int ties = static_cast<int>(need);  // elements equal to kappa to keep
  if (tid == 0) *s_ncand = 0;
  __syncthreads();
  int tie_base = 0;
  constexpr int kPer = 8;
  for (int base = 0; base < V; base += kSelectThreads * kPer) {
    const int first = base + tid * kPer;
    uint32_t keys[kPer];
    int mine = 0;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      keys[q] = first + q < V ? order_key(load_elem<BF16>(rowp, first + q)) : 0u;
      mine += (first + q < V && keys[q] == kappa) ? 1 : 0;
    }
    int total = 0;
    int rank = block_excl_scan<kSelectThreads, int>(mine, s_scan, &total);
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      if (first + q >= V) break;
      bool take = keys[q] > kappa;
      if (keys[q] == kappa) {
        take = tie_base + rank < ties;
        ++rank;
      }
      if (take) {
        const int slot = atomicAdd(s_ncand, 1);
        if (slot < kFiltCap) s_cand[slot] = cand_of(keys[q], static_cast<uint32_t>(first + q));
      }
    }
    tie_base += total;
  }
  __syncthreads();
}

// 2. Per (row, sequence): the top-k, the top-p cut and the kept probabilities.
template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kSelectThreads) filter_select_kernel(FiltParams p) {
  pdl_launch_dependents();
  __shared__ unsigned long long s_cand[kFiltCap];
  __shared__ int s_lane[kFiltLaneCap];
  __shared__ uint32_t s_hist[256];
  __shared__ unsigned long long s_red[kSelectThreads / 32];
  __shared__ double s_dscan[kSelectThreads / 32 + 1];
  __shared__ int s_iscan[kSelectThreads / 32 + 1];
  __shared__ int s_nlane, s_ncand, s_keep, s_misc[2];
  __shared__ double s_kept_mass;

  const int r = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int gamma = p.gamma, nrows = 2 * gamma - 1, V = p.vocab;
  const float T = p.temperature[b];
  const bool greedy = !(T > 0.f);
  if (greedy && r >= gamma) return;
  const int k_in = greedy ? 1 : p.top_k[b];
  const float tp = greedy ? 1.f : p.top_p[b];
  const int64_t rid = static_cast<int64_t>(b) * nrows + r;
  const char* rowp = row_ptr(p, b, r, BF16 ? 2 : 4);
  pdl_wait_prior();  // the lane maxima are written and visible

  const unsigned long long* L = p.lanes + rid * p.nlanes;
  unsigned long long mx = 0;
  for (int i = tid; i < p.nlanes; i += kSelectThreads) {
    const unsigned long long v = L[i];
    mx = v > mx ? v : mx;
  }
  mx = block_max<kSelectThreads>(mx, s_red);
  FiltRow info;
  info.nkeep = 0;
  info.argmax = greedy ? cand_tok(mx) : -1;
  info.flags = 0;
  info.pad = 0;
  if (mx == kBadLane || (!greedy && static_cast<uint32_t>(mx >> 32) <= order_key(-INFINITY)))
    info.flags = kRowBadLogits;  // NaN, +inf (tempered) or no finite logit (tempered)
  else if (!greedy && (k_in < 1 || k_in > p.max_top_k || !(tp > 0.f) || !(tp <= 1.f)))
    info.flags = kRowBadFilter;
  if (greedy || info.flags) {
    if (tid == 0) p.rows[rid] = info;
    return;
  }
  const int K = min(k_in, V);

  // the bound: the high 16 bits of the K-th largest lane key (0: every element)
  uint32_t beta = 0;
  for (int i = tid; i < 256; i += kSelectThreads) s_hist[i] = 0;
  __syncthreads();
  for (int i = tid; i < p.nlanes; i += kSelectThreads) {
    const unsigned long long v = L[i];
    if (v) atomicAdd(&s_hist[static_cast<uint32_t>(v >> 56)], 1u);
  }
  __syncthreads();
  if (tid < 32) {
    uint32_t above = 0;
    const int bin = find_bin_desc(s_hist, static_cast<uint32_t>(K), &above);
    if (tid == 0) {
      s_misc[0] = bin;
      s_misc[1] = static_cast<int>(above);
    }
  }
  __syncthreads();
  const int b1 = s_misc[0];
  if (b1 >= 0) {
    const uint32_t need = static_cast<uint32_t>(K - s_misc[1]);
    __syncthreads();
    for (int i = tid; i < 256; i += kSelectThreads) s_hist[i] = 0;
    __syncthreads();
    for (int i = tid; i < p.nlanes; i += kSelectThreads) {
      const unsigned long long v = L[i];
      if (v && static_cast<int>(v >> 56) == b1) atomicAdd(&s_hist[static_cast<uint32_t>(v >> 48) & 0xffu], 1u);
    }
    __syncthreads();
    if (tid < 32) {
      uint32_t above = 0;
      const int bin = find_bin_desc(s_hist, need, &above);
      if (tid == 0) s_misc[0] = bin;
    }
    __syncthreads();
    beta = (static_cast<uint32_t>(b1) << 24) | (static_cast<uint32_t>(s_misc[0]) << 16);
  }

  // the lanes that can hold a top-K element, then their elements at or above the bound
  if (tid == 0) {
    s_nlane = 0;
    s_ncand = 0;
  }
  __syncthreads();
  for (int i = tid; i < p.nlanes; i += kSelectThreads) {
    const unsigned long long v = L[i];
    if (v && static_cast<uint32_t>(v >> 32) >= beta) {
      const int slot = atomicAdd(&s_nlane, 1);
      if (slot < kFiltLaneCap) s_lane[slot] = i;
    }
  }
  __syncthreads();
  const int nlane = s_nlane;
  if (nlane <= kFiltLaneCap) {
    for (int it = tid; it < nlane * 16; it += kSelectThreads) {
      const int li = s_lane[it >> 4], seg = it & 15;
      const int ch = li >> 5, ln = li & 31;
      const int cstart = ch * kStatsChunk, clen = min(kStatsChunk, V - cstart);
      float x[8];
      int idx[8];
      if (VEC) {
        constexpr int kEpv = BF16 ? 8 : 4;
#pragma unroll
        for (int h = 0; h < 8 / kEpv; ++h) {
          const int g = seg * (8 / kEpv) + h;
          const int e = (g * 32 + ln) * kEpv;
          uint4 v = make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
          if (e < clen) v = __ldg(reinterpret_cast<const uint4*>(rowp + static_cast<int64_t>(cstart + e) * (BF16 ? 2 : 4)));
          const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
          for (int q = 0; q < kEpv; ++q) {
            if (BF16) x[h * kEpv + q] = __uint_as_float((q & 1) ? (wv[q >> 1] & 0xffff0000u) : (wv[q >> 1] << 16));
            else x[h * kEpv + q] = __uint_as_float(wv[q]);
            idx[h * kEpv + q] = e < clen ? cstart + e + q : -1;
          }
        }
      } else {
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const int e = (seg * 8 + q) * 32 + ln;
          idx[q] = e < clen ? cstart + e : -1;
          x[q] = e < clen ? load_elem<BF16>(rowp, cstart + e) : -INFINITY;
        }
      }
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const uint32_t k = order_key(x[q]);
        if (idx[q] >= 0 && k >= beta) {
          const int slot = atomicAdd(&s_ncand, 1);
          if (slot < kFiltCap) s_cand[slot] = cand_of(k, static_cast<uint32_t>(idx[q]));
        }
      }
    }
  }
  __syncthreads();
  if (nlane > kFiltLaneCap || s_ncand > kFiltCap) {
    __syncthreads();
    exact_topk<BF16>(rowp, V, K, s_cand, s_hist, &s_ncand, s_iscan, s_misc);
  }
  const int ncand = min(s_ncand, kFiltCap);
  const int n2 = pow2_at_least(max(ncand, 2));
  for (int i = ncand + tid; i < n2; i += kSelectThreads) s_cand[i] = 0ull;
  __syncthreads();
  bitonic_desc<kSelectThreads>(s_cand, n2);

  // top-p on the renormalised top-K, in fp64: w_j = exp(z_j - z_0), z = l / T
  const int keff = min(K, ncand);
  const double Td = static_cast<double>(T);
  const double z0 = static_cast<double>(key_value(static_cast<uint32_t>(s_cand[0] >> 32))) / Td;
  constexpr int kPer = kFilterMaxTopK / kSelectThreads;  // entries per thread
  double w[kPer], incl[kPer];
  double run = 0.0;
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    const int j = tid * kPer + q;
    w[q] = j < keff ? exp(static_cast<double>(key_value(static_cast<uint32_t>(s_cand[j] >> 32))) / Td - z0) : 0.0;
    run += w[q];
    incl[q] = run;
  }
  double mass = 0.0;
  const double ex = block_excl_scan<kSelectThreads, double>(run, s_dscan, &mass);
  if (tid == 0) s_keep = keff;
  __syncthreads();
  const double tpd = static_cast<double>(tp);
  if (tpd < 1.0) {
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int j = tid * kPer + q;
      if (j < keff && (ex + incl[q]) / mass >= tpd) {
        atomicMin(&s_keep, j + 1);
        break;
      }
    }
  }
  __syncthreads();
  const int keep = s_keep;
#pragma unroll
  for (int q = 0; q < kPer; ++q)
    if (tid * kPer + q == keep - 1) s_kept_mass = ex + incl[q];
  __syncthreads();
  const double S = s_kept_mass;
  int32_t* ids = p.ids + rid * p.max_top_k;
  double* probs = p.probs + rid * p.max_top_k;
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    const int j = tid * kPer + q;
    if (j < keep) {
      ids[j] = cand_tok(s_cand[j]);
      probs[j] = w[q] / S;
    }
  }
  if (tid == 0) {
    info.nkeep = keep;
    info.argmax = cand_tok(s_cand[0]);
    p.rows[rid] = info;
  }
}

// The filtered probability of token t in row rid (0 if not kept), by one warp.
__device__ __forceinline__ double warp_lookup(const FiltParams& p, int64_t rid, int nkeep, int t) {
  const int lane = threadIdx.x & 31;
  const int32_t* ids = p.ids + rid * p.max_top_k;
  const double* probs = p.probs + rid * p.max_top_k;
  double v = 0.0;
  for (int j = lane; j < nkeep; j += 32)
    if (ids[j] == t) v = probs[j];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;  // at most one lane matched
}

// 3. Per sequence: decisions on p'(t_i) / q'(t_i), every output, and the final draw.
__global__ void __launch_bounds__(kFiltDecideThreads) filter_decide_kernel(FiltParams p) {
  constexpr int kMaxGamma = 64;
  constexpr int kThreads = kFiltDecideThreads;
  constexpr int kPer = kFilterMaxTopK / kThreads;
  __shared__ int s_tok[kMaxGamma], s_arg[kMaxGamma], s_nkeep[2 * kMaxGamma];
  __shared__ float s_u[kMaxGamma], s_ptok[kMaxGamma], s_qtok[kMaxGamma];
  __shared__ int sP_id[kFilterMaxTopK], sQ_id[kFilterMaxTopK];
  __shared__ double sP_v[kFilterMaxTopK], sQ_v[kFilterMaxTopK];
  __shared__ double s_dscan[kThreads / 32 + 1];
  __shared__ int s_bad, s_n, s_pick, s_last;

  const int b = blockIdx.x, tid = threadIdx.x;
  const int gamma = p.gamma, V = p.vocab, nrows = 2 * gamma - 1;
  const float T = p.temperature[b];
  const bool greedy = !(T > 0.f);
  if (tid == 0) {
    s_bad = 0;
    s_n = gamma;
    s_pick = INT_MAX;
    s_last = -1;
  }
  // inputs, read while the select kernel still runs
  if (tid < gamma) {
    s_tok[tid] = p.tokens[static_cast<int64_t>(b) * gamma + tid];
    s_u[tid] = p.uniforms[static_cast<int64_t>(b) * gamma + tid];
  }
  pdl_wait_prior();
  __syncthreads();
  const int rows_needed = greedy ? gamma : nrows;
  for (int r = tid; r < rows_needed; r += kThreads) {
    const FiltRow fr = p.rows[static_cast<int64_t>(b) * nrows + r];
    if (fr.flags & kRowBadLogits) atomicOr(&s_bad, 2);
    if (fr.flags & kRowBadFilter) atomicOr(&s_bad, 4);
    s_nkeep[r] = fr.nkeep;
    if (r < gamma) s_arg[r] = fr.argmax;
  }
  if (tid < gamma && (s_tok[tid] < 0 || s_tok[tid] >= V)) atomicOr(&s_bad, 1);
  __syncthreads();

  const int64_t orow = static_cast<int64_t>(b) * (gamma + 1);
  if (s_bad) {
    for (int k = tid; k <= gamma; k += kThreads) p.out_tokens[orow + k] = -1;
    if (p.diag)
      for (int k = tid; k < 2 * gamma; k += kThreads)
        p.diag[static_cast<int64_t>(b) * gamma * 2 + k] = NAN;
    if (tid == 0) {
      p.num_accepted[b] = -1;
      p.num_emitted[b] = 0;
      if (s_bad & 1) set_status(p.status, SPEC_FLAG_BAD_TOKEN);
      if (s_bad & 2) set_status(p.status, SPEC_FLAG_BAD_LOGITS);
      if (s_bad & 4) set_status(p.status, SPEC_FLAG_BAD_FILTER);
    }
    return;
  }

  // the gamma-1 decisions: one warp per draft
  {
    const int warp = tid >> 5, lane = tid & 31;
    for (int i = 1 + warp; i < gamma; i += kThreads / 32) {
      const int t = s_tok[i];
      bool reject;
      float pt, qt;
      if (greedy) {
        reject = t != s_arg[i - 1];
        pt = reject ? 0.f : 1.f;
        qt = 1.f;
      } else {
        const int64_t prow = static_cast<int64_t>(b) * nrows + (i - 1);
        const int64_t qrow = static_cast<int64_t>(b) * nrows + (gamma + i - 1);
        const double pd = warp_lookup(p, prow, s_nkeep[i - 1], t);
        const double qd = warp_lookup(p, qrow, s_nkeep[gamma + i - 1], t);
        // a draft outside q's filtered support: accept iff p'(t) > 0
        const double ratio = qd > 0.0 ? pd / qd : (pd > 0.0 ? INFINITY : 0.0);
        reject = static_cast<double>(s_u[i - 1]) > fmin(1.0, ratio);
        pt = static_cast<float>(pd);
        qt = static_cast<float>(qd);
      }
      if (lane == 0) {
        s_ptok[i] = pt;
        s_qtok[i] = qt;
        if (reject) atomicMin(&s_n, i);
      }
    }
  }
  __syncthreads();
  const int n = s_n;
  for (int k = tid; k <= gamma; k += kThreads) {
    if (k < n) p.out_tokens[orow + k] = s_tok[k];
    else if (k > n) p.out_tokens[orow + k] = -1;
    else if (greedy) p.out_tokens[orow + k] = s_arg[n - 1];
  }
  if (p.diag) {
    for (int i = tid; i < gamma; i += kThreads) {
      const int64_t d = (static_cast<int64_t>(b) * gamma + i) * 2;
      const bool taken = i >= 1 && i <= n && i < gamma;
      p.diag[d] = i == 0 ? 0.f : (taken ? s_ptok[i] : NAN);
      p.diag[d + 1] = i == 0 ? 0.f : (taken ? s_qtok[i] : NAN);
    }
  }
  if (tid == 0) {
    p.num_accepted[b] = n - 1;
    p.num_emitted[b] = n + 1;
  }
  if (greedy) return;

  // the final draw over the kept tokens of p'_n, in ascending token order
  const bool bonus = n == gamma;
  const int64_t prid = static_cast<int64_t>(b) * nrows + (n - 1);
  const int64_t qrid = static_cast<int64_t>(b) * nrows + (gamma + n - 1);
  const int nP = s_nkeep[n - 1];
  const int nQ = bonus ? 0 : s_nkeep[gamma + n - 1];
  const int nP2 = pow2_at_least(max(nP, 2)), nQ2 = pow2_at_least(max(nQ, 2));
  for (int j = tid; j < nP2; j += kThreads) {
    sP_id[j] = j < nP ? p.ids[prid * p.max_top_k + j] : INT_MAX;
    sP_v[j] = j < nP ? p.probs[prid * p.max_top_k + j] : 0.0;
  }
  if (!bonus)
    for (int j = tid; j < nQ2; j += kThreads) {
      sQ_id[j] = j < nQ ? p.ids[qrid * p.max_top_k + j] : INT_MAX;
      sQ_v[j] = j < nQ ? p.probs[qrid * p.max_top_k + j] : 0.0;
    }
  __syncthreads();
  bitonic_pairs_asc<kThreads>(sP_id, sP_v, nP2);
  if (!bonus) bitonic_pairs_asc<kThreads>(sQ_id, sQ_v, nQ2);
  // residual weights [p' - q']_+ (q' by binary search), then their scan
  double w[kPer], incl[kPer];
  double run = 0.0;
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    const int j = tid * kPer + q;
    double x = 0.0;
    if (j < nP) {
      x = sP_v[j];
      if (!bonus) {
        const int t = sP_id[j];
        int lo = 0, hi = nQ;
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (sQ_id[mid] < t) lo = mid + 1;
          else hi = mid;
        }
        const double qv = (lo < nQ && sQ_id[lo] == t) ? sQ_v[lo] : 0.0;
        x = fmax(0.0, x - qv);
      }
    }
    w[q] = x;
    run += x;
    incl[q] = run;
  }
  double S = 0.0;
  double ex = block_excl_scan<kThreads, double>(run, s_dscan, &S);
  if (bonus || !(S > 0.0)) {
    // the bonus draw, or a residual without mass (only through rounding): p'_n itself
    run = 0.0;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int j = tid * kPer + q;
      w[q] = j < nP ? sP_v[j] : 0.0;
      run += w[q];
      incl[q] = run;
    }
    ex = block_excl_scan<kThreads, double>(run, s_dscan, &S);
  }
  const double target = static_cast<double>(s_u[gamma - 1]) * S;
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    const int j = tid * kPer + q;
    if (j < nP && w[q] > 0.0) {
      atomicMax(&s_last, j);
      if (ex + incl[q] >= target) atomicMin(&s_pick, j);
    }
  }
  __syncthreads();
  if (tid == 0) {
    const int j = s_pick != INT_MAX ? s_pick : s_last;  // rounding: the last positive weight
    p.out_tokens[orow + n] = j >= 0 ? sP_id[j] : -1;
  }
}

template <bool BF16, bool VEC>
cudaError_t launch_filtered_typed(const FiltParams& p, cudaStream_t stream, bool overlap_prior) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((p.nchunk + kStatsThreads / 32 - 1) / (kStatsThreads / 32), 2 * p.gamma - 1, p.batch);
  cfg.blockDim = dim3(kStatsThreads);
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = overlap_prior ? 1 : 0;  // beside the attention kernel of a verify step
  cudaError_t e = cudaLaunchKernelEx(&cfg, filter_scan_kernel<BF16, VEC>, p);
  if (e != cudaSuccess) return e;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(2 * p.gamma - 1, p.batch);
  cfg.blockDim = dim3(kSelectThreads);
  e = cudaLaunchKernelEx(&cfg, filter_select_kernel<BF16, VEC>, p);
  if (e != cudaSuccess) return e;
  cfg.gridDim = dim3(p.batch);
  cfg.blockDim = dim3(kFiltDecideThreads);
  e = cudaLaunchKernelEx(&cfg, filter_decide_kernel, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_accept_filtered(const spec_accept_args_t& a, const spec_filter_args_t& f,
                                   const FilterLayout& L, char* ws, cudaStream_t stream,
                                   bool overlap_prior) {
  FiltParams p;
  p.batch = a.batch;
  p.gamma = a.gamma;
  p.vocab = a.vocab;
  p.nchunk = L.nchunk;
  p.nlanes = L.nlanes;
  p.max_top_k = f.max_top_k;
  p.target = a.target_logits;
  p.drafter = a.drafter_logits;
  p.tokens = a.block_tokens;
  p.temperature = a.temperature;
  p.uniforms = a.uniforms;
  p.top_k = f.top_k;
  p.top_p = f.top_p;
  p.num_accepted = a.num_accepted;
  p.out_tokens = a.out_tokens;
  p.num_emitted = a.num_emitted;
  p.diag = a.diag;
  p.status = reinterpret_cast<uint32_t*>(ws);
  p.lanes = reinterpret_cast<unsigned long long*>(ws + L.lanes);
  p.rows = reinterpret_cast<FiltRow*>(ws + L.rows);
  p.ids = reinterpret_cast<int32_t*>(ws + L.ids);
  p.probs = reinterpret_cast<double*>(ws + L.probs);
  const bool bf16 = a.logits_dtype == SPEC_BF16;
  const size_t esz = bf16 ? 2 : 4;
  const bool vec = (static_cast<size_t>(a.vocab) * esz) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(a.target_logits) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(a.drafter_logits) % 16 == 0;
  (void)cudaGetLastError();
  if (bf16)
    return vec ? launch_filtered_typed<true, true>(p, stream, overlap_prior)
               : launch_filtered_typed<true, false>(p, stream, overlap_prior);
  return vec ? launch_filtered_typed<false, true>(p, stream, overlap_prior)
             : launch_filtered_typed<false, false>(p, stream, overlap_prior);
}

}  // namespace specv
