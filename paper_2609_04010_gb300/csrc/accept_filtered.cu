// Top-k / top-p filtered acceptance: the sampling of the paper's evaluations (top-k 50
// and top-p 0.95 for drafting and verification, Sec. 5.1, Sec. 5.2, Appendix C.1)
// applied to the lossless rule of Alg. "Lossless Psi-Spec decoding (Linear Sampler)"
// (Appendix B.3). Each used row's distribution is replaced by its filtered form: the
// top_k tokens by logit (ties to the lower token id), then the shortest prefix of them,
// in rank order, whose renormalised mass reaches top_p, renormalised. The rule then
// runs on the filtered p' and q'.
//
// The filtered distribution needs no vocabulary-wide normaliser: p'(x) is
// exp((l_x - l_max)/T) over the same sum restricted to the kept tokens. So one launch
// does everything, with one or more blocks per (row, sequence) (more when the batch is
// too small to fill the GPU; the row's last block then gathers its parts):
//   1. each block streams its part of the row once with 16-byte loads and keeps the
//      maximum of every lane of 64 contiguous logits in shared memory (greedy rows: only
//      the lowest-index argmax). The k-th largest lane maximum bounds the k-th largest
//      logit from below, since k distinct lanes each hold an element at least that large;
//   2. a two-digit radix select over the lane maxima finds that bound, the block rescans
//      only the lanes that reach it (about k contiguous 128-byte runs, usually still in
//      L2), ranks the candidates, and takes the top-k, the top-p cut and the
//      renormalised probabilities (fp32 sums of weights whose exponent argument is
//      formed in fp64). If the candidates overflow shared memory (many equal logits),
//      an exact radix select over the whole row replaces the bound;
//   3. the block that finishes a sequence's last row (atomic ticket) takes the gamma-1
//      decisions on p'(t_i) / q'(t_i) and draws the final token by inverse CDF, in
//      ascending token order, over the kept tokens of p'_n (weights [p'_n - q'_n]_+,
//      or p'_B). No block waits for another.
#include <cuda_bf16.h>

#include <cfloat>
#include <climits>
#include <cmath>

#include "common.cuh"

namespace specv {

FilterLayout filter_layout(const spec_accept_args_t& a, int max_top_k, size_t base, int sms,
                           bool draw) {
  FilterLayout L;
  L.lane_shift = 0;
  while ((static_cast<int64_t>(a.vocab) + (kFiltLaneElems << L.lane_shift) - 1) /
             (kFiltLaneElems << L.lane_shift) > kFiltMaxLanes)
    ++L.lane_shift;
  const int lane = kFiltLaneElems << L.lane_shift;
  L.nlanes = static_cast<int>((static_cast<int64_t>(a.vocab) + lane - 1) / lane);
  const int64_t rows = static_cast<int64_t>(a.batch) *
                       (draw ? a.gamma : 2 * static_cast<int64_t>(a.gamma) - 1);
  // split rows across blocks until the grid holds about kFiltBlocksPerSm blocks per SM
  int64_t splits = (static_cast<int64_t>(kFiltBlocksPerSm) * sms + rows - 1) / rows;
  splits = splits < 1 ? 1 : (splits > kFiltMaxSplits ? kFiltMaxSplits : splits);
  if (splits > L.nlanes) splits = L.nlanes;
  L.lanes_per_split = static_cast<int>((L.nlanes + splits - 1) / splits);
  L.splits = (L.nlanes + L.lanes_per_split - 1) / L.lanes_per_split;
  L.cand_cap = 512;
  while (L.cand_cap < 4 * max_top_k && L.cand_cap < 2048) L.cand_cap <<= 1;
  // region A holds the lane maxima, then the ranked candidates (8 B each), then the
  // draw's four lists, each padded to a power of two for the bitonic sort
  int mk2 = 1;
  while (mk2 < max_top_k) mk2 <<= 1;
  size_t a_bytes = static_cast<size_t>(L.nlanes) * 4;
  if (static_cast<size_t>(mk2) * 16 > a_bytes) a_bytes = static_cast<size_t>(mk2) * 16;
  L.smem_a = static_cast<int>((a_bytes + 15) / 16 * 16);
  const size_t split_rows = L.splits > 1 ? static_cast<size_t>(rows) : 0;
  L.tickets = base;
  L.rows = ws_round(L.tickets + sizeof(uint32_t) * a.batch);
  L.kept = ws_round(L.rows + sizeof(FiltRow) * rows);
  L.row_tickets = ws_round(L.kept + 8 * rows * max_top_k);
  L.lanes_g = ws_round(L.row_tickets + sizeof(uint32_t) * split_rows);
  L.parts = ws_round(L.lanes_g + sizeof(uint32_t) * split_rows * L.nlanes);
  L.end = ws_round(L.parts + 16 * split_rows * L.splits);
  return L;
}

namespace {

constexpr int kRowUnroll = 8;        // 16-byte loads in flight per thread
constexpr int kRankSortMax = 256;    // candidates ranked by counting; more are sorted bitonically
constexpr uint32_t kRowBadLogits = 1u, kRowBadFilter = 2u;

struct FiltParams {
  int mode;  // 0: verify (target and drafter rows); 1: draw every drafter row's token
  int batch, gamma, vocab, max_top_k, lane_shift, nlanes;
  int splits, lanes_per_split;  // blocks per row and the lanes each scans
  int cand_cap;                 // candidates (and lanes to rescan) one block holds
  int smem_a;                   // bytes of the shared region of lanes / ranks / draw lists
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
  uint32_t* tickets;  // [batch]
  FiltRow* rows;      // [batch][2*gamma-1]
  int2* kept;         // [batch][2*gamma-1][max_top_k]: (token, p' bits), rank order
  uint32_t* row_tickets;  // [batch][2*gamma-1] (splits > 1)
  uint32_t* lanes_g;      // [batch][2*gamma-1][nlanes] lane maxima (splits > 1)
  uint4* parts;           // [batch][2*gamma-1][splits]: (row max candidate, bad) per split
  int32_t* draw_tokens;   // mode 1: [batch][gamma] block tokens
  float* draw_q;          // mode 1: [batch][gamma] their filtered probabilities, or NULL
};

// Small shared arrays of the decision phase (the sequence's last block).
struct DecideSmall {
  int tok[64], arg[64], nkeep[128];
  float u[64], ptok[64], qtok[64];
};
// The kept lists of the final draw, in the block's dynamic shared memory.
struct DrawLists {
  int* P_id;
  int* Q_id;
  float* P_v;
  float* Q_v;
  float* W;    // the draw's weights, in ascending token order (sorted path)
  float* pre;  // their inclusive prefix sums
};

template <bool BF16>
__device__ __forceinline__ float load_elem(const void* base, int64_t i) {
  if (BF16) return bf16_bits_to_f32(static_cast<const uint16_t*>(base)[i]);
  return static_cast<const float*>(base)[i];
}

// Order-preserving key of a float: a larger value has a larger key; -0 shares +0's key
// so that equal values tie. Keys above order_key(+inf) are NaNs; no finite value or
// infinity has key 0.
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

// Row r of sequence b. Verify: target row r for r < gamma, else drafter row
// r - gamma + 1. Draw: drafter row r.
__device__ __forceinline__ const char* row_ptr(const FiltParams& p, int b, int r, int esz) {
  if (p.mode == 1)
    return static_cast<const char*>(p.drafter) + (static_cast<int64_t>(b) * p.gamma + r) * p.vocab * esz;
  const int64_t row = static_cast<int64_t>(b) * p.gamma + (r < p.gamma ? r : r - p.gamma + 1);
  const void* base = r < p.gamma ? p.target : p.drafter;
  return static_cast<const char*>(base) + row * p.vocab * esz;
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

// Warp 0 of the block: the bin of a 256-bin histogram (the sum of nh histograms 256
// apart) that holds the need-th largest item, counting from the top bin down; *above
// receives the items in higher bins. Returns -1 when there are fewer than need items.
__device__ int find_bin_desc(const uint32_t* hist, int nh, uint32_t need, uint32_t* above) {
  const int lane = threadIdx.x & 31;
  uint32_t cnt[8], sum = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    cnt[j] = 0;
    for (int h = 0; h < nh; ++h) cnt[j] += hist[h * 256 + 255 - (lane * 8 + j)];
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
__device__ void bitonic_desc(unsigned long long* s, int n2) {
  for (int k = 2; k <= n2; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n2; i += kRowThreads) {
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
__device__ void bitonic_pairs_asc(int* id, float* val, int n2) {
  for (int k = 2; k <= n2; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n2; i += kRowThreads) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const int x = id[i], y = id[ixj];
          const bool asc = (i & k) == 0;
          if (asc ? x > y : x < y) {
            id[i] = y;
            id[ixj] = x;
            const float t = val[i];
            val[i] = val[ixj];
            val[ixj] = t;
          }
        }
      }
      __syncthreads();
    }
  }
}

// The first of c consecutive slots of a shared list for every lane of the warp (c = 0
// allowed), with one atomic per warp; all lanes of the warp call it.
__device__ __forceinline__ int warp_slots(int c, int* counter) {
  const int lane = threadIdx.x & 31;
  int incl = c;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  const int total = __shfl_sync(0xffffffffu, incl, 31);
  int base = 0;
  if (lane == 31 && total) base = atomicAdd(counter, total);
  base = __shfl_sync(0xffffffffu, base, 31);
  return base + incl - c;
}

__device__ __forceinline__ int pow2_at_least(int n) {
  int m = 1;
  while (m < n) m <<= 1;
  return m;
}

// Exact fallback of the select phase: the K largest candidates of the whole row by a
// four-digit radix select on the keys, then one pass in token order that keeps every
// element above the K-th key and the lowest-id elements equal to it.
template <bool BF16>
__device__ void exact_topk(const char* rowp, int V, int K, unsigned long long* s_cand, int cap,
                           uint32_t* s_hist, int* s_ncand, int* s_scan, int* s_misc) {
  const int tid = threadIdx.x;
  uint32_t prefix = 0, pmask = 0, need = static_cast<uint32_t>(K);
  for (int d = 3; d >= 0; --d) {
    for (int i = tid; i < 256; i += kRowThreads) s_hist[i] = 0;
    __syncthreads();
    for (int i = tid; i < V; i += kRowThreads) {
      const uint32_t k = order_key(load_elem<BF16>(rowp, i));
      if ((k & pmask) == prefix) atomicAdd(&s_hist[(k >> (8 * d)) & 0xffu], 1u);
    }
    __syncthreads();
    if (tid < 32) {
      uint32_t above = 0;
      const int bin = find_bin_desc(s_hist, 1, need, &above);
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
  for (int base = 0; base < V; base += kRowThreads * kPer) {
    const int first = base + tid * kPer;
    uint32_t keys[kPer];
    int mine = 0;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      keys[q] = first + q < V ? order_key(load_elem<BF16>(rowp, first + q)) : 0u;
      mine += (first + q < V && keys[q] == kappa) ? 1 : 0;
    }
    int total = 0;
    int rank = block_excl_scan<kRowThreads, int>(mine, s_scan, &total);
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
        if (slot < cap) s_cand[slot] = cand_of(keys[q], static_cast<uint32_t>(first + q));
      }
    }
    tie_base += total;
  }
  __syncthreads();
}

// The decisions of sequence b on p'(t_i) / q'(t_i), every output, and the final draw;
// run by the block that finished the sequence's last row. Row results written by other
// blocks are read through L2 (__ldcg).
__device__ void decide_sequence(const FiltParams& p, int b, DecideSmall& d, DrawLists L,
                                float* s_fscan, int* s_flags) {
  constexpr int kThreads = kRowThreads;
  const int tid = threadIdx.x;
  const int gamma = p.gamma, V = p.vocab, nrows = 2 * gamma - 1;
  const float T = p.temperature[b];
  const bool greedy = !(T > 0.f);
  if (tid == 0) {
    s_flags[0] = 0;      // bad bits
    s_flags[1] = gamma;  // n
    s_flags[2] = INT_MAX;
    s_flags[3] = -1;
  }
  if (tid < gamma) {
    d.tok[tid] = p.tokens[static_cast<int64_t>(b) * gamma + tid];
    d.u[tid] = p.uniforms[static_cast<int64_t>(b) * gamma + tid];
  }
  __syncthreads();
  const int rows_needed = greedy ? gamma : nrows;
  for (int r = tid; r < rows_needed; r += kThreads) {
    const FiltRow* fr = p.rows + static_cast<int64_t>(b) * nrows + r;
    const uint32_t flags = __ldcg(&fr->flags);
    if (flags & kRowBadLogits) atomicOr(&s_flags[0], 2);
    if (flags & kRowBadFilter) atomicOr(&s_flags[0], 4);
    d.nkeep[r] = __ldcg(&fr->nkeep);
    if (r < gamma) d.arg[r] = __ldcg(&fr->argmax);
  }
  if (tid < gamma && (d.tok[tid] < 0 || d.tok[tid] >= V)) atomicOr(&s_flags[0], 1);
  __syncthreads();

  const int64_t orow = static_cast<int64_t>(b) * (gamma + 1);
  if (s_flags[0]) {
    for (int k = tid; k <= gamma; k += kThreads) p.out_tokens[orow + k] = -1;
    if (p.diag)
      for (int k = tid; k < 2 * gamma; k += kThreads)
        p.diag[static_cast<int64_t>(b) * gamma * 2 + k] = NAN;
    if (tid == 0) {
      p.num_accepted[b] = -1;
      p.num_emitted[b] = 0;
      if (s_flags[0] & 1) set_status(p.status, SPEC_FLAG_BAD_TOKEN);
      if (s_flags[0] & 2) set_status(p.status, SPEC_FLAG_BAD_LOGITS);
      if (s_flags[0] & 4) set_status(p.status, SPEC_FLAG_BAD_FILTER);
    }
    return;
  }

  // the gamma-1 decisions. Tempered: every (draft, side, kept entry) lookup is issued at
  // once, four per thread per round, then one thread per draft decides.
  for (int i = tid; i < gamma; i += kThreads) {
    d.ptok[i] = 0.f;
    d.qtok[i] = 0.f;
  }
  __syncthreads();
  if (!greedy) {
    const int mk = p.max_top_k;
    const int total = (gamma - 1) * 2 * mk;
    for (int it0 = tid; it0 < total; it0 += 4 * kThreads) {
      int2 e[4];
      int side[4], draft[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int it = it0 + u * kThreads;
        e[u] = make_int2(-1, 0);
        draft[u] = 0;
        side[u] = 0;
        if (it < total) {
          const int j = it % mk, sd = (it / mk) & 1, i = it / (2 * mk) + 1;
          const int r = sd ? gamma + i - 1 : i - 1;
          draft[u] = i;
          side[u] = sd;
          if (j < d.nkeep[r]) e[u] = __ldcg(p.kept + (static_cast<int64_t>(b) * nrows + r) * mk + j);
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (e[u].x >= 0 && e[u].x == d.tok[draft[u]]) (side[u] ? d.qtok : d.ptok)[draft[u]] = __int_as_float(e[u].y);
    }
    __syncthreads();
  }
  for (int i = 1 + tid; i < gamma; i += kThreads) {
    const int t = d.tok[i];
    bool reject;
    if (greedy) {
      reject = t != d.arg[i - 1];
      d.ptok[i] = reject ? 0.f : 1.f;
      d.qtok[i] = 1.f;
    } else {
      const float pd = d.ptok[i], qd = d.qtok[i];
      // a draft outside q's filtered support: accept iff p'(t) > 0
      const float ratio = qd > 0.f ? pd / qd : (pd > 0.f ? INFINITY : 0.f);
      reject = d.u[i - 1] > fminf(1.f, ratio);
    }
    if (reject) atomicMin(&s_flags[1], i);
  }
  __syncthreads();
  const int n = s_flags[1];
  for (int k = tid; k <= gamma; k += kThreads) {
    if (k < n) p.out_tokens[orow + k] = d.tok[k];
    else if (k > n) p.out_tokens[orow + k] = -1;
    else if (greedy) p.out_tokens[orow + k] = d.arg[n - 1];
  }
  if (p.diag) {
    for (int i = tid; i < gamma; i += kThreads) {
      const int64_t dd = (static_cast<int64_t>(b) * gamma + i) * 2;
      const bool taken = i >= 1 && i <= n && i < gamma;
      p.diag[dd] = i == 0 ? 0.f : (taken ? d.ptok[i] : NAN);
      p.diag[dd + 1] = i == 0 ? 0.f : (taken ? d.qtok[i] : NAN);
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
  const int nP = d.nkeep[n - 1];
  const int nQ = bonus ? 0 : d.nkeep[gamma + n - 1];
  for (int j = tid; j < nP; j += kThreads) {
    const int2 e = __ldcg(p.kept + prid * p.max_top_k + j);
    L.P_id[j] = e.x;
    L.P_v[j] = __int_as_float(e.y);
  }
  for (int j = tid; j < nQ; j += kThreads) {
    const int2 e = __ldcg(p.kept + qrid * p.max_top_k + j);
    L.Q_id[j] = e.x;
    L.Q_v[j] = __int_as_float(e.y);
  }
  __syncthreads();
  if (nP <= kThreads && nQ <= kThreads) {
    // one kept token per thread: its weight, then its cumulative weight C(x) over the
    // kept tokens with ids <= x (no sort); the token is the smallest x with
    // C(x) >= u * S and a positive weight
    const int j = tid;
    const int my_id = j < nP ? L.P_id[j] : INT_MAX;
    float wj = 0.f;
    if (j < nP) {
      wj = L.P_v[j];
      if (!bonus) {
        float qv = 0.f;
        for (int i = 0; i < nQ; ++i)
          if (L.Q_id[i] == my_id) qv = L.Q_v[i];
        wj = fmaxf(0.f, wj - qv);
      }
    }
    float* W = L.Q_v;  // q' is no longer needed once every thread has its weight
    __syncthreads();
    if (j < nP) W[j] = wj;
    __syncthreads();
    float S = 0.f, C = 0.f;
    for (int i = 0; i < nP; ++i) {
      const float x = W[i];
      S += x;
      if (L.P_id[i] <= my_id) C += x;
    }
    if (bonus || !(S > 0.f)) {
      // the bonus draw, or a residual without mass (only through rounding): p'_n itself
      wj = j < nP ? L.P_v[j] : 0.f;
      S = 0.f;
      C = 0.f;
      for (int i = 0; i < nP; ++i) {
        const float x = L.P_v[i];
        S += x;
        if (L.P_id[i] <= my_id) C += x;
      }
    }
    if (j < nP && wj > 0.f) {
      atomicMax(&s_flags[3], my_id);
      if (C >= d.u[gamma - 1] * S) atomicMin(&s_flags[2], my_id);
    }
    __syncthreads();
    if (tid == 0)  // rounding that leaves u * S above every sum: the last positive weight
      p.out_tokens[orow + n] = s_flags[2] != INT_MAX ? s_flags[2] : s_flags[3];
    return;
  }
  const int nP2 = pow2_at_least(max(nP, 2)), nQ2 = pow2_at_least(max(nQ, 2));
  for (int j = nP + tid; j < nP2; j += kThreads) {
    L.P_id[j] = INT_MAX;
    L.P_v[j] = 0.f;
  }
  for (int j = nQ + tid; j < nQ2; j += kThreads) {
    L.Q_id[j] = INT_MAX;
    L.Q_v[j] = 0.f;
  }
  __syncthreads();
  bitonic_pairs_asc(L.P_id, L.P_v, nP2);
  if (!bonus) bitonic_pairs_asc(L.Q_id, L.Q_v, nQ2);
  // residual weights [p' - q']_+ (q' by binary search), then their prefix sums
  for (int j = tid; j < nP; j += kThreads) {
    float x = L.P_v[j];
    if (!bonus) {
      const int t = L.P_id[j];
      int lo = 0, hi = nQ;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (L.Q_id[mid] < t) lo = mid + 1;
        else hi = mid;
      }
      const float qv = (lo < nQ && L.Q_id[lo] == t) ? L.Q_v[lo] : 0.f;
      x = fmaxf(0.f, x - qv);
    }
    L.W[j] = x;
  }
  float S = 0.f;
  for (int pass = 0; pass < 2; ++pass) {
    __syncthreads();
    float carry = 0.f;
    for (int j0 = 0; j0 < nP; j0 += kThreads) {
      const int j = j0 + tid;
      const float x = j < nP ? L.W[j] : 0.f;
      float tot = 0.f;
      const float ex = block_excl_scan<kThreads, float>(x, s_fscan, &tot);
      if (j < nP) L.pre[j] = carry + ex + x;
      carry += tot;
    }
    S = carry;
    if (pass == 1 || (!bonus && S > 0.f)) break;
    // the bonus draw, or a residual without mass (only through rounding): p'_n itself
    for (int j = tid; j < nP; j += kThreads) L.W[j] = L.P_v[j];
    if (bonus) continue;
  }
  __syncthreads();
  const float target = d.u[gamma - 1] * S;
  for (int j = tid; j < nP; j += kThreads) {
    if (L.W[j] > 0.f) {
      atomicMax(&s_flags[3], j);
      if (L.pre[j] >= target) atomicMin(&s_flags[2], j);
    }
  }
  __syncthreads();
  if (tid == 0) {
    const int j = s_flags[2] != INT_MAX ? s_flags[2] : s_flags[3];  // rounding: last positive
    p.out_tokens[orow + n] = j >= 0 ? L.P_id[j] : -1;
  }
}

// One block per (split, row, sequence): scan, select (the row's last block) and decide
// (the sequence's last block).
template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kRowThreads, 8) filter_row_kernel(FiltParams p) {
  extern __shared__ __align__(16) unsigned char dsm[];
  __shared__ DecideSmall dsmall;
  __shared__ unsigned long long s_red[kRowThreads / 32];
  __shared__ uint32_t s_hist[(kRowThreads / 32) * 256];  // one histogram per warp
  __shared__ float s_fscan[kRowThreads / 32 + 1];
  __shared__ int s_iscan[kRowThreads / 32 + 1];
  __shared__ int s_misc[4];
  __shared__ int s_flags[4];
  __shared__ int s_ncand, s_keep, s_bad, s_last;

  const int split = blockIdx.x, r = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int gamma = p.gamma, nrows = p.mode == 1 ? gamma : 2 * gamma - 1, V = p.vocab;
  const float T = p.temperature[b];
  const bool greedy = !(T > 0.f);
  if (greedy && r >= gamma) return;  // greedy sequences never read drafter rows (verify)
  const float u_draw = p.mode == 1 ? p.uniforms[static_cast<int64_t>(b) * gamma + r] : 0.f;
  const int64_t rid = static_cast<int64_t>(b) * nrows + r;
  const char* rowp = row_ptr(p, b, r, BF16 ? 2 : 4);
  const int lane_elems = kFiltLaneElems << p.lane_shift;
  const int nlanes = p.nlanes;
  const int cap = p.cand_cap;
  const int k_in = greedy ? 1 : p.top_k[b];
  const float tp = greedy ? 1.f : p.top_p[b];
  // dynamic shared memory: region A (lane maxima, then the ranked candidates, then the
  // draw's lists), the candidates, the lanes to rescan
  uint32_t* lanes = reinterpret_cast<uint32_t*>(dsm);
  unsigned long long* cand = reinterpret_cast<unsigned long long*>(dsm + p.smem_a);
  int* qlane = reinterpret_cast<int*>(dsm + p.smem_a + static_cast<size_t>(cap) * 8);
  // this block's lanes [l0, l1) and elements [e_begin, e_end)
  const int l0 = split * p.lanes_per_split;
  const int l1 = min(nlanes, l0 + p.lanes_per_split);
  const int e_begin = l0 * lane_elems;
  const int e_end = min(V, l1 * lane_elems);

  if (tid == 0) s_bad = 0;
  if (!greedy)
    for (int i = tid; i < l1 - l0; i += kRowThreads) lanes[i] = 0u;
  __syncthreads();

  // 1. scan: the maximum (greedy: with its lowest index) and the lane maxima of the
  // block's part of the row
  float m = -INFINITY;
  int a = INT_MAX;
  bool bad = false;
  if (VEC) {
    constexpr int kEpv = BF16 ? 8 : 4;      // elements per 16-byte vector
    constexpr int kGroup = 64 / kEpv;       // vectors (threads) per 64-element lane
    const uint32_t ninf = BF16 ? 0xFF80FF80u : 0xFF800000u;
    // NaN test on packed words: a magnitude above +inf's carries into the top bit
    const uint32_t nan_mask = BF16 ? 0x7FFF7FFFu : 0x7FFFFFFFu;
    const uint32_t nan_add = BF16 ? 0x007F007Fu : 0x007FFFFFu;
    const uint32_t nan_top = BF16 ? 0x80008000u : 0x80000000u;
    const int vpl = lane_elems / kEpv;
    const int vbeg = e_begin / kEpv, vend = e_end / kEpv;
    const uint4* rv = reinterpret_cast<const uint4*>(rowp);
    uint32_t nacc = 0;
    if (vbeg + tid < vend) a = (vbeg + tid) * kEpv;  // a thread's first element starts its argmax
    bool packed = false;
    if constexpr (BF16) {
      if (!greedy) {
        // Sampled bf16 rows need only the lane maxima. Each thread folds each of its
        // vectors to a bf16 pair by packed maxima, then the 8 threads of a lane trade
        // halves in three shuffle rounds (bits 2, 1, 0 of the thread's index in its
        // group), after which thread i of the group holds the maximum of the lane the
        // group read in unroll step i: one conversion, key and shared atomic per lane
        // instead of per vector. The maxima propagate NaNs, so one test per lane finds
        // them.
        static_assert(kRowUnroll == 8 && kGroup == 8, "one lane per thread of a group");
        packed = true;
        const int gi = tid & 7;
        auto hmax = [](uint32_t x, uint32_t y) {
          const __nv_bfloat162 r = __hmax2_nan(*reinterpret_cast<const __nv_bfloat162*>(&x),
                                               *reinterpret_cast<const __nv_bfloat162*>(&y));
          return *reinterpret_cast<const uint32_t*>(&r);
        };
        for (int v0 = vbeg; v0 < vend; v0 += kRowThreads * kRowUnroll) {
          uint4 dv[kRowUnroll];
#pragma unroll
          for (int u = 0; u < kRowUnroll; ++u) {
            const int vi = v0 + u * kRowThreads + tid;
            dv[u] = vi < vend ? __ldg(rv + vi) : make_uint4(ninf, ninf, ninf, ninf);
          }
          uint32_t h[kRowUnroll];
#pragma unroll
          for (int u = 0; u < kRowUnroll; ++u) h[u] = hmax(hmax(dv[u].x, dv[u].y), hmax(dv[u].z, dv[u].w));
#pragma unroll
          for (int half = 4; half >= 1; half >>= 1) {
            const bool up = (gi & half) != 0;
#pragma unroll
            for (int i = 0; i < half; ++i) {
              const uint32_t send = up ? h[i] : h[i + half], keep = up ? h[i + half] : h[i];
              h[i] = hmax(keep, __shfl_xor_sync(0xffffffffu, send, half));
            }
          }
          const int vl = v0 + gi * kRowThreads + (tid & ~7);  // the owned lane's first vector here
          if (vl < vend) {
            nacc |= (h[0] & nan_mask) + nan_add;
            const float lm = fmaxf(__uint_as_float(h[0] << 16), __uint_as_float(h[0] & 0xffff0000u));
            m = fmaxf(m, lm);
            atomicMax(&lanes[vl / vpl - l0], order_key(lm));
          }
        }
      }
    }
    for (int v0 = packed ? vend : vbeg; v0 < vend; v0 += kRowThreads * kRowUnroll) {
      uint4 dv[kRowUnroll];
#pragma unroll
      for (int u = 0; u < kRowUnroll; ++u) {
        const int vi = v0 + u * kRowThreads + tid;
        dv[u] = vi < vend ? __ldg(rv + vi) : make_uint4(ninf, ninf, ninf, ninf);
      }
#pragma unroll
      for (int u = 0; u < kRowUnroll; ++u) {
        const int vi = v0 + u * kRowThreads + tid;
        const uint32_t wv[4] = {dv[u].x, dv[u].y, dv[u].z, dv[u].w};
#pragma unroll
        for (int q = 0; q < 4; ++q) nacc |= (wv[q] & nan_mask) + nan_add;
        if (greedy) {
          // elements in increasing index order: a strict > keeps the lowest index
#pragma unroll
          for (int q = 0; q < kEpv; ++q) {
            const float x = BF16 ? __uint_as_float((q & 1) ? (wv[q >> 1] & 0xffff0000u) : (wv[q >> 1] << 16))
                                 : __uint_as_float(wv[q]);
            if (x > m) { m = x; a = vi * kEpv + q; }
          }
        } else {
          float vm;
          if (BF16) {
            __nv_bfloat162 h = __hmax2(*reinterpret_cast<const __nv_bfloat162*>(&wv[0]),
                                       *reinterpret_cast<const __nv_bfloat162*>(&wv[1]));
            h = __hmax2(h, *reinterpret_cast<const __nv_bfloat162*>(&wv[2]));
            h = __hmax2(h, *reinterpret_cast<const __nv_bfloat162*>(&wv[3]));
            vm = fmaxf(__bfloat162float(h.x), __bfloat162float(h.y));
          } else {
            vm = fmaxf(fmaxf(__uint_as_float(wv[0]), __uint_as_float(wv[1])),
                       fmaxf(__uint_as_float(wv[2]), __uint_as_float(wv[3])));
          }
          m = fmaxf(m, vm);
          // the lane maximum: the kGroup consecutive threads of a lane, then one atomic
          uint32_t key = vi < vend ? order_key(vm) : 0u;
#pragma unroll
          for (int o = 1; o < kGroup; o <<= 1) key = max(key, __shfl_xor_sync(0xffffffffu, key, o));
          if ((tid & (kGroup - 1)) == 0 && vi < vend) atomicMax(&lanes[vi / vpl - l0], key);
        }
      }
    }
    bad = (nacc & nan_top) != 0;
  } else {
    if (e_begin + tid < e_end) a = e_begin + tid;
    for (int e0 = e_begin; e0 < e_end; e0 += kRowThreads * kRowUnroll) {
      float x[kRowUnroll];
#pragma unroll
      for (int u = 0; u < kRowUnroll; ++u) {
        const int ei = e0 + u * kRowThreads + tid;
        x[u] = ei < e_end ? load_elem<BF16>(rowp, ei) : -INFINITY;
      }
#pragma unroll
      for (int u = 0; u < kRowUnroll; ++u) {
        const int ei = e0 + u * kRowThreads + tid;
        bad |= x[u] != x[u];
        if (greedy) {
          if (x[u] > m) { m = x[u]; a = ei; }
        } else {
          m = fmaxf(m, x[u]);
          // a warp's 32 consecutive elements lie in one lane
          uint32_t key = ei < e_end ? order_key(x[u]) : 0u;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) key = max(key, __shfl_xor_sync(0xffffffffu, key, o));
          if ((tid & 31) == 0 && ei < e_end) atomicMax(&lanes[ei / lane_elems - l0], key);
        }
      }
    }
  }
  if (!greedy && m == INFINITY) bad = true;  // +inf leaves a tempered softmax undefined
  // block reduction: the maximum (and its lowest index) and the bad flag
  unsigned long long best = cand_of(order_key(m), static_cast<uint32_t>(a));
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
  for (int k = 1; k < kRowThreads / 32; ++k) best = s_red[k] > best ? s_red[k] : best;

  if (p.splits > 1) {
    // publish this split, and let the row's last block continue with the whole row
    if (!greedy)
      for (int i = tid; i < l1 - l0; i += kRowThreads) p.lanes_g[rid * nlanes + l0 + i] = lanes[i];
    if (tid == 0)
      p.parts[rid * p.splits + split] = make_uint4(static_cast<uint32_t>(best), static_cast<uint32_t>(best >> 32),
                                                   static_cast<uint32_t>(s_bad), 0u);
    __threadfence();
    __syncthreads();
    if (tid == 0) {
      const uint32_t prev = atomicAdd(&p.row_tickets[rid], 1u);
      s_last = prev == static_cast<uint32_t>(p.splits - 1);
      if (s_last) p.row_tickets[rid] = 0;  // leave the counter at zero for the next call
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    if (!greedy)
      for (int i = tid; i < nlanes; i += kRowThreads) lanes[i] = __ldcg(p.lanes_g + rid * nlanes + i);
    best = 0ull;
    uint32_t anybad = 0;
    for (int k = tid; k < p.splits; k += kRowThreads) {
      const uint4 q = __ldcg(p.parts + rid * p.splits + k);
      const unsigned long long c = (static_cast<unsigned long long>(q.y) << 32) | q.x;
      best = c > best ? c : best;
      anybad |= q.z;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long y = __shfl_xor_sync(0xffffffffu, best, o);
      best = y > best ? y : best;
    }
    anybad = __reduce_or_sync(0xffffffffu, anybad);
    __syncthreads();
    if ((tid & 31) == 0) s_red[tid >> 5] = best;
    if (tid == 0) s_bad = 0;
    __syncthreads();
    if ((tid & 31) == 0 && anybad) s_bad = 1;
    __syncthreads();
    best = s_red[0];
#pragma unroll
    for (int k = 1; k < kRowThreads / 32; ++k) best = s_red[k] > best ? s_red[k] : best;
  }

  FiltRow info;
  info.nkeep = 0;
  info.argmax = cand_tok(best);
  info.flags = 0;
  info.pad = 0;
  if (s_bad || (!greedy && static_cast<uint32_t>(best >> 32) <= order_key(-INFINITY)))
    info.flags = kRowBadLogits;  // NaN, +inf (tempered) or no finite logit (tempered)
  else if (!greedy && (k_in < 1 || k_in > p.max_top_k || !(tp > 0.f) || !(tp <= 1.f)))
    info.flags = kRowBadFilter;

  if (!greedy && !info.flags) {
    // 2. select. The bound: the high 16 bits of the K-th largest lane key (0: every
    // element), by two radix digits; each warp counts into its own histogram
    const int K = min(k_in, V);
    uint32_t* my_hist = s_hist + (tid >> 5) * 256;
    for (int i = tid; i < (kRowThreads / 32) * 256; i += kRowThreads) s_hist[i] = 0;
    __syncthreads();
    for (int i = tid; i < nlanes; i += kRowThreads) atomicAdd(&my_hist[lanes[i] >> 24], 1u);
    __syncthreads();
    if (tid < 32) {
      uint32_t above = 0;
      const int bin = find_bin_desc(s_hist, kRowThreads / 32, static_cast<uint32_t>(K), &above);
      if (tid == 0) {
        s_misc[0] = bin;
        s_misc[1] = static_cast<int>(above);
      }
    }
    __syncthreads();
    uint32_t beta = 0;
    const int b1 = s_misc[0];
    if (b1 >= 0) {
      const uint32_t need = static_cast<uint32_t>(K - s_misc[1]);
      for (int i = tid; i < (kRowThreads / 32) * 256; i += kRowThreads) s_hist[i] = 0;
      __syncthreads();
      for (int i = tid; i < nlanes; i += kRowThreads) {
        const uint32_t k = lanes[i];
        if (static_cast<int>(k >> 24) == b1) atomicAdd(&my_hist[(k >> 16) & 0xffu], 1u);
      }
      __syncthreads();
      if (tid < 32) {
        uint32_t above = 0;
        const int bin = find_bin_desc(s_hist, kRowThreads / 32, need, &above);
        if (tid == 0) s_misc[2] = bin;
      }
      __syncthreads();
      beta = (static_cast<uint32_t>(b1) << 24) | (static_cast<uint32_t>(s_misc[2]) << 16);
    }
    // the lanes that can hold a top-K element (counted, then placed by a block scan)
    int mine = 0;
    for (int i = tid; i < nlanes; i += kRowThreads) mine += lanes[i] >= beta ? 1 : 0;
    int nq = 0;
    int slot = block_excl_scan<kRowThreads, int>(mine, s_iscan, &nq);
    if (nq <= cap)
      for (int i = tid; i < nlanes; i += kRowThreads)
        if (lanes[i] >= beta) qlane[slot++] = i;
    if (tid == 0) s_ncand = 0;
    __syncthreads();
    // their elements at or above the bound
    if (nq <= cap) {
      // items of 8 contiguous elements: lane_elems / 8 per lane
      const int ipl = lane_elems / 8;
      for (int it0 = 0; it0 < nq * ipl; it0 += kRowThreads) {
        const int it = it0 + tid;
        const bool live = it < nq * ipl;
        const int e0 = live ? qlane[it / ipl] * lane_elems + (it % ipl) * 8 : V;
        float x[8];
        if (VEC) {
          constexpr int kEpv = BF16 ? 8 : 4;
#pragma unroll
          for (int h = 0; h < 8 / kEpv; ++h) {
            const int e = e0 + h * kEpv;
            uint4 v = make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u);
            if (e < V) v = __ldg(reinterpret_cast<const uint4*>(rowp + static_cast<int64_t>(e) * (BF16 ? 2 : 4)));
            const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int q = 0; q < kEpv; ++q)
              x[h * kEpv + q] = BF16 ? __uint_as_float((q & 1) ? (wv[q >> 1] & 0xffff0000u) : (wv[q >> 1] << 16))
                                     : __uint_as_float(wv[q]);
          }
        } else {
#pragma unroll
          for (int q = 0; q < 8; ++q) x[q] = e0 + q < V ? load_elem<BF16>(rowp, e0 + q) : -INFINITY;
        }
        uint32_t kq[8];
        unsigned takem = 0;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          kq[q] = order_key(x[q]);
          if (e0 + q < V && kq[q] >= beta) takem |= 1u << q;
        }
        int c = warp_slots(__popc(takem), &s_ncand);
#pragma unroll
        for (int q = 0; q < 8; ++q)
          if ((takem >> q) & 1u) {
            if (c < cap) cand[c] = cand_of(kq[q], static_cast<uint32_t>(e0 + q));
            ++c;
          }
      }
    }
    __syncthreads();
    if (nq > cap || s_ncand > cap)
      exact_topk<BF16>(rowp, V, K, cand, cap, s_hist, &s_ncand, s_iscan, s_misc);
    const int ncand = min(s_ncand, cap);
    // the top K candidates in rank order (region A: the lane maxima are no longer needed)
    unsigned long long* ranked = reinterpret_cast<unsigned long long*>(dsm);
    if (ncand <= kRankSortMax) {
      for (int j = tid; j < ncand; j += kRowThreads) {
        const unsigned long long c = cand[j];
        int rank = 0;
        for (int i = 0; i < ncand; ++i) rank += cand[i] > c ? 1 : 0;
        if (rank < K) ranked[rank] = c;
      }
    } else {
      const int n2 = pow2_at_least(ncand);
      for (int i = ncand + tid; i < n2; i += kRowThreads) cand[i] = 0ull;
      __syncthreads();
      bitonic_desc(cand, n2);
      for (int j = tid; j < min(K, ncand); j += kRowThreads) ranked[j] = cand[j];
    }
    __syncthreads();

    // top-p on the renormalised top-K. w_j = exp(z_j - z_0), z = l / T: the argument is
    // formed in fp64 (exact difference, one product) and split into an fp32 pair, so
    // that w_j carries only expf's rounding; sums and ratios are fp32. The weights and
    // their prefix sums live where the candidates and the rescan list were.
    const int keff = min(K, ncand);
    float* wsm = reinterpret_cast<float*>(cand);
    float* pre = reinterpret_cast<float*>(qlane);
    {
      const double cT = 1.0 / static_cast<double>(T);
      const double x0 = static_cast<double>(key_value(static_cast<uint32_t>(ranked[0] >> 32)));
      for (int j = tid; j < keff; j += kRowThreads) {
        const double z = (static_cast<double>(key_value(static_cast<uint32_t>(ranked[j] >> 32))) - x0) * cT;
        const float zh = static_cast<float>(z);
        const float zl = static_cast<float>(z - static_cast<double>(zh));
        wsm[j] = expf(zh) * (1.f + zl);
      }
    }
    __syncthreads();
    float carry = 0.f;
    for (int j0 = 0; j0 < keff; j0 += kRowThreads) {
      const int j = j0 + tid;
      const float x = j < keff ? wsm[j] : 0.f;
      float tot = 0.f;
      const float ex = block_excl_scan<kRowThreads, float>(x, s_fscan, &tot);
      if (j < keff) pre[j] = carry + ex + x;
      carry += tot;
    }
    if (tid == 0) s_keep = keff;
    __syncthreads();
    const float mass = carry;
    if (tp < 1.f)
      for (int j = tid; j < keff; j += kRowThreads)
        if (pre[j] / mass >= tp) atomicMin(&s_keep, j + 1);
    __syncthreads();
    const int keep = s_keep;
    if (p.mode == 1) {
      // the draw: the smallest kept token whose cumulative weight over the kept tokens
      // with ids up to it reaches u * S (every thread sums in the same order)
      if (tid == 0) {
        s_misc[0] = INT_MAX;
        s_misc[1] = -1;
      }
      __syncthreads();
      float Sall = 0.f;
      for (int i = 0; i < keep; ++i) Sall += wsm[i];
      const float target = u_draw * Sall;
      for (int j = tid; j < keep; j += kRowThreads) {
        const int my = cand_tok(ranked[j]);
        float C = 0.f;
        for (int i = 0; i < keep; ++i)
          if (cand_tok(ranked[i]) <= my) C += wsm[i];
        if (wsm[j] > 0.f) {
          atomicMax(&s_misc[1], my);
          if (C >= target) atomicMin(&s_misc[0], my);
        }
      }
      __syncthreads();
      const int tok = s_misc[0] != INT_MAX ? s_misc[0] : s_misc[1];  // rounding: last positive
      for (int j = tid; j < keep; j += kRowThreads)
        if (cand_tok(ranked[j]) == tok) {
          p.draw_tokens[static_cast<int64_t>(b) * gamma + r] = tok;
          if (p.draw_q) p.draw_q[static_cast<int64_t>(b) * gamma + r] = wsm[j] / Sall;
        }
    } else {
      const float S = pre[keep - 1];
      int2* kept = p.kept + rid * p.max_top_k;
      for (int j = tid; j < keep; j += kRowThreads)
        kept[j] = make_int2(cand_tok(ranked[j]), __float_as_int(wsm[j] / S));
    }
    info.nkeep = keep;
    info.argmax = cand_tok(ranked[0]);
  } else if (p.mode == 1 && tid == 0) {
    // a greedy row draws its argmax; a bad row's outputs are set by the sequence's last block
    p.draw_tokens[static_cast<int64_t>(b) * gamma + r] = info.flags ? -1 : info.argmax;
    if (p.draw_q) p.draw_q[static_cast<int64_t>(b) * gamma + r] = info.flags ? NAN : 1.f;
  }
  if (tid == 0) p.rows[rid] = info;

  // 3. the last block of the sequence takes its decisions
  __threadfence();  // this block's row results are visible before its ticket
  __syncthreads();
  if (tid == 0) {
    const uint32_t rows_needed = greedy ? gamma : nrows;
    const uint32_t prev = atomicAdd(&p.tickets[b], 1u);
    s_last = prev == rows_needed - 1;
    if (s_last) p.tickets[b] = 0;  // leave the counter at zero for the next call
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (p.mode == 1) {
    // a sequence with a bad row draws nothing: every token -1 (the oracle's convention)
    if (tid == 0) s_flags[0] = 0;
    __syncthreads();
    for (int k = tid; k < gamma; k += kRowThreads)
      atomicOr(&s_flags[0], static_cast<int>(__ldcg(&p.rows[static_cast<int64_t>(b) * nrows + k].flags)));
    __syncthreads();
    if (s_flags[0]) {
      for (int k = tid; k < gamma; k += kRowThreads) {
        p.draw_tokens[static_cast<int64_t>(b) * gamma + k] = -1;
        if (p.draw_q) p.draw_q[static_cast<int64_t>(b) * gamma + k] = NAN;
      }
      if (tid == 0) {
        if (s_flags[0] & kRowBadLogits) set_status(p.status, SPEC_FLAG_BAD_LOGITS);
        if (s_flags[0] & kRowBadFilter) set_status(p.status, SPEC_FLAG_BAD_FILTER);
      }
    }
    return;
  }
  DrawLists L;
  const int mk2 = pow2_at_least(p.max_top_k);  // list stride: room for the sort's padding
  L.P_id = reinterpret_cast<int*>(dsm);
  L.Q_id = L.P_id + mk2;
  L.P_v = reinterpret_cast<float*>(L.Q_id + mk2);
  L.Q_v = L.P_v + mk2;
  L.W = reinterpret_cast<float*>(cand);  // the candidates' region is free again
  L.pre = L.W + cap;
  decide_sequence(p, b, dsmall, L, s_fscan, s_flags);
}

template <bool BF16, bool VEC>
cudaError_t launch_filtered_typed(const FiltParams& p, cudaStream_t stream, bool overlap_prior) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.splits, p.mode == 1 ? p.gamma : 2 * p.gamma - 1, p.batch);
  cfg.blockDim = dim3(kRowThreads);
  cfg.dynamicSmemBytes = p.smem_a + static_cast<size_t>(p.cand_cap) * 12;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = overlap_prior ? 1 : 0;  // beside the attention kernel of a verify step
  const cudaError_t e = cudaLaunchKernelEx(&cfg, filter_row_kernel<BF16, VEC>, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_accept_filtered(const spec_accept_args_t& a, const spec_filter_args_t& f,
                                   const FilterLayout& L, char* ws, cudaStream_t stream,
                                   bool overlap_prior, int32_t* draw_tokens, float* draw_q) {
  FiltParams p;
  p.mode = draw_tokens ? 1 : 0;
  p.draw_tokens = draw_tokens;
  p.draw_q = draw_q;
  p.batch = a.batch;
  p.gamma = a.gamma;
  p.vocab = a.vocab;
  p.max_top_k = f.max_top_k;
  p.lane_shift = L.lane_shift;
  p.nlanes = L.nlanes;
  p.splits = L.splits;
  p.lanes_per_split = L.lanes_per_split;
  p.cand_cap = L.cand_cap;
  p.smem_a = L.smem_a;
  p.row_tickets = reinterpret_cast<uint32_t*>(ws + L.row_tickets);
  p.lanes_g = reinterpret_cast<uint32_t*>(ws + L.lanes_g);
  p.parts = reinterpret_cast<uint4*>(ws + L.parts);
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
  p.tickets = reinterpret_cast<uint32_t*>(ws + L.tickets);
  p.rows = reinterpret_cast<FiltRow*>(ws + L.rows);
  p.kept = reinterpret_cast<int2*>(ws + L.kept);
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
