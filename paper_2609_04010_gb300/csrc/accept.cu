// Part (b) of the verify step: vocabulary-wide softmax statistics of the target and
// drafter rows and the lossless acceptance rule of Alg. "Lossless Psi-Spec decoding
// (Linear Sampler)" (Appendix B.3; Sec. 4.2).
//
// Three launches, no inter-block waiting (each is a programmatic dependent of the one
// before and waits for it on the device; in a verify step the first is a programmatic
// dependent of the attention kernel and runs beside it):
//   1. row_stats_kernel: one warp per (sequence, row, 4096-entry vocab chunk) reads
//      the chunk once with 16-byte loads and writes its max, its sum of
//      exp((l - max)/T) and (greedy rows) its lowest-index argmax.
//   2. decide_kernel: one block per sequence merges the row statistics and evaluates
//      the gamma-1 decisions r_i > min(1, p_i(t_i)/q_i(t_i)) (fp64 on the few
//      gathered logits), which fixes n; it writes every output except a tempered
//      sequence's final token, and a record of the final draw's normalisers.
//   3. sample_kernel: grid (vocab slice, sequence), tempered sequences only. Each block
//      sums the final draw's weights ([p_n - q_n]_+, or p_B for the bonus) over its
//      slice; the last block of the sequence to finish (atomic ticket) finds the slice
//      where the ascending cumulative sum crosses u * S and rescans that slice with a
//      block-wide scan to pick the token.
#include <cuda_bf16.h>

#include <cfloat>
#include <climits>
#include <cmath>

#include "common.cuh"

namespace specv {

AcceptLayout accept_layout(const spec_accept_args_t& a, size_t base) {
  AcceptLayout L;
  L.nchunk = (a.vocab + kStatsChunk - 1) / kStatsChunk;
  L.nslice = (a.vocab + kSampleSlice - 1) / kSampleSlice;
  const size_t nrows = 2 * static_cast<size_t>(a.gamma) - 1;
  L.tickets = base;
  L.partials = ws_round(L.tickets + sizeof(uint32_t) * a.batch);
  L.records = ws_round(L.partials + sizeof(RowPartial) * a.batch * nrows * L.nchunk);
  L.slice_sums = ws_round(L.records + 32 * static_cast<size_t>(a.batch));
  L.end = ws_round(L.slice_sums + sizeof(float4) * a.batch * L.nslice);
  return L;
}

namespace {

struct SliceSum {  // per (sequence, vocab slice) sums of the final draw's weights
  float w;         // sum of [p_n - q_n]_+ (residual)
  float e;         // sum of exp((l_p - M_p)/T) (bonus, and the empty-residual fallback)
  int32_t wlast;   // last index with positive residual weight, -1 if none
  int32_t elast;   // last index with positive bonus weight, -1 if none
};

struct DecideRecord {  // what the sampling kernel needs of a sequence's decisions
  int32_t n;           // first rejected draft (gamma: all accepted); 0: bad sequence
  float Mp, invSp;     // max and 1 / sum of row p_n (target row n - 1)
  float Mq, invSq;     // the same for q_n (drafter row n); unused for the bonus draw
  int32_t pad[3];
};

struct AcceptParams {
  int batch, gamma, vocab, nchunk, nslice;
  const void* target;
  const void* drafter;
  const int32_t* tokens;
  const float* temperature;
  const float* uniforms;
  int32_t* num_accepted;
  int32_t* out_tokens;
  int32_t* num_emitted;
  float* diag;
  uint32_t* status;
  uint32_t* tickets;
  RowPartial* partials;
  DecideRecord* records;
  SliceSum* slices;
};

template <bool BF16>
__device__ __forceinline__ float load_elem(const void* base, int64_t i) {
  if (BF16) return bf16_bits_to_f32(static_cast<const uint16_t*>(base)[i]);
  return static_cast<const float*>(base)[i];
}

// (m, s) pairs of an online softmax sum in base 2 with scale c: value = s * 2^{c*m}.
__device__ __forceinline__ void merge_ms(float& m, float& s, float m2, float s2, float c) {
  const float mn = fmaxf(m, m2);
  float r = 0.f;
  if (m != -INFINITY) r += s * ex2((m - mn) * c);
  if (m2 != -INFINITY) r += s2 * ex2((m2 - mn) * c);
  m = mn;
  s = r;
}

// Warp-wide combination of the lanes' (m, s) pairs: the maximum by shuffles, then each
// lane's sum rescaled once to it and the sums added (a lane with m = -inf adds 0; a NaN
// or infinite input leaves a NaN sum).
__device__ __forceinline__ void warp_merge_ms(float& m, float& s, float c) {
  float mx = m;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  float sc = m != -INFINITY ? s * ex2((m - mx) * c) : 0.f;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sc += __shfl_xor_sync(0xffffffffu, sc, o);
  m = mx;
  s = sc;
}

__device__ __forceinline__ void merge_arg(float& m, int& a, float m2, int a2) {
  if (m2 > m || (m2 == m && a2 < a)) {
    m = m2;
    a = a2;
  }
}

// Warp-wide lowest-index argmax of the lanes' (m, a) pairs.
__device__ __forceinline__ void warp_merge_arg(float& m, int& a) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const int a2 = __shfl_xor_sync(0xffffffffu, a, o);
    merge_arg(m, a, m2, a2);
  }
}

// One warp per (sequence, row, kStatsChunk-entry chunk), with no block-wide step: the
// warp issues all of its chunk's 16-byte loads together (sixteen per lane and round;
// one round for bf16, two for fp32) and reduces with shuffles. Grid (chunk groups of
// kStatsThreads / 32, row, sequence).
template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kStatsThreads, 5) row_stats_kernel(AcceptParams p) {
  pdl_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int c = blockIdx.x * (kStatsThreads / 32) + (threadIdx.x >> 5);
  const int r = blockIdx.y, b = blockIdx.z;
  if (c >= p.nchunk) return;
  const int nrows = 2 * p.gamma - 1;
  const float T = p.temperature[b];
  const bool greedy = !(T > 0.f);
  if (greedy && r >= p.gamma) return;  // greedy sequences never read drafter rows
  const int64_t row = static_cast<int64_t>(b) * p.gamma + (r < p.gamma ? r : r - p.gamma + 1);
  const void* base = r < p.gamma ? p.target : p.drafter;
  const char* rowp = static_cast<const char*>(base) + row * p.vocab * (BF16 ? 2 : 4);
  const int start = c * kStatsChunk;
  const int len = min(kStatsChunk, p.vocab - start);

  uint32_t bad = 0;
  float m = -INFINITY, s = 0.f;
  int a = INT_MAX;
  const float cs = greedy ? 0.f : kLog2e / T;
  if (VEC) {
    constexpr int kEpv = BF16 ? 8 : 4;  // elements per 16-byte group
    constexpr int kGroups = 16;         // groups per lane and round
    constexpr int kRounds = kStatsChunk / (32 * kGroups * kEpv);
    static_assert(kRounds * 32 * kGroups * kEpv == kStatsChunk, "chunk must fill whole rounds");
    const uint32_t ninf = BF16 ? 0xFF80FF80u : 0xFF800000u;  // -inf padding past the row end
    // greedy: this lane's first element starts the argmax (an all -inf chunk reports
    // its lowest index); a lane past the row end loses every tie
    a = lane * kEpv < len ? start + lane * kEpv : INT_MAX;
#pragma unroll
    for (int rd = 0; rd < kRounds; ++rd) {
      uint32_t w[kGroups * 4];
#pragma unroll
      for (int k = 0; k < kGroups; ++k) {
        const int e = ((rd * kGroups + k) * 32 + lane) * kEpv;  // first element of the group
        const uint4 v = e < len ? __ldg(reinterpret_cast<const uint4*>(rowp + static_cast<int64_t>(start + e) * (BF16 ? 2 : 4)))
                                : make_uint4(ninf, ninf, ninf, ninf);
        w[4 * k] = v.x; w[4 * k + 1] = v.y; w[4 * k + 2] = v.z; w[4 * k + 3] = v.w;
      }
      auto elem = [&](int k, int q) -> float {
        if (BF16) {
          const uint32_t word = w[4 * k + (q >> 1)];
          return __uint_as_float((q & 1) ? (word & 0xffff0000u) : (word << 16));
        }
        return __uint_as_float(w[4 * k + q]);
      };
      if (greedy) {
        // elements in increasing index order: a strict > keeps the lowest index
#pragma unroll
        for (int k = 0; k < kGroups; ++k) {
          const int e = ((rd * kGroups + k) * 32 + lane) * kEpv;
#pragma unroll
          for (int q = 0; q < kEpv; ++q) {
            const float x = elem(k, q);
            bad |= x != x;  // NaN (+inf is a legal maximum for a greedy row)
            if (x > m) { m = x; a = start + e + q; }
          }
        }
      } else {
        // max (NaN is skipped here and caught by the sum below), then the sum
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
        float sr = 0.f;
        if (mr != -INFINITY) {
#pragma unroll
          for (int k = 0; k < kGroups; ++k)
#pragma unroll
            for (int q = 0; q < kEpv; ++q) sr += ex2((elem(k, q) - mr) * cs);
        }
        if (rd == 0) {
          m = mr;
          s = sr;
        } else {
          merge_ms(m, s, mr, sr, cs);
        }
      }
    }
    // NaN anywhere, or +inf (then +inf - +inf), makes the sum NaN
    if (!greedy) bad |= !(s <= FLT_MAX) || !(m <= FLT_MAX);
  } else {
    // element loads (rows not 16-byte aligned): element k * 32 + lane, in batches
    constexpr int kBatch = 16;
    a = lane < len ? start + lane : INT_MAX;
    for (int k0 = 0; k0 < kStatsChunk / 32; k0 += kBatch) {
      float v[kBatch];
#pragma unroll
      for (int k = 0; k < kBatch; ++k) {
        const int e = (k0 + k) * 32 + lane;
        v[k] = e < len ? load_elem<BF16>(rowp, start + e) : -INFINITY;
      }
      if (greedy) {
#pragma unroll
        for (int k = 0; k < kBatch; ++k) {
          bad |= v[k] != v[k];
          if (v[k] > m) { m = v[k]; a = start + (k0 + k) * 32 + lane; }
        }
      } else {
        float mr = -INFINITY;
#pragma unroll
        for (int k = 0; k < kBatch; ++k) {
          bad |= !(v[k] <= FLT_MAX);  // NaN or +inf (padding past the row end is -inf)
          mr = fmaxf(mr, v[k]);
        }
        float sr = 0.f;
        if (mr != -INFINITY) {
#pragma unroll
          for (int k = 0; k < kBatch; ++k) sr += ex2((v[k] - mr) * cs);
        }
        merge_ms(m, s, mr, sr, cs);
      }
    }
  }
  // warp reduction
  bad = __reduce_or_sync(0xffffffffu, bad);
  if (greedy) warp_merge_arg(m, a);
  else warp_merge_ms(m, s, cs);
  if (lane == 0) {
    RowPartial out;
    out.m = m;
    out.s = s;
    out.arg = a;
    out.bad = bad;
    p.partials[(static_cast<int64_t>(b) * nrows + r) * p.nchunk + c] = out;
  }
}

// Block-wide exclusive and inclusive scan of one float per thread, in thread order.
template <int kThreads>
__device__ __forceinline__ void block_scan(float x, float& excl, float& incl, float* sh) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  float in = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, in, o);
    if (lane >= o) in += y;
  }
  float ex = __shfl_up_sync(0xffffffffu, in, 1);
  if (lane == 0) ex = 0.f;
  if (lane == 31) sh[w] = in;
  __syncthreads();
  if (threadIdx.x == 0) {
    float run = 0.f;
    for (int k = 0; k < kThreads / 32; ++k) {
      const float t = sh[k];
      sh[k] = run;
      run += t;
    }
    sh[kThreads / 32] = run;
  }
  __syncthreads();
  excl = sh[w] + ex;
  incl = sh[w] + in;
}

// The weights of the final draw on this thread's contiguous run of one slice.
template <bool BF16, bool VEC>
__device__ __forceinline__ void final_weights(const AcceptParams& p, const void* prow,
                                              const void* qrow, bool bonus, int start, float c,
                                              float Mp, float invSp, float Mq, float invSq,
                                              float* w, float* e, int& first) {
  constexpr int kPer = kSamplePerThread;
  first = start + threadIdx.x * kPer;
  float lp[kPer], lq[kPer];
  const int n = min(kPer, p.vocab - first);
  if (VEC && n == kPer) {
    constexpr int kEpv = BF16 ? 8 : 4;
#pragma unroll
    for (int k = 0; k < kPer / kEpv; ++k) {
      const int64_t off = static_cast<int64_t>(first + k * kEpv) * (BF16 ? 2 : 4);
      const uint4 rp = __ldg(reinterpret_cast<const uint4*>(static_cast<const char*>(prow) + off));
      uint4 rq = make_uint4(0, 0, 0, 0);
      if (!bonus) rq = __ldg(reinterpret_cast<const uint4*>(static_cast<const char*>(qrow) + off));
      const uint32_t wp[4] = {rp.x, rp.y, rp.z, rp.w};
      const uint32_t wq[4] = {rq.x, rq.y, rq.z, rq.w};
#pragma unroll
      for (int q = 0; q < kEpv; ++q) {
        if (BF16) {
          lp[k * kEpv + q] = bf16_bits_to_f32((q & 1) ? (wp[q >> 1] >> 16) : (wp[q >> 1] & 0xffffu));
          lq[k * kEpv + q] = bf16_bits_to_f32((q & 1) ? (wq[q >> 1] >> 16) : (wq[q >> 1] & 0xffffu));
        } else {
          lp[k * kEpv + q] = __uint_as_float(wp[q]);
          lq[k * kEpv + q] = __uint_as_float(wq[q]);
        }
      }
    }
  } else {
#pragma unroll
    for (int k = 0; k < kPer; ++k) {
      lp[k] = k < n ? load_elem<BF16>(prow, first + k) : -INFINITY;
      lq[k] = (k < n && !bonus) ? load_elem<BF16>(qrow, first + k) : -INFINITY;
    }
  }
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const float ep = ex2((lp[k] - Mp) * c);
    e[k] = ep;
    w[k] = bonus ? 0.f : fmaxf(0.f, ep * invSp - ex2((lq[k] - Mq) * c) * invSq);
  }
}

// Decisions: one block per sequence merges the chunk statistics of the rows it uses,
// takes the gamma-1 decisions and writes every output except, for a tempered
// sequence, the final drawn token (left to the sampling kernel with a record).
template <bool BF16>
__global__ void __launch_bounds__(kDecideThreads) decide_kernel(AcceptParams p) {
  pdl_launch_dependents();
  constexpr int kMaxGamma = 64;
  __shared__ float rM[2 * kMaxGamma], rS[2 * kMaxGamma];
  __shared__ int rA[2 * kMaxGamma];
  __shared__ int s_tok[kMaxGamma];
  __shared__ float s_ptok[kMaxGamma], s_qtok[kMaxGamma];
  __shared__ int s_bad, s_n;

  const int b = blockIdx.x, tid = threadIdx.x;
  const int gamma = p.gamma, V = p.vocab, nrows = 2 * gamma - 1;
  const float T = p.temperature[b];
  const bool greedy = !(T > 0.f);
  const float c = greedy ? 0.f : kLog2e / T;
  if (tid == 0) {
    s_bad = 0;
    s_n = gamma;
  }
  // The tokens, the logits at the drafted tokens and the uniforms are inputs, not
  // results of the statistics kernel: they are read while that kernel still runs.
  const int my_tok = tid < gamma ? p.tokens[static_cast<int64_t>(b) * gamma + tid] : 0;
  double my_lp = 0.0, my_lq = 0.0;
  float my_u = 0.f;
  if (!greedy && tid >= 1 && tid < gamma && my_tok >= 0 && my_tok < V) {
    my_lp = load_elem<BF16>(p.target, (static_cast<int64_t>(b) * gamma + tid - 1) * V + my_tok);
    my_lq = load_elem<BF16>(p.drafter, (static_cast<int64_t>(b) * gamma + tid) * V + my_tok);
    my_u = p.uniforms[static_cast<int64_t>(b) * gamma + tid - 1];
  }
  pdl_wait_prior();  // the row statistics kernel has finished and its writes are visible
  __syncthreads();

  // 1. merge the chunk statistics of every row this sequence uses: one warp per row,
  // the lanes load the row's chunk partials in parallel and reduce them with shuffles
  // (chunks are in increasing index order, so ties keep the lowest index)
  const int rows_needed = greedy ? gamma : nrows;
  {
    const int warp = tid >> 5, lane = tid & 31;
    for (int r = warp; r < rows_needed; r += kDecideThreads / 32) {
      const RowPartial* rp = p.partials + (static_cast<int64_t>(b) * nrows + r) * p.nchunk;
      float M = -INFINITY, S = 0.f;
      int A = INT_MAX;
      uint32_t bad = 0;
      for (int k = lane; k < p.nchunk; k += 32) {
        const RowPartial q = rp[k];
        bad |= q.bad;
        if (greedy) merge_arg(M, A, q.m, q.arg);
        else merge_ms(M, S, q.m, q.s, c);
      }
      bad = __reduce_or_sync(0xffffffffu, bad);
      if (greedy) warp_merge_arg(M, A);
      else warp_merge_ms(M, S, c);
      if (!greedy && (M == -INFINITY || !(S > 0.f) || !(S <= FLT_MAX))) bad = 1;
      if (lane == 0) {
        rM[r] = M;
        rS[r] = S;
        rA[r] = A;
        if (bad) atomicOr(&s_bad, 1);
      }
    }
  }
  if (tid < gamma) {
    s_tok[tid] = my_tok;
    if (my_tok < 0 || my_tok >= V) atomicOr(&s_bad, 2);
  }
  __syncthreads();

  const int64_t orow = static_cast<int64_t>(b) * (gamma + 1);
  if (s_bad) {
    for (int k = tid; k <= gamma; k += kDecideThreads) p.out_tokens[orow + k] = -1;
    if (p.diag)
      for (int k = tid; k < 2 * gamma; k += kDecideThreads)
        p.diag[static_cast<int64_t>(b) * gamma * 2 + k] = NAN;
    if (tid == 0) {
      p.num_accepted[b] = -1;
      p.num_emitted[b] = 0;
      set_status(p.status, (s_bad & 2) ? SPEC_FLAG_BAD_TOKEN : SPEC_FLAG_BAD_LOGITS);
      if ((s_bad & 3) == 3) set_status(p.status, SPEC_FLAG_BAD_LOGITS);
      DecideRecord rec = {};
      rec.n = 0;  // nothing to draw
      p.records[b] = rec;
    }
    return;
  }

  // 2. the gamma-1 acceptance decisions, one per thread
  if (tid >= 1 && tid < gamma) {
    const int i = tid, t = s_tok[i];
    bool reject;
    float pt, qt;
    if (greedy) {
      reject = t != rA[i - 1];
      pt = reject ? 0.f : 1.f;
      qt = 1.f;
    } else {
      const double lp = my_lp, lq = my_lq;  // this thread's token is t (fetched above)
      const double Td = static_cast<double>(T);
      const double pd = exp((lp - static_cast<double>(rM[i - 1])) / Td) / static_cast<double>(rS[i - 1]);
      const double qd = exp((lq - static_cast<double>(rM[gamma + i - 1])) / Td) /
                        static_cast<double>(rS[gamma + i - 1]);
      // q_i(t_i) = 0 (underflow): accept iff p_i(t_i) > 0
      const double ratio = qd > 0.0 ? pd / qd : (pd > 0.0 ? INFINITY : 0.0);
      const double u = static_cast<double>(my_u);
      reject = u > fmin(1.0, ratio);
      pt = static_cast<float>(pd);
      qt = static_cast<float>(qd);
    }
    s_ptok[i] = pt;
    s_qtok[i] = qt;
    if (reject) atomicMin(&s_n, i);
  }
  __syncthreads();
  const int n = s_n;

  // every output but the final token of a tempered sequence
  for (int k = tid; k <= gamma; k += kDecideThreads) {
    if (k < n) p.out_tokens[orow + k] = s_tok[k];
    else if (k > n) p.out_tokens[orow + k] = -1;
    else if (greedy) p.out_tokens[orow + k] = rA[n - 1];
  }
  if (p.diag) {
    for (int i = tid; i < gamma; i += kDecideThreads) {
      const int64_t d = (static_cast<int64_t>(b) * gamma + i) * 2;
      const bool taken = i >= 1 && i <= n && i < gamma;
      p.diag[d] = i == 0 ? 0.f : (taken ? s_ptok[i] : NAN);
      p.diag[d + 1] = i == 0 ? 0.f : (taken ? s_qtok[i] : NAN);
    }
  }
  if (tid == 0) {
    p.num_accepted[b] = n - 1;
    p.num_emitted[b] = n + 1;
    if (!greedy) {
      const bool bonus = n == gamma;
      DecideRecord rec = {};
      rec.n = n;
      rec.Mp = rM[n - 1];
      rec.invSp = 1.f / rS[n - 1];
      rec.Mq = bonus ? 0.f : rM[gamma + n - 1];
      rec.invSq = bonus ? 0.f : 1.f / rS[gamma + n - 1];
      p.records[b] = rec;
    }
  }
}

// Sampling: grid (vocab slice, sequence) for tempered sequences. Each block sums the
// final draw's weights over its slice; the last block of the sequence (atomic ticket)
// finds the slice where the ascending cumulative sum crosses u * S and rescans it.
template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kSampleThreads, 5) sample_kernel(AcceptParams p) {
  constexpr int kPer = kSamplePerThread;
  __shared__ int s_last, s_star, s_use_res, s_owner, s_token;
  __shared__ float s_base, s_target;
  __shared__ float sh_scan[kSampleThreads / 32 + 1];
  const int b = blockIdx.y, sl = blockIdx.x, tid = threadIdx.x;
  const int gamma = p.gamma, V = p.vocab;
  const float T = p.temperature[b];
  if (!(T > 0.f)) return;  // greedy: the decide kernel wrote the whole row
  const float c = kLog2e / T;
  if (tid == 0) {
    s_owner = INT_MAX;
    s_token = -1;
  }
  pdl_wait_prior();  // the decide kernel has finished and its writes are visible
  const DecideRecord rec = p.records[b];
  const int n = rec.n;
  if (n < 1) return;  // bad sequence: nothing to draw
  const int64_t orow = static_cast<int64_t>(b) * (gamma + 1);

  // 3. sums of the final draw's weights over this block's slice
  const bool bonus = n == gamma;
  const void* prow = static_cast<const char*>(p.target) +
                     (static_cast<int64_t>(b) * gamma + n - 1) * V * (BF16 ? 2 : 4);
  const void* qrow = bonus ? prow
                           : static_cast<const char*>(p.drafter) +
                                 (static_cast<int64_t>(b) * gamma + n) * V * (BF16 ? 2 : 4);
  const float Mp = rec.Mp, invSp = rec.invSp, Mq = rec.Mq, invSq = rec.invSq;

  float w[kPer], e[kPer];
  int first;
  final_weights<BF16, VEC>(p, prow, qrow, bonus, sl * kSampleSlice, c, Mp, invSp, Mq, invSq, w,
                           e, first);
  float lw = 0.f, le = 0.f;
  int wlast = -1, elast = -1;
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    lw += w[k];
    le += e[k];
    if (w[k] > 0.f) wlast = first + k;
    if (e[k] > 0.f) elast = first + k;
  }
  float ex, inw, ine;
  block_scan<kSampleThreads>(lw, ex, inw, sh_scan);
  const float tot_w = sh_scan[kSampleThreads / 32];
  __syncthreads();
  block_scan<kSampleThreads>(le, ex, ine, sh_scan);
  const float tot_e = sh_scan[kSampleThreads / 32];
  // last positive indices of the slice
  int wl = wlast, el = elast;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    wl = max(wl, __shfl_xor_sync(0xffffffffu, wl, o));
    el = max(el, __shfl_xor_sync(0xffffffffu, el, o));
  }
  __shared__ int sh_wl[kSampleThreads / 32], sh_el[kSampleThreads / 32];
  if ((tid & 31) == 0) {
    sh_wl[tid >> 5] = wl;
    sh_el[tid >> 5] = el;
  }
  __syncthreads();
  if (tid == 0) {
    SliceSum ss;
    ss.w = tot_w;
    ss.e = tot_e;
    ss.wlast = -1;
    ss.elast = -1;
    for (int k = 0; k < kSampleThreads / 32; ++k) {
      ss.wlast = max(ss.wlast, sh_wl[k]);
      ss.elast = max(ss.elast, sh_el[k]);
    }
    p.slices[static_cast<int64_t>(b) * p.nslice + sl] = ss;
    __threadfence();
    const uint32_t prev = atomicAdd(&p.tickets[b], 1u);
    s_last = prev == static_cast<uint32_t>(p.nslice - 1);
    if (s_last) p.tickets[b] = 0;  // leave the counter at zero for the next call
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();

  // 4. the last block: locate the crossing slice (warp 0: the slices' sums in parallel,
  // a warp scan in slice order, a ballot for the first crossing), then the token
  const float u = p.uniforms[static_cast<int64_t>(b) * gamma + gamma - 1];
  if (tid < 32) {
    const int lane = tid;
    const SliceSum* ss = p.slices + static_cast<int64_t>(b) * p.nslice;
    auto scan32 = [&](float v) {
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += y;
      }
      return v;
    };
    // totals, as the end of the inclusive scan in slice order
    float tw = 0.f, te = 0.f;
    for (int k0 = 0; k0 < p.nslice; k0 += 32) {
      const int k = k0 + lane;
      const float vw = k < p.nslice ? __ldcg(&ss[k].w) : 0.f;
      const float ve = k < p.nslice ? __ldcg(&ss[k].e) : 0.f;
      tw += __shfl_sync(0xffffffffu, scan32(vw), 31);
      te += __shfl_sync(0xffffffffu, scan32(ve), 31);
    }
    // residual without mass (only through rounding): draw from p_n itself
    const int use_res = (!bonus && tw > 0.f) ? 1 : 0;
    const float target = u * (use_res ? tw : te);
    float carry = 0.f;
    int star = -1, lastk = -1;
    float base = 0.f;
    for (int k0 = 0; k0 < p.nslice && star < 0; k0 += 32) {
      const int k = k0 + lane;
      const float v = k < p.nslice ? (use_res ? __ldcg(&ss[k].w) : __ldcg(&ss[k].e)) : 0.f;
      const float incl = scan32(v);
      const unsigned hit = __ballot_sync(0xffffffffu, v > 0.f && carry + incl >= target);
      const unsigned pos = __ballot_sync(0xffffffffu, v > 0.f);
      if (pos) lastk = k0 + 31 - __clz(pos);
      if (hit) {
        const int f = __ffs(hit) - 1;
        star = k0 + f;
        base = carry + __shfl_sync(0xffffffffu, incl - v, f);
      }
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) {
      if (star < 0 && lastk >= 0)  // rounding left u*S above every sum: last positive weight
        s_token = use_res ? __ldcg(&ss[lastk].wlast) : __ldcg(&ss[lastk].elast);
      s_star = star;
      s_use_res = use_res;
      s_base = base;
      s_target = target;
    }
  }
  __syncthreads();
  if (s_star >= 0) {
    final_weights<BF16, VEC>(p, prow, qrow, bonus, s_star * kSampleSlice, c, Mp, invSp, Mq,
                             invSq, w, e, first);
    const bool use_res = s_use_res != 0;
    float loc = 0.f;
#pragma unroll
    for (int k = 0; k < kPer; ++k) loc += use_res ? w[k] : e[k];
    float excl, incl;
    block_scan<kSampleThreads>(loc, excl, incl, sh_scan);
    const float base = s_base, target = s_target;
    if (base + incl >= target) atomicMin(&s_owner, tid);
    __syncthreads();
    if (tid == s_owner) {
      float run = 0.f;
      int tok = -1, lastpos = -1;
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        const float x = use_res ? w[k] : e[k];
        run += x;
        if (x > 0.f) {
          lastpos = first + k;
          if (tok < 0 && base + excl + run >= target) tok = first + k;
        }
      }
      s_token = tok >= 0 ? tok : lastpos;
    }
    __syncthreads();
    if (s_token < 0 && tid == 0) {  // no owner: fall back to the slice's last positive weight
      const SliceSum* ss = p.slices + static_cast<int64_t>(b) * p.nslice + s_star;
      s_token = use_res ? __ldcg(&ss->wlast) : __ldcg(&ss->elast);
    }
  }
  __syncthreads();
  if (tid == 0) p.out_tokens[orow + n] = s_token;
}

// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): 10 rounds of two 32x32->64
// multiplies by the Philox constants, with the key advanced by the Weyl constants.
// Returns word g & 3 of the block at counter (g >> 2, 0, 0) under key (seed low, high).
__device__ __forceinline__ uint32_t philox_word(uint64_t seed, uint64_t g) {
  const uint64_t blk = g >> 2;
  uint32_t c0 = static_cast<uint32_t>(blk), c1 = static_cast<uint32_t>(blk >> 32), c2 = 0, c3 = 0;
  uint32_t k0 = static_cast<uint32_t>(seed), k1 = static_cast<uint32_t>(seed >> 32);
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t hi0 = __umulhi(0xD2511F53u, c0), lo0 = 0xD2511F53u * c0;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c2), lo1 = 0xCD9E8D57u * c2;
    const uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
  }
  const uint32_t words[4] = {c0, c1, c2, c3};
  return words[g & 3];
}

__global__ void philox_uniforms_kernel(uint64_t seed, uint64_t offset, int64_t n, float* out) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const uint32_t x = philox_word(seed, offset + static_cast<uint64_t>(i));
  out[i] = static_cast<float>((x >> 8) + 1u) * 5.9604644775390625e-8f;  // * 2^-24
}

// Alg. line 1: noise tokens z ~ U[V], token = floor(x * V / 2^32) of the word x.
__global__ void noise_tokens_kernel(uint64_t seed, uint64_t offset, int64_t n, int32_t vocab,
                                    int32_t* out) {
  const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const uint32_t x = philox_word(seed, offset + static_cast<uint64_t>(i));
  out[i] = static_cast<int32_t>((static_cast<uint64_t>(x) * static_cast<uint32_t>(vocab)) >> 32);
}

template <bool BF16, bool VEC>
cudaError_t launch_typed(const AcceptParams& p, cudaStream_t stream, bool overlap_prior) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  // row statistics: a programmatic dependent of the attention kernel in a verify step
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((p.nchunk + kStatsThreads / 32 - 1) / (kStatsThreads / 32), 2 * p.gamma - 1, p.batch);
  cfg.blockDim = dim3(kStatsThreads);
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = overlap_prior ? 1 : 0;
  cudaError_t e = cudaLaunchKernelEx(&cfg, row_stats_kernel<BF16, VEC>, p);
  if (e != cudaSuccess) return e;
  // decisions (a programmatic dependent of the statistics kernel, which it waits for
  // before reading the partials), then the draws (likewise of the decisions)
  cfg.gridDim = dim3(p.batch);
  cfg.blockDim = dim3(kDecideThreads);
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, decide_kernel<BF16>, p);
  if (e != cudaSuccess) return e;
  cfg.gridDim = dim3(p.nslice, p.batch);
  cfg.blockDim = dim3(kSampleThreads);
  e = cudaLaunchKernelEx(&cfg, sample_kernel<BF16, VEC>, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_accept(const spec_accept_args_t& a, const AcceptLayout& L, char* ws, int,
                          cudaStream_t stream, bool overlap_prior) {
  AcceptParams p;
  p.batch = a.batch;
  p.gamma = a.gamma;
  p.vocab = a.vocab;
  p.nchunk = L.nchunk;
  p.nslice = L.nslice;
  p.target = a.target_logits;
  p.drafter = a.drafter_logits;
  p.tokens = a.block_tokens;
  p.temperature = a.temperature;
  p.uniforms = a.uniforms;
  p.num_accepted = a.num_accepted;
  p.out_tokens = a.out_tokens;
  p.num_emitted = a.num_emitted;
  p.diag = a.diag;
  p.status = reinterpret_cast<uint32_t*>(ws);
  p.tickets = reinterpret_cast<uint32_t*>(ws + L.tickets);
  p.partials = reinterpret_cast<RowPartial*>(ws + L.partials);
  p.records = reinterpret_cast<DecideRecord*>(ws + L.records);
  p.slices = reinterpret_cast<SliceSum*>(ws + L.slice_sums);
  const bool bf16 = a.logits_dtype == SPEC_BF16;
  const size_t esz = bf16 ? 2 : 4;
  const bool vec = (static_cast<size_t>(a.vocab) * esz) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(a.target_logits) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(a.drafter_logits) % 16 == 0;
  if (bf16)
    return vec ? launch_typed<true, true>(p, stream, overlap_prior)
               : launch_typed<true, false>(p, stream, overlap_prior);
  return vec ? launch_typed<false, true>(p, stream, overlap_prior)
             : launch_typed<false, false>(p, stream, overlap_prior);
}

cudaError_t launch_noise(uint64_t seed, uint64_t offset, int64_t n, int32_t vocab, int32_t* out,
                         cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  const int64_t blocks = (n + 255) / 256;
  (void)cudaGetLastError();  // report this launch's error only
  noise_tokens_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(seed, offset, n, vocab, out);
  return cudaGetLastError();
}

cudaError_t launch_philox(uint64_t seed, uint64_t offset, int64_t n, float* out, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  const int64_t blocks = (n + 255) / 256;
  (void)cudaGetLastError();  // report this launch's error only
  philox_uniforms_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(seed, offset, n, out);
  return cudaGetLastError();
}

}  // namespace specv
