// The target's LM head with the acceptance's row statistics fused into it (Sec. 4.2:
// the verifier pass scores the block rows; Appendix B.3: the rule reads p through its
// normaliser, maximum and the logits of drafted tokens).
//
// lm_head_kernel: one block per (224-row vocab tile, 128-row hidden-state tile), two
// blocks per SM. Warp 0 streams 64-column slices of the hidden states and of the weight
// rows by TMA (128-byte swizzle, out-of-range rows read as zeros) into a 2-stage ring;
// warp 1 issues tcgen05.mma (M = 128, N = 224, K = 16) into an fp32 TMEM accumulator; warps
// 2..5 then read one logit row each (a warp reaches the TMEM lanes of its own
// sub-partition) and reduce it, 32 columns at a time, to (max, sum of
// exp((l - max) / T), lowest-index argmax, logit of the row's token), optionally
// writing the logits as bf16. lm_merge_kernel: one warp per row merges the vocab
// tiles' partials.
#include <cuda_bf16.h>

#include <cfloat>
#include <climits>
#include <cmath>

#include "lm_head.cuh"
#include "tc_ptx.cuh"

namespace specv {

LmLayout lm_layout(const spec_lm_head_args_t& a, size_t base) {
  LmLayout L;
  L.ntiles_n = (a.vocab + kLmTileN - 1) / kLmTileN;
  L.ntiles_m = (a.rows + kLmTileM - 1) / kLmTileM;
  L.parts = base;
  L.end = ws_round(L.parts + 16 * static_cast<size_t>(a.rows) * L.ntiles_n);
  return L;
}

namespace {

using namespace tcx;

constexpr int kBK = 64;      // hidden elements per stage: one 128-byte swizzle span
constexpr int kStages = 2;  // 88 KB of shared memory: two blocks per SM, one streams while the other reduces
constexpr uint32_t kABytes = kLmTileM * 128;  // 16 KB of hidden states per stage
constexpr uint32_t kBBytes = kLmTileN * 128;  // 32 KB of weight rows per stage
constexpr uint32_t kOffA = 0;
constexpr uint32_t kOffB = kOffA + kStages * kABytes;
constexpr uint32_t kOffBar = kOffB + kStages * kBBytes;      // full[S], empty[S], acc
constexpr uint32_t kOffMisc = kOffBar + (2 * kStages + 1) * 8;  // TMEM base, abort flag
constexpr size_t kSmem = kOffMisc + 16 + 1024;                // + 1 KB alignment slack
constexpr int kThreads = 192;  // warp 0 TMA, warp 1 MMA, warps 2..5 reduce
// TMEM columns to allocate: a power of two >= 32 that holds the N fp32 accumulator columns
constexpr uint32_t kTmemCols = kLmTileN <= 32 ? 32 : kLmTileN <= 64 ? 64 : kLmTileN <= 128 ? 128
                             : kLmTileN <= 256 ? 256 : 512;

struct LmPart {
  float m, s;   // tile maximum and sum of 2^((l - m) * c2)
  int32_t arg;  // lowest index of the maximum; -2: a non-finite logit in the tile
  float tok;    // the row token's logit if it lies in the tile, else NaN
};

struct LmParams {
  int rows, hidden, vocab, rows_per_seq, ntn, nk;
  const float* temperature;
  const int32_t* tokens;
  __nv_bfloat16* logits;
  LmPart* parts;
  uint32_t* status;
  float* row_max;
  float* row_sum;
  int32_t* row_argmax;
  float* token_logit;
  int starve;  // test hook: the producer issues no copies, so the MMA warp's waits run out
};

__device__ __forceinline__ float row_c2(const LmParams& p, int row) {
  const float T = p.temperature[row / p.rows_per_seq];
  return kLog2e / (T > 0.f ? T : 1.f);
}

// (m, s, a) of two parts, both sums relative to their own maximum; equal maxima keep
// the lower index.
__device__ __forceinline__ void merge_part(float& m, float& s, int& a, float m2, float s2, int a2,
                                           float c2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    s = s2;
    a = a2;
    return;
  }
  const float M = fmaxf(m, m2);
  s = s * ex2((m - M) * c2) + s2 * ex2((m2 - M) * c2);
  a = m2 > m ? a2 : (m > m2 ? a : min(a, a2));
  m = M;
}

__global__ void __launch_bounds__(kThreads)
    lm_head_kernel(const __grid_constant__ CUtensorMap map_h, const __grid_constant__ CUtensorMap map_w,
                   LmParams p) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + kOffBar;
  auto full = [&](int s) { return bar0 + 8u * s; };
  auto empty = [&](int s) { return bar0 + 8u * (kStages + s); };
  const uint32_t acc = bar0 + 8u * (2 * kStages);
  uint32_t* misc = reinterpret_cast<uint32_t*>(smem + kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // blockIdx.x is the row tile, so the row tiles that share a weight tile run together
  // and read it from DRAM once (the others hit L2)
  const int tn = blockIdx.y;  // vocab tile
  const int n0 = tn * kLmTileN, m0 = blockIdx.x * kLmTileM;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full(s), 1);
      mbar_init(empty(s), 1);
    }
    mbar_init(acc, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(misc), kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = misc[0];

  if (warp == 0) {
    // ============================ TMA producer ============================
    if (lane == 0) {
      int k = 0;
      bool ok = true;
      for (; k < p.nk && !p.starve; ++k) {
        const int s = k % kStages;
        if (k >= kStages) ok = mbar_wait(empty(s), ((k / kStages) - 1) & 1, abort_flag, p.status);
        if (!ok) break;
        mbar_arrive_tx(full(s), kABytes + kBBytes);
        tma_load_2d(sbase + kOffA + s * kABytes, &map_h, k * kBK, m0, full(s));
        tma_load_2d(sbase + kOffB + s * kBBytes, &map_w, k * kBK, n0, full(s));
      }
      if (!ok) {  // let the copies still in flight land before the block exits (bounded)
        for (int j = k > kStages ? k - kStages : 0; j < k; ++j) {
          const long long t0 = clock64();
          while (!mbar_try(full(j % kStages), (j / kStages) & 1) && clock64() - t0 < kWaitCycles) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ============================ MMA issuer ============================
    if (lane == 0) {
      constexpr uint32_t kIdesc = idesc_bf16(kLmTileM, kLmTileN, false);
      bool ok = true;
      for (int k = 0; k < p.nk && ok; ++k) {
        const int s = k % kStages;
        ok = mbar_wait(full(s), (k / kStages) & 1, abort_flag, p.status);
        if (!ok) break;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk) {
          const uint64_t ad = desc_sw128(sbase + kOffA + s * kABytes + kk * 32u, 16, 1024);
          const uint64_t bd = desc_sw128(sbase + kOffB + s * kBBytes + kk * 32u, 16, 1024);
          mma_bf16(tmem, ad, bd, kIdesc, (k > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(empty(s));  // the stage is free once these MMAs have read it
      }
      mma_commit(acc);  // the accumulator is complete (or, on abort, idle) after these
    }
    __syncwarp();
  } else {
    // ============================ row reduction ============================
    const int q = warp & 3;  // this warp's TMEM lane quadrant
    const int row = m0 + q * 32 + lane;
    const bool real = row < p.rows;
    const float c2 = real ? row_c2(p, row) : kLog2e;
    const int tok = (real && p.tokens) ? p.tokens[row] : -1;
    const bool ok = mbar_wait(acc, 0, abort_flag, p.status);
    if (ok) {
      tc_fence_after();
      float m = -INFINITY, s = 0.f, tl = __int_as_float(0x7fc00000);
      int a = INT_MAX;
      bool bad = false;
      __nv_bfloat16* lrow = (p.logits && real) ? p.logits + static_cast<int64_t>(row) * p.vocab : nullptr;
#pragma unroll 1
      for (int c = 0; c < kLmTileN / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(tmem + (static_cast<uint32_t>(q * 32) << 16) + c * 32, r);
        tmem_wait_ld();
        const int col0 = n0 + c * 32;
        const int nvalid = min(32, p.vocab - col0);
        float cm = -INFINITY;
        int ca = INT_MAX;
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const float x = __uint_as_float(r[e]);
          if (e < nvalid) {
            bad |= !(fabsf(x) <= FLT_MAX);
            if (x > cm) {
              cm = x;
              ca = col0 + e;
            }
            if (col0 + e == tok) tl = x;
          }
        }
        float cs = 0.f;
        if (cm > -INFINITY) {
          const float mc = cm * c2;
#pragma unroll
          for (int e = 0; e < 32; ++e)
            if (e < nvalid) cs += ex2(fmaf(__uint_as_float(r[e]), c2, -mc));
        }
        merge_part(m, s, a, cm, cs, ca, c2);
        if (lrow && nvalid > 0) {
          if (nvalid == 32 && (p.vocab & 7) == 0) {
            uint4* dst = reinterpret_cast<uint4*>(lrow + col0);
#pragma unroll
            for (int g = 0; g < 4; ++g) {
              uint32_t w[4];
#pragma unroll
              for (int h2 = 0; h2 < 4; ++h2) {
                const __nv_bfloat162 v2 = __floats2bfloat162_rn(__uint_as_float(r[8 * g + 2 * h2]),
                                                                __uint_as_float(r[8 * g + 2 * h2 + 1]));
                w[h2] = *reinterpret_cast<const uint32_t*>(&v2);
              }
              dst[g] = make_uint4(w[0], w[1], w[2], w[3]);
            }
          } else {
#pragma unroll
            for (int e = 0; e < 32; ++e)
              if (e < nvalid) lrow[col0 + e] = __float2bfloat16_rn(__uint_as_float(r[e]));
          }
        }
      }
      if (real) {
        LmPart out;
        out.m = m;
        out.s = s;
        out.arg = bad ? -2 : a;
        out.tok = tl;
        p.parts[static_cast<int64_t>(row) * p.ntn + tn] = out;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// One warp per row: the vocab tiles' partials merged into the row's statistics.
__global__ void __launch_bounds__(128) lm_merge_kernel(LmParams p) {
  const int row = blockIdx.x * 4 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= p.rows) return;
  const float c2 = row_c2(p, row);
  float m = -INFINITY, s = 0.f, tl = __int_as_float(0x7fc00000);
  int a = INT_MAX;
  bool bad = false;
  const LmPart* parts = p.parts + static_cast<int64_t>(row) * p.ntn;
  for (int t = lane; t < p.ntn; t += 32) {
    const LmPart q = parts[t];
    bad |= q.arg == -2;
    if (q.tok == q.tok) tl = q.tok;
    merge_part(m, s, a, q.m, q.s, q.arg, c2);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
    const int a2 = __shfl_xor_sync(0xffffffffu, a, o);
    merge_part(m, s, a, m2, s2, a2, c2);
  }
  const unsigned has_tok = __ballot_sync(0xffffffffu, tl == tl);
  if (has_tok) tl = __shfl_sync(0xffffffffu, tl, __ffs(has_tok) - 1);
  bad = __any_sync(0xffffffffu, bad);
  if (lane == 0) {
    p.row_max[row] = m;
    p.row_sum[row] = s;
    p.row_argmax[row] = bad ? -1 : a;
    if (p.token_logit) p.token_logit[row] = tl;
    if (bad) set_status(p.status, SPEC_FLAG_BAD_LOGITS);
  }
}

}  // namespace

cudaError_t launch_lm_head(const spec_lm_head_args_t& a, const LmLayout& L, char* ws,
                           cudaStream_t stream, bool starve) {
  CUtensorMap mh, mw;
  if (!encode_rows_map(&mh, a.hidden_states, a.rows, a.hidden, kLmTileM) ||
      !encode_rows_map(&mw, a.weight, a.vocab, a.hidden, kLmTileN))
    return cudaErrorInvalidValue;
  LmParams p;
  p.rows = a.rows;
  p.hidden = a.hidden;
  p.vocab = a.vocab;
  p.rows_per_seq = a.rows_per_seq;
  p.ntn = L.ntiles_n;
  p.nk = (a.hidden + kBK - 1) / kBK;
  p.temperature = a.temperature;
  p.tokens = a.tokens;
  p.logits = static_cast<__nv_bfloat16*>(a.logits);
  p.parts = reinterpret_cast<LmPart*>(ws + L.parts);
  p.status = reinterpret_cast<uint32_t*>(ws);
  p.row_max = a.row_max;
  p.row_sum = a.row_sum;
  p.row_argmax = a.row_argmax;
  p.token_logit = a.token_logit;
  p.starve = starve ? 1 : 0;
  (void)cudaGetLastError();
  cudaError_t e = cudaFuncSetAttribute(lm_head_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(kSmem));
  if (e != cudaSuccess) return e;
  lm_head_kernel<<<dim3(L.ntiles_m, L.ntiles_n), kThreads, kSmem, stream>>>(mh, mw, p);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  lm_merge_kernel<<<(a.rows + 3) / 4, 128, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace specv
