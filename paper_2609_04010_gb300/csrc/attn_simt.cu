// Part (a) of the verify step on CUDA cores: block-causal attention of the gamma
// block queries over a paged bf16 KV cache with grouped-query heads (Sec. 4.1: the
// prefix stays in the KV cache while the block is processed; Alg. "Lossless
// Psi-Spec": one causal verifier pass over [x^{L+1}, x~]).
//
// Work unit: (sequence b, KV head g, row tile, KV split). A block holds up to 16 query
// rows of KV head g (row r = block position j * group + head-in-group), so each KV
// page is read once for all heads of the group. KV tiles of 64 keys are gathered
// through the page table with 16-byte cp.async copies into shared memory, double
// buffered. Scores and the online softmax are fp32 (base-2 exponentials); the last
// split of a unit to finish (atomic ticket, no waiting) merges the split partials
// by their log-sum-exp and writes bf16 outputs.
#include <cuda_bf16.h>

#include <cfloat>
#include <cmath>

#include "attn_common.cuh"

namespace specv {
namespace {

constexpr int RT = kSimtRowTile;   // rows per block
constexpr int TK = kSimtKeyTile;   // keys per tile
constexpr int NT = kSimtThreads;   // threads per block

template <int D>
struct SimtSmem {
  static constexpr int kStride = D + 8;  // bf16 elements per staged K/V row (bank spread)
  float q[RT][D];
  __nv_bfloat16 k[2][TK][kStride];
  __nv_bfloat16 v[2][TK][kStride];
  float s[RT][TK];
  float alpha[RT];
  float m[RT];
  float l[RT];
  unsigned long long tmask[RT];  // tree attention: the block keys each row sees
  int bad;
  int last;
};

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool valid) {
  const uint32_t s = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(n));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
__device__ __forceinline__ void cp_async_wait_all_but_one() {
  asm volatile("cp.async.wait_group 1;\n" ::);
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::); }

template <int D>
__device__ __forceinline__ void load_kv_tile(const AttnParams& p, SimtSmem<D>& sm, int buf, int b,
                                             int g, int tile_start, int kv_len) {
  constexpr int kPieces = D / 8;  // 16-byte pieces per key row
  const __nv_bfloat16* kc = static_cast<const __nv_bfloat16*>(p.k_cache);
  const __nv_bfloat16* vc = static_cast<const __nv_bfloat16*>(p.v_cache);
  for (int c = threadIdx.x; c < TK * kPieces; c += NT) {
    const int kk = c / kPieces, piece = c % kPieces;
    const int key = tile_start + kk;
    const bool valid = key < kv_len;
    int64_t off = 0;
    if (valid) {
      const int page = p.page_table[static_cast<int64_t>(b) * p.max_pages + key / p.page_size];
      off = ((static_cast<int64_t>(page) * p.hkv + g) * p.page_size + key % p.page_size) * D +
            piece * 8;
    }
    cp_async16(&sm.k[buf][kk][piece * 8], kc + off, valid);
    cp_async16(&sm.v[buf][kk][piece * 8], vc + off, valid);
  }
}

template <int D>
__global__ void __launch_bounds__(NT) attn_simt_kernel(AttnParams p) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  SimtSmem<D>& sm = *reinterpret_cast<SimtSmem<D>*>(smem_raw);
  pdl_launch_dependents();  // the acceptance kernels of a verify step may start beside us
  const int split = blockIdx.x, g = blockIdx.y;
  const int b = blockIdx.z / p.row_tiles, rt = blockIdx.z % p.row_tiles;
  const int tid = threadIdx.x;
  const int row0 = rt * RT;
  const int nrows = min(RT, p.rows - row0);
  const int kv_len = p.kv_len[b];

  // validity of the sequence and of the pages this split touches
  const int key_begin = split * p.tiles_per_split * TK;
  const bool len_ok = kv_len >= p.gamma && kv_len <= p.max_pages * p.page_size;
  const int key_end = len_ok ? min(kv_len, key_begin + p.tiles_per_split * TK) : 0;
  if (tid == 0) sm.bad = len_ok ? 0 : 2;
  __syncthreads();
  if (len_ok && key_end > key_begin) {
    const int pg0 = key_begin / p.page_size, pg1 = (key_end - 1) / p.page_size;
    for (int pg = pg0 + tid; pg <= pg1; pg += NT) {
      const int id = p.page_table[static_cast<int64_t>(b) * p.max_pages + pg];
      if (id < 0 || id >= p.num_pages) sm.bad = 1;
    }
  }
  // queries of this row tile, fp32, pre-multiplied by scale * log2(e)
  const __nv_bfloat16* qg = static_cast<const __nv_bfloat16*>(p.q);
  for (int i = tid; i < RT * D; i += NT) {
    const int r = i / D, d = i % D;
    float x = 0.f;
    if (r < nrows) {
      const int row = row0 + r, j = row / p.group, hh = row % p.group;
      const int h = g * p.group + hh;
      x = __bfloat162float(qg[((static_cast<int64_t>(b) * p.gamma + j) * p.hq + h) * D + d]) *
          p.scale_log2;
    }
    sm.q[r][d] = x;
  }
  if (tid < RT) {
    sm.m[tid] = -INFINITY;
    sm.l[tid] = 0.f;
    const int j = min(row0 + tid, p.rows - 1) / p.group;
    sm.tmask[tid] = p.tree_mask ? p.tree_mask[static_cast<int64_t>(b) * p.gamma + j] : 0ull;
  }
  __syncthreads();
  const bool bad = sm.bad != 0;
  const int ctx = kv_len - p.gamma;

  // PV ownership: thread -> 8 consecutive dims and rows {rg, rg + RG, ...}
  constexpr int DQ = D / 8;
  constexpr int RG = NT / DQ;
  constexpr int RPT = RT / RG;
  const int dq = tid % DQ, rg = tid / DQ;
  float o[RPT][8];
#pragma unroll
  for (int i = 0; i < RPT; ++i)
#pragma unroll
    for (int e = 0; e < 8; ++e) o[i][e] = 0.f;

  const int ntiles = bad ? 0 : (key_end - key_begin + TK - 1) / TK;
  if (ntiles > 0) {
    load_kv_tile<D>(p, sm, 0, b, g, key_begin, kv_len);
    cp_async_commit();
  }
  // QK ownership: thread -> key kk, rows {hr, hr + 2, ...}
  const int kk = tid % TK, hr = tid / TK;
  for (int it = 0; it < ntiles; ++it) {
    const int buf = it & 1;
    const int tile_start = key_begin + it * TK;
    if (it + 1 < ntiles) {
      load_kv_tile<D>(p, sm, buf ^ 1, b, g, tile_start + TK, kv_len);
      cp_async_commit();
      cp_async_wait_all_but_one();
    } else {
      cp_async_wait_all();
    }
    __syncthreads();
    // scores
    {
      float acc[RT / 2];
#pragma unroll
      for (int i = 0; i < RT / 2; ++i) acc[i] = 0.f;
      const __nv_bfloat16* krow = &sm.k[buf][kk][0];
#pragma unroll 4
      for (int d = 0; d < D; d += 8) {
        const uint4 raw = *reinterpret_cast<const uint4*>(krow + d);
        const uint32_t wv[4] = {raw.x, raw.y, raw.z, raw.w};
        float kf[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          kf[2 * e] = __uint_as_float(wv[e] << 16);
          kf[2 * e + 1] = __uint_as_float(wv[e] & 0xffff0000u);
        }
#pragma unroll
        for (int i = 0; i < RT / 2; ++i) {
          const float4 q0 = *reinterpret_cast<const float4*>(&sm.q[hr + 2 * i][d]);
          const float4 q1 = *reinterpret_cast<const float4*>(&sm.q[hr + 2 * i][d + 4]);
          acc[i] += q0.x * kf[0] + q0.y * kf[1] + q0.z * kf[2] + q0.w * kf[3] + q1.x * kf[4] +
                    q1.y * kf[5] + q1.z * kf[6] + q1.w * kf[7];
        }
      }
      const int key = tile_start + kk;
#pragma unroll
      for (int i = 0; i < RT / 2; ++i) {
        const int r = hr + 2 * i;
        const int j = (row0 + r) / p.group;
        const int rel = key - ctx;  // block position of the key (negative: the prefix)
        const bool vis = r < nrows && (p.tree_mask ? (rel < 0 || (rel < 64 && ((sm.tmask[r] >> rel) & 1ull)))
                                                   : key <= ctx + j);
        sm.s[r][kk] = vis ? acc[i] : -INFINITY;
      }
    }
    __syncthreads();
    // online softmax: warp w owns rows w, w+4, ...
    {
      const int lane = tid & 31, w = tid >> 5;
      for (int r = w; r < RT; r += NT / 32) {
        const float a0 = sm.s[r][lane], a1 = sm.s[r][lane + 32];
        float mx = fmaxf(a0, a1);
#pragma unroll
        for (int o2 = 16; o2 > 0; o2 >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o2));
        const float m_old = sm.m[r];
        const float m_new = fmaxf(m_old, mx);
        float p0 = 0.f, p1 = 0.f, alpha = 1.f;
        if (m_new != -INFINITY) {
          p0 = ex2(a0 - m_new);
          p1 = ex2(a1 - m_new);
          alpha = m_old == -INFINITY ? 0.f : ex2(m_old - m_new);
        }
        float sum = p0 + p1;
#pragma unroll
        for (int o2 = 16; o2 > 0; o2 >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o2);
        sm.s[r][lane] = p0;
        sm.s[r][lane + 32] = p1;
        if (lane == 0) {
          sm.alpha[r] = alpha;
          sm.m[r] = m_new;
          sm.l[r] = sm.l[r] * alpha + sum;
        }
      }
    }
    __syncthreads();
    // O = alpha * O + P V
    {
#pragma unroll
      for (int i = 0; i < RPT; ++i) {
        const float a = sm.alpha[rg + i * RG];
#pragma unroll
        for (int e = 0; e < 8; ++e) o[i][e] *= a;
      }
#pragma unroll 4
      for (int k = 0; k < TK; ++k) {
        const uint4 raw = *reinterpret_cast<const uint4*>(&sm.v[buf][k][dq * 8]);
        const uint32_t wv[4] = {raw.x, raw.y, raw.z, raw.w};
        float vf[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          vf[2 * e] = __uint_as_float(wv[e] << 16);
          vf[2 * e + 1] = __uint_as_float(wv[e] & 0xffff0000u);
        }
#pragma unroll
        for (int i = 0; i < RPT; ++i) {
          const float pk = sm.s[rg + i * RG][k];
#pragma unroll
          for (int e = 0; e < 8; ++e) o[i][e] += pk * vf[e];
        }
      }
    }
    __syncthreads();
  }

  // partial or final output
  float* po = p.partial_o;
  float2* pml = p.partial_ml;
  const int64_t unit = (static_cast<int64_t>(b) * p.hkv + g) * p.row_tiles + rt;
  if (p.nsplit == 1) {
#pragma unroll
    for (int i = 0; i < RPT; ++i) {
      const int r = rg + i * RG;
      if (r < nrows) {
        const float inv = bad ? 0.f : 1.f / sm.l[r];
        write_out_row<D>(p, b, g, row0 + r, dq * 8, o[i], inv);
      }
    }
    if (tid < nrows) write_lse(p, b, g, row0 + tid, bad ? -INFINITY : sm.m[tid], sm.l[tid], bad);
    if (tid == 0 && bad) set_status(p.status, sm.bad == 2 ? SPEC_FLAG_BAD_KV_LEN : SPEC_FLAG_BAD_PAGE);
    return;
  }
  const int64_t slot = unit * p.nsplit + split;
#pragma unroll
  for (int i = 0; i < RPT; ++i) {
    const int r = rg + i * RG;
    float4* dst = reinterpret_cast<float4*>(po + (slot * p.slot_rows + r) * D + dq * 8);
    dst[0] = make_float4(o[i][0], o[i][1], o[i][2], o[i][3]);
    dst[1] = make_float4(o[i][4], o[i][5], o[i][6], o[i][7]);
  }
  if (tid < RT) pml[slot * p.slot_rows + tid] = make_float2(sm.m[tid], bad ? -1.f : sm.l[tid]);
  if (tid == 0 && bad) set_status(p.status, sm.bad == 2 ? SPEC_FLAG_BAD_KV_LEN : SPEC_FLAG_BAD_PAGE);
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const uint32_t prev = atomicAdd(&p.tickets[unit], 1u);
    sm.last = prev == static_cast<uint32_t>(p.nsplit - 1);
    if (sm.last) p.tickets[unit] = 0;
  }
  __syncthreads();
  if (!sm.last) return;
  __threadfence();
  merge_unit<D>(p, b, g, row0, nrows, unit * p.nsplit, p.nsplit, tid, NT);
}

}  // namespace

cudaError_t launch_attn_simt(const spec_attn_args_t& a, const AttnPlan& P, char* ws,
                             cudaStream_t stream) {
  AttnParams p = make_attn_params(a, P, ws);
  const dim3 grid(P.nsplit, a.num_kv_heads, a.batch * P.row_tiles);
  if (a.head_dim == 128) {
    const size_t smem = sizeof(SimtSmem<128>);
    cudaFuncSetAttribute(attn_simt_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         static_cast<int>(smem));
    attn_simt_kernel<128><<<grid, NT, smem, stream>>>(p);
  } else {
    const size_t smem = sizeof(SimtSmem<64>);
    cudaFuncSetAttribute(attn_simt_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         static_cast<int>(smem));
    attn_simt_kernel<64><<<grid, NT, smem, stream>>>(p);
  }
  return cudaGetLastError();
}

}  // namespace specv
