// Internal helpers shared by the CUDA-core and tensor-core attention kernels:
// launch parameters, bf16 output rows, log-sum-exp outputs, and the merge of
// split-KV partials (each split keeps an unnormalised fp32 output, its running
// base-2 max m and its sum l; the merge rescales by 2^{m_s - max m}).
#pragma once

#include <cuda_bf16.h>

#include <cmath>

#include "common.cuh"

namespace specv {

struct AttnParams {
  int batch, gamma, hq, hkv, group, rows, row_tiles, rows_per_cta;
  int page_size, max_pages, num_pages;
  int nsplit, tiles_per_split;
  int slot_rows;     // rows stored per partial slot
  int max_keys;      // max_pages * page_size
  float scale_log2;  // softmax_scale * log2(e)
  const void* q;
  const void* k_cache;
  const void* v_cache;
  const int32_t* page_table;
  const int32_t* kv_len;
  void* out;
  float* lse;
  uint32_t* status;
  uint32_t* tickets;
  float* partial_o;    // [slot][slot_rows][D]
  float2* partial_ml;  // [slot][slot_rows] = (m, l); l = -1 marks a bad sequence
};

inline AttnParams make_attn_params(const spec_attn_args_t& a, const AttnPlan& P, char* ws) {
  AttnParams p;
  p.batch = a.batch;
  p.gamma = a.gamma;
  p.hq = a.num_q_heads;
  p.hkv = a.num_kv_heads;
  p.group = a.num_q_heads / a.num_kv_heads;
  p.rows = P.rows;
  p.row_tiles = P.row_tiles;
  p.rows_per_cta = P.rows_per_cta;
  p.page_size = a.page_size;
  p.max_pages = a.max_pages_per_seq;
  p.num_pages = a.num_pages;
  p.nsplit = P.nsplit;
  p.tiles_per_split = P.tiles_per_split;
  p.slot_rows = P.slot_rows;
  p.max_keys = P.max_keys;
  const float scale = a.softmax_scale != 0.f ? a.softmax_scale : 1.f / sqrtf(static_cast<float>(a.head_dim));
  p.scale_log2 = scale * 1.4426950408889634f;
  p.q = a.q;
  p.k_cache = a.k_cache;
  p.v_cache = a.v_cache;
  p.page_table = a.page_table;
  p.kv_len = a.kv_len;
  p.out = a.out;
  p.lse = a.lse;
  p.status = reinterpret_cast<uint32_t*>(ws);
  p.tickets = reinterpret_cast<uint32_t*>(ws + P.tickets);
  p.partial_o = reinterpret_cast<float*>(ws + P.partial_o);
  p.partial_ml = reinterpret_cast<float2*>(ws + P.partial_ml);
  return p;
}

#ifdef __CUDACC__
// 8 consecutive output dims of unit row `row` (row = j * group + head-in-group).
template <int D>
__device__ __forceinline__ void write_out_row(const AttnParams& p, int b, int g, int row, int d0,
                                              const float* o8, float inv) {
  const int j = row / p.group, h = g * p.group + row % p.group;
  __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(p.out) +
                       ((static_cast<int64_t>(b) * p.gamma + j) * p.hq + h) * D + d0;
  uint32_t w[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const __nv_bfloat162 pr = __floats2bfloat162_rn(o8[2 * e] * inv, o8[2 * e + 1] * inv);
    w[e] = *reinterpret_cast<const uint32_t*>(&pr);
  }
  *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
}

__device__ __forceinline__ void write_lse(const AttnParams& p, int b, int g, int row, float m,
                                          float l, bool bad) {
  if (!p.lse) return;
  const int j = row / p.group, h = g * p.group + row % p.group;
  const float v = (bad || !(l > 0.f)) ? -INFINITY : (m + log2f(l)) * 0.6931471805599453f;
  p.lse[(static_cast<int64_t>(b) * p.gamma + j) * p.hq + h] = v;
}

// Run by the last block to finish a unit: combines the partials in slots
// [slot0, slot0 + nslots) for rows [row0, row0 + nrows) and writes the final
// outputs. Threads tid .. of nthreads cooperate.
template <int D>
__device__ void merge_splits(const AttnParams& p, int b, int g, int row0, int nrows,
                             int64_t slot0, int nslots, int tid, int nthreads) {
  constexpr int DQ = D / 8;
  for (int idx = tid; idx < nrows * DQ; idx += nthreads) {
    const int r = idx / DQ, dq = idx % DQ;
    float M = -INFINITY;
    bool bad = false;
    for (int s = 0; s < nslots; ++s) {
      const float2 ml = __ldcg(&p.partial_ml[(slot0 + s) * p.slot_rows + r]);
      if (ml.y < 0.f) bad = true;
      else if (ml.y > 0.f) M = fmaxf(M, ml.x);
    }
    float L = 0.f, acc[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = 0.f;
    if (!bad) {
      for (int s = 0; s < nslots; ++s) {
        const int64_t slot = (slot0 + s) * p.slot_rows + r;
        const float2 ml = __ldcg(&p.partial_ml[slot]);
        if (!(ml.y > 0.f)) continue;
        const float w = ex2(ml.x - M);
        L += ml.y * w;
        const float4* src = reinterpret_cast<const float4*>(p.partial_o + slot * D + dq * 8);
        const float4 a = __ldcg(src), c = __ldcg(src + 1);
        acc[0] += a.x * w; acc[1] += a.y * w; acc[2] += a.z * w; acc[3] += a.w * w;
        acc[4] += c.x * w; acc[5] += c.y * w; acc[6] += c.z * w; acc[7] += c.w * w;
      }
    }
    const bool dead = bad || !(L > 0.f);
    write_out_row<D>(p, b, g, row0 + r, dq * 8, acc, dead ? 0.f : 1.f / L);
    if (dq == 0) write_lse(p, b, g, row0 + r, M, L, dead);
  }
}
#endif

}  // namespace specv
