// Internal helpers shared by the CUDA-core and tensor-core attention kernels:
// launch parameters, bf16 output rows, log-sum-exp outputs, and the merge of
// split-KV partials (each split keeps an unnormalised fp32 output, its running
// base-2 max m and its sum l; the merge rescales by 2^{m_s - max m}).
#pragma once

#include <cuda.h>  // CUtensorMap
#include <cuda_bf16.h>

#include <cmath>

#include "common.cuh"

namespace specv {

struct AttnParams {
  int batch, gamma, hq, hkv, group, rows, row_tiles, rows_per_cta;
  int hunits;        // KV-head units per sequence: Hkv, or Hkv / 2 when a block serves
                     // two adjacent KV heads together (tensor-core head-pair variant)
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
  int q_tma;           // tensor-core kernel: Q tiles arrive by TMA (else softmax warps load them)
  int unit_overhead;   // tensor-core kernel: tiles charged per unit start in the work list
  const uint64_t* tree_mask;  // [batch][gamma] block keys each query sees, or NULL (causal)
  int starve;  // test hook: the producers issue no copies, so the consumers' waits run out
};

inline AttnParams make_attn_params(const spec_attn_args_t& a, const AttnPlan& P, char* ws) {
  AttnParams p;
  p.batch = a.batch;
  p.gamma = a.gamma;
  p.hq = a.num_q_heads;
  p.hkv = a.num_kv_heads;
  p.hunits = P.head_pair ? a.num_kv_heads / 2 : a.num_kv_heads;
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
  p.q_tma = 0;
  p.unit_overhead = 0;
  p.tree_mask = a.tree_mask;
  p.starve = 0;
  return p;
}

// Tensor maps of the tensor-core kernels (attn_tc.cu): the K or V cache with one page of
// one KV head (or of two adjacent KV heads, heads_per_box = 2) per box, and Q with one
// tile of tile_rows query rows of one KV group per box (false if group does not divide
// tile_rows or the encoder is missing).
bool encode_cache_map(CUtensorMap* map, const void* base, const spec_attn_args_t& a,
                      int heads_per_box = 1);
bool encode_q_map(CUtensorMap* map, const spec_attn_args_t& a, int tile_rows);

#ifdef __CUDACC__
// ---------------------------------------------------------------------------------
// Work list of the persistent tensor-core kernels (TK keys per tile)
// ---------------------------------------------------------------------------------
template <int TK>
__device__ __forceinline__ int unit_tiles(int kv_len, const AttnParams& p) {
  const bool ok = kv_len >= p.gamma && kv_len <= p.max_keys;
  return ok ? (kv_len + TK - 1) / TK : 1;  // a malformed sequence keeps one tile to report it
}

// The work list is virtual: each unit is ovh overhead tiles followed by its real tiles,
// and a block owns an equal range of virtual tiles. A segment is the part of one unit
// inside a block's range. Only a range that ends inside a unit's overhead has a segment
// with no real tile, and then it is the range's last (a first segment without real
// tiles means the block has no work).
struct Seg {
  int b, g, rt;      // sequence, KV head (or head pair), row tile
  int64_t u;         // unit index (b * hunits + g) * row_tiles + rt
  int tile0, ntile;  // first real tile within the unit and real tile count of this segment
  int unit_tiles;    // real tiles of the whole unit
  int kv_len;
  bool len_ok;
  int64_t unit_start;  // virtual index of the unit's first real tile
  int64_t vnext;       // virtual index just past this segment
};

template <int TK>
__device__ __forceinline__ Seg locate(int64_t v, int64_t v1, const AttnParams& p,
                                      const int* pb, int ovh) {
  int lo = 0, hi = p.batch;  // largest b with pb[b] <= v
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (pb[mid] <= v) lo = mid; else hi = mid;
  }
  Seg s;
  s.b = lo;
  s.kv_len = p.kv_len[lo];
  s.len_ok = s.kv_len >= p.gamma && s.kv_len <= p.max_keys;
  s.unit_tiles = unit_tiles<TK>(s.kv_len, p);
  const int vlen = s.unit_tiles + ovh;
  const int64_t rem = v - pb[lo];
  const int ub = static_cast<int>(rem / vlen);
  const int64_t vstart = v - rem % vlen;  // the unit's first (overhead) virtual tile
  s.g = ub / p.row_tiles;
  s.rt = ub % p.row_tiles;
  s.u = static_cast<int64_t>(lo) * p.hunits * p.row_tiles + ub;
  s.unit_start = vstart + ovh;
  const int64_t vend = vstart + vlen;
  s.vnext = vend < v1 ? vend : v1;
  const int64_t lo_real = v > s.unit_start ? v : s.unit_start;
  s.ntile = s.vnext > lo_real ? static_cast<int>(s.vnext - lo_real) : 0;
  s.tile0 = s.ntile > 0 ? static_cast<int>(lo_real - s.unit_start) : 0;
  return s;
}

// Whether real tiles follow segment s in the range ending at v1. A segment ends at its
// unit's end or at v1, so the next one starts a unit, whose real tiles begin ovh virtual
// tiles later; no load is needed.
__device__ __forceinline__ bool has_more(const Seg& s, int64_t v1, int ovh) {
  return v1 - s.vnext > ovh;
}

// Block that owns virtual tile t when `total` virtual tiles are cut into `ctas` ranges
// [c * total / ctas, (c + 1) * total / ctas).
__device__ __forceinline__ int owner_of(int64_t t, int64_t total, int ctas) {
  return static_cast<int>(((t + 1) * ctas - 1) / total);
}

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

// Combines the split-KV partials of one unit, held in slots [slot0, slot0 + nslots), for
// rows [row0, row0 + nrows) and writes the final outputs (nthreads threads from tid
// cooperate; no block synchronization). Row r of the range sits at row prow0 + r of a
// slot (a head-pair unit keeps its second head's rows after the first's). A thread takes
// its (row, 8-column) items IT at a time and walks their slots in batches of SB: the
// (m, l) pairs and output pieces of those items and slots are loaded together, then
// folded into each item's running base-2 max. The merges run at the end of a block
// while the others still stream KV, when an L2 round trip takes about a microsecond:
// units of 128 or more rows (2,048+ items for D = 128) take four items per thread
// (IT = 4, SB = 2) to cut their dependent round trips; smaller ones keep one item per
// thread with up to four slots per batch (IT = 1, SB = 4), which measured faster in the
// fused step for 32-row units.
template <int D, int IT = 1>
__device__ void merge_unit(const AttnParams& p, int b, int g, int row0, int nrows, int64_t slot0,
                           int nslots, int tid, int nthreads, int prow0 = 0) {
  constexpr int C8 = D / 8;
  constexpr int SB = IT == 1 ? 4 : 2;  // slots per batch
  const int nitems = nrows * C8;
  for (int i0 = tid; i0 < nitems; i0 += IT * nthreads) {
    float M[IT], L[IT], acc[IT][8];
    bool bad[IT];
#pragma unroll
    for (int i = 0; i < IT; ++i) {
      M[i] = -INFINITY;
      L[i] = 0.f;
      bad[i] = false;
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[i][e] = 0.f;
    }
    for (int s0 = 0; s0 < nslots; s0 += SB) {
      float2 ml[IT][SB];
      float4 lo[IT][SB], hi[IT][SB];
#pragma unroll
      for (int i = 0; i < IT; ++i) {
        const int idx = i0 + i * nthreads;
        const int r = idx / C8, c8 = idx % C8;
#pragma unroll
        for (int e = 0; e < SB; ++e) {
          if (idx < nitems && s0 + e < nslots) {
            const int64_t slot = (slot0 + s0 + e) * p.slot_rows + prow0 + r;
            ml[i][e] = __ldcg(&p.partial_ml[slot]);
            const float4* src = reinterpret_cast<const float4*>(p.partial_o + slot * D) + 2 * c8;
            lo[i][e] = __ldcg(src);
            hi[i][e] = __ldcg(src + 1);
          } else {
            ml[i][e] = make_float2(-INFINITY, 0.f);
            lo[i][e] = make_float4(0.f, 0.f, 0.f, 0.f);
            hi[i][e] = lo[i][e];
          }
        }
      }
#pragma unroll
      for (int i = 0; i < IT; ++i) {
        float mb = M[i];
#pragma unroll
        for (int e = 0; e < SB; ++e) {
          bad[i] |= ml[i][e].y < 0.f;
          if (ml[i][e].y > 0.f) mb = fmaxf(mb, ml[i][e].x);
        }
        if (mb == -INFINITY) continue;
        const float scale = M[i] == -INFINITY ? 0.f : ex2(M[i] - mb);
        L[i] *= scale;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[i][e] *= scale;
#pragma unroll
        for (int e = 0; e < SB; ++e) {
          if (!(ml[i][e].y > 0.f)) continue;
          const float w = ex2(ml[i][e].x - mb);
          const float4 a = lo[i][e], c = hi[i][e];
          L[i] += ml[i][e].y * w;
          acc[i][0] += a.x * w; acc[i][1] += a.y * w; acc[i][2] += a.z * w; acc[i][3] += a.w * w;
          acc[i][4] += c.x * w; acc[i][5] += c.y * w; acc[i][6] += c.z * w; acc[i][7] += c.w * w;
        }
        M[i] = mb;
      }
    }
#pragma unroll
    for (int i = 0; i < IT; ++i) {
      const int idx = i0 + i * nthreads;
      if (idx >= nitems) break;
      const int r = idx / C8, c8 = idx % C8;
      const bool dead = bad[i] || !(L[i] > 0.f);
      write_out_row<D>(p, b, g, row0 + r, c8 * 8, acc[i], dead ? 0.f : 1.f / L[i]);
      if (c8 == 0) write_lse(p, b, g, row0 + r, M[i], L[i], dead);
    }
  }
}
#endif

}  // namespace specv
