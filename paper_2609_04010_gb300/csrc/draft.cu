// Draft-side steps of Alg. "Lossless Psi-Spec decoding (Linear Sampler)" (Appendix
// B.3): sampling the block tokens from the drafter rows (the free clean token
// x^{L+1} ~ q_0 and the B-1 drafts x~ ~ q, in parallel), and rolling the paged KV cache
// back to the step's accepted prefix.
//
// draft_sample_kernel draws without filtering, in one launch with one or more blocks per
// drafter row. Each block streams its part of the row once and keeps, for every lane of
// 64 (16-byte loads) or 32 (element loads) contiguous logits, the lane's maximum m_i and
// s_i = sum over the lane of exp2((l - m_i) log2(e) / T). These lane summaries give the
// row's normaliser S and the cumulative mass at every lane boundary, so the inverse CDF
// needs no second pass over the row: a block scan finds the lane where the cumulative
// mass crosses u * S, and one warp rescans that lane's logits. The filtered draw is the
// filtered row kernel's draw mode.
//
// commit_kv_kernel is one block: it computes every sequence's new length and page request
// (or release), takes block-wide prefix sums in batch order, and serves the requests that
// fit, so the result is the batch-order definition computed in parallel.
#include <cuda_bf16.h>

#include <cfloat>
#include <climits>
#include <cmath>

#include "common.cuh"

namespace specv {

DraftLayout draft_layout(const spec_draft_args_t& a, size_t base, int sms, bool vec) {
  DraftLayout L;
  L.lane_elems = vec ? 64 : 32;
  L.nlanes = static_cast<int>((static_cast<int64_t>(a.vocab) + L.lane_elems - 1) / L.lane_elems);
  const int64_t rows = static_cast<int64_t>(a.batch) * a.gamma;
  int64_t splits = static_cast<int64_t>(kFiltBlocksPerSm) * sms / rows;  // within one wave
  splits = splits < 1 ? 1 : (splits > kFiltMaxSplits ? kFiltMaxSplits : splits);
  if (splits > L.nlanes) splits = L.nlanes;
  L.lanes_per_split = static_cast<int>((L.nlanes + splits - 1) / splits);
  L.splits = (L.nlanes + L.lanes_per_split - 1) / L.lanes_per_split;
  L.smem = static_cast<size_t>(L.nlanes) * 8;
  const size_t split_rows = L.splits > 1 ? static_cast<size_t>(rows) : 0;
  L.tickets = base;
  L.row_flags = ws_round(L.tickets + sizeof(uint32_t) * a.batch);
  L.row_tickets = ws_round(L.row_flags + sizeof(uint32_t) * rows);
  L.lanes_g = ws_round(L.row_tickets + sizeof(uint32_t) * split_rows);
  L.parts = ws_round(L.lanes_g + 8 * split_rows * L.nlanes);
  L.end = ws_round(L.parts + 16 * split_rows * L.splits);
  return L;
}

namespace {

constexpr int kThreads = kRowThreads;
constexpr int kUnroll = 8;  // 16-byte loads (or elements) in flight per thread
constexpr uint32_t kBadRow = 1u;

struct DraftParams {
  int batch, gamma, vocab, lane_elems, nlanes, splits, lanes_per_split;
  const void* drafter;
  const float* temperature;
  const float* uniforms;
  int32_t* tokens;
  float* q_tok;
  uint32_t* status;
  uint32_t* tickets;      // [batch]
  uint32_t* row_flags;    // [batch][gamma]
  uint32_t* row_tickets;  // [batch][gamma] (splits > 1)
  float2* lanes_g;        // [batch][gamma][nlanes] (splits > 1)
  uint4* parts;           // [batch][gamma][splits]: (row maximum candidate, bad)
};

template <bool BF16>
__device__ __forceinline__ float load_elem(const void* base, int64_t i) {
  if (BF16) return bf16_bits_to_f32(static_cast<const uint16_t*>(base)[i]);
  return static_cast<const float*>(base)[i];
}

// Order-preserving key of a float (-0 shares +0's key); a candidate packs the key above
// 0xffffffff - index, so the larger candidate is the larger value, then the lower index.
__device__ __forceinline__ uint32_t order_key(float x) {
  uint32_t f = __float_as_uint(x);
  if (f == 0x80000000u) f = 0u;
  return (f & 0x80000000u) ? ~f : (f | 0x80000000u);
}
__device__ __forceinline__ unsigned long long cand_of(float x, uint32_t idx) {
  return (static_cast<unsigned long long>(order_key(x)) << 32) | (0xffffffffu - idx);
}
__device__ __forceinline__ int cand_idx(unsigned long long c) {
  return static_cast<int>(0xffffffffu - static_cast<uint32_t>(c));
}

// Block-wide exclusive scan of one float per thread, in thread order; *total gets the sum.
__device__ __forceinline__ float block_excl_scan(float x, float* sh, float* total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  float in = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, in, o);
    if (lane >= o) in += y;
  }
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
  const float ex = sh[w] + in - x;
  *total = sh[kThreads / 32];
  __syncthreads();
  return ex;
}

// One block per (split, drafter row, sequence).
template <bool BF16, bool VEC>
__global__ void __launch_bounds__(kThreads, 8) draft_sample_kernel(DraftParams p) {
  extern __shared__ __align__(16) unsigned char dsm[];
  float2* lanes = reinterpret_cast<float2*>(dsm);
  __shared__ unsigned long long s_red[kThreads / 32];
  __shared__ float s_scan[kThreads / 32 + 1];
  __shared__ int s_bad, s_last, s_pick, s_lastpos, s_tok;
  __shared__ float s_base, s_q;

  const int split = blockIdx.x, j = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int gamma = p.gamma, V = p.vocab, LE = p.lane_elems, nlanes = p.nlanes;
  const int64_t rid = static_cast<int64_t>(b) * gamma + j;
  const char* rowp = static_cast<const char*>(p.drafter) + rid * V * (BF16 ? 2 : 4);
  const float T = p.temperature[b];
  const bool greedy = !(T > 0.f);
  const float c = greedy ? 0.f : kLog2e / T;
  const float u = p.uniforms[rid];
  const int l0 = split * p.lanes_per_split;
  const int l1 = min(nlanes, l0 + p.lanes_per_split);
  const int e_begin = l0 * LE, e_end = min(V, l1 * LE);
  if (tid == 0) s_bad = 0;

  // 1. scan: the maximum (with its lowest index) and, tempered, every lane's (m_i, s_i)
  float m = -INFINITY;
  int a = INT_MAX;
  bool bad = false;
  if (VEC) {
    constexpr int kEpv = BF16 ? 8 : 4;
    constexpr int kGroup = 64 / kEpv;  // threads (vectors) per 64-element lane
    const uint32_t ninf = BF16 ? 0xFF80FF80u : 0xFF800000u;
    const uint32_t nan_mask = BF16 ? 0x7FFF7FFFu : 0x7FFFFFFFu;
    const uint32_t nan_add = BF16 ? 0x007F007Fu : 0x007FFFFFu;
    const uint32_t nan_top = BF16 ? 0x80008000u : 0x80000000u;
    const int vbeg = e_begin / kEpv, vend = e_end / kEpv;
    const uint4* rv = reinterpret_cast<const uint4*>(rowp);
    uint32_t nacc = 0;
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
        float x[kEpv];
#pragma unroll
        for (int q = 0; q < kEpv; ++q)
          x[q] = BF16 ? __uint_as_float((q & 1) ? (wv[q >> 1] & 0xffff0000u) : (wv[q >> 1] << 16))
                      : __uint_as_float(wv[q]);
        if (greedy) {
#pragma unroll
          for (int q = 0; q < 4; ++q) nacc |= (wv[q] & nan_mask) + nan_add;
#pragma unroll
          for (int q = 0; q < kEpv; ++q)
            if (x[q] > m) { m = x[q]; a = vi * kEpv + q; }
        } else {
          float vm = x[0];
#pragma unroll
          for (int q = 1; q < kEpv; ++q) vm = fmaxf(vm, x[q]);
          m = fmaxf(m, vm);
          float lm = vm;
#pragma unroll
          for (int o = 1; o < kGroup; o <<= 1) lm = fmaxf(lm, __shfl_xor_sync(0xffffffffu, lm, o));
          // The lane's weights 2^((x - lm) c), each argument one fused multiply-add. A NaN
          // logit makes its lane's sum NaN (tested once per lane below), except in a lane
          // with no finite maximum, whose words are tested here.
          float ls = 0.f;
          if (lm != -INFINITY) {
            const float nlc = -lm * c;
#pragma unroll
            for (int q = 0; q < kEpv; ++q) ls += ex2(fmaf(x[q], c, nlc));
          } else {
#pragma unroll
            for (int q = 0; q < 4; ++q) nacc |= (wv[q] & nan_mask) + nan_add;
          }
#pragma unroll
          for (int o = 1; o < kGroup; o <<= 1) ls += __shfl_xor_sync(0xffffffffu, ls, o);
          if ((tid & (kGroup - 1)) == 0 && vi < vend) {
            lanes[vi / kGroup - l0] = make_float2(lm, ls);
            bad |= ls != ls;
          }
        }
      }
    }
    bad |= (nacc & nan_top) != 0;
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
        const int ei = e0 + k * kThreads + tid;
        bad |= x[k] != x[k];
        if (greedy) {
          if (x[k] > m) { m = x[k]; a = ei; }
        } else {
          m = fmaxf(m, x[k]);
          // a warp's 32 consecutive elements are one lane
          float lm = x[k];
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) lm = fmaxf(lm, __shfl_xor_sync(0xffffffffu, lm, o));
          float ls = lm != -INFINITY ? exp2f((x[k] - lm) * c) : 0.f;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) ls += __shfl_xor_sync(0xffffffffu, ls, o);
          if ((tid & 31) == 0 && ei < e_end) lanes[ei / 32 - l0] = make_float2(lm, ls);
        }
      }
    }
  }
  if (!greedy && m == INFINITY) bad = true;  // +inf leaves the softmax undefined
  unsigned long long best = cand_of(m, static_cast<uint32_t>(a));
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
    // publish this split; the row's last block continues with the whole row
    if (!greedy)
      for (int i = tid; i < l1 - l0; i += kThreads) p.lanes_g[rid * nlanes + l0 + i] = lanes[i];
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
      for (int i = tid; i < nlanes; i += kThreads) lanes[i] = __ldcg(p.lanes_g + rid * nlanes + i);
    best = 0ull;
    uint32_t anybad = 0;
    for (int k = tid; k < p.splits; k += kThreads) {
      const uint4 q = __ldcg(p.parts + rid * p.splits + k);
      const unsigned long long cq = (static_cast<unsigned long long>(q.y) << 32) | q.x;
      best = cq > best ? cq : best;
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
    for (int k = 1; k < kThreads / 32; ++k) best = s_red[k] > best ? s_red[k] : best;
  }

  // 2. the row's token
  const float M = __uint_as_float((static_cast<uint32_t>(best >> 32) & 0x80000000u)
                                      ? (static_cast<uint32_t>(best >> 32) & 0x7fffffffu)
                                      : ~static_cast<uint32_t>(best >> 32));
  uint32_t flag = s_bad ? kBadRow : 0u;
  if (!greedy && !(M > -INFINITY)) flag = kBadRow;  // no finite logit
  int tok = -1;
  float q = NAN;
  if (!flag && greedy) {
    tok = cand_idx(best);
    q = 1.f;
  } else if (!flag) {
    // cumulative mass at lane boundaries: each thread takes a contiguous run of lanes
    const int per = (nlanes + kThreads - 1) / kThreads;
    const int i0 = min(nlanes, tid * per), i1 = min(nlanes, i0 + per);
    float mine = 0.f;
    for (int i = i0; i < i1; ++i) {
      const float2 ms = lanes[i];
      if (ms.x != -INFINITY) mine += ms.y * exp2f((ms.x - M) * c);
    }
    float S = 0.f;
    const float base = block_excl_scan(mine, s_scan, &S);
    if (tid == 0) {
      s_pick = INT_MAX;
      s_lastpos = -1;
    }
    __syncthreads();
    const float target = u * S;
    float run = base;
    for (int i = i0; i < i1; ++i) {
      const float2 ms = lanes[i];
      const float w = ms.x != -INFINITY ? ms.y * exp2f((ms.x - M) * c) : 0.f;
      run += w;
      if (w > 0.f) {
        atomicMax(&s_lastpos, i);
        if (run >= target) {
          atomicMin(&s_pick, i);
          break;
        }
      }
    }
    __syncthreads();
    const bool crossed = s_pick != INT_MAX;
    const int lane_sel = crossed ? s_pick : s_lastpos;
    if (lane_sel >= i0 && lane_sel < i1) {  // the owner of that lane: its mass before it
      float before = base;
      for (int i = i0; i < lane_sel; ++i) {
        const float2 ms = lanes[i];
        if (ms.x != -INFINITY) before += ms.y * exp2f((ms.x - M) * c);
      }
      s_base = before;
    }
    __syncthreads();
    // warp 0 rescans the lane: element e = lane_sel * LE + 2 * lane + k (k = 0, 1)
    if (tid < 32) {
      const int e0 = lane_sel * LE + 2 * tid;
      float w[2] = {0.f, 0.f};
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int e = e0 + k;
        if (2 * tid + k < LE && e < V) w[k] = exp2f((load_elem<BF16>(rowp, e) - M) * c);
      }
      float incl = w[0] + w[1];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, incl, o);
        if (tid >= o) incl += y;
      }
      const float before = s_base + incl - (w[0] + w[1]);
      int hit = -1, lastk = -1;
      if (w[0] > 0.f) { lastk = 0; if (before + w[0] >= target) hit = 0; }
      if (w[1] > 0.f) { lastk = 1; if (hit < 0 && before + w[0] + w[1] >= target) hit = 1; }
      const unsigned hm = __ballot_sync(0xffffffffu, hit >= 0);
      const unsigned lm = __ballot_sync(0xffffffffu, lastk >= 0);
      int t = -1;
      float wt = 0.f;
      if (crossed && hm) {
        const int src = __ffs(hm) - 1;
        if (tid == src) { t = e0 + hit; wt = w[hit]; }
        t = __shfl_sync(0xffffffffu, t, src);
        wt = __shfl_sync(0xffffffffu, wt, src);
      } else if (lm) {  // rounding left u * S above every sum: the last positive weight
        const int src = 31 - __clz(lm);
        if (tid == src) { t = e0 + lastk; wt = w[lastk]; }
        t = __shfl_sync(0xffffffffu, t, src);
        wt = __shfl_sync(0xffffffffu, wt, src);
      }
      if (tid == 0) {
        s_tok = t;
        s_q = wt / S;
      }
    }
    __syncthreads();
    tok = s_tok;
    q = s_q;
    if (tok < 0) flag = kBadRow;
  }
  if (tid == 0) {
    p.tokens[rid] = flag ? -1 : tok;
    if (p.q_tok) p.q_tok[rid] = flag ? NAN : q;
    p.row_flags[rid] = flag;
  }

  // 3. the sequence's last block: a sequence with a bad row draws nothing
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    const uint32_t prev = atomicAdd(&p.tickets[b], 1u);
    s_last = prev == static_cast<uint32_t>(gamma - 1);
    if (s_last) p.tickets[b] = 0;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid == 0) s_bad = 0;
  __syncthreads();
  for (int k = tid; k < gamma; k += kThreads)
    if (__ldcg(p.row_flags + static_cast<int64_t>(b) * gamma + k)) s_bad = 1;
  __syncthreads();
  if (s_bad) {
    for (int k = tid; k < gamma; k += kThreads) {
      p.tokens[static_cast<int64_t>(b) * gamma + k] = -1;
      if (p.q_tok) p.q_tok[static_cast<int64_t>(b) * gamma + k] = NAN;
    }
    if (tid == 0) set_status(p.status, SPEC_FLAG_BAD_LOGITS);
  }
}

template <bool BF16, bool VEC>
cudaError_t launch_draft_typed(const DraftParams& p, size_t smem, cudaStream_t stream) {
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(draft_sample_kernel<BF16, VEC>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  draft_sample_kernel<BF16, VEC><<<dim3(p.splits, p.gamma, p.batch), kThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------------
// KV commit
// ---------------------------------------------------------------------------------
constexpr int kCommitThreads = 1024;

__device__ __forceinline__ int block_excl_scan_int(int x, int* sh, int* total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int in = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, in, o);
    if (lane >= o) in += y;
  }
  if (lane == 31) sh[w] = in;
  __syncthreads();
  if (threadIdx.x == 0) {
    int run = 0;
    for (int k = 0; k < kCommitThreads / 32; ++k) {
      const int t = sh[k];
      sh[k] = run;
      run += t;
    }
    sh[kCommitThreads / 32] = run;
  }
  __syncthreads();
  const int ex = sh[w] + in - x;
  *total = sh[kCommitThreads / 32];
  __syncthreads();
  return ex;
}

__global__ void __launch_bounds__(kCommitThreads) commit_kv_kernel(spec_commit_args_t a) {
  __shared__ int s_scan[kCommitThreads / 32 + 1];
  __shared__ int s_used;
  const int tid = threadIdx.x, P = a.page_size, G = a.gamma, MP = a.max_pages_per_seq;
  const int count0 = *a.free_count;
  if (tid == 0) s_used = 0;
  int carry = 0;  // pages asked (reserve) or offered (release) by earlier sequences
  for (int b0 = 0; b0 < a.batch; b0 += kCommitThreads) {
    const int b = b0 + tid;
    int flag = 0, kv = 0, nl = 0, have = 0, cnt = 0, from = 0;
    if (b < a.batch) {
      kv = a.kv_len[b];
      const int na = a.num_accepted[b];
      if (kv < G || kv > MP * P || na < -1 || na > G - 1) {
        flag = 1;
      } else {
        nl = kv - G + (na >= 0 ? na + 1 : 0);
        have = (kv + P - 1) / P;
        if (a.reserve) {
          const int want = (nl + G + P - 1) / P;
          if (want > MP) flag = 2;
          else { cnt = want - have; from = have; }
        } else {
          const int keep = (nl + P - 1) / P;
          cnt = have - keep;
          from = keep;
        }
      }
    }
    int total = 0;
    const int before = carry + block_excl_scan_int(cnt, s_scan, &total);
    carry += total;
    if (b < a.batch && flag == 0 && cnt > 0) {
      int32_t* row = a.page_table + static_cast<int64_t>(b) * MP;
      if (a.reserve) {
        if (before + cnt > count0) {
          flag = 2;
        } else {
          for (int i = 0; i < cnt; ++i) row[from + i] = a.free_pages[count0 - 1 - before - i];
          atomicMax(&s_used, before + cnt);
        }
      } else {
        if (count0 + before + cnt > a.free_capacity) {
          flag = 2;
        } else {
          for (int i = 0; i < cnt; ++i) {
            a.free_pages[count0 + before + i] = row[from + i];
            row[from + i] = -1;
          }
          atomicMax(&s_used, before + cnt);
        }
      }
    }
    if (b < a.batch) {
      if (flag != 1) a.kv_len[b] = nl;
      if (a.flags) a.flags[b] = flag;
    }
  }
  __syncthreads();
  if (tid == 0) *a.free_count = a.reserve ? count0 - s_used : count0 + s_used;
}

}  // namespace

cudaError_t launch_draft(const spec_draft_args_t& a, const DraftLayout& L, char* ws,
                         cudaStream_t stream, bool vec) {
  DraftParams p;
  p.batch = a.batch;
  p.gamma = a.gamma;
  p.vocab = a.vocab;
  p.lane_elems = L.lane_elems;
  p.nlanes = L.nlanes;
  p.splits = L.splits;
  p.lanes_per_split = L.lanes_per_split;
  p.drafter = a.drafter_logits;
  p.temperature = a.temperature;
  p.uniforms = a.uniforms;
  p.tokens = a.block_tokens;
  p.q_tok = a.q_tok;
  p.status = reinterpret_cast<uint32_t*>(ws);
  p.tickets = reinterpret_cast<uint32_t*>(ws + L.tickets);
  p.row_flags = reinterpret_cast<uint32_t*>(ws + L.row_flags);
  p.row_tickets = reinterpret_cast<uint32_t*>(ws + L.row_tickets);
  p.lanes_g = reinterpret_cast<float2*>(ws + L.lanes_g);
  p.parts = reinterpret_cast<uint4*>(ws + L.parts);
  (void)cudaGetLastError();
  if (a.logits_dtype == SPEC_BF16)
    return vec ? launch_draft_typed<true, true>(p, L.smem, stream)
               : launch_draft_typed<true, false>(p, L.smem, stream);
  return vec ? launch_draft_typed<false, true>(p, L.smem, stream)
             : launch_draft_typed<false, false>(p, L.smem, stream);
}

cudaError_t launch_commit(const spec_commit_args_t& a, cudaStream_t stream) {
  (void)cudaGetLastError();
  commit_kv_kernel<<<1, kCommitThreads, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace specv
