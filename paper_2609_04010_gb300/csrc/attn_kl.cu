// Part (a) of the verify step on tcgen05 tensor cores, for KV groups of at most 64 query
// rows (group size x gamma <= 64, head_dim 128): block-causal attention of the gamma
// block queries over a paged bf16 KV cache with grouped-query heads (Sec. 4.1: the
// prefix stays in the KV cache while the block is processed; Alg. "Lossless Psi-Spec":
// one causal verifier pass over [x^{L+1}, x~]).
//
// Keys on TMEM lanes. With few query rows per KV head, a tile of M = 128 query rows
// would be mostly padding, and the softmax of the real rows would sit in one or two TMEM
// lane quadrants, i.e. on one or two SM sub-partitions. Here both products are
// transposed so that the 128 keys of a tile are the MMA's M dimension:
//   S^T [128 keys][64 rows] = K_tile [128 keys][D] . Q^T        (A = K, K-major)
//   O^T [D][64 rows]       += V_tile^T [D][128 keys] . P^T      (A = V^T, MN-major)
// so TMEM lane i of S^T holds key i of the tile. Eight softmax warps, two per lane
// quadrant (SM sub-partition), each take the quadrant's 32 keys for half of the rows.
// Row statistics are taken across lanes: the maximum of a row over a warp's keys by a
// shuffle reduce-scatter (lane i ends with row i of the warp's rows), over the four
// quadrants through shared memory (one mbarrier round per tile); the running maximum is
// raised lazily (only when it grows by more than 2^8), and O^T, whose lanes are the head
// dims, is then rescaled by the warp that owns those rows in its quadrant. Each thread
// keeps its key's share of its rows' sums; the shares are reduced once per segment.
//
// This kernel is an alternative to the row-tile kernel (attn_tc.cu), taken only when the
// caller asks for it (SPEC_ATTN_TENSOR_CORES_KEYS_ON_LANES): on GB300 it measured as fast
// as the row-tile kernel at 32 rows per KV head and slower at 64, alone and in the fused
// step, because its five 32 KB K/V stages hold no more bytes in flight than the
// row-tile kernel's ring and its unit starts cost more.
//
// Warp roles (384 threads, one block per SM, persistent):
//   warp 0   K producer: each tile's K pages, one 5-D TMA box (128-byte swizzle) per
//            page, into a ring of KS stages (mbarrier per stage carries the byte count);
//            a stage is free again once the Q K^T MMAs that read it complete.
//   warp 2   V producer: the same for V into a ring of VS stages, freed by the P V MMAs.
//   warp 1   Q K^T issuer (M = 128 keys, N = 64 rows, K = 16 steps over D) into a double
//            buffered fp32 S^T in TMEM; also loads each unit's Q tile by TMA.
//   warp 3   P V issuer (M = D = 128, N = 64 rows, K = 16 steps over keys), V read as an
//            MN-major A operand straight from its stage, P^T from shared memory; it zeroes
//            the V rows of keys past a sequence's end first.
//   warps 4..11  softmax (see above); P^T is written as bf16, one 128-byte row per key
//            (64 rows), double buffered, in the swizzled layout the MMA reads.
// Work balancing (stream-K over all 128-key tiles of all (sequence, KV head) units),
// split-unit partials and their merge, bad-input flags and bounded waits are those of
// the row-tile kernel (attn_tc.cu, attn_common.cuh).
#include <cuda.h>

#include "attn_common.cuh"
#include "tc_ptx.cuh"

namespace specv {
namespace {

using namespace tcx;

constexpr int KT = kKlKeyTile;  // keys per tile (M of the Q K^T MMA)
constexpr int NQ = 64;          // query rows per tile (N of both MMAs)
constexpr int D = 128;

template <int KS, int VS>
struct KlCfg {
  static constexpr int THREADS = 384;  // 4 producer / MMA warps + 8 softmax warps
  static constexpr uint32_t Q_BYTES = 2 * NQ * 128;      // [2 column halves][64 rows][128 B]
  static constexpr uint32_t STAGE_BYTES = KT * D * 2;    // [16 key groups][2 halves][8 keys][128 B]
  static constexpr uint32_t P_BYTES = KT * NQ * 2;       // [128 keys][64 rows] bf16
  static constexpr uint32_t OFF_Q = 0;
  static constexpr uint32_t OFF_K = OFF_Q + Q_BYTES;
  static constexpr uint32_t OFF_V = OFF_K + KS * STAGE_BYTES;
  static constexpr uint32_t OFF_P = OFF_V + VS * STAGE_BYTES;
  static constexpr uint32_t OFF_BAR = OFF_P + 2 * P_BYTES;
  // barriers: k_full[KS], k_empty[KS], v_full[VS], v_empty[VS], s_full[2], s_free[2],
  // p_full[2], pv_done[2], q_full, xch, drain[2], seg flags[8]
  static constexpr int NBAR = 2 * KS + 2 * VS + 8 + 2 + 2 + 8;
  static constexpr uint32_t OFF_MISC = OFF_BAR + NBAR * 8;               // tmem, abort, pending
  static constexpr uint32_t OFF_XMAX = (OFF_MISC + 16 + 15) / 16 * 16;  // f32 [2][4][64]
  static constexpr uint32_t OFF_ROWB = OFF_XMAX + 2 * 4 * NQ * 4;       // f32 [8][32] per warp
  static constexpr uint32_t OFF_ALPHA = OFF_ROWB + 8 * 32 * 4;          // f32 [8][32] per warp
  static constexpr uint32_t OFF_LSUM = OFF_ALPHA + 8 * 32 * 4;          // f32 [4][64]
  static constexpr uint32_t OFF_PEND = OFF_LSUM + 4 * NQ * 4;           // int [2][8]
  static constexpr uint32_t OFF_FLAG = OFF_PEND + 64;                   // int [8]
  static constexpr uint32_t OFF_PB = OFF_FLAG + 32;                     // int [batch + 1]
  static constexpr uint32_t TMEM_COLS = 256;
  static constexpr uint32_t S_COL = 0;     // S^T[buf] at columns buf * 64
  static constexpr uint32_t O_COL = 128;   // O^T at columns 128 .. 191
  // Starting a unit inside a block's range costs about this many tiles (the dependent Q
  // load and the epilogue); measured best among 1, 2, 3, 5 at the high-batch serving shape.
  static constexpr int UNIT_OVERHEAD = 5;
  static size_t smem_bytes(int batch) { return OFF_PB + 4u * (batch + 1) + 1024; }
};

constexpr int kKS = 2, kVS = 3;  // K and V ring stages (5 x 32 KB)

__device__ __forceinline__ void tma_load_page(uint32_t dst, const CUtensorMap* map, int page_head,
                                              uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(0), "r"(0), "r"(0), "r"(page_head),
      "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tma_load_q(uint32_t dst, const CUtensorMap* map, int half, int head0,
                                           int pos0, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(half), "r"(head0), "r"(pos0), "r"(bar)
      : "memory");
}
__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// RH: rows each softmax warp handles (16: rows <= 32, 32: rows <= 64); two warps per TMEM
// lane quadrant split a tile's rows.
template <int RH>
__global__ void __launch_bounds__(384, 1)
    attn_kl_kernel(const __grid_constant__ CUtensorMap tmap_k,
                   const __grid_constant__ CUtensorMap tmap_v,
                   const __grid_constant__ CUtensorMap tmap_q, AttnParams p) {
  using C = KlCfg<kKS, kVS>;
  constexpr int KS = kKS, VS = kVS;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + C::OFF_BAR;
  auto k_full = [&](int s) { return bar0 + 8u * s; };
  auto k_empty = [&](int s) { return bar0 + 8u * (KS + s); };
  auto v_full = [&](int s) { return bar0 + 8u * (2 * KS + s); };
  auto v_empty = [&](int s) { return bar0 + 8u * (2 * KS + VS + s); };
  const uint32_t bar1 = bar0 + 8u * (2 * KS + 2 * VS);
  auto s_full = [&](int b) { return bar1 + 8u * b; };
  auto s_free = [&](int b) { return bar1 + 16u + 8u * b; };
  auto p_full = [&](int b) { return bar1 + 32u + 8u * b; };
  auto pv_done = [&](int b) { return bar1 + 48u + 8u * b; };
  const uint32_t q_full = bar1 + 64u;
  const uint32_t xch = bar1 + 72u;  // the eight softmax warps, once per tile and per epilogue
  auto drain_bar = [&](int i) { return bar1 + 80u + 8u * i; };
  auto flag_bar = [&](int i) { return bar1 + 96u + 8u * i; };
  volatile int* seg_flag = reinterpret_cast<volatile int*>(smem + C::OFF_FLAG);
  uint32_t* misc = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 1);
  volatile int* pend_count = reinterpret_cast<volatile int*>(misc + 2);
  int* pend = reinterpret_cast<int*>(smem + C::OFF_PEND);
  int* pb = reinterpret_cast<int*>(smem + C::OFF_PB);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_launch_dependents();  // the acceptance kernels of a verify step may start beside us

  // ---- prologue: barriers, TMEM, per-sequence tile prefix sums ----
  if (threadIdx.x == 0) {
    for (int s = 0; s < KS; ++s) {
      mbar_init(k_full(s), 1);
      mbar_init(k_empty(s), 1);
    }
    for (int s = 0; s < VS; ++s) {
      mbar_init(v_full(s), 1);
      mbar_init(v_empty(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(s_full(b), 1);
      mbar_init(s_free(b), 8);
      mbar_init(p_full(b), 8);
      mbar_init(pv_done(b), 1);
    }
    mbar_init(q_full, 1);
    mbar_init(xch, 8);
    mbar_init(drain_bar(0), 1);
    mbar_init(drain_bar(1), 1);
    for (int i = 0; i < 8; ++i) mbar_init(flag_bar(i), 1);
    *abort_flag = 0;
    *pend_count = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(misc), C::TMEM_COLS);
  if (warp == 0) {
    int carry = 0;
    for (int b0 = 0; b0 < p.batch; b0 += 32) {
      const int b = b0 + lane;
      int v = b < p.batch ? (unit_tiles<KT>(p.kv_len[b], p) + p.unit_overhead) * p.hunits : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += y;
      }
      if (b < p.batch) pb[b + 1] = carry + v;
      carry += __shfl_sync(0xffffffffu, v, 31);
    }
    if (lane == 0) pb[0] = 0;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = misc[0];

  const int64_t total = pb[p.batch];
  // With no more units than blocks, use a multiple of the unit count (equal-length units
  // then split into equal parts with no unit boundary inside any block's range).
  int ctas = static_cast<int>(total < gridDim.x ? total : gridDim.x);
  {
    const int units = p.batch * p.hunits;
    if (units <= static_cast<int>(gridDim.x)) {
      const int aligned = units * (static_cast<int>(gridDim.x) / units);
      if (aligned < ctas) ctas = aligned;
    }
  }
  const int cta = blockIdx.x;
  const int64_t t0 = cta < ctas ? static_cast<int64_t>(cta) * total / ctas : 0;
  const int64_t t1 = cta < ctas ? static_cast<int64_t>(cta + 1) * total / ctas : 0;
  const int OVH = p.unit_overhead;

  if (warp == 0 || warp == 2) {
    // ============================ KV producers ============================
    const bool isv = warp == 2;
    const int NS = isv ? VS : KS;
    const uint32_t ring = sbase + (isv ? C::OFF_V : C::OFF_K);
    const CUtensorMap* map = isv ? &tmap_v : &tmap_k;
    uint32_t it = 0;
    bool ok = true;
    // page ids are read 32 at a time (lane i holds page cache_base + i of sequence cache_b)
    int cache_b = -1, cache_base = 0, cache_val = 0;
    auto page_of = [&](int b, int pi) -> int {  // warp-uniform
      if (b != cache_b || pi < cache_base || pi >= cache_base + 32) {
        cache_b = b;
        cache_base = pi;
        const int idx = pi + lane;
        cache_val = idx < p.max_pages ? __ldg(&p.page_table[static_cast<int64_t>(b) * p.max_pages + idx]) : 0;
      }
      return __shfl_sync(0xffffffffu, cache_val, pi - cache_base);
    };
    const uint32_t box_bytes = static_cast<uint32_t>(p.page_size) * D * 2;  // one page of one head
    uint32_t seg_no = 0;
    for (Seg s = locate<KT>(t0, t1, p, pb, OVH); s.ntile > 0 && ok; ++seg_no) {
      const bool bad = !s.len_ok;  // nothing to read
      bool flag = bad;             // ... or a page id out of range (read as page 0)
      for (int k = 0; k < s.ntile && ok; ++k, ++it) {
        const int st = static_cast<int>(it % NS);
        if (it >= static_cast<uint32_t>(NS))
          ok = mbar_wait(isv ? v_empty(st) : k_empty(st), ((it / NS) - 1) & 1, abort_flag, p.status);
        if (!ok) break;
        const uint32_t full = isv ? v_full(st) : k_full(st);
        if (bad) {
          if (lane == 0) mbar_arrive(full);
        } else {
          const int key0 = (s.tile0 + k) * KT;
          const int npg = KT / p.page_size;
          int nvalid = 0;
          for (int q = 0; q < npg; ++q) nvalid += (key0 + q * p.page_size) < s.kv_len;
          if (lane == 0) mbar_arrive_tx(full, static_cast<uint32_t>(nvalid) * box_bytes);
          for (int q = 0; q < nvalid; ++q) {
            const int raw = page_of(s.b, key0 / p.page_size + q);
            const bool in_range = raw >= 0 && raw < p.num_pages;
            flag |= !in_range;
            const int page = in_range ? raw : 0;
            if (lane == 0)
              tma_load_page(ring + st * C::STAGE_BYTES + static_cast<uint32_t>(q) * box_bytes, map,
                            page * p.hkv + s.g, full);
          }
        }
        __syncwarp();
      }
      if (ok && !isv && lane == 0) {  // both producers see every page; the K one publishes
        seg_flag[seg_no & 7] = flag ? 1 : 0;
        mbar_arrive(flag_bar(seg_no & 7));
      }
      if (!has_more(s, t1, OVH)) break;
      s = locate<KT>(s.vnext, t1, p, pb, OVH);
    }
    if (!ok) {  // drain this warp's copies still in flight (bounded)
      for (uint32_t x = it > static_cast<uint32_t>(NS) ? it - NS : 0; x < it; ++x) {
        const long long t_0 = clock64();
        const uint32_t full = isv ? v_full(x % NS) : k_full(x % NS);
        while (!mbar_try(full, (x / NS) & 1) && clock64() - t_0 < kWaitCycles) {
        }
      }
    }
  } else if (warp == 1 || warp == 3) {
    // ============================ MMA issuers ============================
    // K and V stages hold a tile as [8-key group][128-byte column half][8 keys][128 B]:
    // the 8-key groups sit 2 KB apart and the column halves 1 KB apart.
    constexpr uint32_t kGroup = 2048u;
    constexpr uint32_t kIdescQK = idesc_bf16(KT, NQ, false, false);  // A = K, B = Q: K-major
    constexpr uint32_t kIdescPV = idesc_bf16(D, NQ, true, true);     // A = V^T, B = P^T: MN-major
    const bool qk_role = warp == 1;
    uint32_t it = 0, seg_no = 0;
    bool ok = true, issued = false;
    auto issue_q = [&](const Seg& sg) {  // both column halves of the unit's Q tile
      if (lane == 0) {
        mbar_arrive_tx(q_full, C::Q_BYTES);
        for (int half = 0; half < 2; ++half)
          tma_load_q(sbase + C::OFF_Q + half * (NQ * 128u), &tmap_q, half, sg.g * p.group,
                     sg.b * p.gamma, q_full);
      }
      __syncwarp();
    };
    if (qk_role) {
      const Seg s0 = locate<KT>(t0, t1, p, pb, OVH);
      if (s0.ntile > 0) issue_q(s0);
    }
    for (Seg s = locate<KT>(t0, t1, p, pb, OVH); s.ntile > 0 && ok;) {
      if (qk_role) {
        ok = mbar_wait(q_full, seg_no & 1, abort_flag, p.status);
        if (!ok) break;
        tc_fence_after();
      }
      for (int k = 0; k < s.ntile && ok; ++k) {
        const uint32_t x = it + k;
        if (qk_role) {
          // S^T = K Q^T for tile x into S^T[x & 1]
          const int st = static_cast<int>(x % KS);
          ok = mbar_wait(k_full(st), (x / KS) & 1, abort_flag, p.status);
          if (ok && x >= 2) ok = mbar_wait(s_free(x & 1), ((x >> 1) - 1) & 1, abort_flag, p.status);
          if (!ok) break;
          tc_fence_after();
          if (lane == 0) {
            const uint32_t d_tmem = tmem + C::S_COL + (x & 1) * NQ;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const uint32_t ka = sbase + C::OFF_K + st * C::STAGE_BYTES + (kk / 4) * 1024u + (kk % 4) * 32u;
              const uint32_t qb = sbase + C::OFF_Q + (kk / 4) * (NQ * 128u) + (kk % 4) * 32u;
              mma_bf16(d_tmem, desc_sw128(ka, 16, kGroup), desc_sw128(qb, 16, 1024), kIdescQK,
                       kk > 0 ? 1u : 0u);
            }
            mma_commit(s_full(x & 1));
            mma_commit(k_empty(st));
            issued = true;
          }
          __syncwarp();
          if (k == s.ntile - 1 && has_more(s, t1, OVH)) {
            // the segment's last scores are done with its Q tile: fetch the next one
            ok = mbar_wait(s_full(x & 1), (x >> 1) & 1, abort_flag, p.status);
            if (!ok) break;
            issue_q(locate<KT>(s.vnext, t1, p, pb, OVH));
          }
        } else {
          // O^T += V^T P^T for tile x
          const int st = static_cast<int>(x % VS);
          ok = mbar_wait(v_full(st), (x / VS) & 1, abort_flag, p.status);
          if (!ok) break;
          // keys past the end of the sequence: zero their V rows so that P = 0 meets
          // finite V (their slots hold other data or stale stages)
          const int key0 = (s.tile0 + k) * KT;
          const int nvalid = s.len_ok ? min(KT, max(0, s.kv_len - key0)) : KT;
          if (nvalid < KT) {
            unsigned char* vst = smem + C::OFF_V + st * C::STAGE_BYTES;
            for (int i = lane; i < (KT - nvalid) * 16; i += 32) {
              const int key = nvalid + (i >> 4), h = (i >> 3) & 1, c = i & 7;
              *reinterpret_cast<uint4*>(vst + (key >> 3) * kGroup + h * 1024u + (key & 7) * 128u +
                                        c * 16u) = make_uint4(0, 0, 0, 0);
            }
            fence_async_smem();
          }
          __syncwarp();
          ok = mbar_wait(p_full(x & 1), (x >> 1) & 1, abort_flag, p.status);
          if (!ok) break;
          tc_fence_after();
          if (lane == 0) {
#pragma unroll
            for (int ks = 0; ks < KT / 16; ++ks) {
              const uint32_t va = sbase + C::OFF_V + st * C::STAGE_BYTES + ks * 2u * kGroup;
              const uint32_t pbm = sbase + C::OFF_P + (x & 1) * C::P_BYTES + ks * 2048u;
              mma_bf16(tmem + C::O_COL, desc_sw128(va, 1024, kGroup), desc_sw128(pbm, 1024, 1024),
                       kIdescPV, (k > 0 || ks > 0) ? 1u : 0u);
            }
            mma_commit(pv_done(x & 1));
            mma_commit(v_empty(st));
            issued = true;
          }
          __syncwarp();
        }
      }
      it += s.ntile;
      ++seg_no;
      if (!ok || !has_more(s, t1, OVH)) break;
      s = locate<KT>(s.vnext, t1, p, pb, OVH);
    }
    if (!ok && __any_sync(0xffffffffu, issued)) {  // drain this warp's MMAs (bounded)
      const uint32_t db = drain_bar(qk_role ? 0 : 1);
      if (lane == 0) mma_commit(db);
      __syncwarp();
      const long long t_0 = clock64();
      while (!mbar_try(db, 0) && clock64() - t_0 < kWaitCycles) {
      }
    }
  } else {
    // ============ softmax (warps 4..11: keys 32q..32q+31, rows row0..row0+RH-1) ============
    const int q = (warp - 4) & 3, hr = (warp - 4) >> 2;
    const int row0 = hr * RH;
    const int kt = q * 32 + lane;  // this thread's key within a tile (its TMEM lane)
    const int rl = row0 + (lane % RH);  // the row whose statistics this lane keeps
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(q * 32) << 16);
    float* xmax = reinterpret_cast<float*>(smem + C::OFF_XMAX);                  // [2][4][64]
    float* rowb = reinterpret_cast<float*>(smem + C::OFF_ROWB) + (warp - 4) * 32;   // this warp's
    float* alph = reinterpret_cast<float*>(smem + C::OFF_ALPHA) + (warp - 4) * 32;  // this warp's
    float* lsum = reinterpret_cast<float*>(smem + C::OFF_LSUM);                  // [4][64]
    const float c = p.scale_log2;
    const int R = p.rows;
    constexpr uint32_t kNegInf = 0xFF800000u;
    auto tld = [&](uint32_t addr, uint32_t* r) {
      if constexpr (RH == 32) tmem_ld32(addr, r); else tmem_ld16(addr, r);
    };
    auto tst = [&](uint32_t addr, const uint32_t* r) {
      if constexpr (RH == 32) tmem_st32(addr, r); else tmem_st16(addr, r);
    };
    uint32_t it = 0, xph = 0, seg_no = 0;
    bool ok = true;
    for (Seg s = locate<KT>(t0, t1, p, pb, OVH); s.ntile > 0 && ok;) {
      const int ctx = s.kv_len - p.gamma;
      float m = -INFINITY;  // running maximum (scaled, base 2) of row rl, the same in every warp
      float psum[RH];       // this thread's key's share of each of this warp's row sums
#pragma unroll
      for (int r = 0; r < RH; ++r) psum[r] = 0.f;
      for (int k = 0; k < s.ntile; ++k) {
        const uint32_t x = it + k;
        const int buf = static_cast<int>(x & 1);
        ok = mbar_wait(s_full(buf), (x >> 1) & 1, abort_flag, p.status);
        if (!ok) break;
        tc_fence_after();
        // keys a row cannot see: row r sees key ctx + d iff d <= r / group, i.e. r >= d * group
        // (every row sees the prefix); padding rows are dropped
        const int key0 = (s.tile0 + k) * KT;
        const bool masked = key0 + KT - 1 > ctx || R < row0 + RH;  // warp-uniform
        const int rmin = (key0 + kt - ctx) * p.group;
        const uint32_t scol = lane_base + C::S_COL + buf * NQ + row0;
        auto apply_mask = [&](uint32_t* sr) {
#pragma unroll
          for (int e = 0; e < RH; ++e)
            if (!(row0 + e >= rmin && row0 + e < R)) sr[e] = kNegInf;
        };
        // pass 1: the tile's row maxima over this warp's keys, then over the four quadrants
        {
          uint32_t sr[RH];
          tld(scol, sr);
          tmem_wait_ld();
          if (masked) apply_mask(sr);
          float v[RH];
#pragma unroll
          for (int e = 0; e < RH; ++e) v[e] = __uint_as_float(sr[e]);
          if constexpr (RH == 16) {
#pragma unroll
            for (int e = 0; e < 16; ++e) v[e] = fmaxf(v[e], __shfl_xor_sync(0xffffffffu, v[e], 16));
          }
          // reduce-scatter over the lanes: lane i ends with the maximum of row row0 + i % RH
#pragma unroll
          for (int off = RH / 2; off >= 1; off >>= 1) {
            const bool hi = (lane & off) != 0;
#pragma unroll
            for (int e = 0; e < off; ++e) {
              const float send = hi ? v[e] : v[e + off];
              const float keep = hi ? v[e + off] : v[e];
              v[e] = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, off));
            }
          }
          if (lane < RH) xmax[(buf * 4 + q) * NQ + row0 + lane] = v[0];
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(xch);
        ok = mbar_wait(xch, xph & 1, abort_flag, p.status);
        ++xph;
        if (!ok) break;
        const float* xt = xmax + buf * 4 * NQ;
        const float tmx =
            fmaxf(fmaxf(xt[rl], xt[NQ + rl]), fmaxf(xt[2 * NQ + rl], xt[3 * NQ + rl])) * c;
        // lazy rescale: the reference maximum moves only when the row grows by more than 8
        // (2^8 in the weights), or at the segment's first tile
        const bool grow = k == 0 || tmx > m + 8.f;
        float al = 1.f;
        if (grow) {
          const float mn = fmaxf(m, tmx);
          al = m == -INFINITY ? 0.f : ex2(m - mn);
          m = mn;
        }
        const bool rescale = k > 0 && __any_sync(0xffffffffu, grow);  // this warp's rows
        if (lane < RH) {
          rowb[lane] = m == -INFINITY ? 0.f : m;
          if (rescale) alph[lane] = al;
        }
        __syncwarp();
        if (rescale) {
          // O^T must hold every earlier tile before it is scaled: wait for the P V of
          // tile x - 1 (which also frees this tile's P buffer)
          ok = mbar_wait(pv_done((x - 1) & 1), ((x - 1) >> 1) & 1, abort_flag, p.status);
          if (!ok) break;
          tc_fence_after();
          uint32_t o[RH];
          tld(lane_base + C::O_COL + row0, o);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < RH; ++e) {
            const float a = alph[e];
            o[e] = __float_as_uint(__uint_as_float(o[e]) * a);
            psum[e] *= a;
          }
          tst(lane_base + C::O_COL + row0, o);
          tmem_wait_st();
        } else if (x >= 2) {
          // the P V that last read this P buffer (tile x - 2) is complete
          ok = mbar_wait(pv_done(buf), ((x - 2) >> 1) & 1, abort_flag, p.status);
          if (!ok) break;
          tc_fence_after();
        }
        // pass 2: the weights of this thread's key for the warp's rows, from a second read
        // of S^T, 8 rows (one 16-byte piece of its P^T row) at a time
        {
          uint32_t sr[RH];
          tld(scol, sr);
          tmem_wait_ld();
          if (masked) apply_mask(sr);
          unsigned char* prow = smem + C::OFF_P + buf * C::P_BYTES + kt * 128u;
#pragma unroll
          for (int r = 0; r < RH; r += 8) {
            const float4 ma = *reinterpret_cast<const float4*>(rowb + r);
            const float4 mb = *reinterpret_cast<const float4*>(rowb + r + 4);
            const float mm[8] = {ma.x, ma.y, ma.z, ma.w, mb.x, mb.y, mb.z, mb.w};
            float w[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              w[e] = ex2(fmaf(__uint_as_float(sr[r + e]), c, -mm[e]));
              psum[r + e] += w[e];
            }
            *reinterpret_cast<uint4*>(prow + ((((row0 + r) >> 3) ^ (kt & 7)) << 4)) =
                make_uint4(pack_bf16(w[0], w[1]), pack_bf16(w[2], w[3]), pack_bf16(w[4], w[5]),
                           pack_bf16(w[6], w[7]));
          }
        }
        fence_async_smem();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(s_free(buf));  // both reads of S^T[buf] are done
          mbar_arrive(p_full(buf));
        }
      }
      if (!ok) break;
      // ---- epilogue: row sums, then O^T (TMEM) -> output or partial ----
      const uint32_t xl = it + s.ntile - 1;
      ok = mbar_wait(pv_done(xl & 1), (xl >> 1) & 1, abort_flag, p.status);
      if (!ok) break;
      tc_fence_after();
      ok = mbar_wait(flag_bar(seg_no & 7), (seg_no >> 3) & 1, abort_flag, p.status);
      if (!ok) break;
      const bool bad = seg_flag[seg_no & 7] != 0;
      // this warp's share of each of its row sums: reduce-scatter over the lanes (lane i
      // ends with row row0 + i % RH), then the four quadrants through shared memory
      {
        float* v = psum;
        if constexpr (RH == 16) {
#pragma unroll
          for (int e = 0; e < 16; ++e) v[e] += __shfl_xor_sync(0xffffffffu, v[e], 16);
        }
#pragma unroll
        for (int off = RH / 2; off >= 1; off >>= 1) {
          const bool hi = (lane & off) != 0;
#pragma unroll
          for (int e = 0; e < off; ++e) {
            const float send = hi ? v[e] : v[e + off];
            const float keep = hi ? v[e + off] : v[e];
            v[e] = keep + __shfl_xor_sync(0xffffffffu, send, off);
          }
        }
        if (lane < RH) lsum[q * NQ + row0 + lane] = v[0];
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(xch);
      ok = mbar_wait(xch, xph & 1, abort_flag, p.status);
      ++xph;
      if (!ok) break;
      const float L = lsum[rl] + lsum[NQ + rl] + lsum[2 * NQ + rl] + lsum[3 * NQ + rl];
      const bool whole = s.tile0 == 0 && s.ntile == s.unit_tiles;
      const int c_first = owner_of(s.unit_start, total, ctas);
      const int c_last = owner_of(s.unit_start + s.unit_tiles - 1, total, ctas);
      const int64_t slot = s.u + cta;
      if (bad && warp == 4 && lane == 0 && (whole || cta == c_first))
        set_status(p.status, s.len_ok ? SPEC_FLAG_BAD_PAGE : SPEC_FLAG_BAD_KV_LEN);
      // 1 / L of the warp's rows for the output scaling (a bad segment writes exact zeros)
      if (whole && lane < RH) rowb[lane] = (bad || !(L > 0.f)) ? 0.f : 1.f / L;
      __syncwarp();
      // this thread's head dim d = kt of O^T, for the warp's rows
      const int d = kt;
      {
        uint32_t o[RH];
        tld(lane_base + C::O_COL + row0, o);
        tmem_wait_ld();
#pragma unroll
        for (int e = 0; e < RH; ++e) {
          const int row = row0 + e;
          if (row >= R) break;
          const float ov = __uint_as_float(o[e]);
          if (whole) {
            const int j = row / p.group, h = s.g * p.group + row % p.group;
            const float val = bad ? 0.f : ov * rowb[e];
            static_cast<__nv_bfloat16*>(p.out)[((static_cast<int64_t>(s.b) * p.gamma + j) * p.hq + h) * D + d] =
                __float2bfloat16_rn(val);
          } else {
            p.partial_o[(slot * p.slot_rows + row) * D + d] = ov;
          }
        }
      }
      tc_fence_before();
      if (q == 0 && lane < RH && rl < R) {
        if (whole) write_lse(p, s.b, s.g, rl, m, L, bad);
        else p.partial_ml[slot * p.slot_rows + rl] = make_float2(m, bad ? -1.f : L);
      }
      if (!whole && warp == 4 && lane == 0) {
        // the ticket of a split unit is taken at the end of the block, after a fence
        int* e = pend + 8 * (*pend_count);
        e[0] = s.b; e[1] = s.g; e[2] = 0; e[3] = R;
        e[4] = static_cast<int>(s.u + c_first); e[5] = c_last - c_first + 1;
        e[6] = static_cast<int>(s.u); e[7] = 0;
        *pend_count = *pend_count + 1;
      }
      it += s.ntile;
      ++seg_no;
      if (!has_more(s, t1, OVH)) break;
      s = locate<KT>(s.vnext, t1, p, pb, OVH);
    }
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
  // Split units: every thread makes its partial writes visible, then the block takes
  // one ticket per unit it wrote; the block that completes a unit merges it.
  if (!*abort_flag) {
    const int np = *pend_count;  // block-uniform
    if (np > 0) {
      __threadfence();
      __syncthreads();
      if (threadIdx.x == 0) {
        for (int i = 0; i < np; ++i) {
          int* e = pend + 8 * i;
          const uint32_t prev = atomicAdd(&p.tickets[e[6]], 1u);
          e[7] = prev == static_cast<uint32_t>(e[5] - 1);
          if (e[7]) p.tickets[e[6]] = 0;  // leave the counter at zero for the next call
        }
      }
      __syncthreads();
      bool any = false;
      for (int i = 0; i < np; ++i) any |= pend[8 * i + 7] != 0;
      if (any) __threadfence();
      for (int i = 0; i < np; ++i) {
        const int* e = pend + 8 * i;
        if (e[7]) merge_unit<D>(p, e[0], e[1], e[2], e[3], e[4], e[5], threadIdx.x, C::THREADS);
      }
    }
  }
}

template <int RH>
cudaError_t launch_rh(const spec_attn_args_t& a, const AttnPlan& P, char* ws, cudaStream_t stream) {
  using Cf = KlCfg<kKS, kVS>;
  CUtensorMap mk, mv, mq;
  if (!encode_cache_map(&mk, a.k_cache, a) || !encode_cache_map(&mv, a.v_cache, a) ||
      !encode_q_map(&mq, a, NQ))
    return cudaErrorInvalidValue;
  AttnParams p = make_attn_params(a, P, ws);
  p.q_tma = 1;
  const int64_t units = static_cast<int64_t>(a.batch) * a.num_kv_heads;
  p.unit_overhead = units > P.grid ? Cf::UNIT_OVERHEAD : 0;
  const size_t smem = Cf::smem_bytes(a.batch);
  auto kernel = attn_kl_kernel<RH>;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  kernel<<<P.grid, Cf::THREADS, smem, stream>>>(mk, mv, mq, p);
  return cudaGetLastError();
}

}  // namespace

size_t kl_smem_bytes(int rows, int batch) {
  (void)rows;
  return KlCfg<kKS, kVS>::smem_bytes(batch);
}

cudaError_t launch_attn_kl(const spec_attn_args_t& a, const AttnPlan& P, char* ws,
                           cudaStream_t stream) {
  return P.rows <= 32 ? launch_rh<16>(a, P, ws, stream) : launch_rh<32>(a, P, ws, stream);
}

}  // namespace specv
