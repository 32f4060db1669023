// Part (a) of the verify step on tcgen05 tensor cores: block-causal attention of the
// gamma block queries over a paged bf16 KV cache with grouped-query heads (Sec. 4.1:
// the prefix stays in the KV cache while the block is processed; Alg. "Lossless
// Psi-Spec": one causal verifier pass over [x^{L+1}, x~]).
//
// One block holds every query row of one KV head (row r = block position j * group +
// head-in-group), padded to M = 128 rows per tensor-core tile (two tiles when the
// group has up to 256 rows), so each KV page is read from HBM once. When a group has 33
// to 64 rows and Hkv is even, the head-pair variant serves two adjacent KV heads in
// one M tile (the first head's rows in TMEM lanes 0..63, the second's in 64..127): the
// cache stores the heads of a page next to each other, so one copy brings a page of both
// (8 KB instead of 4 KB with 16-token pages; the copy engine's rate grows with the size
// of its copies). Each head has its own Q K^T and P V MMAs over the whole tile (the rows
// of the other head are computed and ignored, as the padding rows of a 64-row group are
// otherwise). P stays in tensor memory, written as bf16 over the first head's S columns
// of its tile and read by the P V MMAs from there, so the shared memory of the P buffers
// holds one more V stage; K and V stages have separate rings.
//
// Warp roles (one block per SM, persistent):
//   warps 0,2   KV producers: gather each 64-key tile of K and V page by page through
//               the page table, one 5-D cp.async.bulk.tensor box (128-byte swizzle) per
//               (page, K or V), spread over two issuing warps (one issuer cannot keep
//               the copy engine busy with page-sized boxes), into a multi-stage ring; an
//               mbarrier per stage carries the byte count. The box lays a page out in
//               8-key groups so that the MMAs below can span pages.
//   warp 1      Q K^T issuer: S = Q K^T (tcgen05.mma kind::f16, M = 128, N = 64, K = 16
//               steps over D) into a double-buffered fp32 TMEM accumulator.
//   warp 3      P V issuer: O += P V (N = D) with V read MN-major and P from shared
//               memory, or, with two M tiles or a head pair, from tensor memory.
//   warps 4..11 softmax, one thread per query row; with one M tile two warps share a
//               32-row quadrant, one per half of each tile's keys, each with its own
//               online softmax and O (merged at the end of a unit); with two M tiles
//               one warp per quadrant. Load S from TMEM, scale and mask, online
//               softmax in base 2 with lazy rescale of O (only when the running max
//               grows by more than 2^8), write P as bf16 (in the swizzled shared-memory
//               layout the MMA reads, double-buffered, with one M tile of one head;
//               otherwise over the first 32 columns of the tile's S buffer in TMEM,
//               double-buffered with S), and at the end of a unit read O from TMEM and
//               write the output. Warps without real rows idle.
// Work is balanced across blocks "stream-K" style: all 64-key tiles of all (sequence,
// KV head, row tile) units form one list that is cut into equal contiguous ranges; a
// unit split between blocks is merged from fp32 partials by the last block to finish
// it (atomic ticket, no waiting; a head pair's slots are first brought into the idle
// K/V stages by bulk copies). Every mbarrier wait is bounded: a wait that runs out
// sets SPEC_FLAG_TIMEOUT, drains the block's own copies and MMAs, frees TMEM and exits.
#include <cuda.h>  // CUtensorMap and its encoder's signature (resolved at run time)

#include "attn_common.cuh"
#include "tc_ptx.cuh"

namespace specv {
namespace {

constexpr int TK = kTcKeyTile;               // keys per tile


// QR: query rows one Q or P buffer of an M tile holds: 128, or 64 when a KV group has at
// most 64 query rows. The MMAs still read M = 128 rows; with QR = 64 the buffers are laid
// out Q, P, K/V stages, so that the 64 padding rows each read comes from the next
// buffer (their scores and outputs are never used), and the freed 32 KB (D = 128) holds
// one more K/V stage: more bytes in flight per SM.
// HP: KV heads per block (2: the head-pair variant; QR = 64, one M tile of 2 x 64 rows).
template <int D, int MT, int QR = 128, int HP = 1>
struct TcCfg {
  static_assert(QR == 128 || (QR == 64 && MT == 1), "64-row buffers only with one M tile");
  static_assert(HP == 1 || (HP == 2 && QR == 64), "head pairs only with groups of <= 64 rows");
  static constexpr int DH = D / 64;                   // 128-byte column halves of a row
  // Softmax warps per 32-row quadrant. With one M tile of one head, two warps share each
  // quadrant, one per half of the tile's keys, each with its own online-softmax state
  // and its own O accumulator (merged once per unit); otherwise one warp per quadrant
  // (with two heads the second O pair would not fit in TMEM).
  static constexpr int SPLIT = (MT == 1 && HP == 1) ? 2 : 1;
  static constexpr int KH = TK / SPLIT;               // keys of a tile per softmax warp
  // P in tensor memory (head pairs, two M tiles): P of M tile mt over the first 32
  // columns of its (first head's) S buffer of the tile, which then stays busy until the
  // tile's P V MMAs complete; double-buffered with S
  static constexpr bool PTMEM = HP == 2 || MT == 2;
  static constexpr int PB = (MT == 1 || PTMEM) ? 2 : 1;  // P buffers
  static constexpr int MR = QR * HP;                  // rows of a Q or P buffer
  // one ring of K+V stages (HP = 1), or KST stages of K and VST of V (HP = 2); two M tiles
  // with P in TMEM have the P buffer's 32 KB as a fourth stage
  static constexpr int STAGES = QR == 64 ? 5 : ((D == 64 && MT == 1) ? 3 : 4);
  static constexpr int KST = HP == 2 ? (D == 128 ? 3 : 4) : STAGES;
  static constexpr int VST = HP == 2 ? (D == 128 ? 3 : 4) : STAGES;
  static constexpr int RINGBARS = HP == 2 ? 2 * (KST + VST) : 2 * STAGES;
  static constexpr int THREADS = 128 + 256;           // 4 producer / MMA warps + 8 softmax
  // Starting a unit inside a block's range costs about this many tiles of time (its Q
  // tile, the pipeline refill and the previous unit's epilogue). When blocks hold
  // several unit starts the work list charges it, so that blocks stay balanced.
  static constexpr int UNIT_OVERHEAD = MT == 1 ? 3 : 2;
  static constexpr uint32_t QHALF = MR * 128u;          // one column half of an M tile's Q
  static constexpr uint32_t PBUF = MR * 128u;           // one P buffer of an M tile
  static constexpr uint32_t Q_BYTES = MT * DH * QHALF;  // [MT][DH][MR rows x 128 B]
  // one stage of K (or V): [8-key group][head][DH][8 keys x 128 B]
  static constexpr uint32_t KV_BYTES = HP * DH * 8192;
  static constexpr uint32_t P_BYTES = PTMEM ? 0 : PB * MT * PBUF;  // [PB][MT][MR rows x 128 B]
  static constexpr uint32_t OFF_Q = 0;
  static constexpr uint32_t OFF_P = QR == 64 ? OFF_Q + Q_BYTES : OFF_Q + Q_BYTES + 2 * STAGES * KV_BYTES;
  static constexpr uint32_t OFF_K = QR == 64 ? OFF_P + P_BYTES : OFF_Q + Q_BYTES;
  static constexpr uint32_t OFF_V = OFF_K + KST * KV_BYTES;
  static constexpr uint32_t OFF_BAR = QR == 64 ? OFF_V + VST * KV_BYTES : OFF_P + P_BYTES;
  // the K and V stages, contiguous from OFF_K; at a block's end they stage the partials
  // of the units it merges
  static constexpr uint32_t RING_BYTES = (KST + VST) * KV_BYTES;
  // barriers: ring (kv_full[S], kv_empty[S], or k_full[KST], v_full[VST], k_empty[KST],
  // v_empty[VST]), s_full[MT][2], s_free[MT][2], p_full[MT][PB], pv_done[MT][PB],
  // seg_ready, drain[2], xch[4], q_full, seg_flag_ready[8], merge_staged (HP = 2)
  static constexpr int NBAR = RINGBARS + 4 * MT + 2 * MT * PB + 3 + 4 + 1 + 8 + (HP == 2 ? 1 : 0);
  static constexpr uint32_t OFF_MISC = OFF_BAR + NBAR * 8;  // tmem base, abort, pending count
  static constexpr uint32_t OFF_XCH = OFF_MISC + 16;        // [4][2][32] float2 (m, l) per half
  static constexpr uint32_t OFF_PEND = OFF_XCH + (SPLIT == 2 ? 4 * 2 * 32 * 8 : 0);  // [2][8]
  static constexpr uint32_t OFF_FLAG = OFF_PEND + 64;  // [8] bad flags of segments
  static constexpr uint32_t OFF_PB = (OFF_FLAG + 32 + 15) / 16 * 16;
  // accumulators a = mt * HP + head: S[a][buf] at (a * 2 + buf) * 64, O[a][half] at
  // O_COL + (a * SPLIT + half) * D
  static constexpr uint32_t TMEM_NEED = MT * HP * 128 + MT * HP * SPLIT * D;
  static constexpr uint32_t TMEM_COLS = TMEM_NEED <= 256 ? 256 : 512;
  static_assert(TMEM_NEED <= 512, "TMEM holds 512 columns");
  static constexpr uint32_t S_COL = 0;
  static constexpr uint32_t O_COL = MT * HP * 128;
  static size_t smem_bytes(int batch) { return OFF_PB + 4u * (batch + 1) + 1024; }
};

// ---------------------------------------------------------------------------------
// PTX wrappers (the generic ones are in tc_ptx.cuh)
// ---------------------------------------------------------------------------------
using namespace tcx;
constexpr long long kWaitLimitCycles = kWaitCycles;
// One page of one KV head, or of two adjacent ones (box of the 5-D view of the cache, see
// encode_cache_map), landing as [8-row group][head][128-byte column half][8 rows][128 B],
// 128-byte swizzle.
// The page-and-head coordinate is the map's last dimension with one head per box and
// its fourth with two (see encode_cache_map).
template <int HP>
__device__ __forceinline__ void tma_load_page(uint32_t dst, const CUtensorMap* map, int page_head,
                                              uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(0), "r"(0), "r"(HP == 2 ? page_head : 0),
      "r"(HP == 2 ? 0 : page_head), "r"(bar)
      : "memory");
}
// Rows of one M tile of Q: 128 / group block positions of `group` heads, one
// 128-byte column half (box of the 4-D view of Q, see encode_q_map).
__device__ __forceinline__ void tma_load_q(uint32_t dst, const CUtensorMap* map, int half, int head0,
                                           int pos0, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(half), "r"(head0), "r"(pos0), "r"(bar)
      : "memory");
}
// Contiguous global -> shared copy by the copy engine, completing on bar (16-byte aligned
// addresses, size a multiple of 16).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}
// Orders this thread's view of global memory (generic proxy) before its later copies
// by the copy engine (async proxy).
__device__ __forceinline__ void fence_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}
__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// Merge of one unit from its partial slots staged in shared memory: so[nsl][slot_rows][D]
// and sml[nsl][slot_rows] = (m, l), row r of [row0, row0 + nrows) at slot row prow0 + r.
// The same combination as merge_unit, with every load from shared memory.
template <int D>
__device__ void merge_staged(const AttnParams& p, int b, int g, int row0, int nrows, const float* so,
                             const float2* sml, int nsl, int prow0, int tid, int nthreads) {
  constexpr int C8 = D / 8;
  for (int idx = tid; idx < nrows * C8; idx += nthreads) {
    const int r = idx / C8, c8 = idx % C8, pr = prow0 + r;
    float mx = -INFINITY;
    bool bad = false;
    for (int i = 0; i < nsl; ++i) {
      const float2 ml = sml[i * p.slot_rows + pr];
      bad |= ml.y < 0.f;
      if (ml.y > 0.f) mx = fmaxf(mx, ml.x);
    }
    float L = 0.f, acc[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = 0.f;
    if (mx != -INFINITY) {
      for (int i = 0; i < nsl; ++i) {
        const float2 ml = sml[i * p.slot_rows + pr];
        if (!(ml.y > 0.f)) continue;
        const float w = ex2(ml.x - mx);
        const float4* src = reinterpret_cast<const float4*>(so + (static_cast<size_t>(i) * p.slot_rows + pr) * D) + 2 * c8;
        const float4 a = src[0], c = src[1];
        L += ml.y * w;
        acc[0] += a.x * w; acc[1] += a.y * w; acc[2] += a.z * w; acc[3] += a.w * w;
        acc[4] += c.x * w; acc[5] += c.y * w; acc[6] += c.z * w; acc[7] += c.w * w;
      }
    }
    const bool dead = bad || !(L > 0.f);
    write_out_row<D>(p, b, g, row0 + r, c8 * 8, acc, dead ? 0.f : 1.f / L);
    if (c8 == 0) write_lse(p, b, g, row0 + r, mx, L, dead);
  }
}

// ---------------------------------------------------------------------------------
// The kernel
// ---------------------------------------------------------------------------------
// TREE: tree attention (a per-row mask over the block keys) instead of the causal block.
template <int D, int MT, bool TREE, int QR, int HP>
__global__ void __launch_bounds__(TcCfg<D, MT, QR, HP>::THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmap_k,
                   const __grid_constant__ CUtensorMap tmap_v,
                   const __grid_constant__ CUtensorMap tmap_q, AttnParams p) {
  using C = TcCfg<D, MT, QR, HP>;
  constexpr int SPLIT = C::SPLIT, KH = C::KH, PB = C::PB;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + C::OFF_BAR;
  // HP = 1: one ring of K+V stages
  auto kv_full = [&](int s) { return bar0 + 8u * s; };
  auto kv_empty = [&](int s) { return bar0 + 8u * (C::STAGES + s); };
  // HP = 2: a ring of K stages (freed by the Q K^T MMAs) and a ring of V stages
  auto k_full = [&](int s) { return bar0 + 8u * s; };
  auto v_full = [&](int s) { return bar0 + 8u * (C::KST + s); };
  auto k_empty = [&](int s) { return bar0 + 8u * (C::KST + C::VST + s); };
  auto v_empty = [&](int s) { return bar0 + 8u * (2 * C::KST + C::VST + s); };
  constexpr uint32_t RB = C::RINGBARS;
  auto s_full = [&](int mt, int bf) { return bar0 + 8u * (RB + mt * 2 + bf); };
  auto s_free = [&](int mt, int bf) { return bar0 + 8u * (RB + 2 * MT + mt * 2 + bf); };
  // P buffer pb of M tile mt: written by the softmax warps, read by the P V MMAs
  auto p_full = [&](int mt, int pb) { return bar0 + 8u * (RB + 4 * MT + mt * PB + pb); };
  auto pv_done = [&](int mt, int pb) {
    return bar0 + 8u * (RB + 4 * MT + MT * PB + mt * PB + pb);
  };
  const uint32_t seg_ready = bar0 + 8u * (RB + 4 * MT + 2 * MT * PB);
  auto drain_bar = [&](int i) { return seg_ready + 8 + 8u * i; };  // per MMA issuer
  auto xch_bar = [&](int q) { return seg_ready + 24 + 8u * q; };   // the two halves of quadrant q
  const uint32_t q_full = seg_ready + 56;  // Q tile of the next segment landed (TMA)
  // segment flags: the producer publishes whether a segment reads a bad page or has a
  // malformed length (ring of 8, far more than the producer can run ahead)
  auto flag_bar = [&](int i) { return seg_ready + 64 + 8u * i; };
  const uint32_t merge_bar = seg_ready + 128;  // a unit's partials staged in the ring
  volatile int* seg_flag = reinterpret_cast<volatile int*>(smem + C::OFF_FLAG);
  uint32_t* misc = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 1);
  volatile int* pend_count = reinterpret_cast<volatile int*>(misc + 2);
  // split units this block wrote partials for (only a block's first and last segments
  // can be split): b, g, row0, nrows, first slot, slots, unit, merge-here flag
  int* pend = reinterpret_cast<int*>(smem + C::OFF_PEND);
  int* pb = reinterpret_cast<int*>(smem + C::OFF_PB);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_launch_dependents();  // the acceptance kernels of a verify step may start beside us

  // ---- roles ----
  // Softmax warps take part only as far as the row tile has real rows (32 per warp).
  // With a head pair, quadrants 0-1 hold the first head's rows and 2-3 the second's.
  const int rows_cta = min(p.rows_per_cta, p.rows);
  int nact[MT];  // active quadrants of each M tile
  int nact_total = 0;
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
    nact[mt] = HP == 2 ? 2 * min(2, (rows_cta + 31) / 32) : min(4, max(0, (rows_cta - 128 * mt + 31) / 32));
    nact_total += nact[mt];
  }
  const int nsoft = nact_total * SPLIT;  // active softmax warps
  auto soft_active = [&](int sw) {  // softmax warp sw = warp - 4 has real rows
    if (HP == 2) return sw < 4 && (sw & 1) * 32 < rows_cta;
    return (sw & 3) < nact[(sw >> 2) / SPLIT];
  };
  constexpr int nprod = 2;  // KV producer warps 0 and 2
  const int pw = warp == 0 ? 0 : (warp == 2 ? 1 : -1);

  // ---- prologue: barriers, TMEM, per-sequence tile prefix sums ----
  if (threadIdx.x == 0) {
    if (HP == 2) {
      for (int s = 0; s < C::KST; ++s) {
        mbar_init(k_full(s), 1);
        mbar_init(k_empty(s), 1);
      }
      for (int s = 0; s < C::VST; ++s) {
        mbar_init(v_full(s), 1);
        mbar_init(v_empty(s), 1);
      }
    } else {
      for (int s = 0; s < C::STAGES; ++s) {
        mbar_init(kv_full(s), nprod);
        mbar_init(kv_empty(s), 1);
      }
    }
    for (int mt = 0; mt < MT; ++mt) {
      const uint32_t nw = nact[mt] > 0 ? nact[mt] * SPLIT : 1;
      for (int bf = 0; bf < 2; ++bf) {
        mbar_init(s_full(mt, bf), 1);
        mbar_init(s_free(mt, bf), nw);
      }
      for (int pb = 0; pb < PB; ++pb) {
        mbar_init(p_full(mt, pb), nw);
        mbar_init(pv_done(mt, pb), 1);
      }
    }
    mbar_init(seg_ready, nsoft);
    mbar_init(drain_bar(0), 1);
    mbar_init(drain_bar(1), 1);
    for (int q = 0; q < 4; ++q) mbar_init(xch_bar(q), 2);
    mbar_init(q_full, 1);
    for (int i = 0; i < 8; ++i) mbar_init(flag_bar(i), 1);
    if (HP == 2) mbar_init(merge_bar, 1);
    *abort_flag = 0;
    *pend_count = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(smem_u32(misc), C::TMEM_COLS);
  if (warp == 0) {
    const int per_b = p.hunits * p.row_tiles;
    int carry = 0;
    for (int b0 = 0; b0 < p.batch; b0 += 32) {
      const int b = b0 + lane;
      int v = b < p.batch ? (unit_tiles<TK>(p.kv_len[b], p) + p.unit_overhead) * per_b : 0;
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
  // With no more units than blocks, use a multiple of the unit count: equal-length
  // units then split into equal parts with no unit boundary inside any block's range
  // (a few SMs idle; measured faster than spreading boundaries and extra merges over
  // every SM). Ranges stay equal in tiles, so ragged lengths stay balanced.
  int ctas = static_cast<int>(total < gridDim.x ? total : gridDim.x);
  {
    const int units = p.batch * p.hunits * p.row_tiles;
    if (units <= static_cast<int>(gridDim.x)) {
      const int aligned = units * (static_cast<int>(gridDim.x) / units);
      if (aligned < ctas) ctas = aligned;
    }
  }
  const int cta = blockIdx.x;
  const int64_t t0 = cta < ctas ? static_cast<int64_t>(cta) * total / ctas : 0;
  const int64_t t1 = cta < ctas ? static_cast<int64_t>(cta + 1) * total / ctas : 0;
  const int OVH = p.unit_overhead;

  if (pw >= 0) {
    // ============================ KV producers ============================
    // A tile needs one box per (page, K or V): producer 0 issues the K boxes, producer 1
    // the V boxes (one issuer cannot keep the copy engine busy with page-sized boxes).
    // With one head both fill the same K+V stage; with a head pair each has its own ring.
    uint32_t it = 0;
    bool ok = true;
    // Page ids are read 32 at a time (lane i holds page cache_base + i of sequence
    // cache_b) so that one L2 round trip serves several tiles.
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
    // one page of HP heads
    const uint32_t box_bytes = static_cast<uint32_t>(p.page_size) * D * 2 * HP;
    const uint32_t RS = HP == 2 ? (pw == 0 ? C::KST : C::VST) : C::STAGES;  // ring stages
    auto ring_full = [&](uint32_t st) {
      return HP == 2 ? (pw == 0 ? k_full(st) : v_full(st)) : kv_full(st);
    };
    auto ring_empty = [&](uint32_t st) {
      return HP == 2 ? (pw == 0 ? k_empty(st) : v_empty(st)) : kv_empty(st);
    };
    const uint32_t ring_base = sbase + (pw == 0 ? C::OFF_K : C::OFF_V);
    const CUtensorMap* map = pw == 0 ? &tmap_k : &tmap_v;
    uint32_t seg_no = 0;
    for (Seg s = locate<TK>(t0, t1, p, pb, OVH); s.ntile > 0 && ok && !p.starve; ++seg_no) {
      const bool bad = !s.len_ok;  // nothing to read
      bool flag = bad;             // ... or a page id out of range (read as page 0)
      for (int k = 0; k < s.ntile && ok; ++k, ++it) {
        const uint32_t st = it % RS;
        if (it >= RS) ok = mbar_wait(ring_empty(st), ((it / RS) - 1) & 1, abort_flag, p.status);
        if (!ok) break;
        if (bad) {
          if (lane == 0) mbar_arrive(ring_full(st));
        } else {
          const int key0 = (s.tile0 + k) * TK;
          const int npg = TK / p.page_size;
          int nvalid = 0;
          for (int q = 0; q < npg; ++q) nvalid += (key0 + q * p.page_size) < s.kv_len;
          if (lane == 0) mbar_arrive_tx(ring_full(st), static_cast<uint32_t>(nvalid) * box_bytes);
          for (int q = 0; q < nvalid; ++q) {
            const int raw = page_of(s.b, key0 / p.page_size + q);
            const bool in_range = raw >= 0 && raw < p.num_pages;
            flag |= !in_range;
            const int page = in_range ? raw : 0;
            if (lane == 0)
              tma_load_page<HP>(ring_base + st * C::KV_BYTES + static_cast<uint32_t>(q) * box_bytes, map,
                                page * p.hkv + s.g * HP, ring_full(st));
          }
        }
        __syncwarp();
      }
      if (ok && pw == 0 && lane == 0) {  // both producers see every page; one publishes
        seg_flag[seg_no & 7] = flag ? 1 : 0;
        mbar_arrive(flag_bar(seg_no & 7));
      }
      if (!has_more(s, t1, OVH)) break;
      s = locate<TK>(s.vnext, t1, p, pb, OVH);
    }
    if (!ok) {  // drain this producer's copies still in flight (bounded)
      for (uint32_t x = it > RS ? it - RS : 0; x < it; ++x) {
        const long long t_0 = clock64();
        while (!mbar_try(ring_full(x % RS), (x / RS) & 1) && clock64() - t_0 < kWaitLimitCycles) {
        }
      }
    }
  } else if (warp == 1 || warp == 3) {
    // ============================ MMA issuers ============================
    // Two issuing warps feed the tensor pipe: warp 1 issues S = Q K^T as soon as a
    // tile's K has landed and its S buffer is free (so it runs up to two tiles ahead),
    // warp 3 issues O += P V as soon as a tile's P is written. A blocked issue of one
    // kind never delays the other.
    // K and V stages hold a tile as [8-key group][head][128-byte column half][8 keys]
    // [128 B]: 8-key groups sit at a uniform stride of HP * DH KB across pages, so Q K^T
    // runs with N = 64 keys and P V reads V MN-major with the column halves 1 KB apart.
    constexpr uint32_t kGroup = HP * C::DH * 1024u;
    constexpr uint32_t kHead = C::DH * 1024u;  // the second head of a pair in a key group
    constexpr uint32_t kIdescQK = idesc_bf16(128, TK, false);
    constexpr uint32_t kIdescPV = idesc_bf16(128, D, true);
    const bool qk_role = warp == 1;
    uint32_t it = 0, seg_no = 0;
    bool ok = true;
    bool issued = false;
    // Q tiles of a segment (all M tiles, both column halves, each head of a pair) by TMA,
    // on q_full
    auto issue_q = [&](const Seg& sg) {
      if (lane == 0) {
        mbar_arrive_tx(q_full, C::Q_BYTES);
        for (int mt = 0; mt < MT; ++mt)
          for (int half = 0; half < C::DH; ++half)
            for (int h = 0; h < HP; ++h)
              tma_load_q(sbase + C::OFF_Q + (mt * C::DH + half) * C::QHALF + h * (QR * 128u), &tmap_q,
                         half, (sg.g * HP + h) * p.group,
                         sg.b * p.gamma + (sg.rt * p.rows_per_cta + mt * 128) / p.group, q_full);
      }
      __syncwarp();
    };
    // keys past the end of the sequence: zero their V rows so that P = 0 meets finite V
    auto zero_v_tail = [&](uint32_t vstage, const Seg& sg, int k) {
      const int key0 = (sg.tile0 + k) * TK;
      const int nvalid = sg.len_ok ? min(TK, max(0, sg.kv_len - key0)) : TK;
      if (nvalid < TK) {
        unsigned char* vst = smem + C::OFF_V + vstage * C::KV_BYTES;
        constexpr int kPieces = HP * C::DH * 8;  // 16-byte pieces of one key's rows
        for (int i = lane; i < (TK - nvalid) * kPieces; i += 32) {
          const int key = nvalid + i / kPieces, r = i % kPieces;
          const int h = r / (C::DH * 8), hh = (r / 8) % C::DH, c = r % 8;
          *reinterpret_cast<uint4*>(vst + (key >> 3) * kGroup + h * kHead + hh * 1024u +
                                    (key & 7) * 128u + c * 16u) = make_uint4(0, 0, 0, 0);
        }
        fence_async_smem();
      }
      __syncwarp();
    };
    if (qk_role && p.q_tma) {
      const Seg s0 = locate<TK>(t0, t1, p, pb, OVH);
      if (s0.ntile > 0) issue_q(s0);
    }
    for (Seg s = locate<TK>(t0, t1, p, pb, OVH); s.ntile > 0 && ok;) {
      if (qk_role) {
        ok = mbar_wait(p.q_tma ? q_full : seg_ready, seg_no & 1, abort_flag, p.status);
        if (!ok) break;
        tc_fence_after();
      }
      for (int k = 0; k < s.ntile && ok; ++k) {
        const uint32_t x = it + k;
        if (qk_role) {
          // S = Q K^T for tile x into S[mt * HP + h][x & 1]
          const uint32_t st = x % C::KST;
          ok = HP == 2 ? mbar_wait(k_full(st), (x / C::KST) & 1, abort_flag, p.status)
                       : mbar_wait(kv_full(st), (x / C::STAGES) & 1, abort_flag, p.status);
          if (!ok) break;
          if (HP == 1) zero_v_tail(st, s, k);  // the stage's V has landed with its K
          // S[x & 1] is free once tile x - 2's softmax has read it (and, with P in TMEM,
          // once that tile's P V MMAs have read its P)
          if (x >= 2)
            for (int mt = 0; mt < MT && ok; ++mt)
              ok = mbar_wait(C::PTMEM ? pv_done(mt, x & 1) : s_free(mt, x & 1), ((x >> 1) - 1) & 1,
                             abort_flag, p.status);
          if (!ok) break;
          tc_fence_after();
          if (lane == 0) {
            for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
              for (int h = 0; h < HP; ++h) {
                const uint32_t d_tmem = tmem + C::S_COL + ((mt * HP + h) * 2 + (x & 1)) * TK;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                  const uint32_t qa = sbase + C::OFF_Q + (mt * C::DH + kk / 4) * C::QHALF + (kk % 4) * 32u;
                  const uint32_t kb = sbase + C::OFF_K + st * C::KV_BYTES + h * kHead + (kk / 4) * 1024u +
                                      (kk % 4) * 32u;
                  mma_bf16(d_tmem, desc_sw128(qa, 16, 1024), desc_sw128(kb, 16, kGroup), kIdescQK, kk > 0);
                }
              }
              mma_commit(s_full(mt, x & 1));
            }
            if (HP == 2) mma_commit(k_empty(st));
            issued = true;
          }
          __syncwarp();
          if (p.q_tma && k == s.ntile - 1 && has_more(s, t1, OVH)) {
            // the segment's last scores are done with its Q tile: fetch the next one
            for (int mt = 0; mt < MT && ok; ++mt)
              ok = mbar_wait(s_full(mt, x & 1), (x >> 1) & 1, abort_flag, p.status);
            if (!ok) break;
            issue_q(locate<TK>(s.vnext, t1, p, pb, OVH));
          }
        } else {
          // O += P V for tile x (its P implies its S, hence its landed K stage; with a
          // head pair the V stage has its own barrier)
          const uint32_t st = x % C::VST;
          if (HP == 2) {
            ok = mbar_wait(v_full(st), (x / C::VST) & 1, abort_flag, p.status);
            if (!ok) break;
            zero_v_tail(st, s, k);
          }
          const int pbuf = static_cast<int>(x % PB);
          for (int mt = 0; mt < MT && ok; ++mt)
            ok = mbar_wait(p_full(mt, pbuf), (x / PB) & 1, abort_flag, p.status);
          if (!ok) break;
          tc_fence_after();
          if (lane == 0) {
            for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
              for (int h = 0; h < HP; ++h) {
#pragma unroll
                for (int hf = 0; hf < SPLIT; ++hf) {
                  // each key half accumulates into its own O
                  const uint32_t d_tmem = tmem + C::O_COL + ((mt * HP + h) * SPLIT + hf) * D;
#pragma unroll
                  for (int kk = 0; kk < KH / 16; ++kk) {
                    const int kg = hf * (KH / 16) + kk;  // 16-key step within the tile
                    const uint32_t vb = sbase + C::OFF_V + st * C::KV_BYTES + h * kHead + kg * 2u * kGroup;
                    if constexpr (C::PTMEM) {  // P from TMEM: 8 columns per 16 keys
                      mma_bf16_ta(d_tmem, tmem + C::S_COL + (mt * HP * 2 + pbuf) * TK + kg * 8u,
                                  desc_sw128(vb, 1024, kGroup), kIdescPV, (k > 0 || kk > 0) ? 1u : 0u);
                    } else {
                      const uint32_t pa = sbase + C::OFF_P + (pbuf * MT + mt) * C::PBUF + kg * 32u;
                      mma_bf16(d_tmem, desc_sw128(pa, 16, 1024), desc_sw128(vb, 1024, kGroup), kIdescPV,
                               (k > 0 || kk > 0) ? 1u : 0u);
                    }
                  }
                }
              }
              mma_commit(pv_done(mt, pbuf));
            }
            mma_commit(HP == 2 ? v_empty(st) : kv_empty(st));
            issued = true;
          }
          __syncwarp();
        }
      }
      it += s.ntile;
      ++seg_no;
      if (!has_more(s, t1, OVH)) break;
      s = locate<TK>(s.vnext, t1, p, pb, OVH);
    }
    if (!ok && __any_sync(0xffffffffu, issued)) {  // drain this warp's MMAs (bounded)
      const uint32_t db = drain_bar(qk_role ? 0 : 1);
      if (lane == 0) mma_commit(db);
      __syncwarp();
      const long long t_0 = clock64();
      while (!mbar_try(db, 0) && clock64() - t_0 < kWaitLimitCycles) {
      }
    }
  } else if (warp >= 4 && soft_active(warp - 4)) {
    // ====================== softmax (warps with real rows) ======================
    const int sw = warp - 4, q4 = sw & 3;
    const int mt = HP == 2 ? 0 : (sw >> 2) / SPLIT, hf = HP == 2 ? 0 : (sw >> 2) % SPLIT;
    const int hp = HP == 2 ? q4 >> 1 : 0;  // head of the pair
    const int row = q4 * 32 + lane;        // TMEM lane = row of this M tile
    // row within the unit's row tile (of its head)
    const int lrow = HP == 2 ? (q4 & 1) * 32 + lane : mt * 128 + row;
    const int acc = mt * HP + hp;          // this row's S and O accumulators
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(q4 * 32) << 16);
    const uint32_t ocol = lane_base + C::O_COL + (acc * SPLIT + hf) * D;  // this half's O
    const uint32_t o0col = lane_base + C::O_COL + acc * SPLIT * D;        // first half's O
    const int prow = hp * p.rows + lrow;  // row within a partial slot
    constexpr int kChunks = D / 8 / SPLIT;  // 16-byte pieces of a query row per warp
    uint32_t it = 0, xphase = 0;
    bool ok = true;
    // A row of a segment: the unit row it holds and whether it is a real query row.
    struct RowOf {
      int urow, j, h, kvh;
      bool real;
    };
    auto row_of = [&](const Seg& sg) {
      RowOf r;
      r.urow = sg.rt * p.rows_per_cta + lrow;
      r.real = r.urow < p.rows && lrow < p.rows_per_cta;
      r.j = r.urow / p.group;
      r.kvh = sg.g * HP + hp;
      r.h = r.kvh * p.group + r.urow % p.group;
      return r;
    };
    // this warp's share of a query row (zeros for padding rows)
    auto load_q = [&](const Seg& sg, uint4* qr) {
      const RowOf r = row_of(sg);
      const uint4* src = reinterpret_cast<const uint4*>(
          static_cast<const __nv_bfloat16*>(p.q) +
          ((static_cast<int64_t>(sg.b) * p.gamma + (r.real ? r.j : 0)) * p.hq + (r.real ? r.h : 0)) * D);
#pragma unroll
      for (int c2 = 0; c2 < kChunks; ++c2)
        qr[c2] = r.real ? __ldg(src + hf * kChunks + c2) : make_uint4(0, 0, 0, 0);
    };
    // ... into the swizzled Q tile, then tell the MMA warp the segment may start
    auto store_q = [&](const uint4* qr) {
#pragma unroll
      for (int c2 = 0; c2 < kChunks; ++c2) {
        const int c = hf * kChunks + c2, half = c >> 3, ch = c & 7;
        *reinterpret_cast<uint4*>(smem + C::OFF_Q + (mt * C::DH + half) * C::QHALF + row * 128u +
                                  ((ch ^ (row & 7)) << 4)) = qr[c2];
      }
      fence_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(seg_ready);
    };
    uint4 qr[kChunks];
    uint32_t seg_no = 0;
    Seg s = locate<TK>(t0, t1, p, pb, OVH);
    if (s.ntile > 0 && !p.q_tma) {
      load_q(s, qr);
      store_q(qr);
    }
    while (s.ntile > 0 && ok) {
      const bool has_next = has_more(s, t1, OVH);
      const RowOf ro = row_of(s);
      const int ctx = s.kv_len - p.gamma;
      // tree attention: the block keys this row sees (one bit per block position)
      const unsigned long long tmask =
          TREE ? __ldg(p.tree_mask + static_cast<int64_t>(s.b) * p.gamma + (ro.real ? ro.j : 0)) : 0ull;
      float m = -INFINITY, l = 0.f;
      for (int k = 0; k < s.ntile; ++k) {
        const uint32_t x = it + k;
        ok = mbar_wait(s_full(mt, x & 1), (x >> 1) & 1, abort_flag, p.status);
        if (!ok) break;
        tc_fence_after();
        float v[KH];
        {
          uint32_t r[32];
          const uint32_t col = C::S_COL + (acc * 2 + (x & 1)) * TK + hf * KH;
#pragma unroll
          for (int q = 0; q < KH / 32; ++q) {
            tmem_ld32(lane_base + col + q * 32, r);
            tmem_wait_ld();
#pragma unroll
            for (int c = 0; c < 32; ++c) v[q * 32 + c] = __uint_as_float(r[c]);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0 && !C::PTMEM) mbar_arrive(s_free(mt, x & 1));
        // scale to base 2 and mask keys past ctx + j
        const int key0 = (s.tile0 + k) * TK + hf * KH;
        const int lim = ctx + ro.j - key0;  // keys c <= lim are visible
        float tmax = -INFINITY;
        if (TREE) {
          const int rel0 = key0 - ctx;  // block position of element 0 (negative: the prefix)
#pragma unroll
          for (int c = 0; c < KH; ++c) {
            const int rel = rel0 + c;
            const bool vis = rel < 0 || (rel < 64 && ((tmask >> rel) & 1ull));
            v[c] = vis ? v[c] * p.scale_log2 : -INFINITY;
            tmax = fmaxf(tmax, v[c]);
          }
        } else {
#pragma unroll
          for (int c = 0; c < KH; ++c) {
            v[c] = c <= lim ? v[c] * p.scale_log2 : -INFINITY;
            tmax = fmaxf(tmax, v[c]);
          }
        }
        const float m_new = fmaxf(m, tmax);
        const bool want = k > 0 && m_new > m + 8.f;
        const bool rescale = __any_sync(0xffffffffu, want);
        float alpha = 1.f;
        if (k == 0) {
          m = m_new;
        } else if (rescale) {
          alpha = m == -INFINITY ? 0.f : ex2(m - m_new);
          m = m_new;
        }
        const float msub = m == -INFINITY ? 0.f : m;
        uint32_t pk[KH / 2];
        float sum = 0.f;
#pragma unroll
        for (int c = 0; c < KH / 2; ++c) {
          const float a = ex2(v[2 * c] - msub), b2 = ex2(v[2 * c + 1] - msub);
          sum += a + b2;
          pk[c] = pack_bf16(a, b2);
        }
        l = l * alpha + sum;
        const int pbuf = static_cast<int>(x % PB);
        if (k >= PB) {  // the P V that last read this P buffer is complete
          ok = mbar_wait(pv_done(mt, pbuf), ((x - PB) / PB) & 1, abort_flag, p.status);
          if (!ok) break;
          tc_fence_after();
        }
        if (rescale) {  // k > 0: O must hold every earlier tile before it is scaled
          if (PB > 1) {
            ok = mbar_wait(pv_done(mt, (x - 1) % PB), ((x - 1) / PB) & 1, abort_flag, p.status);
            if (!ok) break;
            tc_fence_after();
          }
#pragma unroll
          for (int cc = 0; cc < D / 32; ++cc) {
            uint32_t r[32];
            tmem_ld32(ocol + cc * 32, r);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
            tmem_st32(ocol + cc * 32, r);
          }
          tmem_wait_st();
        }
        if constexpr (C::PTMEM) {
          // P as bf16 pairs over the first 32 columns of the M tile's (first head's) S
          // buffer of this tile (this row's lane)
          tmem_st32(lane_base + C::S_COL + (mt * HP * 2 + (x & 1)) * TK, pk);
          tmem_wait_st();
        } else {
          unsigned char* prow = smem + C::OFF_P + (pbuf * MT + mt) * C::PBUF + row * 128u;
#pragma unroll
          for (int c2 = 0; c2 < KH / 8; ++c2) {
            const int c = hf * (KH / 8) + c2;
            *reinterpret_cast<uint4*>(prow + ((c ^ (row & 7)) << 4)) =
                make_uint4(pk[4 * c2], pk[4 * c2 + 1], pk[4 * c2 + 2], pk[4 * c2 + 3]);
          }
          fence_async_smem();
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(p_full(mt, pbuf));
      }
      if (!ok) break;
      // The next segment's scores may start now: every Q K^T of this segment is done
      // (its last S was read above), so its Q tile can be replaced while this
      // segment's epilogue runs. Its first P V waits for this epilogue (program order).
      Seg sn;
      sn.ntile = 0;
      if (has_next) {
        sn = locate<TK>(s.vnext, t1, p, pb, OVH);
        if (!p.q_tma) {
          load_q(sn, qr);
          store_q(qr);
        }
      }
      // ---- epilogue: O (TMEM) -> output or partial ----
      const uint32_t xl = it + s.ntile - 1;
      ok = mbar_wait(pv_done(mt, xl % PB), (xl / PB) & 1, abort_flag, p.status);
      if (!ok) break;
      tc_fence_after();
      ok = mbar_wait(flag_bar(seg_no & 7), (seg_no >> 3) & 1, abort_flag, p.status);
      if (!ok) break;
      const bool bad = seg_flag[seg_no & 7] != 0;
      // statistics of the whole tile range: the two key halves merged (identically in
      // both warps of the quadrant)
      float M = m, L = l, sc0 = 1.f, sc1 = 0.f;
      if (SPLIT == 2) {
        float2* xch = reinterpret_cast<float2*>(smem + C::OFF_XCH);
        xch[(q4 * 2 + hf) * 32 + lane] = make_float2(m, l);
        __syncwarp();
        if (lane == 0) mbar_arrive(xch_bar(q4));
        ok = mbar_wait(xch_bar(q4), xphase & 1, abort_flag, p.status);
        ++xphase;
        if (!ok) break;
        const float2 other = xch[(q4 * 2 + (hf ^ 1)) * 32 + lane];
        const float m0 = hf == 0 ? m : other.x, l0 = hf == 0 ? l : other.y;
        const float m1 = hf == 0 ? other.x : m, l1 = hf == 0 ? other.y : l;
        M = fmaxf(m0, m1);
        sc0 = m0 == -INFINITY ? 0.f : ex2(m0 - M);
        sc1 = m1 == -INFINITY ? 0.f : ex2(m1 - M);
        L = l0 * sc0 + l1 * sc1;
      }
      const bool whole = s.tile0 == 0 && s.ntile == s.unit_tiles;
      const int c_first = owner_of(s.unit_start, total, ctas);
      const int c_last = owner_of(s.unit_start + s.unit_tiles - 1, total, ctas);
      const int64_t slot = s.u + cta;
      if (bad && sw == 0 && lane == 0 && (whole || cta == c_first))
        set_status(p.status, s.len_ok ? SPEC_FLAG_BAD_PAGE : SPEC_FLAG_BAD_KV_LEN);
      // this warp writes output columns [hf * D / SPLIT, (hf + 1) * D / SPLIT)
#pragma unroll 1
      for (int cc = hf * (D / 32 / SPLIT); cc < (hf + 1) * (D / 32 / SPLIT); ++cc) {
        uint32_t r[32];
        float o[32];
        tmem_ld32(o0col + cc * 32, r);
        tmem_wait_ld();
#pragma unroll
        for (int e = 0; e < 32; ++e) o[e] = __uint_as_float(r[e]) * sc0;
        if (SPLIT == 2) {
          tmem_ld32(o0col + D + cc * 32, r);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = fmaf(__uint_as_float(r[e]), sc1, o[e]);
        }
        if (!ro.real) continue;
        if (whole) {
          // a bad segment's scores came from stale stages: write exact zeros
          const float inv = bad ? 0.f : 1.f / L;
          if (bad) {
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] = 0.f;
          }
#pragma unroll
          for (int e = 0; e < 32; e += 8) write_out_row<D>(p, s.b, ro.kvh, ro.urow, cc * 32 + e, o + e, inv);
        } else {
          float4* dst = reinterpret_cast<float4*>(p.partial_o + (slot * p.slot_rows + prow) * D + cc * 32);
#pragma unroll
          for (int e = 0; e < 8; ++e)
            dst[e] = make_float4(o[4 * e], o[4 * e + 1], o[4 * e + 2], o[4 * e + 3]);
        }
      }
      tc_fence_before();
      if (ro.real && hf == 0) {
        if (whole) write_lse(p, s.b, ro.kvh, ro.urow, M, L, bad);
        else p.partial_ml[slot * p.slot_rows + prow] = make_float2(M, bad ? -1.f : L);
      }
      if (!whole && sw == 0 && lane == 0) {
        // the ticket of a split unit is taken at the end of the block, after a fence
        int* e = pend + 8 * (*pend_count);
        const int row0 = s.rt * p.rows_per_cta;
        e[0] = s.b; e[1] = s.g; e[2] = row0; e[3] = min(p.rows_per_cta, p.rows - row0);
        e[4] = static_cast<int>(s.u + c_first); e[5] = c_last - c_first + 1;
        e[6] = static_cast<int>(s.u); e[7] = 0;
        *pend_count = *pend_count + 1;
      }
      it += s.ntile;
      s = sn;
      ++seg_no;
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
      uint32_t mphase = 0;
      for (int i = 0; i < np; ++i) {
        const int* e = pend + 8 * i;
        if (!e[7]) continue;
        // Head pairs: the unit's slots are consecutive, and when they fit in the idle K/V
        // stages thread 0 brings them in with two bulk copies (one round trip instead of
        // one per item batch) and every thread merges from shared memory. The (m, l) rows
        // of a slot are 16-byte multiples only for an even slot_rows. (Measured slower in
        // the fused llama8b step for 32-row units, so the one-head kernels keep the
        // global merge.)
        if constexpr (HP == 2) {
          const uint32_t slot_bytes = static_cast<uint32_t>(p.slot_rows) * D * 4;
          const uint32_t ml_bytes = static_cast<uint32_t>(p.slot_rows) * 8;
          const int nsl = e[5];
          if (p.slot_rows % 2 == 0 && static_cast<uint64_t>(nsl) * (slot_bytes + ml_bytes) <= C::RING_BYTES) {
            float* so = reinterpret_cast<float*>(smem + C::OFF_K);
            float2* sml = reinterpret_cast<float2*>(smem + C::OFF_K + nsl * slot_bytes);
            if (threadIdx.x == 0) {
              fence_async_global();  // the partials (generic stores) before the copy engine reads them
              mbar_arrive_tx(merge_bar, nsl * (slot_bytes + ml_bytes));
              bulk_load(smem_u32(so), p.partial_o + static_cast<int64_t>(e[4]) * p.slot_rows * D, nsl * slot_bytes,
                        merge_bar);
              bulk_load(smem_u32(sml), p.partial_ml + static_cast<int64_t>(e[4]) * p.slot_rows, nsl * ml_bytes,
                        merge_bar);
            }
            const bool landed = mbar_wait(merge_bar, mphase & 1, abort_flag, p.status);
            ++mphase;
            if (landed) {
              merge_staged<D>(p, e[0], 2 * e[1], e[2], e[3], so, sml, nsl, 0, threadIdx.x, C::THREADS);
              merge_staged<D>(p, e[0], 2 * e[1] + 1, e[2], e[3], so, sml, nsl, p.rows, threadIdx.x, C::THREADS);
            }
            __syncthreads();  // the staging area is free for the next unit
            continue;
          }
        }
        // units of 128+ rows (a head pair, two M tiles) keep four items per thread in flight
        constexpr int kItems = (HP == 2 || MT == 2) ? 4 : 1;
        if (HP == 2) {  // the pair's heads, the second's rows after the first's in a slot
          merge_unit<D, kItems>(p, e[0], 2 * e[1], e[2], e[3], e[4], e[5], threadIdx.x, C::THREADS, 0);
          merge_unit<D, kItems>(p, e[0], 2 * e[1] + 1, e[2], e[3], e[4], e[5], threadIdx.x, C::THREADS,
                                p.rows);
        } else {
          merge_unit<D, kItems>(p, e[0], e[1], e[2], e[3], e[4], e[5], threadIdx.x, C::THREADS);
        }
      }
    }
  }
}

// ---------------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------------
template <int D, int MT, int QR, int HP>
cudaError_t launch_typed(const spec_attn_args_t& a, const AttnPlan& P, char* ws,
                         cudaStream_t stream, bool starve) {
  using Cf = TcCfg<D, MT, QR, HP>;
  CUtensorMap mk, mv, mq;
  if (!encode_cache_map(&mk, a.k_cache, a, HP) || !encode_cache_map(&mv, a.v_cache, a, HP))
    return cudaErrorInvalidValue;
  AttnParams p = make_attn_params(a, P, ws);
  p.starve = starve ? 1 : 0;
  p.q_tma = encode_q_map(&mq, a, QR) ? 1 : 0;
  // Charge unit starts only when blocks hold several of them; when every unit is spread
  // over several blocks, a block holds at most one start and the charge would mostly
  // move real tiles away from blocks that pay no boundary.
  const int64_t units = static_cast<int64_t>(a.batch) * p.hunits * P.row_tiles;
  p.unit_overhead = units > P.grid ? Cf::UNIT_OVERHEAD : 0;
  if (!p.q_tma) mq = mk;  // unused
  const size_t smem = Cf::smem_bytes(a.batch);
  auto kernel = a.tree_mask ? attn_tc_kernel<D, MT, true, QR, HP> : attn_tc_kernel<D, MT, false, QR, HP>;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  kernel<<<P.grid, Cf::THREADS, smem, stream>>>(mk, mv, mq, p);
  return cudaGetLastError();
}

}  // namespace

// K or V cache viewed as a 5-D tensor of bf16 whose box is one page of one KV head:
// (64 columns; 8 rows at stride D*2 bytes; D/64 column halves at stride 128 bytes;
// page/8 groups of 8 rows at stride 8*D*2 bytes; page * Hkv + head at stride page*D*2).
// The box lands in shared memory as [row group][column half][8 rows][128 B], so the
// 8-row groups of a 64-key tile sit at a uniform stride whatever the page size.
// With heads_per_box = 2 the last two dimensions swap places and the box takes two
// adjacent heads (8 KB contiguous in the cache with 16-token pages, D = 128), landing as
// [row group][head][column half][8 rows][128 B]: the groups of one head keep a uniform
// stride, and the heads sit DH KB apart within a group.
bool encode_cache_map(CUtensorMap* map, const void* base, const spec_attn_args_t& a,
                      int heads_per_box) {
  tcx::EncodeTiledFn enc = tcx::encoder();
  if (!enc) return false;
  const cuuint64_t D = static_cast<cuuint64_t>(a.head_dim);
  const cuuint64_t groups = static_cast<cuuint64_t>(a.page_size / 8);
  const cuuint64_t page_heads = static_cast<cuuint64_t>(a.num_pages) * a.num_kv_heads;
  const cuuint64_t page_stride = static_cast<cuuint64_t>(a.page_size) * D * 2;
  const bool pair = heads_per_box == 2;
  const cuuint64_t dims[5] = {64, 8, D / 64, pair ? page_heads : groups, pair ? groups : page_heads};
  const cuuint64_t strides[4] = {D * 2, 128, pair ? page_stride : 8 * D * 2, pair ? 8 * D * 2 : page_stride};
  const cuuint32_t box[5] = {64, 8, static_cast<cuuint32_t>(D / 64),
                             pair ? 2u : static_cast<cuuint32_t>(groups),
                             pair ? static_cast<cuuint32_t>(groups) : 1u};
  const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Q [batch][gamma][Hq][D] viewed as a 4-D tensor (64 columns; D/64 column halves at
// stride 128 bytes; Hq heads at stride D*2; batch*gamma block positions at stride
// Hq*D*2) whose box is one tile of one column half: the group's heads at
// tile_rows/group consecutive block positions, landing as tile_rows rows of 128 bytes
// (row = j * group + head) with the 128-byte swizzle. Needs group to divide tile_rows;
// positions past the end read zeros and only fill padding rows.
bool encode_q_map(CUtensorMap* map, const spec_attn_args_t& a, int tile_rows) {
  const int group = a.num_q_heads / a.num_kv_heads;
  if (group < 1 || tile_rows % group != 0) return false;
  tcx::EncodeTiledFn enc = tcx::encoder();
  if (!enc) return false;
  const cuuint64_t D = static_cast<cuuint64_t>(a.head_dim);
  const cuuint64_t dims[4] = {64, D / 64, static_cast<cuuint64_t>(a.num_q_heads),
                              static_cast<cuuint64_t>(a.batch) * a.gamma};
  const cuuint64_t strides[3] = {128, D * 2, static_cast<cuuint64_t>(a.num_q_heads) * D * 2};
  const cuuint32_t box[4] = {64, 1, static_cast<cuuint32_t>(group),
                             static_cast<cuuint32_t>(tile_rows / group)};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(a.q), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The buffer configuration of the row-tile kernel: two M tiles, one M tile with 128-row
// buffers, one M tile with 64-row buffers (at most 64 query rows per KV group), or one M
// tile of two KV heads' 64-row groups.
enum TcVariant { kTwoTiles, kOneTile, kOneTileHalf, kHeadPair };
TcVariant tc_variant(int rows_per_cta, int rows, bool head_pair) {
  return head_pair ? kHeadPair : rows_per_cta > 128 ? kTwoTiles : (rows <= 64 ? kOneTileHalf : kOneTile);
}

template <int D>
size_t smem_of(TcVariant v, int batch) {
  return v == kTwoTiles     ? TcCfg<D, 2>::smem_bytes(batch)
         : v == kOneTile    ? TcCfg<D, 1>::smem_bytes(batch)
         : v == kOneTileHalf ? TcCfg<D, 1, 64>::smem_bytes(batch)
                             : TcCfg<D, 1, 64, 2>::smem_bytes(batch);
}

size_t tc_smem_bytes(int head_dim, int rows_per_cta, int rows, int batch, bool head_pair) {
  const TcVariant v = tc_variant(rows_per_cta, rows, head_pair);
  return head_dim == 128 ? smem_of<128>(v, batch) : smem_of<64>(v, batch);
}

// With at most 32 rows per group a pair would leave two lane quadrants idle and give each
// softmax warp a whole tile's keys where the one-head kernel splits them over two warps
// (measured slower at 32 rows: llama8b attention 50.7 against 48.1 us).
bool tc_head_pair(int head_dim, int rows, int num_kv_heads, int batch) {
  return rows > 32 && rows <= 64 && num_kv_heads % 2 == 0 &&
         tc_smem_bytes(head_dim, 128, rows, batch, true) <= kTcMaxSmem;
}

int tc_ctas_per_sm(int head_dim, int rows_per_cta, int rows, int batch, bool head_pair) {
  // Shared memory bounds residency (227 KB usable per SM); TMEM (512 columns) too.
  const size_t smem = tc_smem_bytes(head_dim, rows_per_cta, rows, batch, head_pair);
  int by_smem = static_cast<int>(kTcMaxSmem / (smem + 1024));
  const TcVariant v = tc_variant(rows_per_cta, rows, head_pair);
  const uint32_t cols =
      head_dim == 128
          ? (v == kTwoTiles ? TcCfg<128, 2>::TMEM_COLS
             : v == kHeadPair ? TcCfg<128, 1, 64, 2>::TMEM_COLS : TcCfg<128, 1>::TMEM_COLS)
          : (v == kTwoTiles ? TcCfg<64, 2>::TMEM_COLS
             : v == kHeadPair ? TcCfg<64, 1, 64, 2>::TMEM_COLS : TcCfg<64, 1>::TMEM_COLS);
  const int by_tmem = static_cast<int>(512 / cols);
  int n = by_smem < by_tmem ? by_smem : by_tmem;
  return n < 1 ? 1 : n;
}

template <int D>
cudaError_t launch_d(TcVariant v, const spec_attn_args_t& a, const AttnPlan& P, char* ws,
                     cudaStream_t stream, bool starve) {
  return v == kTwoTiles     ? launch_typed<D, 2, 128, 1>(a, P, ws, stream, starve)
         : v == kOneTile    ? launch_typed<D, 1, 128, 1>(a, P, ws, stream, starve)
         : v == kOneTileHalf ? launch_typed<D, 1, 64, 1>(a, P, ws, stream, starve)
                             : launch_typed<D, 1, 64, 2>(a, P, ws, stream, starve);
}

cudaError_t launch_attn_tc(const spec_attn_args_t& a, const AttnPlan& P, char* ws,
                           cudaStream_t stream, bool starve) {
  const TcVariant v = tc_variant(P.rows_per_cta, P.rows, P.head_pair != 0);
  return a.head_dim == 128 ? launch_d<128>(v, a, P, ws, stream, starve)
                           : launch_d<64>(v, a, P, ws, stream, starve);
}

}  // namespace specv
