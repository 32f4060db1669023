// The C ABI of libspecverify (include/spec_verify.h): host-side argument checks,
// workspace layout, kernel selection and launches. No entry point allocates device
// memory; all state lives in the caller's workspace.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <climits>
#include <cstring>

#include "common.cuh"
#include "lm_head.cuh"

namespace specv {

namespace {
constexpr int kSmCacheDevices = 64;
std::atomic<int> g_sms[kSmCacheDevices];  // cached multiprocessor counts (0 = unknown)
}  // namespace

int device_sm_count(int dev) {
  if (dev < 0 || dev >= kSmCacheDevices) return 148;
  int n = g_sms[dev].load(std::memory_order_relaxed);
  if (n > 0) return n;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) {
    (void)cudaGetLastError();
    n = 148;
  }
  g_sms[dev].store(n, std::memory_order_relaxed);
  return n;
}

// (Hq/Hkv) * gamma at and above which SPEC_ATTN_AUTO picks the tensor-core kernel.
// Measured on GB300: the tensor-core kernel is never slower, from 4 rows per kv head
// (equal time, both latency-bound) to 32 (6x faster: the CUDA-core kernel re-reads
// each KV tile once per 16-row tile and issues the dot products on the FMA pipes), so
// AUTO takes it whenever its shape limits allow.
constexpr int kTcMinRows = 1;
int tc_min_rows() { return kTcMinRows; }

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// The fused step's second stream: one per (host thread, device, caller stream), with a
// fork and a join event, made on first use. Keyed on the caller's stream so that two
// steps issued on two different streams never queue behind each other on a shared side
// stream; per thread, so that calls from different threads never record the same
// event. A call's fork and join also work under stream capture (the side stream joins
// the capture through the fork event). A thread keeps at most kSideCacheSize of them;
// the least recently used one that is not capturing is released to make room (a
// stream or event released with work pending is freed once that work completes).
struct SideStream {
  int dev = -1;
  cudaStream_t caller = nullptr;
  cudaStream_t stream = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
  uint64_t last_use = 0;
};
constexpr int kSideCacheSize = 16;

void release_side(SideStream& ss) {
  if (ss.fork) cudaEventDestroy(ss.fork);
  if (ss.join) cudaEventDestroy(ss.join);
  if (ss.stream) cudaStreamDestroy(ss.stream);
  ss = SideStream();
}

SideStream* side_stream(int dev, cudaStream_t caller) {
  thread_local SideStream cache[kSideCacheSize];
  thread_local uint64_t clock = 0;
  ++clock;
  SideStream* victim = nullptr;
  for (SideStream& ss : cache) {
    if (ss.stream && ss.dev == dev && ss.caller == caller) {
      ss.last_use = clock;
      return &ss;
    }
  }
  for (SideStream& ss : cache) {
    if (!ss.stream) {
      victim = &ss;
      break;
    }
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(ss.stream, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone)
      continue;
    if (!victim || ss.last_use < victim->last_use) victim = &ss;
  }
  if (!victim) return nullptr;
  if (victim->stream) release_side(*victim);
  cudaStream_t st = nullptr;
  cudaEvent_t f = nullptr, j = nullptr;
  if (cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking) != cudaSuccess) return nullptr;
  if (cudaEventCreateWithFlags(&f, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&j, cudaEventDisableTiming) != cudaSuccess) {
    if (f) cudaEventDestroy(f);
    cudaStreamDestroy(st);
    return nullptr;
  }
  victim->dev = dev;
  victim->caller = caller;
  victim->stream = st;
  victim->fork = f;
  victim->join = j;
  victim->last_use = clock;
  return victim;
}

spec_status_t check_attn(const spec_attn_args_t* a) {
  if (!a) return SPEC_ERR_INVALID_ARGUMENT;
  if (a->batch < 1 || a->gamma < 1 || a->num_q_heads < 1 || a->num_kv_heads < 1 ||
      a->max_pages_per_seq < 1 || a->num_pages < 1 || a->page_size < 1 || a->head_dim < 1)
    return SPEC_ERR_INVALID_ARGUMENT;
  if (a->num_q_heads % a->num_kv_heads != 0) return SPEC_ERR_INVALID_ARGUMENT;
  if (!a->q || !a->k_cache || !a->v_cache || !a->page_table || !a->kv_len || !a->out)
    return SPEC_ERR_INVALID_ARGUMENT;
  if (!aligned16(a->q) || !aligned16(a->k_cache) || !aligned16(a->v_cache) || !aligned16(a->out))
    return SPEC_ERR_INVALID_ARGUMENT;
  if (!(a->softmax_scale == 0.f || (a->softmax_scale > 0.f && a->softmax_scale < 1e30f)))
    return SPEC_ERR_INVALID_ARGUMENT;
  if (a->path < SPEC_ATTN_AUTO || a->path > SPEC_ATTN_TENSOR_CORES_KEYS_ON_LANES)
    return SPEC_ERR_INVALID_ARGUMENT;
  if ((a->path == SPEC_ATTN_TENSOR_CORES || a->path == SPEC_ATTN_TENSOR_CORES_KEYS_ON_LANES) &&
      a->batch > kTcMaxBatch)
    return SPEC_ERR_UNSUPPORTED;
  if (a->gamma > 64) return SPEC_ERR_UNSUPPORTED;
  if (a->head_dim != 64 && a->head_dim != 128) return SPEC_ERR_UNSUPPORTED;
  if (a->page_size != 16 && a->page_size != 32 && a->page_size != 64) return SPEC_ERR_UNSUPPORTED;
  const int64_t max_keys = static_cast<int64_t>(a->max_pages_per_seq) * a->page_size;
  if (max_keys > (1 << 30)) return SPEC_ERR_UNSUPPORTED;
  const int64_t rows = static_cast<int64_t>(a->num_q_heads / a->num_kv_heads) * a->gamma;
  const int64_t z = static_cast<int64_t>(a->batch) * ((rows + kSimtRowTile - 1) / kSimtRowTile);
  if (z > 65535 || a->num_kv_heads > 65535) return SPEC_ERR_UNSUPPORTED;
  if (static_cast<int64_t>(a->num_pages) * a->num_kv_heads * a->page_size > INT32_MAX)
    return SPEC_ERR_UNSUPPORTED;
  return SPEC_OK;
}

spec_status_t check_draft(const spec_draft_args_t* d) {
  if (!d) return SPEC_ERR_INVALID_ARGUMENT;
  if (d->batch < 1 || d->gamma < 1 || d->vocab < 1) return SPEC_ERR_INVALID_ARGUMENT;
  if (d->logits_dtype != SPEC_F32 && d->logits_dtype != SPEC_BF16) return SPEC_ERR_INVALID_ARGUMENT;
  if (!d->drafter_logits || !d->temperature || !d->uniforms || !d->block_tokens)
    return SPEC_ERR_INVALID_ARGUMENT;
  if (d->gamma > 64 || d->batch > 65535) return SPEC_ERR_UNSUPPORTED;
  return SPEC_OK;
}

// The acceptance arguments the filtered row kernel reads in its draw mode.
spec_accept_args_t draft_as_accept(const spec_draft_args_t& d) {
  spec_accept_args_t a = {};
  a.batch = d.batch;
  a.gamma = d.gamma;
  a.vocab = d.vocab;
  a.logits_dtype = d.logits_dtype;
  a.target_logits = d.drafter_logits;
  a.drafter_logits = d.drafter_logits;
  a.temperature = d.temperature;
  a.uniforms = d.uniforms;
  return a;
}

constexpr size_t kDraftMaxSmem = 200 * 1024;  // lane summaries of one unfiltered draw block

size_t draft_bytes(const spec_draft_args_t& d, const spec_filter_args_t* f, int sms, bool vec) {
  if (f) return filter_layout(draft_as_accept(d), f->max_top_k, kWsHeader, sms, true).end;
  return draft_layout(d, kWsHeader, sms, vec).end;
}

spec_status_t check_tree(const spec_tree_accept_args_t* t) {
  if (!t) return SPEC_ERR_INVALID_ARGUMENT;
  if (t->batch < 1 || t->num_nodes < 1 || t->vocab < 1) return SPEC_ERR_INVALID_ARGUMENT;
  if (t->logits_dtype != SPEC_F32 && t->logits_dtype != SPEC_BF16) return SPEC_ERR_INVALID_ARGUMENT;
  if (!t->target_logits || !t->tokens || !t->parents || !t->path || !t->num_accepted ||
      !t->out_tokens || !t->num_emitted)
    return SPEC_ERR_INVALID_ARGUMENT;
  if (t->num_nodes > 64 || t->batch > 65535) return SPEC_ERR_UNSUPPORTED;
  if (t->temperature && !t->uniforms) return SPEC_ERR_INVALID_ARGUMENT;
  return SPEC_OK;
}

// Nodes the positions can hold: sum over d = 1 .. gamma-1 of min(top_k, vocab)^d, saturated.
int64_t tree_capacity(const spec_tree_build_args_t* t) {
  const int64_t k = std::min(t->top_k, t->vocab);
  int64_t total = 0, level = 1;
  for (int d = 1; d < t->gamma && total < 64; ++d) {
    level = std::min<int64_t>(level * k, 64);
    total += level;
  }
  return total;
}

spec_status_t check_tree_build(const spec_tree_build_args_t* t) {
  if (!t) return SPEC_ERR_INVALID_ARGUMENT;
  if (t->batch < 1 || t->gamma < 1 || t->vocab < 1 || t->top_k < 1 || t->num_nodes < 1)
    return SPEC_ERR_INVALID_ARGUMENT;
  if (t->logits_dtype != SPEC_F32 && t->logits_dtype != SPEC_BF16) return SPEC_ERR_INVALID_ARGUMENT;
  if (!t->drafter_logits || !t->temperature || !t->root_tokens || !t->tokens || !t->parents)
    return SPEC_ERR_INVALID_ARGUMENT;
  if (t->num_nodes > 64 || t->batch > 65535) return SPEC_ERR_UNSUPPORTED;
  if (tree_capacity(t) < t->num_nodes - 1) return SPEC_ERR_INVALID_ARGUMENT;
  return SPEC_OK;
}

spec_status_t check_lm_head(const spec_lm_head_args_t* a) {
  if (!a) return SPEC_ERR_INVALID_ARGUMENT;
  if (a->rows < 1 || a->hidden < 8 || a->hidden % 8 != 0 || a->vocab < 1 || a->rows_per_seq < 1)
    return SPEC_ERR_INVALID_ARGUMENT;
  if (!a->hidden_states || !a->weight || !a->temperature || !a->row_max || !a->row_sum ||
      !a->row_argmax)
    return SPEC_ERR_INVALID_ARGUMENT;
  if ((reinterpret_cast<uintptr_t>(a->hidden_states) | reinterpret_cast<uintptr_t>(a->weight)) & 15u)
    return SPEC_ERR_INVALID_ARGUMENT;
  if ((a->vocab + kLmTileN - 1) / kLmTileN > 65535) return SPEC_ERR_UNSUPPORTED;  // grid y
  return SPEC_OK;
}

spec_status_t check_filter(const spec_filter_args_t* f) {
  if (!f || !f->top_k || !f->top_p) return SPEC_ERR_INVALID_ARGUMENT;
  if (f->max_top_k < 1) return SPEC_ERR_INVALID_ARGUMENT;
  if (f->max_top_k > SPEC_FILTER_MAX_TOP_K) return SPEC_ERR_UNSUPPORTED;
  return SPEC_OK;
}

}  // namespace

// Also the host check of spec_accept_block_noalloc (accept_noalloc.cu).
spec_status_t check_accept(const spec_accept_args_t* a) {
  if (!a) return SPEC_ERR_INVALID_ARGUMENT;
  if (a->batch < 1 || a->gamma < 1 || a->vocab < 1) return SPEC_ERR_INVALID_ARGUMENT;
  if (a->logits_dtype != SPEC_F32 && a->logits_dtype != SPEC_BF16) return SPEC_ERR_INVALID_ARGUMENT;
  if (!a->target_logits || !a->drafter_logits || !a->block_tokens || !a->temperature ||
      !a->uniforms || !a->num_accepted || !a->out_tokens || !a->num_emitted)
    return SPEC_ERR_INVALID_ARGUMENT;
  if (a->gamma > 64 || a->batch > 65535) return SPEC_ERR_UNSUPPORTED;
  const int64_t nchunk = (static_cast<int64_t>(a->vocab) + kStatsChunk - 1) / kStatsChunk;
  if (static_cast<int64_t>(a->batch) * (2 * a->gamma - 1) * nchunk > INT32_MAX)
    return SPEC_ERR_UNSUPPORTED;
  const int64_t nslice = (static_cast<int64_t>(a->vocab) + kSampleSlice - 1) / kSampleSlice;
  if (nslice > 65535) return SPEC_ERR_UNSUPPORTED;
  return SPEC_OK;
}

AttnPlan attn_plan(const spec_attn_args_t& a, size_t base, int num_sms, int path_override) {
  AttnPlan P;
  P.head_pair = 0;
  P.rows = (a.num_q_heads / a.num_kv_heads) * a.gamma;
  int path = path_override;
  if (path == SPEC_ATTN_AUTO)
    path = (P.rows >= tc_min_rows() && a.batch <= kTcMaxBatch) ? SPEC_ATTN_TENSOR_CORES
                                                               : SPEC_ATTN_CUDA_CORES;
  // the keys-on-lanes kernel, when asked for, takes the KV groups of at most 64 query rows
  const int group = a.num_q_heads / a.num_kv_heads;
  P.keys_on_lanes = path == SPEC_ATTN_TENSOR_CORES_KEYS_ON_LANES && a.head_dim == 128 &&
                    P.rows <= kKlMaxRows && kKlMaxRows % group == 0 && a.batch <= kKlMaxBatch &&
                    !a.tree_mask;
  if (path == SPEC_ATTN_TENSOR_CORES_KEYS_ON_LANES) path = SPEC_ATTN_TENSOR_CORES;
  P.path = path;
  P.max_keys = a.max_pages_per_seq * a.page_size;
  int64_t units;
  if (path == SPEC_ATTN_CUDA_CORES) {
    // static split grid (splits, Hkv, batch * row tiles), two blocks per SM
    P.rows_per_cta = kSimtRowTile;
    P.key_tile = kSimtKeyTile;
    P.row_tiles = (P.rows + P.rows_per_cta - 1) / P.rows_per_cta;
    const int max_tiles = (P.max_keys + P.key_tile - 1) / P.key_tile;
    units = static_cast<int64_t>(a.batch) * a.num_kv_heads * P.row_tiles;
    int64_t nsplit = static_cast<int64_t>(num_sms) * 2 / units;
    if (nsplit < 1) nsplit = 1;
    if (nsplit > max_tiles) nsplit = max_tiles;
    P.tiles_per_split = static_cast<int>((max_tiles + nsplit - 1) / nsplit);
    P.nsplit = (max_tiles + P.tiles_per_split - 1) / P.tiles_per_split;
    P.grid = 0;
    P.slot_rows = P.rows_per_cta;
    P.slots = P.nsplit > 1 ? units * P.nsplit : 0;
  } else if (P.keys_on_lanes) {
    // persistent grid, one block per SM; one unit per (sequence, KV head)
    P.rows_per_cta = kKlMaxRows;
    P.key_tile = kKlKeyTile;
    P.row_tiles = 1;
    units = static_cast<int64_t>(a.batch) * a.num_kv_heads;
    P.nsplit = 1;
    P.tiles_per_split = 0;
    P.grid = num_sms;
    P.slot_rows = P.rows;
    P.slots = units + P.grid;
  } else {
    // persistent grid; the tile list of all units is cut into equal ranges
    P.rows_per_cta = P.rows <= 128 ? 128 : kTcMaxRows;
    P.key_tile = kTcKeyTile;
    P.row_tiles = (P.rows + P.rows_per_cta - 1) / P.rows_per_cta;
    P.head_pair = tc_head_pair(a.head_dim, P.rows, a.num_kv_heads, a.batch) ? 1 : 0;
    units = static_cast<int64_t>(a.batch) * (a.num_kv_heads / (1 + P.head_pair)) * P.row_tiles;
    P.nsplit = 1;
    P.tiles_per_split = 0;
    P.grid = num_sms * tc_ctas_per_sm(a.head_dim, P.rows_per_cta, P.rows, a.batch, P.head_pair != 0);
    // a slot keeps a unit's rows (a head pair's second head after its first)
    P.slot_rows = (P.rows < P.rows_per_cta ? P.rows : P.rows_per_cta) * (1 + P.head_pair);
    P.slots = units + P.grid;
  }
  P.tickets = base;
  P.partial_o = ws_round(P.tickets + sizeof(uint32_t) * units);
  P.partial_ml =
      ws_round(P.partial_o + static_cast<size_t>(P.slots) * P.slot_rows * a.head_dim * 4);
  P.end = ws_round(P.partial_ml + static_cast<size_t>(P.slots) * P.slot_rows * sizeof(float2));
  return P;
}

}  // namespace specv

using namespace specv;

namespace {

size_t attn_region(const spec_attn_args_t& a, size_t base, int sms) {
  size_t end = base;
  for (int path : {SPEC_ATTN_CUDA_CORES, SPEC_ATTN_TENSOR_CORES, SPEC_ATTN_TENSOR_CORES_KEYS_ON_LANES}) {
    if (path != SPEC_ATTN_CUDA_CORES && a.batch > kTcMaxBatch) continue;
    const AttnPlan P = attn_plan(a, base, sms, path);
    if (P.end > end) end = P.end;
  }
  return end;
}

size_t required_bytes(const spec_attn_args_t* attn, const spec_accept_args_t* accept,
                      const spec_filter_args_t* filter, int sms, size_t* attn_base) {
  size_t end = kWsHeader;
  if (accept)
    end = filter ? filter_layout(*accept, filter->max_top_k, kWsHeader, sms).end
                 : accept_layout(*accept, kWsHeader).end;
  if (attn_base) *attn_base = end;
  if (attn) end = attn_region(*attn, end, sms);
  return end;
}

spec_status_t run(const spec_attn_args_t* attn, const spec_accept_args_t* accept,
                  const spec_filter_args_t* filter, void* ws, size_t ws_bytes,
                  spec_stream_t stream_) {
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  if (!attn && !accept) return SPEC_ERR_INVALID_ARGUMENT;
  if (filter) {
    const spec_status_t s = check_filter(filter);
    if (s != SPEC_OK) return s;
  }
  if (attn) {
    const spec_status_t s = check_attn(attn);
    if (s != SPEC_OK) return s;
  }
  if (accept) {
    const spec_status_t s = check_accept(accept);
    if (s != SPEC_OK) return s;
  }
  if (!ws || (reinterpret_cast<uintptr_t>(ws) % kWsAlign) != 0) return SPEC_ERR_INVALID_ARGUMENT;
  // without attention the size does not depend on the device: check it on the host
  if (!attn && required_bytes(nullptr, accept, filter, 0, nullptr) > ws_bytes)
    return SPEC_ERR_WORKSPACE_TOO_SMALL;
  DeviceScope scope(stream);
  if (!scope.ok) return SPEC_ERR_CUDA;
  const int sms = scope.sms;
  (void)cudaGetLastError();  // a failed call before this one must not fail our launches
  size_t attn_base = 0;
  if (required_bytes(attn, accept, filter, sms, &attn_base) > ws_bytes)
    return SPEC_ERR_WORKSPACE_TOO_SMALL;
  char* w = static_cast<char*>(ws);
  // A whole step forks: the acceptance kernels run on a side stream (this thread's, for
  // this caller stream) beside the attention kernel (they share no data: the logits are
  // inputs), on the SM resources it leaves free, and the caller's stream waits for both.
  // On one stream the decisions, which wait for their inputs with griddepcontrol.wait,
  // would also wait for the attention kernel before them.
  cudaStream_t acc_stream = stream;
  SideStream* side = nullptr;
  if (attn && accept) {
    // Without a side stream (it could not be created) both parts run on `stream`, in
    // order: the same results, without the overlap.
    side = side_stream(scope.dev, stream);
    if (!side) (void)cudaGetLastError();
  }
  if (side) {
    if (cudaEventRecord(side->fork, stream) != cudaSuccess ||
        cudaStreamWaitEvent(side->stream, side->fork, 0) != cudaSuccess)
      return SPEC_ERR_CUDA;
    acc_stream = side->stream;
  }
  // Order of the two launches: the acceptance first when its logits are a sizeable
  // share of the step's bytes (at least a sixth of the most KV the attention can read):
  // its statistics then stream on the whole GPU before the attention blocks take it,
  // and the decisions and draws run beside the attention. Otherwise the attention first
  // (its start would wait for a comparatively short statistics pass).
  bool accept_first = false;
  if (side) {
    const size_t esz = accept->logits_dtype == SPEC_BF16 ? 2 : 4;
    const double logits = static_cast<double>(accept->batch) * (2.0 * accept->gamma - 1) *
                          accept->vocab * static_cast<double>(esz);
    const double kv = static_cast<double>(attn->batch) * attn->max_pages_per_seq * attn->page_size *
                      attn->num_kv_heads * attn->head_dim * 4.0;
    accept_first = 6.0 * logits >= kv;
  }
  auto launch_attention = [&]() -> bool {
    if (!attn) return true;
    const AttnPlan P = attn_plan(*attn, attn_base, sms, attn->path);
    const cudaError_t e = P.path != SPEC_ATTN_TENSOR_CORES ? launch_attn_simt(*attn, P, w, stream)
                          : P.keys_on_lanes                 ? launch_attn_kl(*attn, P, w, stream)
                                                            : launch_attn_tc(*attn, P, w, stream);
    return e == cudaSuccess;
  };
  auto launch_acceptance = [&]() -> bool {
    if (accept && filter) {
      const FilterLayout L = filter_layout(*accept, filter->max_top_k, kWsHeader, sms);
      return launch_accept_filtered(*accept, *filter, L, w, acc_stream, false) == cudaSuccess;
    }
    if (accept) {
      const AcceptLayout L = accept_layout(*accept, kWsHeader);
      return launch_accept(*accept, L, w, sms, acc_stream, false) == cudaSuccess;
    }
    return true;
  };
  if (accept_first) {
    if (!launch_acceptance() || !launch_attention()) return SPEC_ERR_CUDA;
  } else {
    if (!launch_attention() || !launch_acceptance()) return SPEC_ERR_CUDA;
  }
  if (side && (cudaEventRecord(side->join, side->stream) != cudaSuccess ||
               cudaStreamWaitEvent(stream, side->join, 0) != cudaSuccess))
    return SPEC_ERR_CUDA;
  return SPEC_OK;
}

size_t workspace_bytes(const spec_attn_args_t* attn, const spec_accept_args_t* accept,
                       const spec_filter_args_t* filter) {
  if (attn && check_attn(attn) != SPEC_OK) return 0;
  if (accept && check_accept(accept) != SPEC_OK) return 0;
  if (filter && (!accept || check_filter(filter) != SPEC_OK)) return 0;
  // The split count depends on the SM count; size for the larger of the current
  // device's and a 160-SM part so that a workspace fits every device it may meet.
  int dev = 0, sms = 160;
  if (cudaGetDevice(&dev) == cudaSuccess) {
    const int n = device_sm_count(dev);
    if (n > sms) sms = n;
  } else {
    cudaGetLastError();
  }
  size_t need = required_bytes(attn, accept, filter, sms, nullptr);
  for (int s : {148, 152, sms}) {
    const size_t x = required_bytes(attn, accept, filter, s, nullptr);
    if (x > need) need = x;
  }
  return need;
}

}  // namespace

extern "C" {

size_t spec_workspace_size(const spec_attn_args_t* attn, const spec_accept_args_t* accept) {
  return workspace_bytes(attn, accept, nullptr);
}

spec_status_t spec_workspace_init(void* ws, size_t ws_bytes, spec_stream_t stream) {
  if (!ws) return SPEC_ERR_INVALID_ARGUMENT;
  return cudaMemsetAsync(ws, 0, ws_bytes, reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
             ? SPEC_OK
             : SPEC_ERR_CUDA;
}

spec_status_t spec_verify_attention(const spec_attn_args_t* attn, void* ws, size_t ws_bytes,
                                    spec_stream_t stream) {
  if (!attn) return SPEC_ERR_INVALID_ARGUMENT;
  return run(attn, nullptr, nullptr, ws, ws_bytes, stream);
}

spec_status_t spec_accept_block(const spec_accept_args_t* accept, void* ws, size_t ws_bytes,
                                spec_stream_t stream) {
  if (!accept) return SPEC_ERR_INVALID_ARGUMENT;
  return run(nullptr, accept, nullptr, ws, ws_bytes, stream);
}

spec_status_t spec_test_attention_wait_timeout(const spec_attn_args_t* attn, void* ws,
                                               size_t ws_bytes, spec_stream_t stream_) {
  if (!attn) return SPEC_ERR_INVALID_ARGUMENT;
  const spec_status_t st = check_attn(attn);
  if (st != SPEC_OK) return st;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) % kWsAlign) != 0) return SPEC_ERR_INVALID_ARGUMENT;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  DeviceScope scope(stream);
  if (!scope.ok) return SPEC_ERR_CUDA;
  (void)cudaGetLastError();
  size_t attn_base = 0;
  if (required_bytes(attn, nullptr, nullptr, scope.sms, &attn_base) > ws_bytes)
    return SPEC_ERR_WORKSPACE_TOO_SMALL;
  const AttnPlan P = attn_plan(*attn, attn_base, scope.sms, SPEC_ATTN_TENSOR_CORES);
  if (P.path != SPEC_ATTN_TENSOR_CORES || P.keys_on_lanes) return SPEC_ERR_UNSUPPORTED;
  return launch_attn_tc(*attn, P, static_cast<char*>(ws), stream, /*starve=*/true) == cudaSuccess
             ? SPEC_OK
             : SPEC_ERR_CUDA;
}

spec_status_t spec_verify_step(const spec_attn_args_t* attn, const spec_accept_args_t* accept,
                               void* ws, size_t ws_bytes, spec_stream_t stream) {
  return run(attn, accept, nullptr, ws, ws_bytes, stream);
}

size_t spec_filtered_workspace_size(const spec_attn_args_t* attn, const spec_accept_args_t* accept,
                                    const spec_filter_args_t* filter) {
  if (!accept || !filter) return 0;
  return workspace_bytes(attn, accept, filter);
}

spec_status_t spec_accept_block_filtered(const spec_accept_args_t* accept,
                                         const spec_filter_args_t* filter, void* ws,
                                         size_t ws_bytes, spec_stream_t stream) {
  if (!accept || !filter) return SPEC_ERR_INVALID_ARGUMENT;
  return run(nullptr, accept, filter, ws, ws_bytes, stream);
}

spec_status_t spec_verify_step_filtered(const spec_attn_args_t* attn,
                                        const spec_accept_args_t* accept,
                                        const spec_filter_args_t* filter, void* ws,
                                        size_t ws_bytes, spec_stream_t stream) {
  if (!accept || !filter) return SPEC_ERR_INVALID_ARGUMENT;
  return run(attn, accept, filter, ws, ws_bytes, stream);
}

spec_status_t spec_noise_tokens(uint64_t seed, uint64_t offset, int64_t n, int32_t vocab,
                                int32_t* out_dev, spec_stream_t stream) {
  if (n < 0 || vocab < 1 || (n > 0 && !out_dev)) return SPEC_ERR_INVALID_ARGUMENT;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  DeviceScope scope(s);
  if (!scope.ok) return SPEC_ERR_CUDA;
  return launch_noise(seed, offset, n, vocab, out_dev, s) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

size_t spec_draft_workspace_size(const spec_draft_args_t* draft, const spec_filter_args_t* filter) {
  if (check_draft(draft) != SPEC_OK || (filter && check_filter(filter) != SPEC_OK)) return 0;
  int dev = 0, sms = 160;
  if (cudaGetDevice(&dev) == cudaSuccess) {
    const int n = device_sm_count(dev);
    if (n > sms) sms = n;
  } else {
    cudaGetLastError();
  }
  size_t need = 0;
  for (int s : {148, 152, sms})
    for (bool vec : {false, true}) {
      const size_t x = draft_bytes(*draft, filter, s, vec);
      if (x > need) need = x;
    }
  return need;
}

spec_status_t spec_sample_block(const spec_draft_args_t* draft, const spec_filter_args_t* filter,
                                void* ws, size_t ws_bytes, spec_stream_t stream_) {
  spec_status_t st = check_draft(draft);
  if (st != SPEC_OK) return st;
  if (filter && (st = check_filter(filter)) != SPEC_OK) return st;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) % kWsAlign) != 0) return SPEC_ERR_INVALID_ARGUMENT;
  const size_t esz = draft->logits_dtype == SPEC_BF16 ? 2 : 4;
  const bool vec = (static_cast<size_t>(draft->vocab) * esz) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(draft->drafter_logits) % 16 == 0;
  if (!filter && draft_layout(*draft, kWsHeader, 1, vec).smem > kDraftMaxSmem) return SPEC_ERR_UNSUPPORTED;
  if (draft_bytes(*draft, filter, 1, vec) > ws_bytes) return SPEC_ERR_WORKSPACE_TOO_SMALL;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  DeviceScope scope(stream);
  if (!scope.ok) return SPEC_ERR_CUDA;
  const int sms = scope.sms;
  (void)cudaGetLastError();
  if (draft_bytes(*draft, filter, sms, vec) > ws_bytes) return SPEC_ERR_WORKSPACE_TOO_SMALL;
  char* w = static_cast<char*>(ws);
  if (filter) {
    const spec_accept_args_t a = draft_as_accept(*draft);
    const FilterLayout L = filter_layout(a, filter->max_top_k, kWsHeader, sms, true);
    return launch_accept_filtered(a, *filter, L, w, stream, false, draft->block_tokens,
                                  draft->q_tok) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
  }
  const DraftLayout L = draft_layout(*draft, kWsHeader, sms, vec);
  return launch_draft(*draft, L, w, stream, vec) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

size_t spec_tree_workspace_size(const spec_tree_accept_args_t* t) {
  if (check_tree(t) != SPEC_OK) return 0;
  int dev = 0, sms = 160;
  if (cudaGetDevice(&dev) == cudaSuccess) {
    const int n = device_sm_count(dev);
    if (n > sms) sms = n;
  } else {
    cudaGetLastError();
  }
  size_t need = 0;
  for (int s : {148, 152, sms})
    for (bool vec : {false, true}) {
      const size_t x = tree_layout(t->batch, t->num_nodes, t->vocab, kWsHeader, s, vec).end;
      if (x > need) need = x;
    }
  return need;
}

spec_status_t spec_accept_tree(const spec_tree_accept_args_t* t, void* ws, size_t ws_bytes,
                               spec_stream_t stream_) {
  const spec_status_t st = check_tree(t);
  if (st != SPEC_OK) return st;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) % kWsAlign) != 0) return SPEC_ERR_INVALID_ARGUMENT;
  const size_t esz = t->logits_dtype == SPEC_BF16 ? 2 : 4;
  const bool vec = (static_cast<size_t>(t->vocab) * esz) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(t->target_logits) % 16 == 0;
  if (tree_layout(t->batch, t->num_nodes, t->vocab, kWsHeader, 1, vec).end > ws_bytes)
    return SPEC_ERR_WORKSPACE_TOO_SMALL;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  DeviceScope scope(stream);
  if (!scope.ok) return SPEC_ERR_CUDA;
  const int sms = scope.sms;
  const TreeLayout L = tree_layout(t->batch, t->num_nodes, t->vocab, kWsHeader, sms, vec);
  if (L.end > ws_bytes) return SPEC_ERR_WORKSPACE_TOO_SMALL;
  return launch_tree_greedy(*t, L, static_cast<char*>(ws), stream, vec) == cudaSuccess
             ? SPEC_OK
             : SPEC_ERR_CUDA;
}

size_t spec_tree_build_workspace_size(const spec_tree_build_args_t* t) {
  if (check_tree_build(t) != SPEC_OK) return 0;
  int dev = 0, sms = 160;
  if (cudaGetDevice(&dev) == cudaSuccess) {
    const int n = device_sm_count(dev);
    if (n > sms) sms = n;
  } else {
    cudaGetLastError();
  }
  size_t need = 0;
  for (int s : {148, 152, sms}) need = std::max(need, tree_build_layout(*t, kWsHeader, s).end);
  return need;
}

spec_status_t spec_build_tree(const spec_tree_build_args_t* t, void* ws, size_t ws_bytes,
                              spec_stream_t stream_) {
  const spec_status_t st = check_tree_build(t);
  if (st != SPEC_OK) return st;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) % kWsAlign) != 0) return SPEC_ERR_INVALID_ARGUMENT;
  if (tree_build_layout(*t, kWsHeader, 1).end > ws_bytes) return SPEC_ERR_WORKSPACE_TOO_SMALL;
  const size_t esz = t->logits_dtype == SPEC_BF16 ? 2 : 4;
  const bool vec = (static_cast<size_t>(t->vocab) * esz) % 16 == 0 &&
                   reinterpret_cast<uintptr_t>(t->drafter_logits) % 16 == 0;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  DeviceScope scope(stream);
  if (!scope.ok) return SPEC_ERR_CUDA;
  const int sms = scope.sms;
  const TreeBuildLayout L = tree_build_layout(*t, kWsHeader, sms);
  if (L.end > ws_bytes) return SPEC_ERR_WORKSPACE_TOO_SMALL;
  return launch_tree_build(*t, L, static_cast<char*>(ws), stream, vec) == cudaSuccess ? SPEC_OK
                                                                                       : SPEC_ERR_CUDA;
}

size_t spec_lm_head_workspace_size(const spec_lm_head_args_t* a) {
  if (check_lm_head(a) != SPEC_OK) return 0;
  return lm_layout(*a, kWsHeader).end;
}

spec_status_t spec_lm_head_stats(const spec_lm_head_args_t* a, void* ws, size_t ws_bytes,
                                 spec_stream_t stream_) {
  const spec_status_t st = check_lm_head(a);
  if (st != SPEC_OK) return st;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) % kWsAlign) != 0) return SPEC_ERR_INVALID_ARGUMENT;
  const LmLayout L = lm_layout(*a, kWsHeader);
  if (L.end > ws_bytes) return SPEC_ERR_WORKSPACE_TOO_SMALL;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  DeviceScope scope(stream);
  if (!scope.ok) return SPEC_ERR_CUDA;
  return launch_lm_head(*a, L, static_cast<char*>(ws), stream) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

spec_status_t spec_test_lm_head_wait_timeout(const spec_lm_head_args_t* a, void* ws,
                                             size_t ws_bytes, spec_stream_t stream_) {
  const spec_status_t st = check_lm_head(a);
  if (st != SPEC_OK) return st;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) % kWsAlign) != 0) return SPEC_ERR_INVALID_ARGUMENT;
  const LmLayout L = lm_layout(*a, kWsHeader);
  if (L.end > ws_bytes) return SPEC_ERR_WORKSPACE_TOO_SMALL;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  DeviceScope scope(stream);
  if (!scope.ok) return SPEC_ERR_CUDA;
  return launch_lm_head(*a, L, static_cast<char*>(ws), stream, /*starve=*/true) == cudaSuccess
             ? SPEC_OK
             : SPEC_ERR_CUDA;
}

spec_status_t spec_commit_tree_kv(const spec_tree_commit_args_t* c, spec_stream_t stream) {
  if (!c || c->batch < 1 || c->num_nodes < 1 || c->num_nodes > 64 || c->num_kv_heads < 1 ||
      c->page_size < 1 || c->max_pages_per_seq < 1 || c->num_pages < 1 || !c->k_cache ||
      !c->v_cache || !c->page_table || !c->kv_len || !c->path || !c->num_accepted)
    return SPEC_ERR_INVALID_ARGUMENT;
  if (c->head_dim != 64 && c->head_dim != 128) return SPEC_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(c->k_cache) | reinterpret_cast<uintptr_t>(c->v_cache)) & 15u)
    return SPEC_ERR_INVALID_ARGUMENT;
  if (c->batch > 65535) return SPEC_ERR_UNSUPPORTED;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  DeviceScope scope(s);
  if (!scope.ok) return SPEC_ERR_CUDA;
  return launch_tree_commit(*c, s) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

spec_status_t spec_commit_kv(const spec_commit_args_t* c, spec_stream_t stream) {
  if (!c || c->batch < 1 || c->gamma < 1 || c->page_size < 1 || c->max_pages_per_seq < 1 ||
      c->free_capacity < 0 || !c->kv_len || !c->num_accepted || !c->page_table ||
      !c->free_pages || !c->free_count || (c->reserve != 0 && c->reserve != 1))
    return SPEC_ERR_INVALID_ARGUMENT;
  if (static_cast<int64_t>(c->max_pages_per_seq) * c->page_size + c->gamma > INT32_MAX)
    return SPEC_ERR_UNSUPPORTED;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  DeviceScope scope(s);
  if (!scope.ok) return SPEC_ERR_CUDA;
  return launch_commit(*c, s) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

spec_status_t spec_philox_uniforms(uint64_t seed, uint64_t offset, int64_t n, float* out_dev,
                                   spec_stream_t stream) {
  if (n < 0 || (n > 0 && !out_dev)) return SPEC_ERR_INVALID_ARGUMENT;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  DeviceScope scope(s);
  if (!scope.ok) return SPEC_ERR_CUDA;
  return launch_philox(seed, offset, n, out_dev, s) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}

spec_status_t spec_read_device_status(void* ws, spec_stream_t stream, uint32_t* flags_out) {
  if (!ws || !flags_out) return SPEC_ERR_INVALID_ARGUMENT;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  DeviceScope scope(s);
  if (!scope.ok) return SPEC_ERR_CUDA;
  uint32_t flags = 0;
  if (cudaMemcpyAsync(&flags, ws, sizeof(flags), cudaMemcpyDeviceToHost, s) != cudaSuccess)
    return SPEC_ERR_CUDA;
  if (cudaMemsetAsync(ws, 0, sizeof(flags), s) != cudaSuccess) return SPEC_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return SPEC_ERR_CUDA;
  *flags_out = flags;
  if (flags & SPEC_FLAG_TIMEOUT) return SPEC_ERR_TIMEOUT;
  return flags ? SPEC_ERR_DEVICE_INPUT : SPEC_OK;
}

const char* spec_status_string(spec_status_t status) {
  switch (status) {
    case SPEC_OK: return "SPEC_OK";
    case SPEC_ERR_INVALID_ARGUMENT: return "SPEC_ERR_INVALID_ARGUMENT";
    case SPEC_ERR_UNSUPPORTED: return "SPEC_ERR_UNSUPPORTED";
    case SPEC_ERR_WORKSPACE_TOO_SMALL: return "SPEC_ERR_WORKSPACE_TOO_SMALL";
    case SPEC_ERR_CUDA: return "SPEC_ERR_CUDA";
    case SPEC_ERR_DEVICE_INPUT: return "SPEC_ERR_DEVICE_INPUT";
    case SPEC_ERR_TIMEOUT: return "SPEC_ERR_TIMEOUT";
  }
  return "unknown spec_status_t";
}

int32_t spec_attn_tensor_core_min_rows(void) { return specv::tc_min_rows(); }

}  // extern "C"
