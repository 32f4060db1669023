// Internal declarations shared by the CUDA translation units of libspecverify.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "spec_verify.h"

namespace specv {

// ----------------------------------------------------------------------------------
// Workspace layout. Every region starts on a 256-byte boundary. The header holds the
// status word; counters are per-call tickets that the last arriving block resets.
// ----------------------------------------------------------------------------------
constexpr size_t kWsAlign = 256;
constexpr size_t kWsHeader = 256;  // [0] = status word (uint32)

inline size_t ws_round(size_t x) { return (x + kWsAlign - 1) / kWsAlign * kWsAlign; }

// --- acceptance ---
// 128-thread blocks with few registers, so that they fit beside a resident attention
// block when the verify step overlaps the two parts.
constexpr int kStatsThreads = 128;
constexpr int kStatsChunk = 4096;                          // vocab elements per row item
constexpr int kSampleThreads = 128;
constexpr int kDecideThreads = 512;                        // one block per sequence
constexpr int kSampleSlice = 4096;                         // vocab elements per sample block
constexpr int kSamplePerThread = kSampleSlice / kSampleThreads;  // contiguous per thread

struct RowPartial {  // one (sequence, row, vocab chunk) item of the row statistics
  float m;           // max raw logit of the chunk (-inf if none finite)
  float s;           // sum exp((l - m) / T) over the chunk (T > 0 rows)
  int32_t arg;       // lowest index of the chunk maximum (greedy rows)
  uint32_t bad;      // NaN / +inf seen
};

struct AcceptLayout {
  size_t tickets;      // uint32 [batch]
  size_t partials;     // RowPartial [batch][2*gamma-1][nchunk]
  size_t records;      // 32-byte decision record [batch] (n and the final draw's normalisers)
  size_t slice_sums;   // float4 [batch][nslice] = (residual sum, p sum, residual last, p last)
  size_t end;
  int nchunk, nslice;
};

AcceptLayout accept_layout(const spec_accept_args_t& a, size_t base);

// --- filtered acceptance ---
constexpr int kFilterMaxTopK = SPEC_FILTER_MAX_TOP_K;
constexpr int kFiltLaneElems = 64;    // contiguous logits per lane (at the smallest lane size)
constexpr int kFiltMaxLanes = 4096;   // lane maxima one row block keeps in shared memory
constexpr int kFiltBlocksPerSm = 8;   // row blocks resident per SM (128 threads each)
constexpr int kFiltMaxSplits = 16;    // blocks one row may be split across
constexpr int kRowThreads = 128;      // threads of a filtered row block

struct FiltRow {    // one (sequence, row) result of the filtered row kernel
  int32_t nkeep;    // kept tokens (top-k, then top-p)
  int32_t argmax;   // lowest index of the row maximum
  uint32_t flags;   // 1: NaN / +inf / no finite logit; 2: top_k or top_p out of range
  int32_t pad;
};

struct FilterLayout {
  size_t tickets;  // uint32 [batch]: rows of the sequence finished (reset by the last)
  size_t rows;     // FiltRow [batch][2*gamma-1]
  size_t kept;     // (int32 token, fp32 p') [batch][2*gamma-1][max_top_k], rank order
  size_t row_tickets;  // uint32 [batch][2*gamma-1]: splits of the row finished (splits > 1)
  size_t lanes_g;  // uint32 [batch][2*gamma-1][nlanes]: lane maxima (splits > 1)
  size_t parts;    // 16 B [batch][2*gamma-1][splits]: each split's maximum and bad flag
  size_t end;
  int lane_shift;  // lanes hold kFiltLaneElems << lane_shift logits
  int nlanes;      // ceil(vocab / lane size) <= kFiltMaxLanes
  int splits;      // blocks per row
  int lanes_per_split;
  int cand_cap;    // candidates one block holds (a power of two)
  int smem_a;      // bytes of the first dynamic shared region
};

// draw = true: the layout of the draft-side draw (gamma drafter rows per sequence).
FilterLayout filter_layout(const spec_accept_args_t& a, int max_top_k, size_t base, int sms,
                           bool draw = false);

// --- draft-side sampling ---
struct DraftLayout {
  size_t tickets;      // uint32 [batch]: rows of the sequence finished (reset by the last)
  size_t row_flags;    // uint32 [batch][gamma]
  size_t row_tickets;  // uint32 [batch][gamma]: splits of the row finished (splits > 1)
  size_t lanes_g;      // float2 [batch][gamma][nlanes]: lane (max, sum) (splits > 1)
  size_t parts;        // 16 B [batch][gamma][splits]: each split's maximum and bad flag
  size_t end;
  size_t smem;         // dynamic shared memory of one block: nlanes x 8 B
  int lane_elems;      // 64 with 16-byte loads, 32 with element loads
  int nlanes, splits, lanes_per_split;
};

DraftLayout draft_layout(const spec_draft_args_t& a, size_t base, int sms, bool vec);
cudaError_t launch_draft(const spec_draft_args_t& a, const DraftLayout& L, char* ws,
                         cudaStream_t stream, bool vec);
cudaError_t launch_commit(const spec_commit_args_t& a, cudaStream_t stream);

// --- tree verification ---
struct TreeLayout {
  size_t tickets;      // uint32 [batch]: node rows of the sequence finished
  size_t row_tickets;  // uint32 [batch][nodes]: splits of the row finished
  size_t parts;        // 16 B [batch][nodes][splits]: (argmax key, max key, bad, sum of 2^..)
  size_t argmax;       // int32 [batch][nodes]
  size_t rowstat;      // float2 [batch][nodes]: (max logit, sum of 2^((l - max) log2e / T))
  size_t end;
  int splits, elems_per_split;
};

TreeLayout tree_layout(int batch, int nodes, int vocab, size_t base, int sms, bool vec);
cudaError_t launch_tree_greedy(const spec_tree_accept_args_t& a, const TreeLayout& L, char* ws,
                               cudaStream_t stream, bool vec);
cudaError_t launch_tree_commit(const spec_tree_commit_args_t& a, cudaStream_t stream);

constexpr int kTreeCandCap = 512;  // candidates of one row part ranked in shared memory

struct TreeBuildLayout {
  size_t tickets;      // uint32 [batch]: position rows of the sequence finished
  size_t seq_flags;    // uint32 [batch]: flags its rows raised
  size_t row_tickets;  // uint32 [batch][rows]: parts of the row finished
  size_t keys;         // uint64 [batch][rows][splits][64]: each part's ranked candidate keys
  size_t stats;        // float4 [batch][rows][splits]: (max, sum of exponentials, bad, -)
  size_t table;        // int2 [batch][rows][64]: the position's (token, log q), ranked
  size_t end;
  int rows;            // positions that can hold a node: min(gamma - 1, num_nodes - 1)
  int keff;            // candidates used per position: min(top_k, vocab, num_nodes - 1)
  int splits, elems_per_split;
  int smem;            // dynamic shared memory of a block, bytes
};

TreeBuildLayout tree_build_layout(const spec_tree_build_args_t& t, size_t base, int sms);
cudaError_t launch_tree_build(const spec_tree_build_args_t& t, const TreeBuildLayout& L, char* ws,
                              cudaStream_t stream, bool vec);

// --- attention ---
struct AttnPlan {
  int path;          // SPEC_ATTN_CUDA_CORES or SPEC_ATTN_TENSOR_CORES
  int keys_on_lanes; // tensor cores: the keys-on-lanes kernel (attn_kl.cu), else row tiles
  int head_pair;     // row tiles: one block serves two adjacent KV heads (8 KB page boxes)
  int rows;          // (Hq/Hkv) * gamma
  int rows_per_cta;  // rows one block handles (a row tile)
  int row_tiles;     // ceil(rows / rows_per_cta)
  int key_tile;      // keys per pipeline step
  int max_keys;      // max_pages_per_seq * page_size
  int nsplit;        // KV splits per (sequence, kv head, row tile) (CUDA-core path)
  int tiles_per_split;
  int grid;          // blocks launched
  int slot_rows;     // rows per partial slot
  int64_t slots;     // partial slots
  size_t tickets, partial_o, partial_ml, end;
};

AttnPlan attn_plan(const spec_attn_args_t& a, size_t base, int num_sms, int path_override);

// ----------------------------------------------------------------------------------
// Launchers (defined in the .cu files); all return cudaGetLastError() of the launch.
// ----------------------------------------------------------------------------------
// overlap_prior: launch the acceptance kernels as programmatic dependents of the kernel
// just launched on the stream (the attention kernel of the same verify step, which
// reads none of their inputs and writes none of their outputs).
cudaError_t launch_accept(const spec_accept_args_t& a, const AcceptLayout& L, char* ws,
                          int num_sms, cudaStream_t stream, bool overlap_prior = false);
// With draw_tokens set, draws every drafter row's token instead of verifying (only the
// logits, temperature, uniforms and batch shape of a are read).
cudaError_t launch_accept_filtered(const spec_accept_args_t& a, const spec_filter_args_t& f,
                                   const FilterLayout& L, char* ws, cudaStream_t stream,
                                   bool overlap_prior = false, int32_t* draw_tokens = nullptr,
                                   float* draw_q = nullptr);
cudaError_t launch_attn_simt(const spec_attn_args_t& a, const AttnPlan& P, char* ws,
                             cudaStream_t stream);
// starve (test hook only): the kernel's producers issue no copies, so its bounded waits
// run out and it returns with SPEC_FLAG_TIMEOUT set.
cudaError_t launch_attn_tc(const spec_attn_args_t& a, const AttnPlan& P, char* ws,
                           cudaStream_t stream, bool starve = false);
cudaError_t launch_attn_kl(const spec_attn_args_t& a, const AttnPlan& P, char* ws,
                           cudaStream_t stream);
cudaError_t launch_philox(uint64_t seed, uint64_t offset, int64_t n, float* out, cudaStream_t s);
cudaError_t launch_noise(uint64_t seed, uint64_t offset, int64_t n, int32_t vocab, int32_t* out,
                         cudaStream_t s);

// Rows of one CUDA-core block and of one tensor-core block.
constexpr int kSimtRowTile = 16;
constexpr int kSimtKeyTile = 64;
constexpr int kSimtThreads = 128;
constexpr int kTcKeyTile = 64;
constexpr int kTcMaxRows = 256;  // two M = 128 tiles per block
// The keys-on-lanes tensor-core kernel (attn_kl.cu): 128 keys per tile, at most 64 query
// rows per KV head, head_dim 128, batch prefix sums in shared memory.
constexpr int kKlKeyTile = 128;
constexpr int kKlMaxRows = 64;
constexpr int kKlMaxBatch = 2048;
size_t kl_smem_bytes(int rows, int batch);

int tc_min_rows();

// The device a stream belongs to. cudaStreamGetDevice is not allowed on a capturing
// stream (it invalidates the capture), so a stream under capture is taken to belong
// to the current device, the one its captured work must run on.
inline cudaError_t stream_device(cudaStream_t stream, int* dev) {
  if (stream != nullptr) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    const cudaError_t e = cudaStreamIsCapturing(stream, &cs);
    if (e != cudaSuccess) return e;
    if (cs == cudaStreamCaptureStatusNone) return cudaStreamGetDevice(stream, dev);
  }
  return cudaGetDevice(dev);
}
// Cached multiprocessor count of a device (asked once per device).
int device_sm_count(int dev);

// Makes the device of `stream` current for the duration of one entry point and puts
// the caller's current device back when it goes out of scope, so that no call changes
// which device the calling thread has current. `ok` is false when the device could
// not be found or selected.
struct DeviceScope {
  int dev = 0, prev = -1, sms = 0;
  bool ok = false;
  explicit DeviceScope(cudaStream_t stream) {
    if (cudaGetDevice(&prev) != cudaSuccess) { prev = -1; return; }
    if (stream_device(stream, &dev) != cudaSuccess) return;
    if (dev != prev && cudaSetDevice(dev) != cudaSuccess) return;
    sms = device_sm_count(dev);
    ok = true;
  }
  ~DeviceScope() {
    if (prev >= 0 && dev != prev) cudaSetDevice(prev);
  }
  DeviceScope(const DeviceScope&) = delete;
  DeviceScope& operator=(const DeviceScope&) = delete;
};

int tc_ctas_per_sm(int head_dim, int rows_per_cta, int rows, int batch, bool head_pair);
size_t tc_smem_bytes(int head_dim, int rows_per_cta, int rows, int batch, bool head_pair);
// Whether the row-tile kernel serves two adjacent KV heads per block: KV groups of 33 to
// 64 rows, an even Hkv, and the batch's prefix sums fit beside its stages.
bool tc_head_pair(int head_dim, int rows, int num_kv_heads, int batch);
constexpr int kTcMaxBatch = 4096;  // batch prefix sums live in shared memory
constexpr size_t kTcMaxSmem = 227u * 1024u;  // dynamic shared memory of one block

}  // namespace specv

// ----------------------------------------------------------------------------------
// Device helpers
// ----------------------------------------------------------------------------------
#ifdef __CUDACC__
namespace specv {

__device__ __forceinline__ float bf16_bits_to_f32(uint32_t h) { return __uint_as_float(h << 16); }

// 2^x via the PTX approximate base-2 exponential (relative error about 2^-22;
// results below 2^-126 flush to zero).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Programmatic dependent launch: let the next kernel on the stream start now / wait for
// the kernel this one depends on (no-ops for kernels launched without the attribute).
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait_prior() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ void set_status(uint32_t* status, uint32_t flag) {
  atomicOr(status, flag);
}

constexpr float kLog2e = 1.4426950408889634f;

}  // namespace specv
#endif
