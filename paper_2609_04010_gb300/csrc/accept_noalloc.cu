// spec_accept_block_noalloc: the acceptance step with its scratch in a fixed device
// array that this library owns, for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc (or any allocating routine) at the point where
// they verify a block: for example, code running inside a memory pool or a
// pre-planned arena whose allocations are frozen, or code that must not trigger an
// allocator at all. This entry point takes the same arguments as spec_accept_block
// minus the workspace; its scratch (row statistics, slice sums, tickets, status word)
// lives in kScratchBytes of device memory declared below, which every GPU that loads
// the library keeps until the process exits.
#include <atomic>
#include <mutex>

#include "common.cuh"

namespace specv {

// The argument check of spec_accept_block (api.cu): the same limits and error codes.
spec_status_t check_accept(const spec_accept_args_t* a);

namespace {

constexpr size_t kScratchBytes = SPEC_NOALLOC_SCRATCH_BYTES;

// The scratch array. Host code must not use this name as a device address: the first
// call on each device looks up its address with cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_accept_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

// The device address of the scratch array on `dev` (which is current); looked up once.
cudaError_t scratch_address(int dev, void** out) {
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_scratch_ptr[dev]) {
    void* ptr = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&ptr, g_accept_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = ptr;
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

}  // namespace
}  // namespace specv

using namespace specv;

extern "C" spec_status_t spec_accept_block_noalloc(const spec_accept_args_t* accept,
                                                   spec_stream_t stream_) {
  const spec_status_t st = check_accept(accept);
  if (st != SPEC_OK) return st;
  // The same scratch layout spec_accept_block uses inside a caller's workspace.
  const AcceptLayout L = accept_layout(*accept, kWsHeader);
  if (L.end > kScratchBytes) return SPEC_ERR_WORKSPACE_TOO_SMALL;  // beyond the fixed array
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  // the stream's device is current until this call returns; the caller's is restored
  DeviceScope scope(stream);
  if (!scope.ok) return SPEC_ERR_CUDA;
  void* ptr = nullptr;
  if (scratch_address(scope.dev, &ptr) != cudaSuccess) return SPEC_ERR_CUDA;
  (void)cudaGetLastError();  // a failed call before this one must not fail our launches
  char* ws = static_cast<char*>(ptr);
  // The status word and the tickets must start at zero; the array keeps whatever the
  // previous call (possibly an interrupted one) left, so clear them on the stream.
  if (cudaMemsetAsync(ws, 0, L.partials, stream) != cudaSuccess) return SPEC_ERR_CUDA;
  return launch_accept(*accept, L, ws, scope.sms, stream) == cudaSuccess ? SPEC_OK : SPEC_ERR_CUDA;
}
