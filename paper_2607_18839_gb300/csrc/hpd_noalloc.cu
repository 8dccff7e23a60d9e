// hpd_noalloc.cu -- hpd_branch_attn_noalloc: the branch-attention step for
// callers that cannot allocate device memory.
//
// Some callers have no way to obtain a scratch buffer: a plugin whose host
// engine owns every device allocation and hands it only input and output
// buffers, or code on a path where a cudaMalloc (which may synchronise the
// device) is not allowed.  This entry point gives them the same step with
// its scratch in a fixed file-scope device array instead of a caller-provided
// workspace.  The array is HPD_NOALLOC_WORKSPACE_BYTES long; every GPU that
// loads libhpd keeps it until the process exits.
#include <atomic>
#include <mutex>

#include "common.cuh"

namespace {

// Scratch shared by every hpd_branch_attn_noalloc call on a device.
__device__ __align__(256) uint8_t g_noalloc_scratch[HPD_NOALLOC_WORKSPACE_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
std::atomic<void *> g_scratch_ptr[kMaxDevices];

// Device address of the scratch array on the current device.  In host code
// the array's name is only a host-side stand-in, so the address has to come
// from cudaGetSymbolAddress, once per device, with that device current.
cudaError_t scratch_address(void **out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  void *p = g_scratch_ptr[dev].load(std::memory_order_acquire);
  if (!p) {
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    p = g_scratch_ptr[dev].load(std::memory_order_acquire);
    if (!p) {
      e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
      if (e != cudaSuccess) return e;
      g_scratch_ptr[dev].store(p, std::memory_order_release);
    }
  }
  *out = p;
  return cudaSuccess;
}

}  // namespace

extern "C" hpd_status hpd_branch_attn_noalloc(const hpd_branch_attn_args *args,
                                              hpd_stream_t stream) {
  if (!args) return HPD_ERR_INVALID_ARG;
  hpd_branch_attn_args a = *args;
  a.workspace = nullptr;
  a.workspace_bytes = 0;
  // A call that is refused enqueues nothing, not even the clear of the
  // shared array below: every argument check comes first.
  const hpd_status st = hpd::check_call_args(&a);
  if (st != HPD_OK) return st;
  const size_t need = hpd_branch_attn_workspace_size(&a);
  if (need == 0) return HPD_ERR_INVALID_ARG;
  if (need > HPD_NOALLOC_WORKSPACE_BYTES) return HPD_ERR_WORKSPACE;

  void *scratch = nullptr;
  cudaError_t e = scratch_address(&scratch);
  if (e != cudaSuccess) return hpd::record_cuda_error(e);
  // The array keeps the previous call's contents; the error word and the
  // arrival tickets at its head must start at zero.
  e = cudaMemsetAsync(scratch, 0, hpd::workspace_zero_bytes(&a),
                      reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return hpd::record_cuda_error(e);
  a.workspace = scratch;
  a.workspace_bytes = HPD_NOALLOC_WORKSPACE_BYTES;
  return hpd_branch_attn(&a, stream);
}
