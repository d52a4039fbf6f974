// noalloc.cu — strided_dense_attn_noalloc: the strided dense attention for
// callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc or cudaMallocAsync: processes whose
// device memory is owned and pooled by another allocator (an inference
// framework's caching allocator, a runtime with a fixed memory budget reserved
// at start-up) and code that must not allocate on its hot path.  They still
// own their inputs and outputs, but have no way to hand this library the
// split-K scratch (partial rows, merge tickets, the work-item counter) that
// strided_dense_attn() takes as a workspace.  This entry point keeps that
// scratch in a fixed file-scope device array instead, so a call allocates
// nothing.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "delta_attn.h"

namespace {

// Fixed scratch: 16 MiB, held by every GPU that loads this library until the
// process exits.  All calls share it.
constexpr size_t kScratchBytes = size_t(16) << 20;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
void* g_scratch_ptr[kMaxDevices];
std::once_flag g_scratch_once[kMaxDevices];
cudaError_t g_scratch_err[kMaxDevices];

// The device address of the scratch array on the current device.  The host
// symbol g_noalloc_scratch is only a host-side stand-in, never a device
// address; the address is looked up once per device, with that device
// current, on its first call.
int scratch_for_current_device(void** ptr) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DA_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return DA_ERR_UNSUPPORTED;
  std::call_once(g_scratch_once[dev], [dev] {
    void* p = nullptr;
    g_scratch_err[dev] = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    g_scratch_ptr[dev] = (g_scratch_err[dev] == cudaSuccess) ? p : nullptr;
  });
  if (g_scratch_err[dev] != cudaSuccess || g_scratch_ptr[dev] == nullptr) return DA_ERR_CUDA;
  *ptr = g_scratch_ptr[dev];
  return DA_OK;
}

}  // namespace

extern "C" int strided_dense_attn_noalloc(const void* Q, const void* K, const void* V, float* D_sampled, int B,
                                          int Hq, int Hkv, int64_t N, int d, int gamma, void* stream) {
  size_t need = 0;
  int rc = strided_dense_workspace_size(B, Hq, Hkv, N, d, gamma, &need);
  if (rc != DA_OK) return rc;
  if (need > kScratchBytes) return DA_ERR_WORKSPACE;  // this shape needs more than the fixed scratch
  void* scratch = nullptr;
  if ((rc = scratch_for_current_device(&scratch)) != DA_OK) return rc;
  // strided_dense_attn zeroes the tickets and the item counter in the scratch
  // on `stream` before its kernel runs, and allocates nothing when it is given
  // a workspace.
  return strided_dense_attn(Q, K, V, D_sampled, B, Hq, Hkv, N, d, gamma, scratch, kScratchBytes, stream);
}
