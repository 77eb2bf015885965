// dd_attn_bwd_noalloc: the attention backward for callers that cannot
// allocate device memory.
//
// Who needs it: a host runtime that owns every byte of device memory through
// its own allocator and only hands this library the tensors it already holds
// (there is no way for it to pass an allocator across a plain C boundary), or
// a step loop run under a fixed device-memory budget where a cudaMalloc at
// step time is not allowed (it can fail when the budget is spent and it
// synchronises the device). Such a caller cannot provide the backward's
// workspace, so this entry point brings its own: a fixed-size array in device
// global memory that the library reserves for itself.
//
// The array is a file-scope __device__ variable, so every GPU on which this
// library's device code is loaded holds kNoallocScratchBytes of it until the
// process exits. Host code cannot use the array's name as a device address:
// the address is looked up once per device with cudaGetSymbolAddress, with
// that device current, on the first call made on that device. That first
// call should therefore come before any stream capture. The looked-up address
// belongs to the device's current context: after cudaDeviceReset (which
// destroys that context and unloads the module) it is stale, so this entry
// point must not be used on a device that has been reset in this process.
//
// All calls share the one array and it keeps the previous call's contents:
// the status word is cleared at the start of every call and the backward's
// first kernel zeroes the dQ accumulator and rewrites the per-row vectors.
// Calls whose kernels overlap on the GPU (other streams, or other host
// threads) race on the array; the caller must order them.
#include <mutex>

#include <cuda_runtime.h>

#include "../../include/ddattn.h"

namespace ddattn {
dd_status validate_desc(const dd_attn_desc* desc);  // api.cu
}

namespace {

constexpr size_t kNoallocScratchBytes = size_t(32) << 20;  // 32 MiB per device
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up once).
void* scratch_on_current_device() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return nullptr;
    g_scratch_addr[dev] = p;
  }
  return g_scratch_addr[dev];
}

}  // namespace

extern "C" dd_status dd_attn_bwd_noalloc(const dd_attn_desc* desc, const void* q, const void* k, const void* v,
                                         const void* o, const void* dO, const float* lse, void* dq, void* dk,
                                         void* dv, int32_t* device_status, void* stream) {
  // The same code dd_attn_bwd returns for a bad descriptor, then the size limit.
  const dd_status valid = ddattn::validate_desc(desc);
  if (valid != DD_OK) return valid;
  if (dd_attn_workspace_size(desc, 1) > kNoallocScratchBytes) return DD_ERR_WORKSPACE;
  if (!q || !k || !v || !o || !dO || !lse || !dq || !dk || !dv) return DD_ERR_INVALID_ARG;
  void* scratch = scratch_on_current_device();
  if (!scratch) return DD_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(scratch, 0, sizeof(int32_t), s) != cudaSuccess) return DD_ERR_CUDA;
  dd_status st = dd_attn_bwd_phases(desc, q, k, v, o, dO, lse, dq, dk, dv, scratch, kNoallocScratchBytes,
                                    DD_BWD_ALL, stream);
  if (st != DD_OK) return st;
  if (device_status &&
      cudaMemcpyAsync(device_status, scratch, sizeof(int32_t), cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return DD_ERR_CUDA;
  return DD_OK;
}
