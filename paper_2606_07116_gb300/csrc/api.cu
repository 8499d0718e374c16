// Status strings, ABI version and the device status word.
#include <mutex>

#include "offq.h"
#include "offq_host.h"

namespace {

// One status word per device. Kernels write OFFQ_ERR_TIMEOUT here when a
// bounded wait runs out; offq_get_device_status reads and clears it.
__device__ int g_device_status = 0;

std::mutex g_mu;
int* g_status_ptr[offq::kMaxDevices] = {};

}  // namespace

namespace offq {

int* device_status_ptr() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_status_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_device_status) != cudaSuccess) return nullptr;
    g_status_ptr[dev] = static_cast<int*>(p);
  }
  return g_status_ptr[dev];
}

}  // namespace offq

extern "C" int offq_get_device_status(void* stream) {
  int* p = offq::device_status_ptr();
  if (p == nullptr) return OFFQ_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int host = 0;
  if (cudaMemcpyAsync(&host, p, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess) return OFFQ_ERR_CUDA;
  if (cudaMemsetAsync(p, 0, sizeof(int), s) != cudaSuccess) return OFFQ_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return OFFQ_ERR_CUDA;
  return host;
}

extern "C" const char* offq_status_string(int status) {
  switch (status) {
    case OFFQ_OK: return "OFFQ_OK";
    case OFFQ_ERR_INVALID_ARG: return "OFFQ_ERR_INVALID_ARG";
    case OFFQ_ERR_UNSUPPORTED: return "OFFQ_ERR_UNSUPPORTED";
    case OFFQ_ERR_MISALIGNED: return "OFFQ_ERR_MISALIGNED";
    case OFFQ_ERR_CUDA: return "OFFQ_ERR_CUDA";
    case OFFQ_ERR_TIMEOUT: return "OFFQ_ERR_TIMEOUT";
    default: return "OFFQ_UNKNOWN_STATUS";
  }
}

extern "C" int offq_abi_version(void) { return OFFQ_ABI_VERSION; }
