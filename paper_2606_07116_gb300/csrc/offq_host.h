// Host-side helpers shared by the OffQ translation units (not part of the ABI).
#pragma once

#include <atomic>
#include <cstdint>
#include <mutex>
#include <utility>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include "offq.h"

namespace offq {

// Device address of the status word of the current device (set up once per
// device). Returns nullptr if the runtime call failed.
int* device_status_ptr();

inline bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

inline bool is_pow2(int64_t v) { return v > 0 && (v & (v - 1)) == 0; }

inline int elem_bytes(int dtype) {
  switch (dtype) {
    case OFFQ_F32: return 4;
    case OFFQ_BF16: return 2;
    case OFFQ_F16: return 2;
    default: return 0;
  }
}

inline int launch_status() {
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? OFFQ_OK : OFFQ_ERR_CUDA;
}

// Launches kern<<<grid, block, smem, stream>>>(args...) with programmatic
// stream serialization: the kernel may be scheduled while the previous kernel
// in the stream finishes, and waits for it (griddepcontrol.wait) before its
// first global-memory access. Returns the launch's status.
template <typename... KArgs, typename... Args>
inline int launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                      Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...) == cudaSuccess ? OFFQ_OK : OFFQ_ERR_CUDA;
}

constexpr int kMaxDevices = 64;

// Opts kKernel in to `bytes` of dynamic shared memory on the current device.
// The attribute belongs to the device's context, so it is set once per device
// (not once per process): a process that launches on a second GPU sets it
// there too. Returns false if the device query or the attribute call failed.
template <auto kKernel>
inline bool smem_optin(int bytes) {
  static std::atomic<bool> done[kMaxDevices] = {};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return false;
  if (done[dev].load(std::memory_order_acquire)) return true;
  std::lock_guard<std::mutex> lock(mu);
  if (!done[dev].load(std::memory_order_relaxed)) {
    if (cudaFuncSetAttribute(kKernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) != cudaSuccess)
      return false;
    done[dev].store(true, std::memory_order_release);
  }
  return true;
}

// Decode form of offq_w4a4_linear (csrc/gemm_decode.cu): tokens it takes at
// most, and the launch for 1 <= T <= decode_max_tokens() with arguments
// already checked by offq_w4a4_linear.
int decode_max_tokens();
// MXFP4 activation rows on the persistent warp-per-1024-channel layout; 1 when
// the shape or row count does not suit it (csrc/quant.cu).
int quantize_mx_rows_fast(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx, int32_t g, int32_t flags,
                          uint8_t* codes, uint8_t* shifts, float* row_scale, float* offset, cudaStream_t s);
int w4a4_linear_decode(const uint8_t* a_codes, const float* a_scale, const float* a_offset, int64_t T, int64_t N,
                       int64_t K, int32_t g, const uint8_t* w_codes, const float* w_scale, const float* w_offsum,
                       void* out, int out_dtype, int64_t ldo, int32_t* acc_debug, cudaStream_t stream);

// Rows of the g = 1024 rotating quantizer on the tensor cores (bf16 input, one
// head; csrc/quant_mma.cu). Returns 1 when the shape, alignment or row count
// does not suit it, else the launch status.
struct MmaQuantRows {
  const void* x;       // bf16 [rows][ld_t]
  int64_t ld_t;
  int64_t rows;
  int K;
  int flags;           // OFFQ_OFFSET (OFFQ_ROTATE implied)
  uint8_t* codes;
  float* scale;
  float* offset;       // [rows][K / 1024] or nullptr
  int tiled;
  float inv_sqrt_g;
  float scale_mul;
  int* status;
  long long wait_cycles;
};
int quantize_rows_mma(const MmaQuantRows& p, cudaStream_t s);

// cuTensorMapEncodeTiled from the driver (nullptr if unavailable; csrc/kv_rot.cu).
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder();

// Largest input dimension the row quantizer stages in shared memory.
constexpr int64_t kMaxQuantK = 32768;
// Largest K of the GEMM: every partial sum stays an integer below 2^24.
constexpr int64_t kMaxGemmK = 65536;

}  // namespace offq
