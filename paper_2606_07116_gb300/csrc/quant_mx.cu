// MXFP4 residual quantizer of the OffQ extension to micro-scaling formats
// (paper Sec. 3.4 "Generality on Data Formats": a zero-point per block lets
// MXFP4 absorb the outlier offset as the integer grid does).
//
// Per token row (or weight row):
//   y = x_b H_g / sqrt(g) per block b of g channels   (OFFQ_ROTATE)
//   o[b] = mean(y_b)  (OFFQ_OFFSET; with the rotation = x_b[0] / sqrt(g)),  r = y - o
// then per 32 channels j of r:
//   X_j = floor(log2(max |r_j|)) - 2,  kept within 6 of the row's largest X;
//   e = E2M1 code of r / 2^X_j (nearest magnitude of 0, .5, 1, 1.5, 2, 3, 4, 6,
//       ties to the even mantissa, saturating at 6), sign in bit 3.
// Stored: codes two per byte (even channel low) in the tiled operand layout,
// shift_j = X_j - (Xmax - 6) in 0..6 (tiled, see offq.h), row scale 2^(Xmax - 6),
// offsets. For weights, also the block sums of the operand values e * 2^shift.
//
// One CTA per row, the row staged as fp32 in shared memory: the Sylvester
// transform runs as log2(g) in-place butterfly stages; then a warp per 32-channel
// block finds the block's exponent, and after the row's maximum is known, its
// codes. This form serves the format's correctness and the GEMM's inputs; it is
// not bandwidth-tuned like the per-token quantizer.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cmath>
#include <type_traits>

#include "offq.h"
#include "offq_device.cuh"
#include "offq_host.h"

namespace {

using namespace offq;

constexpr int kMxThreads = 256;
constexpr int kMxWarps = kMxThreads / 32;
constexpr int kMxBlock = 32;
constexpr int kMxSpan = 6;
constexpr int kMxMaxK = 32768;

struct MxArgs {
  const void* x;
  int64_t ldx;
  int64_t rows;
  int K, g, log2g, G;
  int flags;
  float inv_sqrt_g;
  uint8_t* codes;      // tiled [ceil(rows/32)*32][K/2]
  uint8_t* shifts;     // tiled shift bytes
  float* row_scale;    // [rows]
  float* offset;       // [rows][G] or nullptr
  float* offsum;       // [G][rows] or nullptr (weights)
};

template <typename Tin>
__device__ __forceinline__ float load_elem(const Tin* p) {
  if constexpr (sizeof(Tin) == 4) {
    return __ldg(reinterpret_cast<const float*>(p));
  } else if constexpr (std::is_same<Tin, __nv_bfloat16>::value) {
    return __bfloat162float(*p);
  } else {
    return __half2float(*p);
  }
}

// E2M1 magnitude code of m = |v| / 2^X >= 0: the number of decision points below m,
// with ties going to the even code (0.25 -> 0, 0.75 -> 2, 1.25 -> 2, 1.75 -> 4,
// 2.5 -> 4, 3.5 -> 6, 5 -> 6) and everything above 5 to 6.0 (code 7).
__device__ __forceinline__ int e2m1_mag_code(float m) {
  return (m > 0.25f) + (m >= 0.75f) + (m > 1.25f) + (m >= 1.75f) + (m > 2.5f) + (m >= 3.5f) + (m > 5.0f);
}

__device__ __forceinline__ float e2m1_mag_value(int c) {
  const float lo = c < 2 ? 0.5f * c : (c < 4 ? 1.0f + 0.5f * (c - 2) : (c < 6 ? 2.0f + (c - 4) : 4.0f + 2.0f * (c - 6)));
  return lo;
}

// floor(log2(a)) for a normal positive fp32 a, from its exponent field.
__device__ __forceinline__ int floor_log2(float a) { return static_cast<int>((__float_as_uint(a) >> 23) & 0xFF) - 127; }

// 2^e as fp32 for -126 <= e <= 127.
__device__ __forceinline__ float pow2f(int e) { return __uint_as_float(static_cast<uint32_t>(e + 127) << 23); }

template <typename Tin>
__global__ void __launch_bounds__(kMxThreads) quantize_mx_kernel(const MxArgs a) {
  extern __shared__ float row[];  // [K] fp32, then [kMxWarps] ints, then [G] floats
  int* wmax = reinterpret_cast<int*>(row + a.K);
  float* gsum = reinterpret_cast<float*>(wmax + kMxWarps);
  griddep_wait();
  griddep_launch_dependents();
  const int64_t r = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int K = a.K, g = a.g;
  const bool rotate = (a.flags & OFFQ_ROTATE) != 0;
  const bool offs = (a.flags & OFFQ_OFFSET) != 0;
  const Tin* x = static_cast<const Tin*>(a.x) + r * a.ldx;
  for (int i = tid; i < K; i += kMxThreads) row[i] = load_elem(x + i);
  for (int b = tid; b < a.G; b += kMxThreads) gsum[b] = 0.f;
  __syncthreads();

  // Offsets: with the rotation the block-leading channel over sqrt(g) (its value is
  // zeroed so the transform yields sqrt(g) times the residual); without it the block mean.
  if (rotate) {
    if (offs) {
      for (int b = tid; b < a.G; b += kMxThreads) {
        const float x0 = row[b * g];
        if (a.offset != nullptr) a.offset[r * a.G + b] = x0 * a.inv_sqrt_g;
        row[b * g] = 0.f;
      }
    } else if (a.offset != nullptr) {
      for (int b = tid; b < a.G; b += kMxThreads) a.offset[r * a.G + b] = 0.f;
    }
    __syncthreads();
    for (int h = 1; h < g; h <<= 1) {
      for (int p = tid; p < K / 2; p += kMxThreads) {
        const int i = (p / h) * 2 * h + (p % h);
        const float u = row[i], v = row[i + h];
        row[i] = u + v;
        row[i + h] = u - v;
      }
      __syncthreads();
    }
    for (int i = tid; i < K; i += kMxThreads) row[i] *= a.inv_sqrt_g;
    __syncthreads();
  } else if (offs) {
    // Block sums: a warp per block, each lane's g/32 values by a pairwise tree
    // (a power of two of them), then a shuffle tree: depth log2(g).
    for (int b = warp; b < a.G; b += kMxWarps) {
      float lvl[9];
      int n = 0;
      for (int i = lane; i < g; i += 32) {
        float c = row[b * g + i];
        bool carry = true;
#pragma unroll
        for (int k = 0; k < 9; ++k) {
          const bool full = (n >> k) & 1;
          if (carry && full) c = lvl[k] + c;
          if (carry && !full) lvl[k] = c;
          carry = carry && full;
        }
        ++n;
      }
      float s = 0.f;
#pragma unroll
      for (int k = 0; k < 9; ++k) {
        if (n == (1 << k)) s = lvl[k];
      }
#pragma unroll
      for (int m = 16; m > 0; m >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, m);
      const float o = s * (1.0f / static_cast<float>(g));
      if (lane == 0 && a.offset != nullptr) a.offset[r * a.G + b] = o;
      for (int i = lane; i < g; i += 32) row[b * g + i] -= o;
    }
    __syncthreads();
  } else if (a.offset != nullptr) {
    for (int b = tid; b < a.G; b += kMxThreads) a.offset[r * a.G + b] = 0.f;
  }

  // Block exponents and the row's largest.
  const int nblk = K / kMxBlock;
  int my_max = -1000;
  for (int j = warp; j < nblk; j += kMxWarps) {
    float m = fabsf(row[j * kMxBlock + lane]);
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, s));
    if (m > 0.f) my_max = max(my_max, floor_log2(m) - 2);
  }
  if (lane == 0) wmax[warp] = my_max;
  __syncthreads();
  int xmax = -1000;
  for (int w = 0; w < kMxWarps; ++w) xmax = max(xmax, wmax[w]);
  if (xmax == -1000) xmax = 0;  // an all-zero row: any exponent
  const int xlo = xmax - kMxSpan;
  if (tid == 0) a.row_scale[r] = pow2f(xlo);

  // Codes, shifts and (weights) the operand block sums.
  const int nkt = K / 128;
  uint8_t* crow = a.codes + (r >> 5) * (K / 32) * 512 + (r & 31) * 16;
  for (int j = warp; j < nblk; j += kMxWarps) {
    const float v = row[j * kMxBlock + lane];
    float m = fabsf(v);
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, s));
    const int X = m > 0.f ? max(floor_log2(m) - 2, xlo) : xlo;
    const int mag = e2m1_mag_code(fabsf(v) * pow2f(-X));
    const uint32_t nib = static_cast<uint32_t>(mag | (v < 0.f && mag > 0 ? 8 : 0));
    // Eight codes per 32-bit word, code k in nibble k: OR-reduce over aligned groups of 8 lanes.
    uint32_t word = nib << (4 * (lane & 7));
#pragma unroll
    for (int s = 1; s < 8; s <<= 1) word |= __shfl_xor_sync(0xFFFFFFFFu, word, s);
    if ((lane & 7) == 0) reinterpret_cast<uint32_t*>(crow + j * 512)[lane >> 3] = word;
    if (lane == 0) {
      const int sh = X - xlo;
      a.shifts[(((r >> 5) * nkt + (j >> 2)) * 32 + (r & 31)) * 4 + (j & 3)] = static_cast<uint8_t>(sh);
    }
    if (a.offsum != nullptr) {
      // Operand value e * 2^shift: a multiple of 1/2 below 2^9, so these sums are exact.
      float ov = e2m1_mag_value(mag) * pow2f(X - xlo);
      if (v < 0.f) ov = -ov;
#pragma unroll
      for (int s = 16; s > 0; s >>= 1) ov += __shfl_xor_sync(0xFFFFFFFFu, ov, s);
      if (lane == 0) atomicAdd(&gsum[(j * kMxBlock) / g], ov);
    }
  }
  if (a.offsum != nullptr) {
    __syncthreads();
    for (int b = tid; b < a.G; b += kMxThreads) a.offsum[static_cast<int64_t>(b) * a.rows + r] = gsum[b];
  }
}

int ilog2i(int v) {
  int l = 0;
  while ((1 << l) < v) ++l;
  return l;
}

template <typename Tin>
int launch_mx(const MxArgs& a, cudaStream_t s) {
  const size_t smem = static_cast<size_t>(a.K) * 4 + kMxWarps * 4 + static_cast<size_t>(a.G) * 4;
  if (smem > 48 * 1024 && !smem_optin<quantize_mx_kernel<Tin>>(kMxMaxK * 4 + kMxWarps * 4 + (kMxMaxK / 32) * 4))
    return OFFQ_ERR_CUDA;
  return launch_pdl(quantize_mx_kernel<Tin>, dim3(static_cast<unsigned>(a.rows)), dim3(kMxThreads), smem, s, a);
}

int run_mx(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx, int32_t g, int32_t flags, uint8_t* codes,
           uint8_t* shifts, float* row_scale, float* offset, float* offsum, bool zero_pad, cudaStream_t s) {
  const int eb = elem_bytes(dtype);
  if (eb == 0 || rows < 0 || K <= 0 || ldx < K || (flags & ~(OFFQ_ROTATE | OFFQ_OFFSET)) != 0)
    return OFFQ_ERR_INVALID_ARG;
  if (!is_pow2(g) || g < 32 || g > 8192 || K % g != 0 || K % 128 != 0) return OFFQ_ERR_INVALID_ARG;
  if (K > kMxMaxK || rows > 0x7FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  if (rows == 0) return OFFQ_OK;
  if (x == nullptr || codes == nullptr || shifts == nullptr || row_scale == nullptr ||
      ((flags & OFFQ_OFFSET) != 0 && offset == nullptr))
    return OFFQ_ERR_INVALID_ARG;
  if (!aligned(x, 16) || (ldx * eb) % 16 != 0 || !aligned(codes, 16) || !aligned(shifts, 4) ||
      !aligned(row_scale, 4) || (offset != nullptr && !aligned(offset, 4)) || (offsum != nullptr && !aligned(offsum, 4)))
    return OFFQ_ERR_MISALIGNED;
  if (zero_pad && rows % 32 != 0) {
    // The last 32-row block's padding rows read as zero codes and shifts: clear
    // that block's codes and shifts before the kernel writes its real rows.
    const int64_t last = rows / 32;
    if (cudaMemsetAsync(codes + last * (K / 32) * 512, 0, static_cast<size_t>((K / 32) * 512), s) != cudaSuccess ||
        cudaMemsetAsync(shifts + last * (K / 128) * 128, 0, static_cast<size_t>((K / 128) * 128), s) != cudaSuccess)
      return OFFQ_ERR_CUDA;
  }
  MxArgs a{};
  a.x = x;
  a.ldx = ldx;
  a.rows = rows;
  a.K = static_cast<int>(K);
  a.g = g;
  a.log2g = ilog2i(g);
  a.G = static_cast<int>(K / g);
  a.flags = flags;
  a.inv_sqrt_g = (flags & OFFQ_ROTATE) ? static_cast<float>(1.0 / std::sqrt(static_cast<double>(g))) : 1.0f;
  a.codes = codes;
  a.shifts = shifts;
  a.row_scale = row_scale;
  a.offset = offset;
  a.offsum = offsum;
  switch (dtype) {
    case OFFQ_F32: return launch_mx<float>(a, s);
    case OFFQ_BF16: return launch_mx<__nv_bfloat16>(a, s);
    case OFFQ_F16: return launch_mx<__half>(a, s);
    default: return OFFQ_ERR_INVALID_ARG;
  }
}

}  // namespace

extern "C" int offq_quantize_act_mx(const void* x, int x_dtype, int64_t T, int64_t K, int64_t ldx, int32_t g,
                                    int32_t flags, uint8_t* codes, uint8_t* shifts, float* row_scale, float* offset,
                                    void* stream) {
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // Prefill-sized inputs of 1024-multiple widths take the persistent form; the
  // arguments are checked by run_mx's rules first (a dry check with zero rows).
  const int chk = run_mx(x, x_dtype, 0, K, ldx, g, flags, codes, shifts, row_scale, offset, nullptr, false, s);
  if (chk != OFFQ_OK) return chk;
  if (T > 0 && x != nullptr && codes != nullptr && shifts != nullptr && row_scale != nullptr &&
      ((flags & OFFQ_OFFSET) == 0 || offset != nullptr) && aligned(x, 16) && (ldx * elem_bytes(x_dtype)) % 16 == 0 &&
      aligned(codes, 16) && aligned(row_scale, 4) && (offset == nullptr || aligned(offset, 4))) {
    const int st = quantize_mx_rows_fast(x, x_dtype, T, K, ldx, g, flags, codes, shifts, row_scale, offset, s);
    if (st != 1) return st;
  }
  return run_mx(x, x_dtype, T, K, ldx, g, flags, codes, shifts, row_scale, offset, nullptr, false, s);
}

extern "C" int offq_prepare_weight_mx(const void* w, int dtype, int64_t N, int64_t K, int32_t g, int32_t rotate,
                                      uint8_t* w_codes, uint8_t* w_shifts, float* w_scale, float* w_offsum,
                                      void* stream) {
  if (N < 1 || w_offsum == nullptr) return OFFQ_ERR_INVALID_ARG;
  return run_mx(w, dtype, N, K, K, g, rotate ? OFFQ_ROTATE : 0, w_codes, w_shifts, w_scale, nullptr, w_offsum, true,
                static_cast<cudaStream_t>(stream));
}

extern "C" int64_t offq_mx_shift_bytes(int64_t R, int64_t K) {
  if (R < 0 || K <= 0 || K % 128 != 0) return -1;
  return (R + 31) / 32 * 32 * (K / 32);
}
