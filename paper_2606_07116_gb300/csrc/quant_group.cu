// Per-group asymmetric activation quantizer (offq_quantize_act_group) and the
// per-group weight row sums its GEMM needs (offq_weight_group_sums).
//
// The paper's evaluated activation setting (Sec. 4): every group of 128
// channels of a (rotated) token row is quantized with Eq. 1's zero-point,
//   s = (max - min) / 15,   z = -rne(min / s),   u = clamp(rne(y / s) + z, 0, 15),
// so the constant offset the rotation leaves in a block (Eq. 5) is absorbed by
// the zero-point (Sec. 3.2 footnote: the grid need not hold 0). A constant
// group gets s = 0, z = 0, u = 0.
//
// One warp takes one 512-channel chunk of a row: lane l holds 16 consecutive
// channels, a group is 8 lanes. With the rotation on (block g a power of two)
// the Sylvester transform runs in place: index bits 0-3 inside the lane, bits
// 4-8 across lanes (shuffle partner l ^ 2^(b-4)), and for g >= 1024 bits 9..
// across the warps of the CTA, which holds whole blocks (a shared-memory
// exchange per bit). The codes are decided on the unnormalised transform
// (y / s is the same ratio) and only the stored scale carries the 1/sqrt(g).
//
// Eq. 1's y / s is evaluated as 15 y / (max - min), the same real number
// without s rounded first: for bf16 / f16 inputs 15 y and max - min are exact
// in fp32, so a ratio that is exactly a half-integer (frequent on those
// grids) stays one and rounds half to even; so does -min / s for z.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <type_traits>

#include "offq.h"
#include "offq_device.cuh"
#include "offq_host.h"

namespace {

using namespace offq;

constexpr int kQGroup = 128;
constexpr int kChunk = 512;          // channels per warp
constexpr int kPerLane = kChunk / 32;  // 16
constexpr int kQWarps = 8;           // warps per CTA for blocks up to 4096 (16 for 8192)
constexpr int kMaxQWarps = 16;

struct GroupQuantArgs {
  const void* x;
  int64_t ldx;
  int64_t T;
  int K;
  int Gq;        // K / 128
  int log2g;     // rotation block, 0 = no rotation
  float inv_sqrt_g;
  uint8_t* codes;  // tiled [ceil(T/32)*32][K/2]
  float* scale;    // [T][Gq]
  float* zero;     // [T][Gq]
};

template <typename Tin>
__device__ __forceinline__ void load16(const Tin* src, float (&v)[kPerLane]) {
  if constexpr (sizeof(Tin) == 4) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float4 f = __ldg(reinterpret_cast<const float4*>(src) + i);
      v[4 * i] = f.x;
      v[4 * i + 1] = f.y;
      v[4 * i + 2] = f.z;
      v[4 * i + 3] = f.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const uint4 u = __ldg(reinterpret_cast<const uint4*>(src) + i);
      const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        if constexpr (std::is_same<Tin, __nv_bfloat16>::value) {
          v[8 * i + 2 * k] = __uint_as_float(w[k] << 16);
          v[8 * i + 2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
        } else {
          const __half2 h = *reinterpret_cast<const __half2*>(&w[k]);
          const float2 f = __half22float2(h);
          v[8 * i + 2 * k] = f.x;
          v[8 * i + 2 * k + 1] = f.y;
        }
      }
    }
  }
}

template <typename Tin>
__global__ void __launch_bounds__(kMaxQWarps * 32) quantize_group_kernel(const GroupQuantArgs a) {
  extern __shared__ float xchg[];  // cross-warp stages: [warps][512]
  griddep_wait();
  griddep_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int warps = blockDim.x >> 5;
  const int chunks = (a.K + kChunk - 1) / kChunk;
  const int64_t item = static_cast<int64_t>(blockIdx.x) * warps + warp;
  // Blocks of g >= 1024 span g / 512 warps of one CTA: every warp takes part in
  // the exchange barriers, so none returns early then. (A CTA's first item and
  // a row's chunk count are multiples of g / 512, so a block never straddles
  // CTAs, and an item past the end lies in a block with no valid item.)
  const bool cross = a.log2g > 9;
  const bool valid = item < a.T * chunks;
  if (!valid && !cross) return;  // warp-uniform
  const int64_t row = valid ? item / chunks : 0;
  const int ch = valid ? static_cast<int>(item - row * chunks) : 0;
  const int c0 = ch * kChunk + lane * kPerLane;
  const bool active = valid && c0 < a.K;  // uniform over each 8-lane group (K % 128 == 0)

  float v[kPerLane];
  if (active) {
    load16(static_cast<const Tin*>(a.x) + row * a.ldx + c0, v);
  } else {
#pragma unroll
    for (int i = 0; i < kPerLane; ++i) v[i] = 0.f;
  }

  // Sylvester transform of each block of g = 2^log2g channels (unnormalised).
  if (a.log2g > 0) {
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      if (b < a.log2g) {
        const int h = 1 << b;
#pragma unroll
        for (int i = 0; i < kPerLane; ++i) {
          if ((i & h) == 0) {
            const float x0 = v[i], x1 = v[i + h];
            v[i] = x0 + x1;
            v[i + h] = x0 - x1;
          }
        }
      }
    }
    const int lane_bits = a.log2g < 9 ? a.log2g : 9;
    for (int b = 4; b < lane_bits; ++b) {
      const int m = 1 << (b - 4);
      const bool upper = (lane & m) != 0;
#pragma unroll
      for (int i = 0; i < kPerLane; ++i) {
        const float o = __shfl_xor_sync(0xFFFFFFFFu, v[i], m);
        v[i] = upper ? o - v[i] : v[i] + o;
      }
    }
    // Bits 9.. of the block index: the partner warp is warp ^ 2^(b-9), through
    // shared memory (element i of lane l of warp w at w*512 + i*32 + l).
    for (int b = 9; b < a.log2g; ++b) {
      const int m = 1 << (b - 9);
      const bool upper = (warp & m) != 0;
      float* mine = xchg + warp * kChunk + lane;
      const float* theirs = xchg + (warp ^ m) * kChunk + lane;
#pragma unroll
      for (int i = 0; i < kPerLane; ++i) mine[i * 32] = v[i];
      __syncthreads();
#pragma unroll
      for (int i = 0; i < kPerLane; ++i) {
        const float o = theirs[i * 32];
        v[i] = upper ? o - v[i] : v[i] + o;
      }
      __syncthreads();
    }
  }

  // Group range: 16 values in the lane, then the 8 lanes of the group.
  float mn = v[0], mx = v[0];
#pragma unroll
  for (int i = 1; i < kPerLane; ++i) {
    mn = fminf(mn, v[i]);
    mx = fmaxf(mx, v[i]);
  }
#pragma unroll
  for (int m = 1; m < 8; m <<= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xFFFFFFFFu, mn, m));
    mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, m));
  }
  // s = range / 15; the decisions take y / s as 15 y / range (one rounding).
  const float range = mx - mn;
  const float su = __fdiv_rn(range, 15.0f);
  float z = 0.f;
  if (su > 0.f) z = -rintf(__fdiv_rn(15.0f * mn, range));
  uint32_t packed[2] = {0u, 0u};
#pragma unroll
  for (int i = 0; i < kPerLane; ++i) {
    const float q = su > 0.f ? fminf(fmaxf(rintf(__fdiv_rn(15.0f * v[i], range)) + z, 0.f), 15.f) : 0.f;
    packed[i >> 3] |= static_cast<uint32_t>(q) << (4 * (i & 7));
  }
  if (!active) return;
  // Tiled layout: byte j of row r at ((r/32) (K/32) + j/16) 512 + (r%32) 16 + j%16.
  const int64_t j = c0 / 2;  // first byte of this lane's 16 codes (8 bytes)
  uint8_t* dst = a.codes + ((row >> 5) * (a.K / 32) + (j >> 4)) * 512 + (row & 31) * 16 + (j & 15);
  *reinterpret_cast<uint2*>(dst) = make_uint2(packed[0], packed[1]);
  if ((lane & 7) == 0) {
    const int64_t gi = row * a.Gq + c0 / kQGroup;
    a.scale[gi] = su * a.inv_sqrt_g;
    a.zero[gi] = z;
  }
}

// R[j][n] = sum over group j of the weight codes of row n, decoded from the
// interleaved sign-magnitude layout: per 8 channels in bytes B0..B3, Bj holds
// |q(c_2j)| in bits 0-2 with its sign in bit 7, |q(c_2j+1)| in bits 4-6, and
// in bit 3 the sign of q(c_(2j-1) mod 8).
__global__ void weight_group_sums_kernel(const uint8_t* __restrict__ codes, float* __restrict__ sums, int64_t N,
                                         int K, int group) {
  griddep_wait();
  griddep_launch_dependents();
  const int Gq = K / group;
  const int64_t id = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (id >= N * Gq) return;
  const int64_t jg = id / N;
  const int64_t n = id - jg * N;
  const uint8_t* tile_row = codes + (n >> 5) * (K / 32) * 512 + (n & 31) * 16;
  int sum = 0;
  for (int i = 0; i < group / 8; ++i) {
    const int64_t bo = jg * (group / 2) + 4 * i;
    const uint32_t u = *reinterpret_cast<const uint32_t*>(tile_row + (bo >> 4) * 512 + (bo & 15));
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const uint32_t byte = (u >> (8 * b)) & 0xFFu;
      const uint32_t next = (u >> (8 * ((b + 1) & 3))) & 0xFFu;
      const int m_even = static_cast<int>(byte & 7u), m_odd = static_cast<int>((byte >> 4) & 7u);
      sum += (byte & 0x80u) ? -m_even : m_even;
      sum += (next & 0x08u) ? -m_odd : m_odd;
    }
  }
  sums[jg * N + n] = static_cast<float>(sum);
}

int ilog2(int v) {
  int l = 0;
  while ((1 << l) < v) ++l;
  return l;
}

}  // namespace

extern "C" int offq_quantize_act_group(const void* x, int x_dtype, int64_t T, int64_t K, int64_t ldx, int32_t g,
                                       int32_t group, int32_t flags, uint8_t* codes, float* scale, float* zero,
                                       void* stream) {
  const int eb = elem_bytes(x_dtype);
  if (eb == 0 || T < 0 || K <= 0 || ldx < K || (flags & ~OFFQ_ROTATE) != 0) return OFFQ_ERR_INVALID_ARG;
  if (group != kQGroup) return group > 0 ? OFFQ_ERR_UNSUPPORTED : OFFQ_ERR_INVALID_ARG;
  if (K % kQGroup != 0) return OFFQ_ERR_INVALID_ARG;
  const bool rotate = (flags & OFFQ_ROTATE) != 0;
  if (rotate) {
    if (!is_pow2(g) || g < 32 || g > 8192 || K % g != 0) return OFFQ_ERR_INVALID_ARG;
  }
  if (K > kMaxGemmK || T > 0x3FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  if (T == 0) return OFFQ_OK;
  if (x == nullptr || codes == nullptr || scale == nullptr || zero == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(x, 16) || (ldx * eb) % 16 != 0 || !aligned(codes, 16) || !aligned(scale, 4) || !aligned(zero, 4))
    return OFFQ_ERR_MISALIGNED;
  GroupQuantArgs a{};
  a.x = x;
  a.ldx = ldx;
  a.T = T;
  a.K = static_cast<int>(K);
  a.Gq = static_cast<int>(K / kQGroup);
  a.log2g = rotate ? ilog2(g) : 0;
  a.inv_sqrt_g = rotate ? 1.0f / sqrtf(static_cast<float>(g)) : 1.0f;
  a.codes = codes;
  a.scale = scale;
  a.zero = zero;
  const int64_t items = T * ((K + kChunk - 1) / kChunk);
  // g >= 1024: a CTA holds whole blocks (g / 512 warps each); 16 warps for g = 8192.
  const int warps = rotate && g > kQWarps * kChunk ? static_cast<int>(g / kChunk) : kQWarps;
  const size_t smem = rotate && g > kChunk ? static_cast<size_t>(warps) * kChunk * sizeof(float) : 0;
  const dim3 grid(static_cast<unsigned>((items + warps - 1) / warps));
  const dim3 block(static_cast<unsigned>(warps * 32));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  switch (x_dtype) {
    case OFFQ_F32: return launch_pdl(quantize_group_kernel<float>, grid, block, smem, s, a);
    case OFFQ_BF16: return launch_pdl(quantize_group_kernel<__nv_bfloat16>, grid, block, smem, s, a);
    case OFFQ_F16: return launch_pdl(quantize_group_kernel<__half>, grid, block, smem, s, a);
    default: return OFFQ_ERR_INVALID_ARG;
  }
}

extern "C" int offq_weight_group_sums(const uint8_t* w_codes, int64_t N, int64_t K, int32_t group, float* w_groupsum,
                                      void* stream) {
  if (N < 1 || K <= 0 || !is_pow2(group) || group < 32 || K % group != 0 || K % 32 != 0)
    return OFFQ_ERR_INVALID_ARG;
  if (K > kMaxGemmK || N > 0x3FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  if (w_codes == nullptr || w_groupsum == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(w_codes, 16) || !aligned(w_groupsum, 4)) return OFFQ_ERR_MISALIGNED;
  const int64_t units = N * (K / group);
  const int threads = 256;
  return launch_pdl(weight_group_sums_kernel, dim3(static_cast<unsigned>((units + threads - 1) / threads)),
                    dim3(threads), 0, static_cast<cudaStream_t>(stream), w_codes, w_groupsum, N,
                    static_cast<int>(K), static_cast<int>(group));
}
