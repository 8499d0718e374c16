// Offline transform builder (paper Sec. 3.1 top-1 PCA, Sec. 3.2 group-wise
// offsetting, Sec. 3.3 Steps 1-2): from calibration activations to the
// rotation M = U1 P1 H1 fused into the weights.
//
//   offq_top1_tokens      per sequence, the token of largest L-infinity norm
//   offq_top1_direction   leading eigenvector of X^T X by power iteration
//   offq_reflect_rows     A U1, U1 the reflection with U1 e_1 = v / |v|
//   offq_column_absmax    per-channel absolute maxima
//   offq_sorted_grouping  the sorted-grouping permutation (host)
//   offq_fuse_rotation    W U1 P1 blockdiag(H_g) / sqrt(g)
//
// None of these is on the timed inference path; they run once per model.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>
#include <cmath>
#include <numeric>
#include <type_traits>
#include <vector>

#include "offq.h"
#include "offq_device.cuh"
#include "offq_host.h"

namespace {

using namespace offq;

template <typename Tin>
__device__ __forceinline__ float to_f(Tin v) {
  if constexpr (std::is_same<Tin, float>::value) return v;
  else if constexpr (std::is_same<Tin, __nv_bfloat16>::value) return __bfloat162float(v);
  else return __half2float(v);
}

constexpr int kTopThreads = 256;
constexpr int kTopChunks = 16;  // CTAs per sequence in the scan

template <typename Tin>
__device__ __forceinline__ float absmax16b(const Tin* p) {
  const uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
  float m = 0.f;
  if constexpr (sizeof(Tin) == 4) {
#pragma unroll
    for (int k = 0; k < 4; ++k) m = fmaxf(m, fabsf(__uint_as_float(w[k])));
  } else {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      if constexpr (std::is_same<Tin, __nv_bfloat16>::value) {
        m = fmaxf(m, fmaxf(fabsf(__uint_as_float(w[k] << 16)), fabsf(__uint_as_float(w[k] & 0xFFFF0000u))));
      } else {
        const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[k]));
        m = fmaxf(m, fmaxf(fabsf(f.x), fabsf(f.y)));
      }
    }
  }
  return m;
}

// Pass 1: CTA (c, s) scans tokens c, c + kTopChunks, ... of sequence s, a warp
// per token (16-byte loads when the rows allow them), and leaves its largest
// L-inf norm and first token index in rows[s][2c], rows[s][2c + 1] (the output
// rows hold the partials until pass 2 overwrites them).
template <typename Tin>
__global__ void __launch_bounds__(kTopThreads) top1_scan_kernel(const Tin* __restrict__ x, int64_t L, int64_t D,
                                                                int64_t ld_token, int64_t ld_seq, int vec,
                                                                float* __restrict__ rows) {
  __shared__ float best_v[kTopThreads / 32];
  __shared__ int64_t best_i[kTopThreads / 32];
  griddep_wait();
  griddep_launch_dependents();
  const int64_t s = blockIdx.y;
  const int c = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const Tin* xs = x + s * ld_seq;
  constexpr int kPer16 = 16 / sizeof(Tin);
  float bv = -1.f;
  int64_t bi = 0;
  for (int64_t l = c + static_cast<int64_t>(warp) * kTopChunks; l < L; l += static_cast<int64_t>(kTopChunks) * (kTopThreads / 32)) {
    const Tin* row = xs + l * ld_token;
    float m = 0.f;
    if (vec) {
      for (int64_t d = static_cast<int64_t>(lane) * kPer16; d < D; d += 32 * kPer16) m = fmaxf(m, absmax16b(row + d));
    } else {
      for (int64_t d = lane; d < D; d += 32) m = fmaxf(m, fabsf(to_f(row[d])));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
    if (m > bv) {  // a warp visits its tokens in increasing order: first on ties
      bv = m;
      bi = l;
    }
  }
  if (lane == 0) {
    best_v[warp] = bv;
    best_i[warp] = bi;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float v = best_v[0];
    int64_t i = best_i[0];
    for (int w = 1; w < kTopThreads / 32; ++w)
      if (best_v[w] > v || (best_v[w] == v && best_i[w] < i)) {
        v = best_v[w];
        i = best_i[w];
      }
    rows[s * D + 2 * c] = v;
    rows[s * D + 2 * c + 1] = __int_as_float(static_cast<int>(i));
  }
}

// Pass 2: per sequence, the best of the partials (first index on ties), then
// that token copied into rows[s].
template <typename Tin>
__global__ void __launch_bounds__(kTopThreads) top1_pick_kernel(const Tin* __restrict__ x, int64_t L, int64_t D,
                                                                int64_t ld_token, int64_t ld_seq,
                                                                int32_t* __restrict__ index,
                                                                float* __restrict__ rows) {
  __shared__ int64_t sel;
  griddep_wait();
  griddep_launch_dependents();
  const int64_t s = blockIdx.x;
  if (threadIdx.x == 0) {
    float v = -2.f;
    int64_t i = 0;
    for (int c = 0; c < kTopChunks && c < L; ++c) {
      const float pv = rows[s * D + 2 * c];
      const int64_t pi = __float_as_int(rows[s * D + 2 * c + 1]);
      if (pv > v || (pv == v && pi < i)) {
        v = pv;
        i = pi;
      }
    }
    sel = i;
    index[s] = static_cast<int32_t>(i);
  }
  __syncthreads();
  const Tin* row = x + s * ld_seq + sel * ld_token;
  for (int64_t d = threadIdx.x; d < D; d += kTopThreads) rows[s * D + d] = to_f(row[d]);
}

// u[n] = X[n] . v, one warp per row.
__global__ void matvec_rows_kernel(const float* __restrict__ X, int64_t N, int64_t D, const float* __restrict__ v,
                                   float* __restrict__ u) {
  griddep_wait();
  griddep_launch_dependents();
  const int64_t n = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (n >= N) return;
  float acc = 0.f;
  for (int64_t d = lane; d < D; d += 32) acc = fmaf(X[n * D + d], v[d], acc);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
  if (lane == 0) u[n] = acc;
}

// v[d] = sum_n X[n][d] u[n], one thread per column (rows in order).
__global__ void matvec_cols_kernel(const float* __restrict__ X, int64_t N, int64_t D, const float* __restrict__ u,
                                   float* __restrict__ v) {
  griddep_wait();
  griddep_launch_dependents();
  const int64_t d = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (d >= D) return;
  float acc = 0.f;
  for (int64_t n = 0; n < N; ++n) acc = fmaf(X[n * D + d], u[n], acc);
  v[d] = acc;
}

// v /= |v|; with fix_sign, also make the largest-magnitude entry positive.
__global__ void __launch_bounds__(1024) normalize_kernel(float* __restrict__ v, int64_t D, int fix_sign) {
  __shared__ float red[32];
  __shared__ float big[32];
  __shared__ int64_t bigi[32];
  griddep_wait();
  griddep_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float ss = 0.f, bm = -1.f;
  int64_t bi = 0;
  for (int64_t d = threadIdx.x; d < D; d += blockDim.x) {
    const float a = v[d];
    ss = fmaf(a, a, ss);
    if (fabsf(a) > bm) {
      bm = fabsf(a);
      bi = d;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    ss += __shfl_xor_sync(0xFFFFFFFFu, ss, o);
    const float om = __shfl_xor_sync(0xFFFFFFFFu, bm, o);
    const int64_t oi = __shfl_xor_sync(0xFFFFFFFFu, bi, o);
    if (om > bm || (om == bm && oi < bi)) {
      bm = om;
      bi = oi;
    }
  }
  if (lane == 0) {
    red[warp] = ss;
    big[warp] = bm;
    bigi[warp] = bi;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f, m = -1.f;
    int64_t mi = 0;
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) {
      t += red[w];
      if (big[w] > m || (big[w] == m && bigi[w] < mi)) {
        m = big[w];
        mi = bigi[w];
      }
    }
    float sc = t > 0.f ? 1.0f / sqrtf(t) : 0.f;
    if (fix_sign && v[mi] < 0.f) sc = -sc;
    red[0] = sc;
  }
  __syncthreads();
  const float sc = red[0];
  for (int64_t d = threadIdx.x; d < D; d += blockDim.x) v[d] *= sc;
}

// Shared by the row kernels: the reflection's unit w direction pieces. With
// vh = v / |v|: w = vh - e_1, |w|^2 = 2 - 2 vh_0, and a U1 = a - 2 (a.w) w / |w|^2.
__device__ __forceinline__ float block_sum(float x, float* red) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
  __syncthreads();
  if (lane == 0) red[warp] = x;
  __syncthreads();
  float t = 0.f;
  for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) t += red[w];
  return t;
}

// out[r] = A[r] U1 (reflection), and with perm / g also the permutation and
// the normalised block Hadamard; one CTA per row, the row in shared memory.
__global__ void __launch_bounds__(1024) row_transform_kernel(const float* __restrict__ A, int64_t D,
                                                             const float* __restrict__ v,
                                                             const int32_t* __restrict__ perm, int log2g,
                                                             float* __restrict__ out) {
  extern __shared__ float buf[];  // 2 D floats
  __shared__ float red[32];
  griddep_wait();
  griddep_launch_dependents();
  const int64_t r = blockIdx.x;
  const float* a = A + r * D;
  float* x = buf;
  float* y = buf + D;
  float vv = 0.f, av = 0.f;
  for (int64_t d = threadIdx.x; d < D; d += blockDim.x) {
    const float ad = a[d], vd = v[d];
    x[d] = ad;
    vv = fmaf(vd, vd, vv);
    av = fmaf(ad, vd, av);
  }
  vv = block_sum(vv, red);
  av = block_sum(av, red);
  const float inv = vv > 0.f ? 1.0f / sqrtf(vv) : 0.f;
  const float v0 = v[0] * inv;
  const float ww = 2.f - 2.f * v0;                    // |vh - e_1|^2
  const float aw = av * inv - x[0];                   // a . (vh - e_1), x[0] read before any write
  const float coef = ww > 1e-30f ? 2.f * aw / ww : 0.f;
  __syncthreads();
  for (int64_t d = threadIdx.x; d < D; d += blockDim.x) {
    const float wd = v[d] * inv - (d == 0 ? 1.f : 0.f);
    x[d] = fmaf(-coef, wd, x[d]);
  }
  __syncthreads();
  if (perm == nullptr) {
    for (int64_t d = threadIdx.x; d < D; d += blockDim.x) out[r * D + d] = x[d];
    return;
  }
  for (int64_t d = threadIdx.x; d < D; d += blockDim.x) y[d] = x[perm[d]];
  __syncthreads();
  // Sylvester transform of every block of 2^log2g entries, in place in y.
  for (int b = 0; b < log2g; ++b) {
    const int64_t h = int64_t{1} << b;
    for (int64_t i = threadIdx.x; i < D / 2; i += blockDim.x) {
      const int64_t lo = (i / h) * 2 * h + (i % h);
      const float p = y[lo], q = y[lo + h];
      y[lo] = p + q;
      y[lo + h] = p - q;
    }
    __syncthreads();
  }
  const float hs = 1.0f / sqrtf(static_cast<float>(int64_t{1} << log2g));
  for (int64_t d = threadIdx.x; d < D; d += blockDim.x) out[r * D + d] = y[d] * hs;
}

// mag[d] = max_r |A[r][d]|, one thread per column.
__global__ void column_absmax_kernel(const float* __restrict__ A, int64_t R, int64_t D, float* __restrict__ mag) {
  griddep_wait();
  griddep_launch_dependents();
  const int64_t d = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (d >= D) return;
  float m = 0.f;
  for (int64_t r = 0; r < R; ++r) m = fmaxf(m, fabsf(A[r * D + d]));
  mag[d] = m;
}

constexpr int64_t kMaxRowD = 16384;  // two rows of floats in shared memory

}  // namespace

extern "C" int offq_top1_tokens(const void* x, int dtype, int64_t S, int64_t L, int64_t D, int64_t ld_token,
                                int64_t ld_seq, int32_t* index, float* rows, void* stream) {
  const int eb = elem_bytes(dtype);
  if (eb == 0 || S < 0 || L < 1 || D < 1 || ld_token < D || ld_seq < L * ld_token) return OFFQ_ERR_INVALID_ARG;
  if (D < 2 * kTopChunks) return OFFQ_ERR_UNSUPPORTED;  // the partials live in rows[s]
  if (L > 0x7FFFFFFF || S > 65535) return OFFQ_ERR_UNSUPPORTED;
  if (S == 0) return OFFQ_OK;
  if (x == nullptr || index == nullptr || rows == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(x, eb) || !aligned(index, 4) || !aligned(rows, 4)) return OFFQ_ERR_MISALIGNED;
  const int vec = aligned(x, 16) && (ld_token * eb) % 16 == 0 && (ld_seq * eb) % 16 == 0 && (D * eb) % 16 == 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const dim3 scan_grid(kTopChunks, static_cast<unsigned>(S)), pick_grid(static_cast<unsigned>(S)), block(kTopThreads);
  int rc;
  switch (dtype) {
    case OFFQ_F32: {
      const float* p = static_cast<const float*>(x);
      rc = launch_pdl(top1_scan_kernel<float>, scan_grid, block, 0, s, p, L, D, ld_token, ld_seq, vec, rows);
      return rc != OFFQ_OK ? rc : launch_pdl(top1_pick_kernel<float>, pick_grid, block, 0, s, p, L, D, ld_token,
                                             ld_seq, index, rows);
    }
    case OFFQ_BF16: {
      const __nv_bfloat16* p = static_cast<const __nv_bfloat16*>(x);
      rc = launch_pdl(top1_scan_kernel<__nv_bfloat16>, scan_grid, block, 0, s, p, L, D, ld_token, ld_seq, vec, rows);
      return rc != OFFQ_OK ? rc : launch_pdl(top1_pick_kernel<__nv_bfloat16>, pick_grid, block, 0, s, p, L, D,
                                             ld_token, ld_seq, index, rows);
    }
    case OFFQ_F16: {
      const __half* p = static_cast<const __half*>(x);
      rc = launch_pdl(top1_scan_kernel<__half>, scan_grid, block, 0, s, p, L, D, ld_token, ld_seq, vec, rows);
      return rc != OFFQ_OK ? rc : launch_pdl(top1_pick_kernel<__half>, pick_grid, block, 0, s, p, L, D, ld_token,
                                             ld_seq, index, rows);
    }
    default: return OFFQ_ERR_INVALID_ARG;
  }
}

extern "C" int offq_top1_direction(const float* X, int64_t N, int64_t D, int32_t iters, const float* v0, float* v,
                                   float* proj, void* stream) {
  if (N < 1 || D < 1 || iters < 1) return OFFQ_ERR_INVALID_ARG;
  if (N > 0x7FFFFFFF || D > 0x7FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  if (X == nullptr || v0 == nullptr || v == nullptr || proj == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(X, 4) || !aligned(v0, 4) || !aligned(v, 4) || !aligned(proj, 4)) return OFFQ_ERR_MISALIGNED;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(v, v0, D * sizeof(float), cudaMemcpyDeviceToDevice, s) != cudaSuccess) return OFFQ_ERR_CUDA;
  const dim3 rows_grid(static_cast<unsigned>((N * 32 + 255) / 256)), cols_grid(static_cast<unsigned>((D + 255) / 256));
  int rc = launch_pdl(normalize_kernel, dim3(1), dim3(1024), 0, s, v, D, 0);
  for (int it = 0; it < iters && rc == OFFQ_OK; ++it) {
    rc = launch_pdl(matvec_rows_kernel, rows_grid, dim3(256), 0, s, X, N, D, static_cast<const float*>(v), proj);
    if (rc == OFFQ_OK) rc = launch_pdl(matvec_cols_kernel, cols_grid, dim3(256), 0, s, X, N, D,
                                       static_cast<const float*>(proj), v);
    if (rc == OFFQ_OK) rc = launch_pdl(normalize_kernel, dim3(1), dim3(1024), 0, s, v, D, it == iters - 1 ? 1 : 0);
  }
  if (rc == OFFQ_OK)
    rc = launch_pdl(matvec_rows_kernel, rows_grid, dim3(256), 0, s, X, N, D, static_cast<const float*>(v), proj);
  return rc;
}

extern "C" int offq_reflect_rows(const float* A, int64_t R, int64_t D, const float* v, float* out, void* stream) {
  if (R < 0 || D < 1) return OFFQ_ERR_INVALID_ARG;
  if (D > kMaxRowD || R > 0x7FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  if (R == 0) return OFFQ_OK;
  if (A == nullptr || v == nullptr || out == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(A, 4) || !aligned(v, 4) || !aligned(out, 4)) return OFFQ_ERR_MISALIGNED;
  const size_t smem = 2 * static_cast<size_t>(D) * sizeof(float);
  if (cudaFuncSetAttribute(row_transform_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return OFFQ_ERR_CUDA;
  return launch_pdl(row_transform_kernel, dim3(static_cast<unsigned>(R)), dim3(1024), smem,
                    static_cast<cudaStream_t>(stream), A, D, v, static_cast<const int32_t*>(nullptr), 0, out);
}

extern "C" int offq_column_absmax(const float* A, int64_t R, int64_t D, float* mag, void* stream) {
  if (R < 1 || D < 1) return OFFQ_ERR_INVALID_ARG;
  if (A == nullptr || mag == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(A, 4) || !aligned(mag, 4)) return OFFQ_ERR_MISALIGNED;
  return launch_pdl(column_absmax_kernel, dim3(static_cast<unsigned>((D + 255) / 256)), dim3(256), 0,
                    static_cast<cudaStream_t>(stream), A, R, D, mag);
}

extern "C" int offq_sorted_grouping(const float* mag, int64_t D, int32_t G, int32_t* perm) {
  if (D < 1 || G < 1 || D % G != 0 || mag == nullptr || perm == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (D > 0x7FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  std::vector<int64_t> order(static_cast<size_t>(D));
  std::iota(order.begin(), order.end(), int64_t{0});
  auto a = [&](int64_t i) { return std::fabs(static_cast<double>(mag[i])); };
  std::stable_sort(order.begin(), order.end(), [&](int64_t i, int64_t j) { return a(i) > a(j); });
  std::vector<int64_t> rest(order.begin() + G, order.end());
  std::stable_sort(rest.begin(), rest.end(), [&](int64_t i, int64_t j) { return a(i) < a(j); });
  const int64_t size = D / G;
  for (int64_t gi = 0; gi < G; ++gi) {
    perm[gi * size] = static_cast<int32_t>(order[static_cast<size_t>(gi)]);
    for (int64_t k = 1; k < size; ++k)
      perm[gi * size + k] = static_cast<int32_t>(rest[static_cast<size_t>(gi * (size - 1) + k - 1)]);
  }
  return OFFQ_OK;
}

extern "C" int offq_fuse_rotation(const float* W, int64_t N, int64_t D, const float* v, const int32_t* perm,
                                  int32_t g, float* out, void* stream) {
  if (N < 0 || D < 1 || !is_pow2(g) || g < 2 || D % g != 0) return OFFQ_ERR_INVALID_ARG;
  if (D > kMaxRowD || N > 0x7FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  if (N == 0) return OFFQ_OK;
  if (W == nullptr || v == nullptr || perm == nullptr || out == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(W, 4) || !aligned(v, 4) || !aligned(perm, 4) || !aligned(out, 4)) return OFFQ_ERR_MISALIGNED;
  int log2g = 0;
  while ((1 << log2g) < g) ++log2g;
  const size_t smem = 2 * static_cast<size_t>(D) * sizeof(float);
  if (cudaFuncSetAttribute(row_transform_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return OFFQ_ERR_CUDA;
  return launch_pdl(row_transform_kernel, dim3(static_cast<unsigned>(N)), dim3(1024), smem,
                    static_cast<cudaStream_t>(stream), W, D, v, perm, log2g, out);
}
