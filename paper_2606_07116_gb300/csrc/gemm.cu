// W4A4 GEMM of the OffQ path (offq_w4a4_linear) on the 5th-generation tensor
// cores of sm_103a, with the dequant + offset epilogue fused.
//
//   y[t][n] = s_w[n] * ( s_a[t] * acc'[t][n] + sum_b (o[t][b] - 8 s_a[t]) * R[b][n] )
//   acc'[t][n] = sum_k (q_a[t][k] + 8) * q_w[n][k]
//
// acc' is what the tensor cores accumulate: activation codes are stored as
// u = q + 8 (1..15) and weight codes as sign-magnitude q (-7..7). Both widen to
// E4M3 bytes whose values are exact integers times 2^-9: bytes 0x00..0x0F are
// the values 0..15 * 2^-9 (subnormals and the first binade share one step), and
// the sign bit negates. Every product and partial sum is then an integer times
// 2^-18 below 2^24 * 2^-18 for K <= 65536, exact in the fp32 accumulator. The
// "+8" is removed in the epilogue with the weight block row sums R, together
// with the offsets: sum_b 8 s_a R[b][n] = 8 s_a sum_k q_w[n][k].
//
// Persistent CTAs (one per SM), tile 128 (tokens) x 256 (channels), k-tile 128
// codes. Warp roles:
//   warp 0       TMA producer: packed int4 tiles of A and B into a 4-stage ring
//   warp 1       TMEM allocation and the single-thread MMA issuer
//   warps 2-9    widen packed codes to E4M3 tiles in the 128-byte-swizzled
//                K-major layout of the MMA (2-stage ring)
//   warps 10-13  epilogue from TMEM (each warp owns one 32-lane quarter of the
//                accumulator); two accumulator buffers (2 x 256 columns) let the
//                epilogue of a tile overlap the main loop of the next
// Every wait is bounded; a wait that runs out aborts the CTA and records
// OFFQ_ERR_TIMEOUT in the device status word.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <mutex>

#include "offq.h"
#include "offq_device.cuh"
#include "offq_host.h"

namespace {

using namespace offq;

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 128;  // codes per k-tile (128 fp8 bytes = one swizzle row)
constexpr int kPackStages = 4;
constexpr int kF8Stages = 2;
constexpr int kConvWarps = 8;
constexpr int kEpiWarps = 4;
constexpr int kConvThreads = kConvWarps * 32;
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr int kFirstConvWarp = 2;
constexpr int kFirstEpiWarp = kFirstConvWarp + kConvWarps;
constexpr int kThreads = (kFirstEpiWarp + kEpiWarps) * 32;
constexpr int kAccCols = BN;          // fp32 accumulator columns per buffer
constexpr int kTmemCols = 2 * kAccCols;  // double-buffered accumulator
constexpr int kMaxEpilogueG = 2048;

constexpr int kAPack = BM * BK / 2;  // 8 KB
constexpr int kBPack = BN * BK / 2;  // 16 KB
constexpr int kAF8 = BM * BK;        // 16 KB
constexpr int kBF8 = BN * BK;        // 32 KB

constexpr int kOffF8A = 0;
constexpr int kOffF8B = kOffF8A + kF8Stages * kAF8;
constexpr int kOffPackA = kOffF8B + kF8Stages * kBF8;
constexpr int kOffPackB = kOffPackA + kPackStages * kAPack;
constexpr int kOffBars = kOffPackB + kPackStages * kBPack;
constexpr int kNumBars = 2 * kPackStages + 2 * kF8Stages + 4;
constexpr int kOffMisc = kOffBars + kNumBars * 8;
constexpr int kSmemBytes = kOffMisc + 64 + 1024;  // + alignment slack for the 1024-byte base

static_assert(kOffPackA % 1024 == 0 && kOffF8B % 1024 == 0, "MMA tiles need 1024-byte alignment");
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
static_assert(BM * 4 % kConvThreads == 0 && BN * 4 % kConvThreads == 0, "even converter split");

constexpr uint32_t kIdesc = idesc_e4m3_f32(BM, BN);

struct GemmParams {
  const float* a_scale;
  const float* a_offset;  // [T][G] or nullptr
  const float* w_scale;
  const float* rowsum;    // [G][N]
  void* out;
  int64_t ldo;
  int32_t* acc_debug;
  int* status;
  int T, N, K, G, out_dtype;
  int m_tiles, n_tiles;
  int vec_ok;  // rowsum and w_scale rows are 16-byte aligned (float4 loads allowed)
};

__device__ __forceinline__ bool mbar_wait_teardown(uint32_t bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (clock64() - t0 > kWaitCycles) return false;
  }
  return true;
}

// Eight activation codes (u = q + 8 nibbles) -> eight E4M3 bytes, ordered
// [c0 c2 c4 c6 | c1 c3 c5 c7]: zero-extending a nibble gives the E4M3 byte of
// u * 2^-9.
__device__ __forceinline__ void widen_act(uint32_t w, uint32_t& lo, uint32_t& hi) {
  lo = w & 0x0F0F0F0Fu;
  hi = (w >> 4) & 0x0F0F0F0Fu;
}

// Eight weight codes (interleaved sign-magnitude) -> eight E4M3 bytes in the
// same channel order: sign at bit 7 and magnitude at bits 0-2 of each byte.
__device__ __forceinline__ void widen_weight(uint32_t w, uint32_t& lo, uint32_t& hi) {
  lo = w & 0x87878787u;
  hi = __funnelshift_r(w, w, 4) & 0x87878787u;
}

__device__ __forceinline__ void sts128(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 r;
  asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "r"(addr)
               : "memory");
  return r;
}

template <int OUT, int CW>
__device__ __forceinline__ void store_out(void* out, int64_t off, const float* y, int nvalid) {
  if (OUT == OFFQ_F32) {
    float* o = static_cast<float*>(out) + off;
    if (nvalid == CW) {
#pragma unroll
      for (int i = 0; i < CW / 4; ++i)
        *reinterpret_cast<float4*>(o + 4 * i) = make_float4(y[4 * i], y[4 * i + 1], y[4 * i + 2], y[4 * i + 3]);
    } else {
#pragma unroll
      for (int i = 0; i < CW; ++i)
        if (i < nvalid) o[i] = y[i];
    }
  } else {
    uint32_t p[CW / 2];
#pragma unroll
    for (int i = 0; i < CW / 2; ++i) {
      if (OUT == OFFQ_BF16) {
        const __nv_bfloat162 h = __floats2bfloat162_rn(y[2 * i], y[2 * i + 1]);
        p[i] = *reinterpret_cast<const uint32_t*>(&h);
      } else {
        const __half2 h = __floats2half2_rn(y[2 * i], y[2 * i + 1]);
        p[i] = *reinterpret_cast<const uint32_t*>(&h);
      }
    }
    uint16_t* o = static_cast<uint16_t*>(out) + off;
    if (nvalid == CW) {
#pragma unroll
      for (int i = 0; i < CW / 8; ++i)
        *reinterpret_cast<uint4*>(o + 8 * i) = make_uint4(p[4 * i], p[4 * i + 1], p[4 * i + 2], p[4 * i + 3]);
    } else {
#pragma unroll
      for (int i = 0; i < CW; ++i)
        if (i < nvalid) o[i] = static_cast<uint16_t>(p[i >> 1] >> (16 * (i & 1)));
    }
  }
}

// Persistent kernel: CTA b processes tiles b, b + gridDim.x, ... (tile index =
// m_tile * n_tiles + n_tile). The k-tile pipeline counters run across tiles, and
// the accumulator alternates between two TMEM buffers so the epilogue of one tile
// overlaps the main loop of the next.
template <int OUT>
__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_kernel(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_b,
                     const GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (base - raw);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nk = (p.K + BK - 1) / BK;
  const int num_tiles = p.m_tiles * p.n_tiles;

  const uint32_t bar0 = base + kOffBars;
  auto full_pack = [&](int s) { return bar0 + 8u * s; };
  auto empty_pack = [&](int s) { return bar0 + 8u * (kPackStages + s); };
  auto full_f8 = [&](int s) { return bar0 + 8u * (2 * kPackStages + s); };
  auto empty_f8 = [&](int s) { return bar0 + 8u * (2 * kPackStages + kF8Stages + s); };
  auto acc_full = [&](int b) { return bar0 + 8u * (2 * kPackStages + 2 * kF8Stages + b); };
  auto acc_empty = [&](int b) { return bar0 + 8u * (2 * kPackStages + 2 * kF8Stages + 2 + b); };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kOffMisc);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + kOffMisc + 16);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kPackStages; ++s) {
      mbar_init(full_pack(s), 1);
      mbar_init(empty_pack(s), kConvThreads);
    }
    for (int s = 0; s < kF8Stages; ++s) {
      mbar_init(full_f8(s), kConvThreads);
      mbar_init(empty_f8(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full(b), 1);
      mbar_init(acc_empty(b), kEpiThreads);
    }
    *abort = 0;
    mbar_fence_init();
    tma_prefetch_desc(&tmap_a);
    tma_prefetch_desc(&tmap_b);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  int issued = 0;     // producer: k-tiles whose TMA loads were issued (global count)
  int mma_tiles = 0;  // MMA issuer: tiles whose accumulation was committed

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      int g = 0;
      for (int tile = blockIdx.x; tile < num_tiles && !*abort; tile += gridDim.x) {
        const int m0 = (tile / p.n_tiles) * BM;
        const int n0 = (tile % p.n_tiles) * BN;
        for (int kt = 0; kt < nk; ++kt, ++g) {
          const int s = g % kPackStages;
          const uint32_t ph = (g / kPackStages) & 1;
          if (!mbar_wait(empty_pack(s), ph ^ 1, abort)) break;
          mbar_arrive_expect_tx(full_pack(s), kAPack + kBPack);
          tma_load_2d(base + kOffPackA + s * kAPack, &tmap_a, full_pack(s), kt * (BK / 2), m0);
          tma_load_2d(base + kOffPackB + s * kBPack, &tmap_b, full_pack(s), kt * (BK / 2), n0);
          issued = g + 1;
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int g = 0, lt = 0;
      for (int tile = blockIdx.x; tile < num_tiles && !*abort; tile += gridDim.x, ++lt) {
        const int ab = lt & 1;
        if (!mbar_wait(acc_empty(ab), ((lt >> 1) & 1) ^ 1, abort)) break;
        tc_fence_after();
        const uint32_t acc = tmem + ab * kAccCols;
        bool ok = true;
        for (int kt = 0; kt < nk; ++kt, ++g) {
          const int s = g % kF8Stages;
          const uint32_t ph = (g / kF8Stages) & 1;
          if (!mbar_wait(full_f8(s), ph, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_addr = base + kOffF8A + s * kAF8;
          const uint32_t b_addr = base + kOffF8B + s * kBF8;
#pragma unroll
          for (int kk = 0; kk < BK / 32; ++kk) {
            mma_f8f6f4(acc, smem_desc_sw128(a_addr + 32 * kk), smem_desc_sw128(b_addr + 32 * kk), kIdesc,
                       (kt | kk) != 0 ? 1u : 0u);
          }
          mma_commit(empty_f8(s));
        }
        mma_commit(acc_full(ab));
        mma_tiles = lt + 1;
        if (!ok) break;
      }
    }
  } else if (warp < kFirstEpiWarp) {
    // ---------------- widen packed codes to E4M3 operand tiles ----------------
    const int ct = threadIdx.x - kFirstConvWarp * 32;
    int g = 0;
    for (int tile = blockIdx.x; tile < num_tiles && !*abort; tile += gridDim.x) {
      for (int kt = 0; kt < nk; ++kt, ++g) {
        const int ps = g % kPackStages;
        const uint32_t pph = (g / kPackStages) & 1;
        const int fs = g % kF8Stages;
        const uint32_t fph = (g / kF8Stages) & 1;
        if (!mbar_wait(full_pack(ps), pph, abort)) break;
        if (!mbar_wait(empty_f8(fs), fph ^ 1, abort)) break;
        const uint32_t pa = base + kOffPackA + ps * kAPack;
        const uint32_t pb = base + kOffPackB + ps * kBPack;
        const uint32_t fa = base + kOffF8A + fs * kAF8;
        const uint32_t fb = base + kOffF8B + fs * kBF8;
#pragma unroll
        for (int it = 0; it < BM * 4 / kConvThreads; ++it) {
          const int i = ct + it * kConvThreads;
          const int r = i >> 2, j = i & 3;
          const uint4 w = lds128(pa + i * 16);
          uint32_t a0, a1, a2, a3, b0, b1, b2, b3;
          widen_act(w.x, a0, a1);
          widen_act(w.y, a2, a3);
          widen_act(w.z, b0, b1);
          widen_act(w.w, b2, b3);
          sts128(fa + r * 128 + (((2 * j) ^ (r & 7)) << 4), a0, a1, a2, a3);
          sts128(fa + r * 128 + (((2 * j + 1) ^ (r & 7)) << 4), b0, b1, b2, b3);
        }
#pragma unroll
        for (int it = 0; it < BN * 4 / kConvThreads; ++it) {
          const int i = ct + it * kConvThreads;
          const int r = i >> 2, j = i & 3;
          const uint4 w = lds128(pb + i * 16);
          uint32_t a0, a1, a2, a3, b0, b1, b2, b3;
          widen_weight(w.x, a0, a1);
          widen_weight(w.y, a2, a3);
          widen_weight(w.z, b0, b1);
          widen_weight(w.w, b2, b3);
          sts128(fb + r * 128 + (((2 * j) ^ (r & 7)) << 4), a0, a1, a2, a3);
          sts128(fb + r * 128 + (((2 * j + 1) ^ (r & 7)) << 4), b0, b1, b2, b3);
        }
        fence_proxy_async_smem();
        mbar_arrive(empty_pack(ps));
        mbar_arrive(full_f8(fs));
      }
    }
  } else {
    // ---------------- epilogue ----------------
    const int quarter = warp & 3;  // TMEM lanes this warp may read
    const int rl = quarter * 32 + lane;
    const int G = p.G;
    int lt = 0;
    for (int tile = blockIdx.x; tile < num_tiles && !*abort; tile += gridDim.x, ++lt) {
      const int ab = lt & 1;
      const int m0 = (tile / p.n_tiles) * BM;
      const int n0 = (tile % p.n_tiles) * BN;
      if (!mbar_wait(acc_full(ab), (lt >> 1) & 1, abort)) break;
      tc_fence_after();
      const int t = m0 + rl;
      const bool row_ok = t < p.T;
      const float sa = row_ok ? __ldg(p.a_scale + t) : 0.f;
      const bool has_off = p.a_offset != nullptr && row_ok;
      const float* orow = has_off ? p.a_offset + static_cast<int64_t>(t) * G : p.a_scale;
      const float o0 = (has_off ? __ldg(orow) : 0.f) - 8.0f * sa;
      const uint32_t acc_tm = tmem + ab * kAccCols + (static_cast<uint32_t>(quarter * 32) << 16);
      constexpr int CW = 16;  // accumulator columns per TMEM load
      for (int c = 0; c < BN / CW; ++c) {
        uint32_t acc[CW];
        tmem_ld_16cols(acc_tm + c * CW, acc);
        tmem_ld_wait();
        const int nb = n0 + c * CW;
        if (!row_ok || nb >= p.N) continue;
        const int nvalid = p.N - nb < CW ? p.N - nb : CW;
        float y[CW];
        if (nvalid == CW && p.vec_ok) {
          const float4* r4 = reinterpret_cast<const float4*>(p.rowsum + nb);
#pragma unroll
          for (int q4 = 0; q4 < CW / 4; ++q4) {
            const float4 rv = __ldg(r4 + q4);
            y[4 * q4] = o0 * rv.x; y[4 * q4 + 1] = o0 * rv.y; y[4 * q4 + 2] = o0 * rv.z; y[4 * q4 + 3] = o0 * rv.w;
          }
          for (int b = 1; b < G; ++b) {
            const float ob = (has_off ? __ldg(orow + b) : 0.f) - 8.0f * sa;
            const float4* rb4 = reinterpret_cast<const float4*>(p.rowsum + static_cast<int64_t>(b) * p.N + nb);
#pragma unroll
            for (int q4 = 0; q4 < CW / 4; ++q4) {
              const float4 rv = __ldg(rb4 + q4);
              y[4 * q4] = fmaf(ob, rv.x, y[4 * q4]);
              y[4 * q4 + 1] = fmaf(ob, rv.y, y[4 * q4 + 1]);
              y[4 * q4 + 2] = fmaf(ob, rv.z, y[4 * q4 + 2]);
              y[4 * q4 + 3] = fmaf(ob, rv.w, y[4 * q4 + 3]);
            }
          }
          const float4* w4 = reinterpret_cast<const float4*>(p.w_scale + nb);
#pragma unroll
          for (int q4 = 0; q4 < CW / 4; ++q4) {
            const float4 wv = __ldg(w4 + q4);
            const float sw4[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const int jj = 4 * q4 + e;
              const float accf = __uint_as_float(acc[jj]) * 262144.0f;  // exact: * 2^18
              y[jj] = sw4[e] * fmaf(sa, accf, y[jj]);
            }
          }
        } else {
#pragma unroll
          for (int jj = 0; jj < CW; ++jj) y[jj] = jj < nvalid ? o0 * __ldg(p.rowsum + nb + jj) : 0.f;
          for (int b = 1; b < G; ++b) {
            const float ob = (has_off ? __ldg(orow + b) : 0.f) - 8.0f * sa;
            const float* rb = p.rowsum + static_cast<int64_t>(b) * p.N + nb;
#pragma unroll
            for (int jj = 0; jj < CW; ++jj)
              if (jj < nvalid) y[jj] = fmaf(ob, __ldg(rb + jj), y[jj]);
          }
#pragma unroll
          for (int jj = 0; jj < CW; ++jj) {
            const float accf = __uint_as_float(acc[jj]) * 262144.0f;
            y[jj] = jj < nvalid ? __ldg(p.w_scale + nb + jj) * fmaf(sa, accf, y[jj]) : 0.f;
          }
        }
        store_out<OUT, CW>(p.out, static_cast<int64_t>(t) * p.ldo + nb, y, nvalid);
        if (p.acc_debug != nullptr) {
          int32_t* d = p.acc_debug + static_cast<int64_t>(t) * p.N + nb;
#pragma unroll
          for (int jj = 0; jj < CW; ++jj)
            if (jj < nvalid) d[jj] = __float2int_rn(__uint_as_float(acc[jj]) * 262144.0f);
        }
      }
      tc_fence_before();
      mbar_arrive(acc_empty(ab));
    }
  }

  // ---------------- teardown ----------------
  if (*abort && warp == 0 && lane == 0) {
    // Let TMA copies still in flight land before the CTA's shared memory goes away.
    for (int g = issued - kPackStages < 0 ? 0 : issued - kPackStages; g < issued; ++g)
      mbar_wait_teardown(full_pack(g % kPackStages), (g / kPackStages) & 1);
  }
  if (*abort && warp == 1 && lane == 0 && mma_tiles > 0) {
    const int lt = mma_tiles - 1;
    mbar_wait_teardown(acc_full(lt & 1), (lt >> 1) & 1);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && *abort && p.status != nullptr) atomicExch(p.status, kErrTimeout);
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  return fn;
}

// 2-D map over a [rows][row_bytes] byte matrix, box = 64 bytes x box_rows.
bool make_code_map(CUtensorMap* m, const void* ptr, int64_t rows, int64_t row_bytes, int box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return false;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(row_bytes), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(row_bytes)};
  const cuuint32_t box[2] = {BK / 2, static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(ptr), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int num_sms() {
  static int sms[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  if (sms[dev] == 0) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    sms[dev] = v;
  }
  return sms[dev];
}

template <int OUT>
int launch_gemm(const CUtensorMap& ma, const CUtensorMap& mb, const GemmParams& p, cudaStream_t s) {
  auto kern = w4a4_gemm_kernel<OUT>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [&] {
    attr_err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  });
  if (attr_err != cudaSuccess) return OFFQ_ERR_CUDA;
  const int sms = num_sms();
  if (sms <= 0) return OFFQ_ERR_CUDA;
  const int tiles = p.m_tiles * p.n_tiles;
  const int grid = tiles < sms ? tiles : sms;
  kern<<<grid, kThreads, kSmemBytes, s>>>(ma, mb, p);
  return launch_status();
}

}  // namespace

extern "C" int offq_w4a4_linear(const uint8_t* a_codes, const float* a_scale, const float* a_offset, int64_t T,
                                int64_t N, int64_t K, int32_t g, const uint8_t* w_codes, const float* w_scale,
                                const float* w_offsum, void* out, int out_dtype, int64_t ldo, int32_t* acc_debug,
                                void* stream) {
  const int ob = elem_bytes(out_dtype);
  if (ob == 0 || T < 0 || N < 1 || !is_pow2(g) || g < 32 || g > 8192) return OFFQ_ERR_INVALID_ARG;
  if (K <= 0 || K % g != 0 || K % 32 != 0 || ldo < N) return OFFQ_ERR_INVALID_ARG;
  if (K > kMaxGemmK || T > 0x7FFFFFFF / 2 || N > 0x7FFFFFFF / 2) return OFFQ_ERR_UNSUPPORTED;
  if (K / g > kMaxEpilogueG) return OFFQ_ERR_UNSUPPORTED;
  if (T == 0) return OFFQ_OK;
  if (a_codes == nullptr || a_scale == nullptr || w_codes == nullptr || w_scale == nullptr || w_offsum == nullptr ||
      out == nullptr)
    return OFFQ_ERR_INVALID_ARG;
  if (!aligned(a_codes, 16) || !aligned(w_codes, 16) || !aligned(out, 16) || (ldo * ob) % 16 != 0 ||
      !aligned(a_scale, 4) || !aligned(w_scale, 4) || !aligned(w_offsum, 4) ||
      (a_offset != nullptr && !aligned(a_offset, 4)) || (acc_debug != nullptr && !aligned(acc_debug, 4)))
    return OFFQ_ERR_MISALIGNED;

  CUtensorMap ma, mb;
  if (!make_code_map(&ma, a_codes, T, K / 2, BM) || !make_code_map(&mb, w_codes, N, K / 2, BN))
    return OFFQ_ERR_CUDA;
  GemmParams p{};
  p.a_scale = a_scale;
  p.a_offset = a_offset;
  p.w_scale = w_scale;
  p.rowsum = w_offsum;
  p.out = out;
  p.ldo = ldo;
  p.acc_debug = acc_debug;
  p.status = device_status_ptr();
  p.T = static_cast<int>(T);
  p.N = static_cast<int>(N);
  p.K = static_cast<int>(K);
  p.G = static_cast<int>(K / g);
  p.out_dtype = out_dtype;
  p.m_tiles = static_cast<int>((T + BM - 1) / BM);
  p.vec_ok = aligned(w_offsum, 16) && aligned(w_scale, 16) && (N % 4 == 0);
  p.n_tiles = static_cast<int>((N + BN - 1) / BN);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  switch (out_dtype) {
    case OFFQ_F32: return launch_gemm<OFFQ_F32>(ma, mb, p, s);
    case OFFQ_BF16: return launch_gemm<OFFQ_BF16>(ma, mb, p, s);
    case OFFQ_F16: return launch_gemm<OFFQ_F16>(ma, mb, p, s);
    default: return OFFQ_ERR_INVALID_ARG;
  }
}
