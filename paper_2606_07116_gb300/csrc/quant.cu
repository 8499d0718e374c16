// Row quantizers of the OffQ path: the online activation quantizer
// (offq_quantize_act), the KV-cache quantizer (offq_kv4_quantize) and the
// offline weight preparation (offq_prepare_weight).
//
// Per row and per block of g channels (paper Sec. 3.2, Eq. 4-5; Sec. 3 Eq. 1):
//   y = x H_g / sqrt(g),  o = mean(y) = x[0] / sqrt(g),  r = y - o,
//   s = max|r| / 7 over the row,  q = rne(r / s),  stored as q + 8.
//
// With the rotation on, the kernel uses that the first row of the Sylvester
// Hadamard is all ones: zeroing x[0] before the transform yields the
// unnormalised residual sqrt(g) * r directly, and the offset is x[0]/sqrt(g).
// The 1/sqrt(g) factor cancels in r / s, so it is applied only to the stored
// scale and offset.
//
// Kernel layouts (per g = 2^L; the Hadamard is a Kronecker product of 2x2
// stages, so the stages may run in any order):
//  * g <= 1024 (quantize_rows_kernel): a thread owns E = 2^ceil((L+3)/2)
//    elements and TPB = g / E threads share a block. Pass 1 loads 16-byte
//    vectors (8 channels, coalesced across the block's threads) and runs the
//    stages of every index bit it holds except bit 0; one swizzled transpose
//    through shared memory gives each thread E contiguous channels, pass 2 runs
//    the stages of bit 0 and of the bits that were spread over threads, and the
//    thread packs its E codes into whole 16-byte chunks of the code buffer.
//    Packed fp32x2 instructions take register pairs that differ in index bit 0,
//    so the bit-0 stage alone runs on scalar adds.
//  * g >= 2048 (quantize_rows_wide_kernel): E = 2^ceil((L+1)/2) elements per
//    thread, the same two passes with pass 2 keeping the lowest one or two
//    index bits, and codes staged in shared memory before the 16-byte writes.
//  * Both come in a one-shot form (a CTA per group of rows) and, for one-head
//    inputs with more row groups than SMs, a persistent form whose CTAs stage
//    their next groups in shared memory by bulk async copies (cp.async.bulk,
//    mbarrier completion) while they compute the current one.
//  * No rotation and one block of g >= 1024 per row
//    (quantize_rows_bulk_kernel): a persistent kernel whose warps stream rows
//    through their own rings of shared-memory slots; offset and absmax from one
//    sweep of the slot, codes from a second. Rows too long for the ring take
//    quantize_rows_stream_kernel (a warp per row, the row in registers).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <type_traits>

#include "offq.h"
#include "offq_device.cuh"
#include "offq_host.h"

namespace {

using namespace offq;

struct QuantArgs {
  const void* x;
  int64_t ld_t;     // elements between consecutive tokens
  int64_t ld_h;     // elements between consecutive heads (0 when H == 1)
  int64_t rows;     // tokens * heads
  int H;            // heads per token (1 for activations)
  int K;            // channels per row
  int G;            // blocks per row
  int flags;
  uint8_t* codes;   // [rows][K/2]
  float* scale;     // [rows]
  float* offset;    // [rows][G] or nullptr
  float inv_sqrt_g; // 1/sqrt(g) with the rotation, else 1
  float scale_mul;  // inv_sqrt_g / 7
  int tpr;          // threads per row (a power of two <= 32 or a multiple of 32)
  int rows_per_cta;
  int tiled;        // codes in the 32-row tiled operand layout (else row-major)
  int* status;      // device status word (bounded waits that run out write here)
  int ring_slots;   // persistent forms: slots of rows_per_cta rows each (1 to 3)
  long long wait_cycles;  // persistent forms: budget of a wait for a staged row (kWaitCycles unless a test sets it)
  uint8_t* shifts;  // MXFP4 form: tiled block shifts (else nullptr)
  int g;            // MXFP4 form: the offset block
};

template <int L>
struct WideGeo {
  static constexpr int kLogE = (L + 2) / 2;
  static constexpr int kE = 1 << kLogE;       // elements per thread
  static constexpr int kP = L - kLogE;        // log2 threads per block
  static constexpr int kTPB = 1 << kP;        // threads per block
  static constexpr int kQ = kLogE - kP;       // low index bits kept in pass 2 (1 or 2)
  static constexpr int kNC = kE / 8;          // 8-element chunks per thread in pass 1
  static constexpr int kMaxThreads = kLogE >= 7 ? 256 : (kLogE == 6 ? 512 : 1024);
  static_assert(kQ >= 1 && kQ <= 2, "pass-2 layout keeps one or two low bits");
  static_assert(kP >= 2, "swizzle assumes at least four threads per block");
};

// ---------------------------------------------------------------------------
// Loads of one 8-element chunk (16 bytes of bf16/f16, 32 bytes of f32).
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 ldg_nc_v4(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ void bf16x2_to_f32(uint32_t w, float& lo, float& hi) {
  lo = __uint_as_float(w << 16);
  hi = __uint_as_float(w & 0xFFFF0000u);
}

__device__ __forceinline__ void f16x2_to_f32(uint32_t w, float& lo, float& hi) {
  __half2 h;
  *reinterpret_cast<uint32_t*>(&h) = w;
  const float2 f = __half22float2(h);
  lo = f.x;
  hi = f.y;
}

__device__ __forceinline__ void load_chunk8(const __nv_bfloat16* p, float* v) {
  const uint4 w = ldg_nc_v4(p);
  bf16x2_to_f32(w.x, v[0], v[1]);
  bf16x2_to_f32(w.y, v[2], v[3]);
  bf16x2_to_f32(w.z, v[4], v[5]);
  bf16x2_to_f32(w.w, v[6], v[7]);
}

__device__ __forceinline__ void load_chunk8(const __half* p, float* v) {
  const uint4 w = ldg_nc_v4(p);
  f16x2_to_f32(w.x, v[0], v[1]);
  f16x2_to_f32(w.y, v[2], v[3]);
  f16x2_to_f32(w.z, v[4], v[5]);
  f16x2_to_f32(w.w, v[6], v[7]);
}

__device__ __forceinline__ void load_chunk8(const float* p, float* v) {
  const uint4 a = ldg_nc_v4(p);
  const uint4 b = ldg_nc_v4(p + 4);
  v[0] = __uint_as_float(a.x); v[1] = __uint_as_float(a.y);
  v[2] = __uint_as_float(a.z); v[3] = __uint_as_float(a.w);
  v[4] = __uint_as_float(b.x); v[5] = __uint_as_float(b.y);
  v[6] = __uint_as_float(b.z); v[7] = __uint_as_float(b.w);
}

// ---------------------------------------------------------------------------
// In-register fast Walsh-Hadamard stages (Sylvester order: (a, b) -> (a+b, a-b)
// for the pair of indices that differ in one bit, the lower index first).
// ---------------------------------------------------------------------------
template <int E, int BIT>
__device__ __forceinline__ void fwht_stage(float (&v)[E]) {
  constexpr int m = 1 << BIT;
  if constexpr (BIT == 0) {
#pragma unroll
    for (int r = 0; r < E; r += 4) butterfly2(v[r], v[r + 2], v[r + 1], v[r + 3]);
  } else {
#pragma unroll
    for (int r = 0; r < E; r += 2) {
      if ((r & m) == 0) butterfly2(v[r], v[r + 1], v[r + m], v[r + m + 1]);
    }
  }
}

template <int E, int LO, int HI>
__device__ __forceinline__ void fwht_bits(float (&v)[E]) {
  if constexpr (LO < HI) {
    fwht_stage<E, LO>(v);
    fwht_bits<E, LO + 1, HI>(v);
  }
}

// Swizzle of the row's fp32 transpose buffer: flips bits 2-4 of the element
// index with higher bits so that both the pass-1 stores and the pass-2 loads of
// a warp spread over the 32 banks. Bits >= 5 are untouched, so it is a bijection.
template <int P>
__device__ __forceinline__ int swz(int idx) {
  return idx ^ (((idx >> 5) & 1) << 2) ^ (((idx >> (3 + P)) & 3) << 3);
}

// Reduction over aligned groups of W consecutive threads (W a power of two up
// to 32, or a multiple of 32). All threads of the CTA must call it.
template <bool kMax>
__device__ __forceinline__ float group_reduce(float v, int W, float* scratch) {
  const int lane = threadIdx.x & 31;
  const int wl = W < 32 ? W : 32;
  for (int o = wl >> 1; o > 0; o >>= 1) {
    const float u = __shfl_xor_sync(0xFFFFFFFFu, v, o);
    v = kMax ? fmaxf(v, u) : v + u;
  }
  if (W > 32) {
    const int warp = threadIdx.x >> 5;
    if (lane == 0) scratch[warp] = v;
    __syncthreads();
    const int nw = W >> 5;
    const int first = (warp / nw) * nw;
    float acc = kMax ? 0.f : 0.f;
    for (int i = 0; i < nw; ++i) {
      const float u = scratch[first + i];
      acc = kMax ? fmaxf(acc, u) : acc + u;
    }
    v = acc;
    __syncthreads();
  }
  return v;
}

// Round-to-nearest-even of x*inv as the integer held in the low mantissa bits
// of fma(x, inv, 1.5 * 2^23 + 8) (the classic magic-number rounding: the
// addend puts the result's ulp at 1). For |x*inv| <= 7 the low nibble is
// rne(x*inv) + 8, the activation code.
constexpr float kMagic8 = 12582920.0f;

// The bit pattern of such a rounded value is 0x4B400000 | (q + 8): bits 4-21
// are zero, so (u1 << 4) + u0 has the byte of two codes in its low 8 bits.
// pack_codes8 returns the 32-bit code word of channels c0..c7 (code of
// channel 2k in the low nibble of byte k, channel 2k+1 in the high nibble).
__device__ __forceinline__ uint32_t pack_codes8(uint32_t u0, uint32_t u1, uint32_t u2, uint32_t u3, uint32_t u4,
                                                uint32_t u5, uint32_t u6, uint32_t u7) {
  const uint32_t b0 = (u1 << 4) + u0, b1 = (u3 << 4) + u2, b2 = (u5 << 4) + u4, b3 = (u7 << 4) + u6;
  return __byte_perm(__byte_perm(b0, b1, 0x0040), __byte_perm(b2, b3, 0x0040), 0x5410);
}

// Packed subtraction {a0 - c, a1 - c}.
__device__ __forceinline__ void sub2(float& a0, float& a1, float c) {
  const uint64_t A = pack2(a0, a1);
  const uint64_t C = pack2(c, c);
  uint64_t R;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(R) : "l"(A), "l"(C));
  unpack2(R, a0, a1);
}

// Butterflies between registers r and r + 2^M (M >= 1) of every pair with bit M
// of r clear, two per packed instruction: the pair (v[r], v[r+1]) against
// (v[r+2^M], v[r+2^M+1]).
template <int E, int M>
__device__ __forceinline__ void fwht_reg_stage(float (&v)[E]) {
  static_assert(M >= 1, "register bit 0 pairs the packed lanes");
  constexpr int d = 1 << M;
#pragma unroll
  for (int r = 0; r < E; r += 2) {
    if ((r & d) == 0) butterfly2(v[r], v[r + 1], v[r + d], v[r + d + 1]);
  }
}

template <int E, int LO, int HI>
__device__ __forceinline__ void fwht_reg_stages(float (&v)[E]) {
  if constexpr (LO < HI) {
    fwht_reg_stage<E, LO>(v);
    fwht_reg_stages<E, LO + 1, HI>(v);
  }
}

// Pairwise sum of N values (a balanced tree of depth log2 N).
template <int N>
__device__ __forceinline__ float tree_sum(const float* v) {
  if constexpr (N == 1) {
    return v[0];
  } else {
    return tree_sum<N / 2>(v) + tree_sum<N / 2>(v + N / 2);
  }
}

// ---------------------------------------------------------------------------
// Row rings of the persistent kernels: shared-memory slots filled by bulk
// asynchronous copies (cp.async.bulk) whose bytes complete on an mbarrier.
// ---------------------------------------------------------------------------
constexpr size_t kMaxDynSmem = 226 * 1024;  // dynamic bytes; the static flag needs a few more

__device__ __forceinline__ void bulk_load_row(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}

// Rows [grp*R, grp*R + R) of a one-head input (those below a.rows) into the
// slot, row l at byte l * K * sizeof(Tin); one copy when the rows are
// contiguous. Called by one thread.
template <typename Tin>
__device__ __forceinline__ void ring_issue(const QuantArgs& a, int64_t grp, int R, uint8_t* slot, uint32_t bar) {
  const int64_t r0 = grp * R;
  const int n = static_cast<int>(a.rows - r0 < R ? a.rows - r0 : R);
  const uint32_t rb = static_cast<uint32_t>(a.K) * static_cast<uint32_t>(sizeof(Tin));
  const Tin* x = static_cast<const Tin*>(a.x);
  mbar_arrive_expect_tx(bar, static_cast<uint32_t>(n) * rb);
  if (a.ld_t == a.K) {
    bulk_load_row(smem_u32(slot), x + r0 * a.K, static_cast<uint32_t>(n) * rb, bar);
  } else {
    for (int l = 0; l < n; ++l) bulk_load_row(smem_u32(slot + static_cast<size_t>(l) * rb), x + (r0 + l) * a.ld_t, rb, bar);
  }
}

// The ring of a persistent row kernel: S slots of R rows, slot k at
// base + k * slot_bytes with its mbarrier at bar0 + 8 k. The CTA's i-th group
// (blockIdx.x + i * gridDim.x) lands in slot i mod S; s and phase name the slot
// of the group being consumed and the parity of its completion.
struct RowRing {
  uint8_t* base;
  uint32_t bar0;
  uint32_t slot_bytes;
  int S;
  int s;
  uint32_t phase;
  __device__ __forceinline__ uint8_t* slot() const { return base + static_cast<size_t>(s) * slot_bytes; }
  __device__ __forceinline__ uint32_t bar() const { return bar0 + 8u * static_cast<uint32_t>(s); }
  __device__ __forceinline__ void advance() {
    if (++s == S) {
      s = 0;
      phase ^= 1u;
    }
  }
};

// Thread 0 initialises the slots' barriers and issues the CTA's first S groups.
template <typename Tin>
__device__ __forceinline__ void ring_start(const QuantArgs& a, const RowRing& ring, int R, int64_t ngroups) {
  if (threadIdx.x != 0) return;
  for (int k = 0; k < ring.S; ++k) {
    const int64_t grp = blockIdx.x + static_cast<int64_t>(k) * gridDim.x;
    if (grp < ngroups) ring_issue<Tin>(a, grp, R, ring.base + static_cast<size_t>(k) * ring.slot_bytes, ring.bar0 + 8u * k);
  }
}

// A slot wait ran out somewhere in the CTA while consuming group grp: thread 0
// lets every copy still in flight land (bounded waits) and reports the timeout.
__device__ __forceinline__ void ring_fail(const RowRing& ring, int64_t grp, int64_t ngroups, int* status) {
  if (threadIdx.x != 0) return;
  for (int d = 0; d < ring.S; ++d) {
    if (grp + static_cast<int64_t>(d) * gridDim.x >= ngroups) break;
    const int k = (ring.s + d) % ring.S;
    const uint32_t parity = ring.s + d < ring.S ? ring.phase : (ring.phase ^ 1u);
    const long long t0 = clock64();
    while (!mbar_try_wait(ring.bar0 + 8u * k, parity) && clock64() - t0 < kWaitCycles) {
    }
  }
  if (status != nullptr) atomicExch(status, kErrTimeout);
}

// One 8-element chunk of a staged row (shared memory) as fp32.
__device__ __forceinline__ void load_chunk8_smem(const __nv_bfloat16* p, float* v) {
  const uint4 w = *reinterpret_cast<const uint4*>(p);
  bf16x2_to_f32(w.x, v[0], v[1]);
  bf16x2_to_f32(w.y, v[2], v[3]);
  bf16x2_to_f32(w.z, v[4], v[5]);
  bf16x2_to_f32(w.w, v[6], v[7]);
}

__device__ __forceinline__ void load_chunk8_smem(const __half* p, float* v) {
  const uint4 w = *reinterpret_cast<const uint4*>(p);
  f16x2_to_f32(w.x, v[0], v[1]);
  f16x2_to_f32(w.y, v[2], v[3]);
  f16x2_to_f32(w.z, v[4], v[5]);
  f16x2_to_f32(w.w, v[6], v[7]);
}

__device__ __forceinline__ void load_chunk8_smem(const float* p, float* v) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

// Geometry of quantize_rows_kernel (g = 2^L <= 512). E >= 2^(3+P) puts a
// thread's in-block position (pass-1 index bits 3..3+P-1) below the bits it
// holds in registers, so a pass-2 thread owns E contiguous channels.
template <int L>
struct NarrowGeo {
  static constexpr int kLogE = (L + 4) / 2;   // ceil((L + 3) / 2)
  static constexpr int kE = 1 << kLogE;       // elements per thread
  static constexpr int kP = L - kLogE;        // log2 threads per block
  static constexpr int kTPB = 1 << kP;
  static constexpr int kNC = kE / 8;          // 8-channel loads per thread
  // 128 blocks of g = 256 or 64 of g = 512; 128 registers of data per thread
  // (g = 1024) need the 255-register limit of 256-thread CTAs.
  static constexpr int kMaxThreads = kE >= 128 ? 256 : 512;
  static_assert(3 + kP <= kLogE && kP >= 1 && kE >= 16, "narrow geometry");
};

// Transpose swizzle of quantize_rows_kernel (float index within the CTA's
// buffer): bits 3-4 take the two lowest pass-2 thread bits, bit 2 the parity of
// the block and of bit 5. Only bits >= 5 feed bits 2-4, so it is a bijection;
// for g = 128 and 256 every quarter-warp of the pass-1 stores and of the
// pass-2 loads hits eight distinct 16-byte bank groups, for g = 64 and 512 at
// most two lanes share one. g = 32 keeps the plain layout.
template <int L, int LOGE>
__device__ __forceinline__ int swz_narrow(int idx) {
  if constexpr (L == 5) {
    return idx;
  } else {
    return idx ^ (((idx >> LOGE) & 3) << 3) ^ ((((idx >> L) ^ (idx >> 5)) & 1) << 2);
  }
}

// kRing: persistent form for one-head inputs. The CTA's rows_per_cta rows of
// group grp (rows grp*R ..) are staged in a shared-memory slot by bulk copies;
// once pass 1 has read them, the copy of the CTA's next group is issued, so
// its HBM reads overlap this group's arithmetic.
template <int L, typename Tin, bool kRing>
__global__ void __launch_bounds__(NarrowGeo<L>::kMaxThreads) quantize_rows_kernel(const QuantArgs a) {
  using GG = NarrowGeo<L>;
  constexpr int E = GG::kE, P = GG::kP, TPB = GG::kTPB, NC = GG::kNC, LOGE = GG::kLogE;
  constexpr int g = 1 << L;

  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ int abort_flag;
  float* red = reinterpret_cast<float*>(smem);          // 32 floats for group_reduce
  float* buf = reinterpret_cast<float*>(smem + 128);    // [rows_per_cta][K] fp32 transpose
  const bool rotate = (a.flags & OFFQ_ROTATE) != 0;
  const bool offs = (a.flags & OFFQ_OFFSET) != 0;
  const int K = a.K;
  const int R = a.rows_per_cta;
  // kRing: ring_slots slots of [R][K] inputs after the transpose buffer, then their barriers.
  RowRing ring;
  ring.base = smem + 128 + static_cast<size_t>(R) * K * 4;
  ring.slot_bytes = static_cast<uint32_t>(R) * K * sizeof(Tin);
  ring.S = a.ring_slots;
  ring.bar0 = smem_u32(ring.base + static_cast<size_t>(ring.S) * ring.slot_bytes);
  ring.s = 0;
  ring.phase = 0;

  const int tid = threadIdx.x;
  const int lrow = tid / a.tpr;
  const int j = tid - lrow * a.tpr;
  const int b = j >> P;
  const int t = j & (TPB - 1);
  const int64_t ngroups = (a.rows + R - 1) / R;
  int64_t grp = blockIdx.x;
  if constexpr (kRing) {
    if (tid == 0) {
      abort_flag = 0;
      for (int k = 0; k < ring.S; ++k) mbar_init(ring.bar0 + 8u * k, 1);
      mbar_fence_init();
    }
    __syncthreads();
  }
  griddep_wait();
  griddep_launch_dependents();
  if constexpr (kRing) ring_start<Tin>(a, ring, R, ngroups);

  while (true) {
    const int64_t row = grp * R + lrow;
    const bool row_ok = row < a.rows;
    const bool active = row_ok && (j < a.G * TPB);

    // Pass 1: register 8i + c holds channel 8t + 8 TPB i + c of block b.
    float v[E];
    if constexpr (kRing) {
      const bool ok = mbar_wait_for(ring.bar(), ring.phase, &abort_flag, a.wait_cycles);
      if (ok && active) {
        const Tin* p = reinterpret_cast<const Tin*>(ring.slot()) + static_cast<size_t>(lrow) * K + b * g + 8 * t;
#pragma unroll
        for (int i = 0; i < NC; ++i) load_chunk8_smem(p + i * 8 * TPB, &v[8 * i]);
      } else {
#pragma unroll
        for (int r = 0; r < E; ++r) v[r] = 0.f;
      }
      if (!__syncthreads_and(ok)) {
        ring_fail(ring, grp, ngroups, a.status);
        return;
      }
      // Every thread has read the slot: it takes the group S turns ahead.
      const int64_t next = grp + static_cast<int64_t>(ring.S) * gridDim.x;
      if (tid == 0 && next < ngroups) ring_issue<Tin>(a, next, R, ring.slot(), ring.bar());
      ring.advance();
    } else {
      if (active) {
        const int64_t tok = row / a.H;
        const int64_t h = row - tok * a.H;
        const Tin* p = static_cast<const Tin*>(a.x) + tok * a.ld_t + h * a.ld_h + static_cast<int64_t>(b) * g + 8 * t;
#pragma unroll
        for (int i = 0; i < NC; ++i) load_chunk8(p + i * 8 * TPB, &v[8 * i]);
      } else {
#pragma unroll
        for (int r = 0; r < E; ++r) v[r] = 0.f;
      }
    }

    float off = 0.f;
    if (rotate) {
      // Offset = x[block start] / sqrt(g); removing it first leaves the residual.
      if (offs && t == 0) {
        off = v[0];
        v[0] = 0.f;
      }
      fwht_reg_stages<E, 1, LOGE>(v);   // channel bits 1, 2 and 3+P .. L-1
    } else if (offs) {
      // Block mean by a pairwise tree (depth log2(E) in the thread, P across threads).
      off = group_reduce<false>(tree_sum<E>(v), TPB, red) * (1.0f / static_cast<float>(g));
    }

    const int base = lrow * K + b * g;
    if (active) {
#pragma unroll
      for (int i = 0; i < NC; ++i) {
        const int e0 = base + 8 * t + 8 * TPB * i;
        *reinterpret_cast<float4*>(buf + swz_narrow<L, LOGE>(e0)) =
            make_float4(v[8 * i], v[8 * i + 1], v[8 * i + 2], v[8 * i + 3]);
        *reinterpret_cast<float4*>(buf + swz_narrow<L, LOGE>(e0 + 4)) =
            make_float4(v[8 * i + 4], v[8 * i + 5], v[8 * i + 6], v[8 * i + 7]);
      }
    }
    __syncwarp();  // a block's TPB <= 8 threads share one warp
    // Pass 2: register r holds channel E t + r of block b.
    if (active) {
#pragma unroll
      for (int m = 0; m < E / 4; ++m) {
        const float4 f = *reinterpret_cast<const float4*>(buf + swz_narrow<L, LOGE>(base + E * t + 4 * m));
        v[4 * m] = f.x;
        v[4 * m + 1] = f.y;
        v[4 * m + 2] = f.z;
        v[4 * m + 3] = f.w;
      }
    }
    if (rotate) {
#pragma unroll
      for (int r = 0; r < E; r += 2) {   // channel bit 0
        const float x0 = v[r], x1 = v[r + 1];
        v[r] = x0 + x1;
        v[r + 1] = x0 - x1;
      }
      fwht_reg_stages<E, 3, 3 + P>(v);   // channel bits 3 .. 3+P-1
    } else if (offs) {
#pragma unroll
      for (int r = 0; r < E; r += 2) sub2(v[r], v[r + 1], off);
    }

    // Per-row absmax of the residual.
    float mx[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int r = 0; r < E; ++r) mx[r & 3] = fmaxf(mx[r & 3], fabsf(v[r]));
    float m = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
    m = group_reduce<true>(m, a.tpr, red);
    const float inv = m > 0.f ? __fdiv_rn(7.0f, m) : 0.f;

#pragma unroll
    for (int r = 0; r < E; r += 2) fma2(v[r], v[r + 1], inv, kMagic8);

    if (active) {
      uint32_t wd[E / 8];
#pragma unroll
      for (int w = 0; w < E / 8; ++w) {
        const float* q = &v[8 * w];
        wd[w] = pack_codes8(__float_as_uint(q[0]), __float_as_uint(q[1]), __float_as_uint(q[2]),
                            __float_as_uint(q[3]), __float_as_uint(q[4]), __float_as_uint(q[5]),
                            __float_as_uint(q[6]), __float_as_uint(q[7]));
      }
      const int es = b * g + E * t;              // first channel of the thread's run
      const int cpr = K / 32;                    // 16-byte chunks per row
      uint8_t* rdst = a.tiled ? a.codes + (row >> 5) * cpr * 512 + (row & 31) * 16
                              : a.codes + row * (K / 2);
      const int cstride = a.tiled ? 512 : 16;    // bytes between consecutive chunks of a row
      if constexpr (E >= 32) {
#pragma unroll
        for (int q = 0; q < E / 32; ++q) {
          *reinterpret_cast<uint4*>(rdst + ((es >> 5) + q) * cstride) =
              make_uint4(wd[4 * q], wd[4 * q + 1], wd[4 * q + 2], wd[4 * q + 3]);
        }
      } else {
        *reinterpret_cast<uint2*>(rdst + (es >> 5) * cstride + (es & 31) / 2) = make_uint2(wd[0], wd[1]);
      }
    }

    if (row_ok && j == 0) a.scale[row] = m * a.scale_mul;
    if (active && t == 0 && a.offset != nullptr) {
      a.offset[row * a.G + b] = offs ? (rotate ? off * a.inv_sqrt_g : off) : 0.f;
    }
    if constexpr (!kRing) break;
    grp += gridDim.x;
    if (grp >= ngroups) break;
  }
}

// kRing: persistent form for one-head inputs, as in quantize_rows_kernel (the
// slot follows the reduction scratch in shared memory).
template <int L, typename Tin, bool kRing>
__global__ void __launch_bounds__(WideGeo<L>::kMaxThreads) quantize_rows_wide_kernel(const QuantArgs a) {
  using GG = WideGeo<L>;
  constexpr int E = GG::kE, P = GG::kP, TPB = GG::kTPB, Q = GG::kQ, NC = GG::kNC, LOGE = GG::kLogE;
  constexpr int g = 1 << L;

  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ int abort_flag;
  const bool rotate = (a.flags & OFFQ_ROTATE) != 0;
  const bool offs = (a.flags & OFFQ_OFFSET) != 0;
  const int R = a.rows_per_cta;
  const int K = a.K;
  float* buf = reinterpret_cast<float*>(smem);                                  // [R][K] fp32 (rotate)
  uint8_t* cbuf = smem + (rotate ? static_cast<size_t>(R) * K * 4 : 0);         // [R][K/2] codes
  float* red = reinterpret_cast<float*>(cbuf + static_cast<size_t>(R) * (K / 2));
  // kRing: ring_slots slots of [R][K] inputs after the reduction scratch, then their barriers.
  RowRing ring;
  ring.base = reinterpret_cast<uint8_t*>(red + 32);
  ring.slot_bytes = static_cast<uint32_t>(R) * K * sizeof(Tin);
  ring.S = a.ring_slots;
  ring.bar0 = smem_u32(ring.base + static_cast<size_t>(ring.S) * ring.slot_bytes);
  ring.s = 0;
  ring.phase = 0;

  const int tid = threadIdx.x;
  const int lrow = tid / a.tpr;
  const int j = tid - lrow * a.tpr;
  const int b = j / TPB;
  const int t1 = j % TPB;
  const int64_t ngroups = (a.rows + R - 1) / R;
  int64_t grp = blockIdx.x;
  if constexpr (kRing) {
    if (tid == 0) {
      abort_flag = 0;
      for (int k = 0; k < ring.S; ++k) mbar_init(ring.bar0 + 8u * k, 1);
      mbar_fence_init();
    }
    __syncthreads();
  }
  griddep_wait();
  griddep_launch_dependents();
  if constexpr (kRing) ring_start<Tin>(a, ring, R, ngroups);

  while (true) {
    const int64_t row = grp * R + lrow;
    const bool row_ok = row < a.rows;
    const bool active = row_ok && (j < a.G * TPB);

    float v[E];
    if constexpr (kRing) {
      const bool ok = mbar_wait_for(ring.bar(), ring.phase, &abort_flag, a.wait_cycles);
      if (ok && active) {
        const Tin* p = reinterpret_cast<const Tin*>(ring.slot()) + static_cast<size_t>(lrow) * K + b * g + 8 * t1;
#pragma unroll
        for (int i = 0; i < NC; ++i) load_chunk8_smem(p + i * 8 * TPB, &v[8 * i]);
      } else {
#pragma unroll
        for (int r = 0; r < E; ++r) v[r] = 0.f;
      }
      if (!__syncthreads_and(ok)) {
        ring_fail(ring, grp, ngroups, a.status);
        return;
      }
      // Every thread has read the slot: it takes the group S turns ahead.
      const int64_t next = grp + static_cast<int64_t>(ring.S) * gridDim.x;
      if (tid == 0 && next < ngroups) ring_issue<Tin>(a, next, R, ring.slot(), ring.bar());
      ring.advance();
    } else {
      if (active) {
        const int64_t t = row / a.H;
        const int64_t h = row - t * a.H;
        const Tin* p = static_cast<const Tin*>(a.x) + t * a.ld_t + h * a.ld_h + static_cast<int64_t>(b) * g + 8 * t1;
#pragma unroll
        for (int i = 0; i < NC; ++i) load_chunk8(p + i * 8 * TPB, &v[8 * i]);
      } else {
#pragma unroll
        for (int r = 0; r < E; ++r) v[r] = 0.f;
      }
    }

    float off = 0.f;
    if (rotate) {
      // Offset = x[block start] / sqrt(g); removing it first leaves the residual.
      if (offs && t1 == 0) {
        off = v[0];
        v[0] = 0.f;
      }
      // Index bits {0,1,2} and {3+P, .., L-1}: bit 0 on scalar adds, the others
      // packed on the (even, odd) register pairs the loads produced.
#pragma unroll
      for (int r = 0; r < E; r += 2) {
        const float x0 = v[r], x1 = v[r + 1];
        v[r] = x0 + x1;
        v[r + 1] = x0 - x1;
      }
      fwht_reg_stages<E, 1, LOGE>(v);
      float* rb = buf + static_cast<size_t>(lrow) * K + static_cast<size_t>(b) * g;
      if (active) {
#pragma unroll
        for (int i = 0; i < NC; ++i) {
          const int e0 = 8 * t1 + 8 * TPB * i;
          *reinterpret_cast<float4*>(rb + swz<P>(e0)) = make_float4(v[8 * i], v[8 * i + 1], v[8 * i + 2], v[8 * i + 3]);
          *reinterpret_cast<float4*>(rb + swz<P>(e0 + 4)) =
              make_float4(v[8 * i + 4], v[8 * i + 5], v[8 * i + 6], v[8 * i + 7]);
        }
      }
      // A block's TPB threads share one warp (TPB <= 32) except for g = 8192.
      if constexpr (TPB <= 32) {
        __syncwarp();
      } else {
        __syncthreads();
      }
      if (active) {
#pragma unroll
        for (int hi = 0; hi < (1 << P); ++hi) {
          const int e = ((t1 & ((1 << (3 - Q)) - 1)) << Q) | (hi << 3) | ((t1 >> (3 - Q)) << (3 + P));
          if constexpr (Q == 2) {
            const float4 f = *reinterpret_cast<const float4*>(rb + swz<P>(e));
            v[4 * hi] = f.x; v[4 * hi + 1] = f.y; v[4 * hi + 2] = f.z; v[4 * hi + 3] = f.w;
          } else {
            const float2 f = *reinterpret_cast<const float2*>(rb + swz<P>(e));
            v[2 * hi] = f.x; v[2 * hi + 1] = f.y;
          }
        }
      }
      fwht_bits<E, Q, LOGE>(v);  // index bits {3, .., 3+P-1}
    } else if (offs) {
      // Block mean by a pairwise tree (depth log2(E) in the thread, P across threads).
      float s = tree_sum<E>(v);
      s = group_reduce<false>(s, TPB, red);
      off = s * (1.0f / static_cast<float>(g));
#pragma unroll
      for (int r = 0; r < E; ++r) v[r] -= off;
    }

    // Per-row absmax of the residual.
    float m = 0.f;
#pragma unroll
    for (int r = 0; r < E; ++r) m = fmaxf(m, fabsf(v[r]));
    m = group_reduce<true>(m, a.tpr, red);
    const float inv = m > 0.f ? __fdiv_rn(7.0f, m) : 0.f;

#pragma unroll
    for (int r = 0; r < E; r += 2) fma2(v[r], v[r + 1], inv, kMagic8);

    uint8_t* crow = cbuf + static_cast<size_t>(lrow) * (K / 2) + static_cast<size_t>(b) * (g / 2);
    if (active) {
      if (rotate) {
#pragma unroll
        for (int hi = 0; hi < (1 << P); ++hi) {
          const int e = ((t1 & ((1 << (3 - Q)) - 1)) << Q) | (hi << 3) | ((t1 >> (3 - Q)) << (3 + P));
          // Bits 4-21 of a rounded value are zero, so (u1 << 4) + u0 carries the
          // byte of two codes in its low 8 bits.
          if constexpr (Q == 2) {
            const uint32_t b0 = (__float_as_uint(v[4 * hi + 1]) << 4) + __float_as_uint(v[4 * hi]);
            const uint32_t b1 = (__float_as_uint(v[4 * hi + 3]) << 4) + __float_as_uint(v[4 * hi + 2]);
            *reinterpret_cast<uint16_t*>(crow + e / 2) = static_cast<uint16_t>(__byte_perm(b0, b1, 0x0040));
          } else {
            crow[e / 2] = static_cast<uint8_t>((__float_as_uint(v[2 * hi + 1]) << 4) + __float_as_uint(v[2 * hi]));
          }
        }
      } else {
#pragma unroll
        for (int i = 0; i < NC; ++i) {
          uint32_t w = 0;
#pragma unroll
          for (int e = 0; e < 8; ++e) w |= (__float_as_uint(v[8 * i + e]) & 0xFu) << (4 * e);
          *reinterpret_cast<uint32_t*>(crow + 4 * t1 + 4 * TPB * i) = w;
        }
      }
    }
    // Each block's TPB threads write the block's g/2 code bytes as 16-byte chunks.
    if constexpr (TPB <= 32) {
      __syncwarp();
    } else {
      __syncthreads();
    }
    if (active) {
      const int cpr = K / 32;       // 16-byte chunks per row
      const int cpb = g / 32;       // 16-byte chunks per block
      for (int c = t1; c < cpb; c += TPB) {
        const int cc = b * cpb + c;
        const uint4 w = *reinterpret_cast<const uint4*>(crow + c * 16);
        uint8_t* dst = a.tiled ? a.codes + ((row >> 5) * cpr + cc) * 512 + (row & 31) * 16
                               : a.codes + row * (K / 2) + cc * 16;
        *reinterpret_cast<uint4*>(dst) = w;
      }
    }

    if (row_ok && j == 0) a.scale[row] = m * a.scale_mul;
    if (active && t1 == 0 && a.offset != nullptr) {
      a.offset[row * a.G + b] = offs ? (rotate ? off * a.inv_sqrt_g : off) : 0.f;
    }
    if constexpr (!kRing) break;
    grp += gridDim.x;
    if (grp >= ngroups) break;
  }
}

// g = 1024 with the rotation, persistent: a warp per block of 1024 channels,
// 32 channels per lane, so a CTA of up to 28 warps holds whole rows in
// registers at 32 data registers a thread (the register file holds two rows
// of 28672 channels). Rows arrive in a ring of shared-memory slots filled by
// bulk copies. Channel e of a block has index bits e0..e9. Pass 1: lane l,
// register j holds e = l + 32 j (conflict-free 2- or 4-byte loads from the
// slot) and runs the stages of e5..e9; a transpose through the warp's 4 KB of
// shared memory gives lane l the channels e = 32 l + j, whose stages (e0..e4)
// pass 2 runs; the lane then owns one whole 16-byte code chunk. The row's
// absmax crosses warps through shared memory (one barrier per row group).
constexpr int k1kMaxWarps = 28;

template <typename Tin>
__device__ __forceinline__ float smem_elem(const Tin* p) {
  if constexpr (sizeof(Tin) == 4) {
    return *reinterpret_cast<const float*>(p);
  } else if constexpr (std::is_same<Tin, __nv_bfloat16>::value) {
    return __uint_as_float(static_cast<uint32_t>(*reinterpret_cast<const uint16_t*>(p)) << 16);
  } else {
    return __half2float(*p);
  }
}

// max(a, b, c) in one instruction.
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// Shared-memory accesses by 32-bit address.
__device__ __forceinline__ void sts_f32(uint32_t addr, float v) {
  asm volatile("st.shared.f32 [%0], %1;" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ float4 lds_f32x4(uint32_t addr) {
  float4 r;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(r.x), "=f"(r.y), "=f"(r.z), "=f"(r.w) : "r"(addr) : "memory");
  return r;
}

// Butterflies of register bit M of quantize_rows_1k_kernel, whose 32 values sit
// in 16 float2 pairs (register 2i in .x, 2i + 1 in .y): bit 0 within each pair,
// bit M >= 1 between pairs i and i + 2^(M-1), two lanes per packed add.
template <int M>
__device__ __forceinline__ void fwht1k_stage(float2 (&v)[16]) {
  if constexpr (M == 0) {
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = make_float2(v[i].x + v[i].y, v[i].x - v[i].y);
  } else {
    constexpr int d = 1 << (M - 1);
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      if ((i & d) == 0) {
        const float2 p = v[i], q = v[i + d];
        v[i] = __fadd2_rn(p, q);
        v[i + d] = __ffma2_rn(q, make_float2(-1.0f, -1.0f), p);  // p - q, one rounding
      }
    }
  }
}

__device__ __forceinline__ void fwht1k_pass(float2 (&v)[16]) {
  fwht1k_stage<0>(v);
  fwht1k_stage<1>(v);
  fwht1k_stage<2>(v);
  fwht1k_stage<3>(v);
  fwht1k_stage<4>(v);
}

template <typename Tin>
__global__ void __launch_bounds__(k1kMaxWarps * 32, 1) quantize_rows_1k_kernel(const QuantArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ int abort_flag;
  __shared__ float wmax[k1kMaxWarps];
  const int K = a.K, G = a.G, R = a.rows_per_cta;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int lrow = warp / G;
  const int b = warp - lrow * G;
  const bool offs = (a.flags & OFFQ_OFFSET) != 0;
  const uint32_t scr32 = smem_u32(smem) + 4096u * warp;  // the warp's transpose scratch
  RowRing ring;
  ring.base = smem + static_cast<size_t>(R) * G * 4096;
  ring.slot_bytes = static_cast<uint32_t>(R) * K * sizeof(Tin);
  ring.S = a.ring_slots;
  ring.bar0 = smem_u32(ring.base + static_cast<size_t>(ring.S) * ring.slot_bytes);
  ring.s = 0;
  ring.phase = 0;
  // Rows fit an int here (the launcher checks), so group and row indices are 32-bit.
  const int ngroups = static_cast<int>((a.rows + R - 1) / R);
  int grp = blockIdx.x;
  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int k = 0; k < ring.S; ++k) mbar_init(ring.bar0 + 8u * k, 1);
    mbar_fence_init();
  }
  __syncthreads();
  griddep_wait();
  griddep_launch_dependents();
  ring_start<Tin>(a, ring, R, ngroups);

  const int cpr = K / 32;
  const int cstride = a.tiled ? 512 : 16;
  const int blk_off = lrow * K + b * 1024 + lane;
  while (true) {
    const int row = grp * R + lrow;
    const bool row_ok = row < a.rows;
    // v[i].x: channel lane + 64 i, v[i].y: channel lane + 64 i + 32 (register j = 2i, 2i + 1).
    float2 v[16];
    const bool ok = mbar_wait_for(ring.bar(), ring.phase, &abort_flag, a.wait_cycles);
    if (ok && row_ok) {
      const Tin* p = reinterpret_cast<const Tin*>(ring.slot()) + blk_off;
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = make_float2(smem_elem(p + 64 * i), smem_elem(p + 64 * i + 32));
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = make_float2(0.f, 0.f);
    }
    // Offset = x[block start] / sqrt(g); removing it first leaves the residual.
    float off = 0.f;
    if (offs && lane == 0) {
      off = v[0].x;
      v[0].x = 0.f;
    }
    fwht1k_pass(v);  // channel bits 5..9
    // Transpose through the warp's scratch: channel e at float e ^ (((e >> 5) & 7) << 2)
    // (the 16-byte chunk index takes bits 5-7 as well, so the stores of one register
    // hit 32 banks and the float4 loads of a quarter-warp 8 distinct chunks). Register j
    // of lane l (e = l + 32 j) lands at byte 128 j + (4 l ^ 16 (j & 7)): eight lane bases,
    // the rest immediate offsets. Lane l then reads its row's float4 k at
    // 128 l + (16 k ^ 16 (l & 7)).
    {
      uint32_t wb[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) wb[q] = scr32 + ((4u * lane) ^ (16u * q));
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        sts_f32(wb[(2 * i) & 7] + 128u * (2 * i), v[i].x);
        sts_f32(wb[(2 * i + 1) & 7] + 128u * (2 * i + 1), v[i].y);
      }
    }
    __syncwarp();
    // Now register j = 4k + c holds channel 32 lane + j.
    {
      const uint32_t rb = scr32 + 128u * lane;
      const uint32_t rx = 16u * (lane & 7);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const float4 f = lds_f32x4(rb + ((16u * k) ^ rx));
        v[2 * k] = make_float2(f.x, f.y);
        v[2 * k + 1] = make_float2(f.z, f.w);
      }
    }
    fwht1k_pass(v);  // channel bits 0..4

    // Row absmax: the lane's, the warp's (non-negative floats order as their
    // bit patterns), then over the row's G warps.
    float mx0 = 0.f, mx1 = 0.f;
#pragma unroll
    for (int i = 0; i < 16; i += 2) {
      mx0 = fmax3(mx0, fabsf(v[i].x), fabsf(v[i].y));
      mx1 = fmax3(mx1, fabsf(v[i + 1].x), fabsf(v[i + 1].y));
    }
    const uint32_t wm = __reduce_max_sync(0xFFFFFFFFu, __float_as_uint(fmaxf(mx0, mx1)));
    if (lane == 0) wmax[warp] = __uint_as_float(wm);
    // One barrier per row group: the warps' maxima are visible, every thread has read
    // the slot (so it takes the group S turns ahead), and a wait that ran out anywhere
    // in the CTA is seen by all.
    if (!__syncthreads_and(ok)) {
      ring_fail(ring, grp, ngroups, a.status);
      return;
    }
    const int next = grp + ring.S * static_cast<int>(gridDim.x);
    if (threadIdx.x == 0 && next < ngroups) ring_issue<Tin>(a, next, R, ring.slot(), ring.bar());
    ring.advance();
    const float m = __uint_as_float(
        __reduce_max_sync(0xFFFFFFFFu, lane < G ? __float_as_uint(wmax[lrow * G + lane]) : 0u));
    const float inv = m > 0.f ? __fdiv_rn(7.0f, m) : 0.f;

    const float2 inv2 = make_float2(inv, inv), mag2 = make_float2(kMagic8, kMagic8);
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __ffma2_rn(v[i], inv2, mag2);
    uint32_t wd[4];
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float2* q = &v[4 * w];
      wd[w] = pack_codes8(__float_as_uint(q[0].x), __float_as_uint(q[0].y), __float_as_uint(q[1].x),
                          __float_as_uint(q[1].y), __float_as_uint(q[2].x), __float_as_uint(q[2].y),
                          __float_as_uint(q[3].x), __float_as_uint(q[3].y));
    }
    if (row_ok) {
      uint8_t* rdst = a.tiled ? a.codes + static_cast<int64_t>(row >> 5) * cpr * 512 + (row & 31) * 16
                              : a.codes + static_cast<int64_t>(row) * (K / 2);
      *reinterpret_cast<uint4*>(rdst + (b * 32 + lane) * cstride) = make_uint4(wd[0], wd[1], wd[2], wd[3]);
      if (b == 0 && lane == 0) a.scale[row] = m * a.scale_mul;
      if (lane == 0 && a.offset != nullptr) a.offset[static_cast<int64_t>(row) * G + b] = offs ? off * a.inv_sqrt_g : 0.f;
    }
    grp += gridDim.x;
    if (grp >= ngroups) break;
  }
}

// MXFP4 rows (the Sec. 3.4 extension), persistent, on the layout of
// quantize_rows_1k_kernel: a warp per 1024 channels, so after the rotation (or,
// without it, straight from the staged row) lane l holds the 32 consecutive
// channels 32 l + j of its warp's span, one whole MX block. Per row: offsets
// (the block-leading channel over sqrt(1024) with the rotation; without it the
// mean over g = 1024 m channels by a balanced tree, across the m warps of the
// block through shared memory), the residual, the lane's block exponent
// X = floor(log2 amax) - 2, the row's largest through shared memory (one
// barrier), X kept within 6 of it, then the codes by the E2M1 conversion
// instruction (round to nearest even, saturating at 6; a code of magnitude 0
// keeps sign 0), one 16-byte store of the block's codes and its shift byte.
// With the rotation the values are 32 r (unnormalised by sqrt(1024) = 2^5,
// exact), so their exponents are offset by 5.

// floor(log2(a)) for a normal positive fp32 a, from its exponent field.
__device__ __forceinline__ int floor_log2(float a) { return static_cast<int>((__float_as_uint(a) >> 23) & 0xFF) - 127; }

// 2^e as fp32 for -126 <= e <= 127.
__device__ __forceinline__ float pow2f(int e) { return __uint_as_float(static_cast<uint32_t>(e + 127) << 23); }

// Two fp32 values -> one byte of E2M1 codes (hi in bits 4-7, lo in bits 0-3).
__device__ __forceinline__ uint32_t e2m1x2(float hi, float lo) {
  uint16_t r;
  asm("{\n.reg .b8 t;\ncvt.rn.satfinite.e2m1x2.f32 t, %1, %2;\nmov.b16 %0, {t, 0};\n}" : "=h"(r) : "f"(hi), "f"(lo));
  return r;
}

// Clears the sign bit of every nibble whose magnitude bits are 0 (E2M1 -0 -> +0).
__device__ __forceinline__ uint32_t e2m1_clear_neg_zero(uint32_t w) {
  const uint32_t mag = w & 0x77777777u;
  const uint32_t nonzero = (mag + 0x77777777u) & 0x88888888u;  // bit 3 of each nibble: magnitude >= 1
  return mag | (w & nonzero);
}

template <typename Tin, bool kRot>
__global__ void __launch_bounds__(k1kMaxWarps * 32, 1) quantize_mx_1k_kernel(const QuantArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ int abort_flag;
  __shared__ float wpart[k1kMaxWarps];  // per-warp block sums (no rotation, g > 1024)
  __shared__ int wmaxx[k1kMaxWarps];    // per-warp largest block exponent (+ 1024)
  const int K = a.K, R = a.rows_per_cta;
  const int nbw = K / 1024;  // warps per row
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int lrow = warp / nbw;
  const int b = warp - lrow * nbw;          // 1024-channel span of this warp
  const int m = a.g / 1024;                 // warps per offset block (no rotation)
  const int G = a.G;
  const bool offs = (a.flags & OFFQ_OFFSET) != 0;
  const uint32_t scr32 = smem_u32(smem) + 4096u * warp;  // the warp's transpose scratch (rotation)
  RowRing ring;
  ring.base = smem + (kRot ? static_cast<size_t>(R) * nbw * 4096 : 0);
  ring.slot_bytes = static_cast<uint32_t>(R) * K * sizeof(Tin);
  ring.S = a.ring_slots;
  ring.bar0 = smem_u32(ring.base + static_cast<size_t>(ring.S) * ring.slot_bytes);
  ring.s = 0;
  ring.phase = 0;
  const int ngroups = static_cast<int>((a.rows + R - 1) / R);
  int grp = blockIdx.x;
  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int k = 0; k < ring.S; ++k) mbar_init(ring.bar0 + 8u * k, 1);
    mbar_fence_init();
  }
  __syncthreads();
  griddep_wait();
  griddep_launch_dependents();
  ring_start<Tin>(a, ring, R, ngroups);

  const int cpr = K / 32;
  const int nkt = K / 128;
  while (true) {
    const int row = grp * R + lrow;
    const bool row_ok = row < a.rows;
    float2 v[16];  // v[i] = channels (32 lane + 2i, 32 lane + 2i + 1) of the span, after pass 2
    const bool ok = mbar_wait_for(ring.bar(), ring.phase, &abort_flag, a.wait_cycles);
    float off = 0.f;
    if constexpr (kRot) {
      if (ok && row_ok) {
        const Tin* p = reinterpret_cast<const Tin*>(ring.slot()) + static_cast<size_t>(lrow) * K + b * 1024 + lane;
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = make_float2(smem_elem(p + 64 * i), smem_elem(p + 64 * i + 32));
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = make_float2(0.f, 0.f);
      }
      if (offs && lane == 0) {
        off = v[0].x;
        v[0].x = 0.f;
      }
      fwht1k_pass(v);  // channel bits 5..9
      {
        uint32_t wb[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) wb[q] = scr32 + ((4u * lane) ^ (16u * q));
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          sts_f32(wb[(2 * i) & 7] + 128u * (2 * i), v[i].x);
          sts_f32(wb[(2 * i + 1) & 7] + 128u * (2 * i + 1), v[i].y);
        }
      }
      __syncwarp();
      {
        const uint32_t rb = scr32 + 128u * lane;
        const uint32_t rx = 16u * (lane & 7);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const float4 f = lds_f32x4(rb + ((16u * k) ^ rx));
          v[2 * k] = make_float2(f.x, f.y);
          v[2 * k + 1] = make_float2(f.z, f.w);
        }
      }
      fwht1k_pass(v);  // channel bits 0..4
    } else {
      if (ok && row_ok) {
        const Tin* p = reinterpret_cast<const Tin*>(ring.slot()) + static_cast<size_t>(lrow) * K + b * 1024 + 32 * lane;
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          float f[8];
          load_chunk8_smem(p + 8 * c, f);
#pragma unroll
          for (int e = 0; e < 4; ++e) v[4 * c + e] = make_float2(f[2 * e], f[2 * e + 1]);
        }
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = make_float2(0.f, 0.f);
      }
      if (offs) {
        // Block mean over g = 1024 m channels: a tree over the lane's 32, the warp's
        // 32 lanes, then the m warps of the block.
        float2 t8[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) t8[i] = __fadd2_rn(v[i], v[i + 8]);
#pragma unroll
        for (int i = 0; i < 4; ++i) t8[i] = __fadd2_rn(t8[i], t8[i + 4]);
#pragma unroll
        for (int i = 0; i < 2; ++i) t8[i] = __fadd2_rn(t8[i], t8[i + 2]);
        t8[0] = __fadd2_rn(t8[0], t8[1]);
        float sum = t8[0].x + t8[0].y;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
        if (m > 1) {
          if (lane == 0) wpart[warp] = sum;
          __syncthreads();
          const int w0 = lrow * nbw + (b / m) * m;  // first warp of this offset block
          float part[8];
          for (int i = 0; i < 8; ++i) part[i] = i < m ? wpart[w0 + i] : 0.f;
          // m is a power of two <= 8: pairwise
          for (int h = 4; h > 0; h >>= 1)
            for (int i = 0; i < h; ++i) part[i] += part[i + h];
          sum = part[0];
          __syncthreads();  // wpart is read before the next row writes it
        }
        off = sum * (1.0f / static_cast<float>(a.g));
        const float2 o2 = make_float2(off, off);
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = __fadd2_rn(v[i], make_float2(-o2.x, -o2.y));
      }
    }

    // The lane's block exponent, then the row's largest.
    float mx0 = 0.f, mx1 = 0.f;
#pragma unroll
    for (int i = 0; i < 16; i += 2) {
      mx0 = fmax3(mx0, fabsf(v[i].x), fabsf(v[i].y));
      mx1 = fmax3(mx1, fabsf(v[i + 1].x), fabsf(v[i + 1].y));
    }
    const float amax = fmaxf(mx0, mx1);
    constexpr int kUnnorm = kRot ? 5 : 0;  // values are 2^5 r with the rotation
    const int xl = amax > 0.f ? floor_log2(amax) - 2 - kUnnorm : -1000;
    const uint32_t wx = __reduce_max_sync(0xFFFFFFFFu, static_cast<uint32_t>(xl + 1024));
    if (lane == 0) wmaxx[warp] = static_cast<int>(wx);
    if (!__syncthreads_and(ok)) {
      ring_fail(ring, grp, ngroups, a.status);
      return;
    }
    const int next = grp + ring.S * static_cast<int>(gridDim.x);
    if (threadIdx.x == 0 && next < ngroups) ring_issue<Tin>(a, next, R, ring.slot(), ring.bar());
    ring.advance();
    int xmax = static_cast<int>(__reduce_max_sync(0xFFFFFFFFu, lane < nbw ? static_cast<uint32_t>(wmaxx[lrow * nbw + lane]) : 0u)) - 1024;
    if (xmax < -900) xmax = 0;  // an all-zero row: any exponent
    const int xlo = xmax - 6;
    const int X = xl > xlo ? xl : xlo;
    const float sc = pow2f(-(X + kUnnorm));
    uint32_t wd[4];
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      uint32_t bytes[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 f = v[4 * w + q];
        bytes[q] = e2m1x2(f.y * sc, f.x * sc);
      }
      wd[w] = e2m1_clear_neg_zero(bytes[0] | (bytes[1] << 8) | (bytes[2] << 16) | (bytes[3] << 24));
    }
    if (row_ok) {
      const int mb = b * 32 + lane;  // the row's MX block
      uint8_t* rdst = a.codes + static_cast<int64_t>(row >> 5) * cpr * 512 + (row & 31) * 16;
      *reinterpret_cast<uint4*>(rdst + static_cast<int64_t>(mb) * 512) = make_uint4(wd[0], wd[1], wd[2], wd[3]);
      a.shifts[((static_cast<int64_t>(row >> 5) * nkt + (mb >> 2)) * 32 + (row & 31)) * 4 + (mb & 3)] =
          static_cast<uint8_t>(X - xlo);
      if (b == 0 && lane == 0) a.scale[row] = pow2f(xlo);
      if (lane == 0 && a.offset != nullptr) {
        if constexpr (kRot) {
          a.offset[static_cast<int64_t>(row) * G + b] = offs ? off * 0.03125f : 0.f;
        } else {
          if (b % m == 0) a.offset[static_cast<int64_t>(row) * G + b / m] = offs ? off : 0.f;
        }
      }
    }
    grp += gridDim.x;
    if (grp >= ngroups) break;
  }
}

// Rows without the rotation whose offset block is the whole row (g == K): one
// warp per row. Each lane issues the loads of up to CB 8-element chunks at once
// and keeps them (raw) in registers, so a row of up to 256*CB elements costs one
// trip to memory; longer rows are read twice in batches of CB chunks (the
// second time from L2). Since rounding is monotonic,
// max_k |fl(x_k - o)| = max(fl(max x - o), fl(o - min x)), so the first sweep
// already yields the row's residual absmax.
template <typename Tin>
struct RawChunk {
  static constexpr int kWords = sizeof(Tin) == 4 ? 8 : 4;  // 32-bit words per 8-element chunk
  uint32_t w[kWords];
  __device__ __forceinline__ void load(const Tin* p) {
    const uint4 a = ldg_nc_v4(p);
    w[0] = a.x; w[1] = a.y; w[2] = a.z; w[3] = a.w;
    if constexpr (kWords == 8) {
      const uint4 b = ldg_nc_v4(p + 4);
      w[4] = b.x; w[5] = b.y; w[6] = b.z; w[7] = b.w;
    }
  }
  __device__ __forceinline__ void load_smem(const uint8_t* p) {
    const uint4 a = *reinterpret_cast<const uint4*>(p);
    w[0] = a.x; w[1] = a.y; w[2] = a.z; w[3] = a.w;
    if constexpr (kWords == 8) {
      const uint4 b = *reinterpret_cast<const uint4*>(p + 16);
      w[4] = b.x; w[5] = b.y; w[6] = b.z; w[7] = b.w;
    }
  }
  __device__ __forceinline__ void unpack(float (&v)[8]) const {
    if constexpr (kWords == 8) {
#pragma unroll
      for (int e = 0; e < 8; ++e) v[e] = __uint_as_float(w[e]);
    } else if constexpr (std::is_same<Tin, __half>::value) {
#pragma unroll
      for (int e = 0; e < 4; ++e) f16x2_to_f32(w[e], v[2 * e], v[2 * e + 1]);
    } else {
#pragma unroll
      for (int e = 0; e < 4; ++e) bf16x2_to_f32(w[e], v[2 * e], v[2 * e + 1]);
    }
  }
};

// Running min and max over raw input words: packed bf16x2 / f16x2 (exact) for
// the 16-bit types, one fp32 value per word for fp32.
template <typename Tin>
struct RowMinMax {
  uint32_t lo, hi;
  __device__ __forceinline__ RowMinMax() {
    if constexpr (std::is_same<Tin, __half>::value) {
      lo = 0x7BFF7BFFu;  // +65504 twice
      hi = 0xFBFFFBFFu;
    } else {
      lo = 0x7F7F7F7Fu;  // largest finite bf16 twice
      hi = 0xFF7FFF7Fu;
    }
  }
  __device__ __forceinline__ void add_word(uint32_t w) {
    if constexpr (std::is_same<Tin, __half>::value) {
      asm("min.f16x2 %0, %0, %1;" : "+r"(lo) : "r"(w));
      asm("max.f16x2 %0, %0, %1;" : "+r"(hi) : "r"(w));
    } else {
      asm("min.bf16x2 %0, %0, %1;" : "+r"(lo) : "r"(w));
      asm("max.bf16x2 %0, %0, %1;" : "+r"(hi) : "r"(w));
    }
  }
  __device__ __forceinline__ void result(float& mn, float& mx) const {
    float a, b, c, d;
    if constexpr (std::is_same<Tin, __half>::value) {
      f16x2_to_f32(lo, a, b);
      f16x2_to_f32(hi, c, d);
    } else {
      bf16x2_to_f32(lo, a, b);
      bf16x2_to_f32(hi, c, d);
    }
    mn = fminf(a, b);
    mx = fmaxf(c, d);
  }
};

template <>
struct RowMinMax<float> {
  float mn = 3.402823466e38f, mx = -3.402823466e38f;
  __device__ __forceinline__ void add_word(uint32_t w) {
    mn = fminf(mn, __uint_as_float(w));
    mx = fmaxf(mx, __uint_as_float(w));
  }
  __device__ __forceinline__ void result(float& a, float& b) const {
    a = mn;
    b = mx;
  }
};

// Packed accumulation {a0 + b0, a1 + b1}.
__device__ __forceinline__ void add2(float& a0, float& a1, float b0, float b1) {
  const uint64_t A = pack2(a0, a1);
  const uint64_t B = pack2(b0, b1);
  uint64_t R;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(R) : "l"(A), "l"(B));
  unpack2(R, a0, a1);
}

// Pairwise summation over a stream of values whose count is a power of two
// (at most 2^L): level k holds the sum of the last complete run of 2^k values,
// so each value joins a balanced tree and the total, read at level
// log2(count), has depth log2(count).
template <int L>
struct PairwiseSum {
  float lvl[L + 1];
  int n = 0;
  __device__ __forceinline__ void add(float c) {
    bool carry = true;
#pragma unroll
    for (int k = 0; k <= L; ++k) {
      const bool full = (n >> k) & 1;
      if (carry && full) c = lvl[k] + c;
      if (carry && !full) lvl[k] = c;
      carry = carry && full;
    }
    ++n;
  }
  // The total once n is a power of two.
  __device__ __forceinline__ float total() const {
    float t = 0.f;
#pragma unroll
    for (int k = 0; k <= L; ++k) {
      if (n == (1 << k)) t = lvl[k];
    }
    return t;
  }
};

// Sum of the 8 values of a chunk by a tree of depth 3.
__device__ __forceinline__ float chunk_sum8(float (&v)[8]) {
  add2(v[0], v[1], v[2], v[3]);
  add2(v[4], v[5], v[6], v[7]);
  add2(v[0], v[1], v[4], v[5]);
  return v[0] + v[1];
}

template <typename Tin, int CB>
__global__ void __launch_bounds__(256) quantize_rows_stream_kernel(const QuantArgs a) {
  griddep_wait();
  griddep_launch_dependents();
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t row = static_cast<int64_t>(blockIdx.x) * 8 + warp;
  if (row >= a.rows) return;
  const bool offs = (a.flags & OFFQ_OFFSET) != 0;
  const int K = a.K;
  const int nch = K / 8;  // 8-element chunks per row
  const int64_t t = row / a.H;
  const int64_t h = row - t * a.H;
  const Tin* xr = static_cast<const Tin*>(a.x) + t * a.ld_t + h * a.ld_h;
  const bool resident = nch <= 32 * CB;

  RawChunk<Tin> raw[CB];
  RowMinMax<Tin> mm;
  PairwiseSum<6> ps;  // the batches' sums (a power of two of them)
  for (int c0 = 0; c0 < nch; c0 += 32 * CB) {
#pragma unroll
    for (int i = 0; i < CB; ++i) {
      const int c = c0 + lane + 32 * i;
      if (c < nch) raw[i].load(xr + 8 * c);
    }
    float cs[CB];
#pragma unroll
    for (int i = 0; i < CB; ++i) {
      const int c = c0 + lane + 32 * i;
      cs[i] = 0.f;
      if (c < nch) {
#pragma unroll
        for (int e = 0; e < RawChunk<Tin>::kWords; ++e) mm.add_word(raw[i].w[e]);
        float v[8];
        raw[i].unpack(v);
        cs[i] = chunk_sum8(v);
      }
    }
    // The batch's chunks present are its first min(CB, nch/32) (a power of two): the
    // zeros after them add exactly, so the tree's depth over real terms is log2 of that.
    ps.add(tree_sum<CB>(cs));
  }
  // Row sum: depth 3 in the chunk, log2 over the lane's chunks, 5 over the warp.
  float sum = ps.total(), mn, mx;
  mm.result(mn, mx);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
    mn = fminf(mn, __shfl_xor_sync(0xFFFFFFFFu, mn, o));
    mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
  }
  const float off = offs ? sum * (1.0f / static_cast<float>(K)) : 0.f;  // K is a power of two
  const float m = fmaxf(fmaxf(mx - off, off - mn), 0.f);
  const float inv = m > 0.f ? __fdiv_rn(7.0f, m) : 0.f;

  const int cpr = K / 32;
  uint8_t* tile_row = a.tiled ? a.codes + (row >> 5) * cpr * 512 + (row & 31) * 16 : a.codes + row * (K / 2);
  for (int c0 = 0; c0 < nch; c0 += 32 * CB) {
    if (!resident) {
#pragma unroll
      for (int i = 0; i < CB; ++i) {
        const int c = c0 + lane + 32 * i;
        if (c < nch) raw[i].load(xr + 8 * c);
      }
    }
#pragma unroll
    for (int i = 0; i < CB; ++i) {
      const int c = c0 + lane + 32 * i;
      if (c < nch) {
        float v[8];
        raw[i].unpack(v);
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
          sub2(v[e], v[e + 1], off);
          fma2(v[e], v[e + 1], inv, kMagic8);
        }
        const uint32_t w = pack_codes8(__float_as_uint(v[0]), __float_as_uint(v[1]), __float_as_uint(v[2]),
                                       __float_as_uint(v[3]), __float_as_uint(v[4]), __float_as_uint(v[5]),
                                       __float_as_uint(v[6]), __float_as_uint(v[7]));
        const int bo = 4 * c;  // byte of the row-major row
        uint8_t* dst = a.tiled ? tile_row + (bo >> 4) * 512 + (bo & 15) : tile_row + bo;
        *reinterpret_cast<uint32_t*>(dst) = w;
      }
    }
  }
  if (lane == 0) {
    a.scale[row] = m * a.scale_mul;
    if (a.offset != nullptr) a.offset[row] = off;
  }
}

// The same rows (no rotation, one offset block g == K) when a row fits a
// shared-memory slot: a persistent kernel whose warps each own a ring of S row
// slots. Lane 0 fills the slots with bulk asynchronous copies (cp.async.bulk,
// completion counted in bytes on the slot's mbarrier) up to S - 1 rows ahead of
// the row the warp quantizes, so HBM keeps streaming later rows while the
// warp runs both sweeps of the current one out of shared memory. Rows are
// dealt to the grid's warps round-robin.
constexpr int kBulkRingBytes = 192 * 1024;  // ring bytes per CTA at most

// CPL = K / 256: the 8-channel chunks each lane sweeps (a power of two, 4 to 32).
template <typename Tin, int CPL>
__global__ void __launch_bounds__(256) quantize_rows_bulk_kernel(const QuantArgs a, int S) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ int abort_flag;
  constexpr int kChunkBytes = 8 * static_cast<int>(sizeof(Tin));
  const int W = static_cast<int>(blockDim.x >> 5);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int K = a.K;
  const uint32_t rb = static_cast<uint32_t>(K) * static_cast<uint32_t>(sizeof(Tin));  // a multiple of 64
  constexpr int cpl = CPL;                                                            // chunks per lane
  uint8_t* ring = smem + static_cast<size_t>(warp) * S * rb;
  const uint32_t bar0 = smem_u32(smem + static_cast<size_t>(W) * S * rb) + 8u * static_cast<uint32_t>(warp * S);
  if (threadIdx.x == 0) abort_flag = 0;
  if (lane < S) mbar_init(bar0 + 8u * lane, 1);
  mbar_fence_init();
  __syncthreads();
  griddep_wait();
  griddep_launch_dependents();

  const bool offs = (a.flags & OFFQ_OFFSET) != 0;
  const int64_t TW = static_cast<int64_t>(gridDim.x) * W;
  const int64_t r0 = static_cast<int64_t>(blockIdx.x) * W + warp;
  const Tin* x = static_cast<const Tin*>(a.x);
  auto row_src = [&](int64_t r) {
    const int64_t t = r / a.H;
    return x + t * a.ld_t + (r - t * a.H) * a.ld_h;
  };

  // Prologue: the first S rows of this warp in flight.
  int64_t issued = 0;
  for (int s = 0; s < S; ++s) {
    const int64_t r = r0 + s * TW;
    if (r >= a.rows) break;
    if (lane == 0) {
      mbar_arrive_expect_tx(bar0 + 8u * s, rb);
      bulk_load_row(smem_u32(ring + static_cast<size_t>(s) * rb), row_src(r), rb, bar0 + 8u * s);
    }
    ++issued;
  }

  const int cpr = K / 32;  // 16-byte code chunks per row
  int slot = 0;
  uint32_t phase = 0;
  int64_t done = 0;
  bool ok = true;
  for (int64_t r = r0; r < a.rows; r += TW) {
    const uint32_t bar = bar0 + 8u * slot;
    // Warp-uniform outcome: the sweeps below shuffle across the whole warp.
    if (!__all_sync(0xFFFFFFFFu, mbar_wait_for(bar, phase, &abort_flag, a.wait_cycles))) {
      ok = false;
      break;
    }
    const uint8_t* rowp = ring + static_cast<size_t>(slot) * rb;

    // Sweep 1: packed min / max of the raw values and the fp32 row sum.
    RowMinMax<Tin> mm;
    // Chunk sums as packed pairs (even and odd channels), combined pairwise; fully
    // unrolled, so the carries resolve at compile time and log2(cpl) + 1 pairs stay live.
    float2 lvl[6];
#pragma unroll
    for (int j = 0; j < cpl; ++j) {
      RawChunk<Tin> c;
      c.load_smem(rowp + (lane + 32 * j) * kChunkBytes);
#pragma unroll
      for (int e = 0; e < RawChunk<Tin>::kWords; ++e) mm.add_word(c.w[e]);
      float v[8];
      c.unpack(v);
      add2(v[0], v[1], v[2], v[3]);
      add2(v[4], v[5], v[6], v[7]);
      add2(v[0], v[1], v[4], v[5]);
      float2 p = make_float2(v[0], v[1]);
#pragma unroll
      for (int k = 0; k < 6; ++k) {
        if ((j >> k) & 1) {
          p = __fadd2_rn(lvl[k], p);
        } else {
          lvl[k] = p;
          break;
        }
      }
    }
    // Row sum: depth 3 in the chunk, log2(cpl) over the lane's chunks, 1 for the pair,
    // 5 over the warp.
    float2 tot = lvl[0];
#pragma unroll
    for (int k = 1; k < 6; ++k) {
      if (cpl == (1 << k)) tot = lvl[k];
    }
    float sum = tot.x + tot.y, mn, mx;
    mm.result(mn, mx);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
      mn = fminf(mn, __shfl_xor_sync(0xFFFFFFFFu, mn, o));
      mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
    }
    const float off = offs ? sum * (1.0f / static_cast<float>(K)) : 0.f;  // K is a power of two
    const float m = fmaxf(fmaxf(mx - off, off - mn), 0.f);
    const float inv = m > 0.f ? __fdiv_rn(7.0f, m) : 0.f;

    // Sweep 2: codes, one 4-byte word per 8-channel chunk.
    uint8_t* tile_row = a.tiled ? a.codes + (r >> 5) * cpr * 512 + (r & 31) * 16 : a.codes + r * (K / 2);
#pragma unroll 4
    for (int j = 0; j < cpl; ++j) {
      const int c = lane + 32 * j;
      RawChunk<Tin> ch;
      ch.load_smem(rowp + c * kChunkBytes);
      float v[8];
      ch.unpack(v);
#pragma unroll
      for (int e = 0; e < 8; e += 2) {
        sub2(v[e], v[e + 1], off);
        fma2(v[e], v[e + 1], inv, kMagic8);
      }
      const uint32_t w = pack_codes8(__float_as_uint(v[0]), __float_as_uint(v[1]), __float_as_uint(v[2]),
                                     __float_as_uint(v[3]), __float_as_uint(v[4]), __float_as_uint(v[5]),
                                     __float_as_uint(v[6]), __float_as_uint(v[7]));
      const int bo = 4 * c;  // byte of the row-major row
      uint8_t* dst = a.tiled ? tile_row + (bo >> 4) * 512 + (bo & 15) : tile_row + bo;
      *reinterpret_cast<uint32_t*>(dst) = w;
    }
    if (lane == 0) {
      a.scale[r] = m * a.scale_mul;
      if (a.offset != nullptr) a.offset[r] = off;
    }
    ++done;

    // Every lane has read the slot: refill it with the row S turns ahead.
    __syncwarp();
    const int64_t rn = r + S * TW;
    if (rn < a.rows) {
      if (lane == 0) {
        mbar_arrive_expect_tx(bar, rb);
        bulk_load_row(smem_u32(ring + static_cast<size_t>(slot) * rb), row_src(rn), rb, bar);
      }
      ++issued;
    }
    if (++slot == S) {
      slot = 0;
      phase ^= 1u;
    }
  }
  if (!ok && lane == 0) {
    // A wait ran out: let this warp's copies still in flight land (bounded),
    // then report the timeout.
    for (int64_t j = done; j < issued; ++j) {
      const uint32_t b = bar0 + 8u * static_cast<uint32_t>(j % S);
      const uint32_t p = static_cast<uint32_t>((j / S) & 1);
      const long long t0 = clock64();
      while (!mbar_try_wait(b, p) && clock64() - t0 < kWaitCycles) {
      }
    }
    if (a.status != nullptr) atomicExch(a.status, kErrTimeout);
  }
}

// Asks for the largest shared-memory carveout for a kernel, once per device,
// so that the CTAs' shared memory does not cap residency below the register
// limit.
template <typename F>
int prefer_max_shared(F* kern) {
  static unsigned long long done = 0;  // bit d: set on device d
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return OFFQ_ERR_CUDA;
  if (dev < 64 && (__atomic_load_n(&done, __ATOMIC_ACQUIRE) >> dev) & 1ull) return OFFQ_OK;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared) !=
      cudaSuccess)
    return OFFQ_ERR_CUDA;
  if (dev < 64) __atomic_fetch_or(&done, 1ull << dev, __ATOMIC_ACQ_REL);
  return OFFQ_OK;
}

// Streaming multiprocessors of the current device (queried once per device).
int sm_count() {
  static int cache[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (dev < 64 && cache[dev] > 0) return cache[dev];
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  if (dev < 64) cache[dev] = n;
  return n;
}

constexpr int kNoRing = 1;  // launch_ring: use the one-shot kernel instead

// Launches the persistent (ring) form of a row kernel when the input has one
// head, there are more row groups than SMs, and the slot fits: one CTA per
// resident slot, each looping over the groups grid-stride.
// base_smem is the kernel's shared memory without the ring, slot_bytes one
// slot (rows_per_cta rows of input). The slot count (1 to 3) is the one with
// the most slots per SM, so the most rows in flight; ties take more slots.
template <typename F>
int launch_ring(F* kern, QuantArgs a, int threads, size_t base_smem, size_t slot_bytes, cudaStream_t stream) {
  if (a.H != 1) return kNoRing;
  const int sms = sm_count();
  const int64_t groups = (a.rows + a.rows_per_cta - 1) / a.rows_per_cta;
  if (sms <= 0 || groups <= sms) return kNoRing;
  if (prefer_max_shared(kern) != OFFQ_OK) return OFFQ_ERR_CUDA;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kMaxDynSmem)) !=
      cudaSuccess)
    return OFFQ_ERR_CUDA;
  int best_s = 0, best_per_sm = 0;
  for (int S = 1; S <= 3; ++S) {
    const size_t smem = base_smem + S * (slot_bytes + 8);
    if (smem > kMaxDynSmem) break;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem) != cudaSuccess)
      return OFFQ_ERR_CUDA;
    if (per_sm >= 1 && per_sm * S >= best_per_sm * best_s) {
      best_s = S;
      best_per_sm = per_sm;
    }
  }
  if (best_s == 0) return kNoRing;
  a.ring_slots = best_s;
  const size_t smem = base_smem + best_s * (slot_bytes + 8);
  const int64_t grid = std::min<int64_t>(groups, static_cast<int64_t>(sms) * best_per_sm);
  return launch_pdl(kern, dim3(static_cast<unsigned>(grid)), dim3(threads), smem, stream, a);
}

template <int L, typename Tin>
int launch_narrow(QuantArgs a, cudaStream_t stream) {
  using GG = NarrowGeo<L>;
  const int raw = a.G * GG::kTPB;
  int tpr = 1;
  if (raw <= 32) {
    while (tpr < raw) tpr <<= 1;
  } else {
    tpr = (raw + 31) / 32 * 32;
  }
  if (tpr > GG::kMaxThreads) return OFFQ_ERR_UNSUPPORTED;
  const size_t row_smem = static_cast<size_t>(a.K) * 4;
  int R = std::max(1, 256 / tpr);
  while (R > 1 && static_cast<size_t>(R) * row_smem > 64 * 1024) --R;
  a.tpr = tpr;
  a.rows_per_cta = R;
  const size_t smem = 128 + static_cast<size_t>(R) * row_smem;
  const int rs = launch_ring(quantize_rows_kernel<L, Tin, true>, a, R * tpr, smem,
                             static_cast<size_t>(R) * a.K * sizeof(Tin), stream);
  if (rs != kNoRing) return rs;
  auto kern = quantize_rows_kernel<L, Tin, false>;
  if (prefer_max_shared(kern) != OFFQ_OK) return OFFQ_ERR_CUDA;
  if (smem > 48 * 1024) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) !=
        cudaSuccess)
      return OFFQ_ERR_CUDA;
  }
  const int64_t grid = (a.rows + R - 1) / R;
  if (grid > 0x7FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  return launch_pdl(kern, dim3(static_cast<unsigned>(grid)), dim3(R * tpr), smem, stream, a);
}

template <int L, typename Tin>
int launch_wide(QuantArgs a, cudaStream_t stream) {
  using GG = WideGeo<L>;
  const int raw = a.G * GG::kTPB;
  int tpr = 1;
  if (raw <= 32) {
    while (tpr < raw) tpr <<= 1;
  } else {
    tpr = (raw + 31) / 32 * 32;
  }
  if (tpr > GG::kMaxThreads) return OFFQ_ERR_UNSUPPORTED;
  const bool rotate = (a.flags & OFFQ_ROTATE) != 0;
  const size_t row_smem = (rotate ? static_cast<size_t>(a.K) * 4 : 0) + a.K / 2;
  int R = std::max(1, std::min(GG::kMaxThreads, 256) / tpr);
  while (R > 1 && static_cast<size_t>(R) * row_smem > 64 * 1024) --R;
  a.tpr = tpr;
  a.rows_per_cta = R;
  const size_t smem = static_cast<size_t>(R) * row_smem + 32 * sizeof(float);
  const int rs = launch_ring(quantize_rows_wide_kernel<L, Tin, true>, a, R * tpr, smem,
                             static_cast<size_t>(R) * a.K * sizeof(Tin), stream);
  if (rs != kNoRing) return rs;
  auto kern = quantize_rows_wide_kernel<L, Tin, false>;
  if (smem > 48 * 1024) {
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) !=
        cudaSuccess)
      return OFFQ_ERR_CUDA;
  }
  const int64_t grid = (a.rows + R - 1) / R;
  if (grid > 0x7FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  return launch_pdl(kern, dim3(static_cast<unsigned>(grid)), dim3(R * tpr), smem, stream, a);
}

// quantize_rows_1k_kernel: R rows of G warps per CTA. One row per CTA unless a
// CTA would have fewer than 4 warps: CTAs of G <= 14 warps share an SM and
// drift apart, so one CTA's barrier waits overlap another's arithmetic. The
// ring takes 2 or 3 slots, whichever gives more CTAs per SM (ties: more
// slots); 1 slot only when 2 do not fit. kNoRing when the one-shot kernels
// serve better (one head required, more row groups than SMs).
template <typename Tin>
int launch_1k(QuantArgs a, cudaStream_t stream) {
  if (a.H != 1 || (a.flags & OFFQ_ROTATE) == 0 || a.G > k1kMaxWarps) return kNoRing;
  const int sms = sm_count();
  if (sms <= 0) return OFFQ_ERR_CUDA;
  const int R = std::max(1, 4 / a.G);
  const int64_t groups = (a.rows + R - 1) / R;
  if (groups <= sms || a.rows + R > 0x7FFFFFFF) return kNoRing;
  auto kern = quantize_rows_1k_kernel<Tin>;
  if (prefer_max_shared(kern) != OFFQ_OK) return OFFQ_ERR_CUDA;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kMaxDynSmem)) !=
      cudaSuccess)
    return OFFQ_ERR_CUDA;
  const int threads = R * a.G * 32;
  const size_t fixed = static_cast<size_t>(R) * a.G * 4096;
  const size_t slot = static_cast<size_t>(R) * a.K * sizeof(Tin) + 8;
  int best_s = 0, best_per_sm = 0;
  for (int S = 1; S <= 3; ++S) {
    const size_t smem = fixed + S * slot;
    if (smem > kMaxDynSmem) break;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem) != cudaSuccess)
      return OFFQ_ERR_CUDA;
    if (per_sm < 1) break;
    const bool better = best_s == 0 || (best_s == 1 && S >= 2) || (S >= 2 && per_sm >= best_per_sm);
    if (better) {
      best_s = S;
      best_per_sm = per_sm;
    }
  }
  if (best_s == 0) return kNoRing;
  a.rows_per_cta = R;
  a.ring_slots = best_s;
  a.tpr = a.G * 32;
  const size_t smem = fixed + best_s * slot;
  const int64_t grid = std::min<int64_t>(groups, static_cast<int64_t>(sms) * best_per_sm);
  return launch_pdl(kern, dim3(static_cast<unsigned>(grid)), dim3(threads), smem, stream, a);
}

// quantize_mx_1k_kernel: one row of K/1024 warps per CTA (rows per CTA grow
// while a CTA has fewer than 4 warps), the ring as launch_1k's. kNoRing when the
// shape does not fit it (the generic MX kernel serves those).
template <typename Tin, bool kRot>
int launch_mx_1k(QuantArgs a, cudaStream_t stream) {
  const int nbw = a.K / 1024;
  if (a.H != 1 || a.K % 1024 != 0 || nbw > k1kMaxWarps) return kNoRing;
  if (kRot ? a.g != 1024 : (a.g % 1024 != 0 || a.g / 1024 > 8)) return kNoRing;
  const int sms = sm_count();
  if (sms <= 0) return OFFQ_ERR_CUDA;
  const int R = std::max(1, 4 / nbw);
  const int64_t groups = (a.rows + R - 1) / R;
  if (groups <= sms || a.rows + R > 0x7FFFFFFF) return kNoRing;
  auto kern = quantize_mx_1k_kernel<Tin, kRot>;
  if (prefer_max_shared(kern) != OFFQ_OK) return OFFQ_ERR_CUDA;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kMaxDynSmem)) !=
      cudaSuccess)
    return OFFQ_ERR_CUDA;
  const int threads = R * nbw * 32;
  const size_t fixed = kRot ? static_cast<size_t>(R) * nbw * 4096 : 0;
  const size_t slot = static_cast<size_t>(R) * a.K * sizeof(Tin) + 8;
  int best_s = 0, best_per_sm = 0;
  for (int S = 1; S <= 3; ++S) {
    const size_t smem = fixed + S * slot;
    if (smem > kMaxDynSmem) break;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem) != cudaSuccess)
      return OFFQ_ERR_CUDA;
    if (per_sm < 1) break;
    const bool better = best_s == 0 || (best_s == 1 && S >= 2) || (S >= 2 && per_sm >= best_per_sm);
    if (better) {
      best_s = S;
      best_per_sm = per_sm;
    }
  }
  if (best_s == 0) return kNoRing;
  a.rows_per_cta = R;
  a.ring_slots = best_s;
  a.tpr = nbw * 32;
  const size_t smem = fixed + best_s * slot;
  const int64_t grid = std::min<int64_t>(groups, static_cast<int64_t>(sms) * best_per_sm);
  return launch_pdl(kern, dim3(static_cast<unsigned>(grid)), dim3(threads), smem, stream, a);
}

template <typename Tin>
int launch_stream(const QuantArgs& a, cudaStream_t stream) {
  const int64_t grid = (a.rows + 7) / 8;
  if (grid > 0x7FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  // Up to 16 chunks (64 registers of bf16) per lane stay resident.
  constexpr int CB = sizeof(Tin) == 4 ? 8 : 16;
  return launch_pdl(quantize_rows_stream_kernel<Tin, CB>, dim3(static_cast<unsigned>(grid)), dim3(256), 0, stream, a);
}

constexpr int kNoFit = 1;  // launch_bulk: the row does not fit the ring; use the register kernel

// The ring geometry: the most warps (8 down to 4) whose rings of 2 to 4 row
// slots fit kBulkRingBytes.
template <typename Tin>
int launch_bulk(const QuantArgs& a, cudaStream_t stream) {
  if (a.H != 1) return kNoFit;
  const int64_t rb = static_cast<int64_t>(a.K) * static_cast<int64_t>(sizeof(Tin));
  int W = 8, S = 0;
  for (; W >= 4; --W) {
    S = static_cast<int>(std::min<int64_t>(4, kBulkRingBytes / (W * rb)));
    if (S >= 2) break;
  }
  if (S < 2) return kNoFit;
  const size_t smem = static_cast<size_t>(W) * S * rb + static_cast<size_t>(W) * S * 8;
  decltype(&quantize_rows_bulk_kernel<Tin, 4>) kern = nullptr;
  switch (a.K / 256) {
    case 4: kern = quantize_rows_bulk_kernel<Tin, 4>; break;
    case 8: kern = quantize_rows_bulk_kernel<Tin, 8>; break;
    case 16: kern = quantize_rows_bulk_kernel<Tin, 16>; break;
    case 32: kern = quantize_rows_bulk_kernel<Tin, 32>; break;
    default: return kNoFit;
  }
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) != cudaSuccess)
    return OFFQ_ERR_CUDA;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, W * 32, smem) != cudaSuccess || per_sm < 1)
    return OFFQ_ERR_CUDA;
  const int sms = sm_count();
  if (sms <= 0) return OFFQ_ERR_CUDA;
  const int64_t grid = std::min<int64_t>((a.rows + W - 1) / W, static_cast<int64_t>(sms) * per_sm);
  return launch_pdl(kern, dim3(static_cast<unsigned>(grid)), dim3(W * 32), smem, stream, a, S);
}

template <typename Tin>
int dispatch_g(const QuantArgs& a, int g, cudaStream_t s) {
  if ((a.flags & OFFQ_ROTATE) == 0 && a.G == 1 && g >= 1024) {
    const int st = launch_bulk<Tin>(a, s);
    return st == kNoFit ? launch_stream<Tin>(a, s) : st;
  }
  switch (g) {
    case 32: return launch_narrow<5, Tin>(a, s);
    case 64: return launch_narrow<6, Tin>(a, s);
    case 128: return launch_narrow<7, Tin>(a, s);
    case 256: return launch_narrow<8, Tin>(a, s);
    case 512: return launch_narrow<9, Tin>(a, s);
    case 1024: {
      if constexpr (std::is_same<Tin, __nv_bfloat16>::value) {
        if (a.H == 1 && (a.flags & OFFQ_ROTATE) != 0) {
          MmaQuantRows p{};
          p.x = a.x;
          p.ld_t = a.ld_t;
          p.rows = a.rows;
          p.K = a.K;
          p.flags = a.flags;
          p.codes = a.codes;
          p.scale = a.scale;
          p.offset = a.offset;
          p.tiled = a.tiled;
          p.inv_sqrt_g = a.inv_sqrt_g;
          p.scale_mul = a.scale_mul;
          p.status = a.status;
          p.wait_cycles = a.wait_cycles;
          const int st = quantize_rows_mma(p, s);
          if (st != 1) return st;
        }
      }
      const int st = launch_1k<Tin>(a, s);
      return st == kNoRing ? launch_narrow<10, Tin>(a, s) : st;
    }
    case 2048: return launch_wide<11, Tin>(a, s);
    case 4096: return launch_wide<12, Tin>(a, s);
    case 8192: return launch_wide<13, Tin>(a, s);
    default: return OFFQ_ERR_UNSUPPORTED;
  }
}

// Budget of the persistent kernels' waits for a staged row, in SM cycles
// (offq_set_wait_cycles; kWaitCycles unless a test shortens it).
std::atomic<long long> g_row_wait_cycles{kWaitCycles};

int run_quant(QuantArgs a, int dtype, int g, cudaStream_t s) {
  const double isg = (a.flags & OFFQ_ROTATE) ? 1.0 / std::sqrt(static_cast<double>(g)) : 1.0;
  a.inv_sqrt_g = static_cast<float>(isg);
  a.scale_mul = static_cast<float>(isg / 7.0);
  a.status = device_status_ptr();
  a.wait_cycles = g_row_wait_cycles.load(std::memory_order_relaxed);
  switch (dtype) {
    case OFFQ_BF16: return dispatch_g<__nv_bfloat16>(a, g, s);
    case OFFQ_F16: return dispatch_g<__half>(a, g, s);
    case OFFQ_F32: return dispatch_g<float>(a, g, s);
    default: return OFFQ_ERR_INVALID_ARG;
  }
}

// K and g rules shared by the row quantizers.
int check_row_shape(int64_t K, int32_t g) {
  if (!is_pow2(g) || g < 32 || g > 8192) return OFFQ_ERR_INVALID_ARG;
  if (K <= 0 || K % g != 0 || K % 32 != 0) return OFFQ_ERR_INVALID_ARG;
  if (K > kMaxQuantK || K > 128 * static_cast<int64_t>(g)) return OFFQ_ERR_UNSUPPORTED;
  return OFFQ_OK;
}

// Offline: activation-format codes (q + 8) -> weight format, in place, plus the
// integer block row sums R[b][n]; the padding rows of the last 32-row tile are
// zeroed. Codes are in the tiled operand layout. One thread per (row, block).
// It does not release its dependents early: the few-token GEMM starts reading
// weight codes and row sums before it waits for the kernel ahead of it.
__global__ void weight_repack_kernel(uint8_t* __restrict__ codes, float* __restrict__ rowsum, int64_t N,
                                     int64_t N_pad, int K, int g) {
  griddep_wait();
  const int G = K / g;
  const int64_t id = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (id >= N_pad * G) return;
  const int64_t n = id / G;
  const int b = static_cast<int>(id - n * G);
  const int64_t cpr = K / 32;
  uint8_t* tile_row = codes + (n >> 5) * cpr * 512 + (n & 31) * 16;
  int sum = 0;
  for (int i = 0; i < g / 8; ++i) {
    const int64_t bo = static_cast<int64_t>(b) * (g / 2) + 4 * i;  // byte of the row-major row
    uint32_t* w = reinterpret_cast<uint32_t*>(tile_row + (bo >> 4) * 512 + (bo & 15));
    if (n >= N) {
      *w = 0u;
      continue;
    }
    const uint32_t u = *w;
    uint32_t mag[8], neg[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      const int q = static_cast<int>((u >> (4 * c)) & 0xFu) - 8;
      sum += q;
      mag[c] = static_cast<uint32_t>(q < 0 ? -q : q);
      neg[c] = q < 0 ? 1u : 0u;
    }
    uint32_t out = 0;
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      const uint32_t byte = mag[2 * jj] | (neg[2 * jj] << 7) | (mag[2 * jj + 1] << 4) | (neg[(2 * jj + 7) & 7] << 3);
      out |= byte << (8 * jj);
    }
    *w = out;
  }
  if (n < N) rowsum[static_cast<int64_t>(b) * N + n] = static_cast<float>(sum);
}

}  // namespace

namespace offq {

// The MXFP4 row quantizer on the warp-per-1024-channel layout (arguments checked
// by the caller). Returns 1 when the shape or the row count does not suit it.
int quantize_mx_rows_fast(const void* x, int dtype, int64_t rows, int64_t K, int64_t ldx, int32_t g, int32_t flags,
                          uint8_t* codes, uint8_t* shifts, float* row_scale, float* offset, cudaStream_t s) {
  QuantArgs a{};
  a.x = x;
  a.ld_t = ldx;
  a.ld_h = 0;
  a.rows = rows;
  a.H = 1;
  a.K = static_cast<int>(K);
  a.G = static_cast<int>(K / g);
  a.flags = flags;
  a.codes = codes;
  a.scale = row_scale;
  a.offset = offset;
  a.tiled = 1;
  a.status = device_status_ptr();
  a.wait_cycles = g_row_wait_cycles.load(std::memory_order_relaxed);
  a.shifts = shifts;
  a.g = g;
  const bool rot = (flags & OFFQ_ROTATE) != 0;
  int st = kNoRing;
  switch (dtype) {
    case OFFQ_BF16: st = rot ? launch_mx_1k<__nv_bfloat16, true>(a, s) : launch_mx_1k<__nv_bfloat16, false>(a, s); break;
    case OFFQ_F16: st = rot ? launch_mx_1k<__half, true>(a, s) : launch_mx_1k<__half, false>(a, s); break;
    case OFFQ_F32: st = rot ? launch_mx_1k<float, true>(a, s) : launch_mx_1k<float, false>(a, s); break;
    default: return OFFQ_ERR_INVALID_ARG;
  }
  return st == kNoRing ? 1 : st;
}

}  // namespace offq

extern "C" int offq_quantize_act(const void* x, int x_dtype, int64_t T, int64_t K, int64_t ldx, int32_t g,
                                 int32_t flags, uint8_t* codes, float* scale, float* offset, void* stream) {
  const int eb = elem_bytes(x_dtype);
  if (eb == 0 || T < 0 || (flags & ~(OFFQ_ROTATE | OFFQ_OFFSET)) != 0) return OFFQ_ERR_INVALID_ARG;
  const int st = check_row_shape(K, g);
  if (st != OFFQ_OK) return st;
  if (ldx < K) return OFFQ_ERR_INVALID_ARG;
  if (T == 0) return OFFQ_OK;
  if (x == nullptr || codes == nullptr || scale == nullptr) return OFFQ_ERR_INVALID_ARG;
  if ((flags & OFFQ_OFFSET) && offset == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(x, 16) || (ldx * eb) % 16 != 0 || !aligned(codes, 16) || !aligned(scale, 4) ||
      (offset != nullptr && !aligned(offset, 4)))
    return OFFQ_ERR_MISALIGNED;
  QuantArgs a{};
  a.x = x;
  a.ld_t = ldx;
  a.ld_h = 0;
  a.rows = T;
  a.H = 1;
  a.K = static_cast<int>(K);
  a.G = static_cast<int>(K / g);
  a.flags = flags;
  a.codes = codes;
  a.scale = scale;
  a.offset = offset;
  a.tiled = 1;
  return run_quant(a, x_dtype, g, static_cast<cudaStream_t>(stream));
}

extern "C" int offq_kv4_quantize(const void* kv, int dtype, int64_t T, int32_t H, int32_t head_dim,
                                 int64_t ld_token, int32_t flags, uint8_t* codes, float* scale, float* offset,
                                 void* stream) {
  const int eb = elem_bytes(dtype);
  if (eb == 0 || T < 0 || H < 1 || (flags & ~(OFFQ_ROTATE | OFFQ_OFFSET)) != 0) return OFFQ_ERR_INVALID_ARG;
  const int st = check_row_shape(head_dim, head_dim);
  if (st != OFFQ_OK) return st;
  if (ld_token < static_cast<int64_t>(H) * head_dim) return OFFQ_ERR_INVALID_ARG;
  if (T == 0) return OFFQ_OK;
  if (kv == nullptr || codes == nullptr || scale == nullptr) return OFFQ_ERR_INVALID_ARG;
  if ((flags & OFFQ_OFFSET) && offset == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(kv, 16) || (ld_token * eb) % 16 != 0 || !aligned(codes, 16) || !aligned(scale, 4) ||
      (offset != nullptr && !aligned(offset, 4)))
    return OFFQ_ERR_MISALIGNED;
  QuantArgs a{};
  a.x = kv;
  a.ld_t = ld_token;
  a.ld_h = head_dim;
  a.rows = T * H;
  a.H = H;
  a.K = head_dim;
  a.G = 1;
  a.flags = flags;
  a.codes = codes;
  a.scale = scale;
  a.offset = offset;
  a.tiled = 0;
  return run_quant(a, dtype, head_dim, static_cast<cudaStream_t>(stream));
}

extern "C" int offq_prepare_weight(const void* w, int dtype, int64_t N, int64_t K, int32_t g, int32_t rotate,
                                   uint8_t* w_codes, float* w_scale, float* w_offsum, void* stream) {
  const int eb = elem_bytes(dtype);
  if (eb == 0 || N < 1) return OFFQ_ERR_INVALID_ARG;
  const int st = check_row_shape(K, g);
  if (st != OFFQ_OK) return st;
  if (w == nullptr || w_codes == nullptr || w_scale == nullptr || w_offsum == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(w, 16) || (K * eb) % 16 != 0 || !aligned(w_codes, 16) || !aligned(w_scale, 4) ||
      !aligned(w_offsum, 4))
    return OFFQ_ERR_MISALIGNED;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  QuantArgs a{};
  a.x = w;
  a.ld_t = K;
  a.ld_h = 0;
  a.rows = N;
  a.H = 1;
  a.K = static_cast<int>(K);
  a.G = static_cast<int>(K / g);
  a.flags = rotate ? OFFQ_ROTATE : 0;
  a.codes = w_codes;
  a.scale = w_scale;
  a.offset = nullptr;
  a.tiled = 1;
  int rc = run_quant(a, dtype, g, s);
  if (rc != OFFQ_OK) return rc;
  const int64_t n_pad = (N + 31) / 32 * 32;
  const int64_t units = n_pad * (K / g);
  const int threads = 256;
  return launch_pdl(weight_repack_kernel, dim3(static_cast<unsigned>((units + threads - 1) / threads)),
                    dim3(threads), 0, s, w_codes, w_offsum, N, n_pad, static_cast<int>(K), g);
}

extern "C" int64_t offq_act_codes_bytes(int64_t T, int64_t K) {
  if (T < 0 || K <= 0 || K % 32 != 0) return -1;
  return (T + 31) / 32 * 32 * (K / 2);
}

extern "C" int64_t offq_weight_codes_bytes(int64_t N, int64_t K) {
  if (N < 1 || K <= 0 || K % 32 != 0) return -1;
  return (N + 31) / 32 * 32 * (K / 2);
}

extern "C" int offq_set_wait_cycles(int64_t cycles) {
  if (cycles < 0) return OFFQ_ERR_INVALID_ARG;
  g_row_wait_cycles.store(cycles == 0 || cycles > kWaitCycles ? kWaitCycles : cycles, std::memory_order_relaxed);
  return OFFQ_OK;
}
