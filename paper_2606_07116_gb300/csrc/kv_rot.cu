// Key cache under a dense per-head rotation (offq_kv4_quantize_rotated) and the
// same rotation alone for the queries (offq_rotate_heads).
//
// With bias-induced outliers in the keys, the per-head online Hadamard H3 is
// replaced by M = U3 P3 H3 (paper Sec. 3.3 Step 2 (3)): y = x M for every
// (token, head) vector x of head_dim = 128. Q and K take the same M, so Q K^T
// is unchanged. The key cache is then quantized per (token, head) as with H3
// (Sec. 4.2: the KV group is the head):
//   o = mean(y) (with OFFQ_OFFSET), r = y - o, s = max|r| / 7,
//   q = clamp(rne(r / s), -7, 7), stored as the nibble q + 8.
//
// bf16 keys take the tensor cores: M is split into three bf16 parts,
// M = M1 + M2 + M3 (24 significant bits, M's whole fp32 significand); bf16 x
// bf16 products are exact, so y = x M1 + x M2 + x M3 accumulated in fp32 by
// tcgen05.mma (kind::f16, M 128 tokens x N 128 outputs, K 3 x 128) keeps fp32
// accuracy. A CTA takes one head, stages the three parts once (K-major, 128-byte
// swizzle) and loops over 128-token tiles; in the epilogue each thread owns one
// token's accumulator row in TMEM, so offset, scale and codes need no shuffles.
//
// Other input types (fp32, fp16) would lose bits in bf16 and take the FMA
// kernel: a CTA takes one head and loops over 64-token tiles of it (tiles c, c +
// gridDim.x, ...), so M (64 KB) is staged in shared memory once per CTA. Each
// tile is staged transposed (a warp stores 32 consecutive tokens of one
// channel: conflict-free); each lane accumulates 4 output channels of 8 tokens
// in fp32 (32 FMAs per three 16-byte shared loads), in input-channel order.
// Offset, scale and codes come from warp reductions over the token's 128
// outputs (4 per lane).
#include <cuda_bf16.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>

#include <cmath>
#include <cstring>
#include <mutex>
#include <type_traits>

#include "offq.h"
#include "offq_device.cuh"
#include "offq_host.h"

namespace {

using namespace offq;

constexpr int kHd = 128;
constexpr int kTokTile = 64;
constexpr int kRotWarps = 8;
constexpr int kTokPerWarp = kTokTile / kRotWarps;  // 8
constexpr int kXPitch = kTokTile + 4;              // floats per transposed channel row
constexpr int kRotSmem = (kHd * kHd + kHd * kXPitch) * 4;

struct RotArgs {
  const void* x;
  int64_t ld_token;  // elements between consecutive tokens
  int64_t T;
  int H;
  const float* rot;  // [H][128][128]
  const void* prep;  // the prepared image (tensor-core kernel), or nullptr: split rot in the kernel
  int quantize;      // 1: codes / scale / offset; 0: the rotated values
  int offset;        // subtract the mean (quantize only)
  uint8_t* codes;    // [T][H][64]
  float* scale;      // [T][H]
  float* off;        // [T][H] or nullptr
  void* out;         // [T][ld_out] of out_dtype
  int64_t ld_out;
  int* status;       // device status word (bounded waits of the tensor-core kernel)
};

// Raw 16-byte chunks of 8 channels (two for fp32 input), loaded ahead of use.
template <typename Tin>
struct Chunk8 {
  uint4 u[sizeof(Tin) == 4 ? 2 : 1];
};

template <typename Tin>
__device__ __forceinline__ void load_chunk(const Tin* src, bool ok, Chunk8<Tin>& c) {
#pragma unroll
  for (int k = 0; k < (sizeof(Tin) == 4 ? 2 : 1); ++k)
    c.u[k] = ok ? __ldg(reinterpret_cast<const uint4*>(src) + k) : make_uint4(0u, 0u, 0u, 0u);
}

template <typename Tin>
__device__ __forceinline__ void unpack_chunk(const Chunk8<Tin>& c, float (&v)[8]) {
  if constexpr (sizeof(Tin) == 4) {
    v[0] = __uint_as_float(c.u[0].x); v[1] = __uint_as_float(c.u[0].y);
    v[2] = __uint_as_float(c.u[0].z); v[3] = __uint_as_float(c.u[0].w);
    v[4] = __uint_as_float(c.u[1].x); v[5] = __uint_as_float(c.u[1].y);
    v[6] = __uint_as_float(c.u[1].z); v[7] = __uint_as_float(c.u[1].w);
  } else {
    const uint32_t w[4] = {c.u[0].x, c.u[0].y, c.u[0].z, c.u[0].w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      if constexpr (std::is_same<Tin, __nv_bfloat16>::value) {
        v[2 * k] = __uint_as_float(w[k] << 16);
        v[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
      } else {
        const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[k]));
        v[2 * k] = f.x;
        v[2 * k + 1] = f.y;
      }
    }
  }
}

template <int OUT>
__device__ __forceinline__ void store4(void* out, int64_t off, float a, float b, float c, float d) {
  if constexpr (OUT == OFFQ_F32) {
    *reinterpret_cast<float4*>(static_cast<float*>(out) + off) = make_float4(a, b, c, d);
  } else if constexpr (OUT == OFFQ_BF16) {
    const __nv_bfloat162 lo = __floats2bfloat162_rn(a, b), hi = __floats2bfloat162_rn(c, d);
    *reinterpret_cast<uint2*>(static_cast<uint16_t*>(out) + off) =
        make_uint2(*reinterpret_cast<const uint32_t*>(&lo), *reinterpret_cast<const uint32_t*>(&hi));
  } else {
    const __half2 lo = __floats2half2_rn(a, b), hi = __floats2half2_rn(c, d);
    *reinterpret_cast<uint2*>(static_cast<uint16_t*>(out) + off) =
        make_uint2(*reinterpret_cast<const uint32_t*>(&lo), *reinterpret_cast<const uint32_t*>(&hi));
  }
}

template <typename Tin, int OUT>
__global__ void __launch_bounds__(kRotWarps * 32) rotate_heads_kernel(const RotArgs a) {
  extern __shared__ float4 smem4[];
  float* Ms = reinterpret_cast<float*>(smem4);  // [128][128]
  float* xs = Ms + kHd * kHd;                   // [128][kXPitch], x transposed
  const int h = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  griddep_wait();
  griddep_launch_dependents();

  const float4* Mg = reinterpret_cast<const float4*>(a.rot + static_cast<int64_t>(h) * kHd * kHd);
  for (int i = tid; i < kHd * kHd / 4; i += kRotWarps * 32) smem4[i] = __ldg(Mg + i);
  const int64_t tiles = (a.T + kTokTile - 1) / kTokTile;
  // Thread tid owns chunks c = tid + 256 k of a tile: token c % 64, channels
  // 8 (c / 64) .. + 7. The next tile's chunks are loaded while this one computes.
  constexpr int kChunksPerThread = kTokTile * (kHd / 8) / (kRotWarps * 32);  // 4
  Chunk8<Tin> pre[kChunksPerThread];
  auto load_tile = [&](int64_t tile) {
#pragma unroll
    for (int k = 0; k < kChunksPerThread; ++k) {
      const int c = tid + k * kRotWarps * 32;
      const int64_t tok = tile * kTokTile + c % kTokTile;
      const int i0 = (c / kTokTile) * 8;
      load_chunk(static_cast<const Tin*>(a.x) + (tok < a.T ? tok : 0) * a.ld_token + static_cast<int64_t>(h) * kHd + i0,
                 tok < a.T, pre[k]);
    }
  };
  if (static_cast<int64_t>(blockIdx.x) < tiles) load_tile(blockIdx.x);
  for (int64_t tile = blockIdx.x; tile < tiles; tile += gridDim.x) {
    const int64_t t0 = tile * kTokTile;
    __syncthreads();  // the previous tile's reads of xs are done (and M is staged)
#pragma unroll
    for (int k = 0; k < kChunksPerThread; ++k) {
      const int c = tid + k * kRotWarps * 32;
      const int t = c % kTokTile, i0 = (c / kTokTile) * 8;
      float v[8];
      unpack_chunk(pre[k], v);
#pragma unroll
      for (int e = 0; e < 8; ++e) xs[(i0 + e) * kXPitch + t] = v[e];
    }
    __syncthreads();
    if (tile + gridDim.x < tiles) load_tile(tile + gridDim.x);

    // y[t][j] = sum_i x[t][i] M[i][j], i in order, for this warp's 8 tokens and
    // this lane's outputs j = 4 lane .. 4 lane + 3.
    float acc[kTokPerWarp][4];
#pragma unroll
    for (int t = 0; t < kTokPerWarp; ++t)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[t][c] = 0.f;
    const float* xw = xs + warp * kTokPerWarp;
#pragma unroll 4
    for (int i = 0; i < kHd; ++i) {
      const float4 m = *reinterpret_cast<const float4*>(Ms + i * kHd + 4 * lane);
      const float4 xa = *reinterpret_cast<const float4*>(xw + i * kXPitch);
      const float4 xb = *reinterpret_cast<const float4*>(xw + i * kXPitch + 4);
      const float xv[8] = {xa.x, xa.y, xa.z, xa.w, xb.x, xb.y, xb.z, xb.w};
#pragma unroll
      for (int t = 0; t < kTokPerWarp; ++t) {
        acc[t][0] = fmaf(xv[t], m.x, acc[t][0]);
        acc[t][1] = fmaf(xv[t], m.y, acc[t][1]);
        acc[t][2] = fmaf(xv[t], m.z, acc[t][2]);
        acc[t][3] = fmaf(xv[t], m.w, acc[t][3]);
      }
    }

#pragma unroll
    for (int t = 0; t < kTokPerWarp; ++t) {
      const int64_t tok = t0 + warp * kTokPerWarp + t;
      if (tok >= a.T) break;  // warp-uniform
      const int64_t th = tok * a.H + h;
      if (!a.quantize) {
        store4<OUT>(a.out, tok * a.ld_out + static_cast<int64_t>(h) * kHd + 4 * lane, acc[t][0], acc[t][1],
                    acc[t][2], acc[t][3]);
        continue;
      }
      float o = 0.f;
      if (a.offset) {
        float sum = (acc[t][0] + acc[t][1]) + (acc[t][2] + acc[t][3]);
#pragma unroll
        for (int m = 16; m > 0; m >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, m);
        o = sum * (1.0f / kHd);
      }
      const float r0 = acc[t][0] - o, r1 = acc[t][1] - o, r2 = acc[t][2] - o, r3 = acc[t][3] - o;
      float amax = fmaxf(fmaxf(fabsf(r0), fabsf(r1)), fmaxf(fabsf(r2), fabsf(r3)));
#pragma unroll
      for (int m = 16; m > 0; m >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xFFFFFFFFu, amax, m));
      const float inv = amax > 0.f ? __fdiv_rn(7.0f, amax) : 0.f;
      const float rr[4] = {r0, r1, r2, r3};
      uint32_t packed = 0;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const float q = fminf(fmaxf(rintf(rr[c] * inv), -7.f), 7.f);
        packed |= static_cast<uint32_t>(static_cast<int>(q) + 8) << (4 * c);
      }
      *reinterpret_cast<uint16_t*>(a.codes + th * (kHd / 2) + 2 * lane) = static_cast<uint16_t>(packed);
      if (lane == 0) {
        a.scale[th] = amax * (1.0f / 7.0f);
        if (a.off != nullptr) a.off[th] = o;
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Tensor-core kernel (bf16 keys)
// ---------------------------------------------------------------------------
constexpr int kTM = 128;                       // tokens per MMA tile
constexpr int kParts = 3;                      // bf16 parts of M
constexpr int kAtomBytes = 128 * 128;          // 128 rows x 64 bf16 (one 128-byte swizzle atom column)
constexpr int kOpBytes = 2 * kAtomBytes;       // 128 rows x 128 bf16
constexpr int kPrepBytes = kParts * kOpBytes;  // one head's three parts
constexpr int kAcc = 3;                        // TMEM accumulators
constexpr int kEpi = 3;                        // epilogue warpgroups, group e reading accumulator e
constexpr int kMmaThreads = 64 + 128 * kEpi;   // TMA warp, MMA warp, epilogue
static_assert(kPrepBytes == OFFQ_KEY_ROTATION_BYTES, "prepared image size");
static_assert(kEpi == kAcc, "each epilogue group owns one accumulator and takes its phases in order");

// The structured rotation M = U3 P3 H3 with U3 = I - 2 w w^T (a reflection):
// x M = u - 2 (x . w) w'' with u = x P3 H3 and w'' = (P3 H3)^T w. B holds
// rows n < 128 of sqrt(128) (P3 H)^T (entries +-1, exact in bf16), then the
// three bf16 parts of w (so one MMA also gives x . w), then zero rows to N = 144.
constexpr int kRefRows = 144;
constexpr int kRefAtom = kRefRows * 128;          // one 64-channel atom column of B
constexpr int kRefBBytes = 2 * kRefAtom;
constexpr int kRefImgBytes = kRefBBytes + kHd * 4;  // B, then w'' (fp32)
constexpr float kInvSqrtHd = 0.08838834764831844055f;  // 1 / sqrt(128), rounded to fp32
static_assert(kRefImgBytes == OFFQ_KEY_REFLECTION_BYTES, "prepared reflection size");

// Shared and tensor memory of the two variants: the dense one keeps M's
// three parts (96 KB) and four tile slots, the structured one its 36 KB
// image and five.
template <bool REFLECT>
struct RotLayout {
  static constexpr int kImg = REFLECT ? kRefImgBytes : kPrepBytes;     // bytes copied per head
  static constexpr int kBSmem = (kImg + 1023) / 1024 * 1024;          // ring stays 1024-aligned
  static constexpr int kSlots = REFLECT ? 5 : 4;
  static constexpr int kN = REFLECT ? kRefRows : kHd;                 // MMA N
  static constexpr int kAccCols = REFLECT ? 160 : kHd;               // accumulator stride in TMEM
  static constexpr int kCtrlOff = kBSmem + kSlots * kOpBytes;       // barriers, TMEM address, abort flag
  static constexpr int kCtrlBars = 8 * (1 + 2 * kSlots + 2 * kAcc);
  static constexpr int kSmem = kCtrlOff + kCtrlBars + 8 + 1024;
  // kind::f16: D f32 (bits 4-5 = 1), A and B bf16 (7-9, 10-12 = 1), both
  // K-major, N >> 3 at bit 17, M >> 4 at bit 24.
  static constexpr uint32_t kIdesc =
      (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(kN >> 3) << 17) | ((128u >> 4) << 24);
  static_assert(kSmem <= 232448, "one CTA per SM");
  static_assert(kAcc * kAccCols <= 512, "TMEM columns");
};

__device__ __forceinline__ void sts128v(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

// 1.5 * 2^23 + 8 and the bits of 1.5 * 2^23: fl(x + kRoundMagic) for |x| < 2^21
// is 1.5 * 2^23 + 8 + round_half_even(x), whose bits are kRoundMagicBits + that.
constexpr float kRoundMagic = 12582920.0f;
constexpr uint32_t kRoundMagicBits = 0x4B400000u;

__device__ __forceinline__ uint64_t add2v(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
__device__ __forceinline__ uint64_t sub2v(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

// Shared -> global TMA store of one box (tensor coordinates x, y), tracked in
// this thread's bulk groups; rows past the tensor are not written.
__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, uint32_t src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%2, %3}], [%1];" ::"l"(map),
               "r"(src), "r"(x), "r"(y)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// This thread's bulk stores have read their shared-memory source.
__device__ __forceinline__ void bulk_wait_read_all() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// This thread's bulk stores are complete.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// Barrier over the 128 threads of named barrier `id`.
__device__ __forceinline__ void wg_sync(int id) { asm volatile("bar.sync %0, 128;" ::"r"(id) : "memory"); }

// The same barrier, returning whether `pred` held for any of the 128 threads.
__device__ __forceinline__ bool wg_any(int id, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n"
      ".reg .pred p, q;\n"
      "setp.ne.b32 p, %1, 0;\n"
      "bar.red.or.pred q, %2, 128, p;\n"
      "selp.u32 %0, 1, 0, q;\n"
      "}\n"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(pred)), "r"(id)
      : "memory");
  return r != 0;
}

// Two floats as one 32-bit word of 16-bit values (round to nearest even).
template <int OUT>
__device__ __forceinline__ uint32_t pack16(float a, float b) {
  if constexpr (OUT == OFFQ_BF16) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&v);
  } else {
    const __half2 v = __floats2half2_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&v);
  }
}

// Global -> shared bulk copy (async proxy), completing `bytes` on an mbarrier.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
               "l"(src), "r"(bytes), "r"(bar)
               : "memory");
}

// Waits for this thread's TMEM loads; the registers they fill are operands, so
// no use of them moves above the wait.
__device__ __forceinline__ void tmem_wait_into(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                 "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                 "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                 "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}

// The four 32-column chunks of this thread's 128-column TMEM row: f(v, c) on
// chunk c while chunk c + 1 is loading; last() once all four are loaded.
template <typename F, typename G>
__device__ __forceinline__ void tmem_row_pass(uint32_t row_tm, F&& f, G&& last) {
  uint32_t va[32], vb[32];
  tmem_ld_32cols(row_tm, va);
  tmem_wait_into(va);
  tmem_ld_32cols(row_tm + 32, vb);
  f(va, 0);
  tmem_wait_into(vb);
  tmem_ld_32cols(row_tm + 64, va);
  f(vb, 1);
  tmem_wait_into(va);
  tmem_ld_32cols(row_tm + 96, vb);
  f(va, 2);
  tmem_wait_into(vb);
  last();
  f(vb, 3);
}

// Byte offset of 16-byte chunk c (8 bf16, c = 0..15) of row r in a 128-row
// K-major operand: two 16 KB atom columns, 128-byte rows, chunk swizzle c ^ (r & 7).
__device__ __forceinline__ uint32_t sw_off(int r, int c) {
  return (c >> 3) * kAtomBytes + r * 128 + (((c & 7) ^ (r & 7)) << 4);
}

__device__ __forceinline__ uint32_t bf16_bits(float v) {
  const __nv_bfloat16 b = __float2bfloat16_rn(v);
  return static_cast<uint32_t>(*reinterpret_cast<const uint16_t*>(&b));
}

// m = hi + mid + lo + e with |e| <= 2^-24 |m| roughly: each part rounds what
// the previous ones left (the differences are exact in fp32).
__device__ __forceinline__ void split3(float m, uint32_t& hi, uint32_t& mid, uint32_t& lo) {
  hi = bf16_bits(m);
  const float r1 = m - __uint_as_float(hi << 16);
  mid = bf16_bits(r1);
  const float r2 = r1 - __uint_as_float(mid << 16);
  lo = bf16_bits(r2);
}

// Column n of M, k-chunks c0 .. c0 + 3 (k = 8 c0 .. 8 c0 + 31): w[cc][s] holds
// part s of M[8 (c0 + cc) .. + 7][n] as 8 bf16. The 32 loads of a thread are
// in flight together; across threads (consecutive n) they are coalesced.
__device__ __forceinline__ void split_column(const float* Mh, int n, int c0, uint4 (&w)[4][kParts]) {
  float m[4][8];
#pragma unroll
  for (int cc = 0; cc < 4; ++cc)
#pragma unroll
    for (int e = 0; e < 8; ++e) m[cc][e] = __ldg(Mh + (8 * (c0 + cc) + e) * kHd + n);
#pragma unroll
  for (int cc = 0; cc < 4; ++cc) {
    uint32_t p[kParts][4];
#pragma unroll
    for (int e = 0; e < 8; e += 2) {
      uint32_t h0, m0, l0, h1, m1, l1;
      split3(m[cc][e], h0, m0, l0);
      split3(m[cc][e + 1], h1, m1, l1);
      p[0][e / 2] = h0 | (h1 << 16);
      p[1][e / 2] = m0 | (m1 << 16);
      p[2][e / 2] = l0 | (l1 << 16);
    }
#pragma unroll
    for (int s = 0; s < kParts; ++s) w[cc][s] = make_uint4(p[s][0], p[s][1], p[s][2], p[s][3]);
  }
}

// The prepared image: head h's part s at prep[h][s], B_s[n][k] = part s of
// M[k][n] in the shared-memory operand layout (sw_off), so the tensor-core
// kernel copies it as is. Grid (4, H) x 128 threads: thread n, k-chunks 4 bx .. + 3.
__global__ void __launch_bounds__(128) prepare_rotation_kernel(const float* __restrict__ rot,
                                                               uint8_t* __restrict__ prep) {
  const int h = blockIdx.y, n = threadIdx.x, c0 = 4 * blockIdx.x;
  griddep_wait();
  griddep_launch_dependents();
  uint4 w[4][kParts];
  split_column(rot + static_cast<int64_t>(h) * kHd * kHd, n, c0, w);
  uint8_t* dst = prep + static_cast<int64_t>(h) * kPrepBytes;
#pragma unroll
  for (int cc = 0; cc < 4; ++cc)
#pragma unroll
    for (int s = 0; s < kParts; ++s) *reinterpret_cast<uint4*>(dst + s * kOpBytes + sw_off(n, c0 + cc)) = w[cc][s];
}

// One CTA per (head, share of its tiles), warp-specialised:
//   warp 0    loads the CTA's 128-token tiles by TMA into a ring of kSlots
//             buffers (two 64-channel boxes per tile, 128-byte swizzle) and,
//             with a prepared image, M's three parts by one bulk copy each;
//   warp 1    allocates the accumulators and issues each tile's 3 x 8 MMAs;
//   warps 2.. (kEpi groups of four) read an accumulator, write the codes and
//             free it: group e takes the CTA's tiles e, e + kEpi, ... in
//             accumulator e.
// Without a prepared image the epilogue warps split M into the three parts
// before their first tile. REFLECT: the structured image instead (one MMA of
// N = 144 per 16 channels; the epilogue forms y = u - 2 (x . w) w'').
template <int OUT, bool REFLECT>
__global__ void __launch_bounds__(kMmaThreads, 1)
    rotate_heads_mma_kernel(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ CUtensorMap omap,
                            const RotArgs a) {
  using L = RotLayout<REFLECT>;
  // 16-bit rotated outputs (the query side) are staged in the tile's own ring
  // slot and leave by TMA stores; the slot is freed after the store has read it.
  constexpr bool kStage = OUT != OFFQ_F32;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (base - raw);
  // B: kParts operands B_s[n][k] = part s of M[k][n], or the structured image.
  const uint32_t b_base = base;
  const uint32_t ring = base + L::kBSmem;           // L::kSlots token tiles
  const uint32_t ctrl = base + L::kCtrlOff;
  const uint32_t bar_b = ctrl;                      // B is in shared memory
  const uint32_t full0 = ctrl + 8;                  // [kSlots] a tile has landed
  const uint32_t empty0 = full0 + 8 * L::kSlots;    // [kSlots] its MMAs have read it
  const uint32_t tfull0 = empty0 + 8 * L::kSlots;   // [kAcc] an accumulator holds a tile's product
  const uint32_t tempty0 = tfull0 + 8 * kAcc;       // [kAcc] its four epilogue warps have read it
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::kCtrlOff + L::kCtrlBars);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + L::kCtrlOff + L::kCtrlBars + 4);
  const int h = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const bool prepared = a.prep != nullptr;
  if (tid == 0) {
    mbar_init(bar_b, prepared ? 1 : 128 * kEpi);
#pragma unroll
    for (int s = 0; s < L::kSlots; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
#pragma unroll
    for (int x = 0; x < kAcc; ++x) {
      mbar_init(tfull0 + 8 * x, 1);
      mbar_init(tempty0 + 8 * x, 4);
    }
    *abort = 0;
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  griddep_wait();
  griddep_launch_dependents();

  const int64_t tiles = (a.T + kTM - 1) / kTM;
  const int n_local = static_cast<int>((tiles - blockIdx.x + gridDim.x - 1) / gridDim.x);  // >= 1

  if (warp == 0) {
    if (lane == 0) {
      if (prepared) {
        const uint8_t* src = static_cast<const uint8_t*>(a.prep) + static_cast<int64_t>(h) * L::kImg;
        mbar_arrive_expect_tx(bar_b, L::kImg);
        if constexpr (REFLECT) {
          bulk_load(b_base, src, L::kImg, bar_b);
        } else {
#pragma unroll
          for (int s = 0; s < kParts; ++s) bulk_load(b_base + s * kOpBytes, src + s * kOpBytes, kOpBytes, bar_b);
        }
      }
      tma_prefetch_desc(&xmap);
      int i = 0;
      for (; i < n_local; ++i) {
        const int s = i % L::kSlots;
        if (i >= L::kSlots && !mbar_wait(empty0 + 8 * s, ((i / L::kSlots) - 1) & 1, abort)) break;
        const int y = static_cast<int>((blockIdx.x + static_cast<int64_t>(i) * gridDim.x) * kTM);
        const uint32_t dst = ring + s * kOpBytes;
        mbar_arrive_expect_tx(full0 + 8 * s, kOpBytes);
        tma_load_2d(dst, &xmap, full0 + 8 * s, h * kHd, y);
        tma_load_2d(dst + kAtomBytes, &xmap, full0 + 8 * s, h * kHd + 64, y);
      }
      if (*abort) {
        // Copies still in flight land (bounded) before shared memory is released.
        const long long c0 = clock64();
        for (int j = i - 1; j >= 0 && j >= i - L::kSlots; --j)
          while (!mbar_try_wait(full0 + 8 * (j % L::kSlots), (j / L::kSlots) & 1) && clock64() - c0 < kWaitCycles) {
          }
        if (prepared)
          while (!mbar_try_wait(bar_b, 0) && clock64() - c0 < kWaitCycles) {
          }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      int committed = -1;
      if (mbar_wait(bar_b, 0, abort)) {
        for (int i = 0; i < n_local; ++i) {
          const int s = i % L::kSlots, x = i % kAcc;
          if (!mbar_wait(full0 + 8 * s, (i / L::kSlots) & 1, abort)) break;
          if (i >= kAcc && !mbar_wait(tempty0 + 8 * x, ((i / kAcc) - 1) & 1, abort)) break;
          tc_fence_after();
          const uint32_t at = ring + s * kOpBytes, acc = tmem + x * L::kAccCols;
          if constexpr (REFLECT) {
#pragma unroll
            for (int kk = 0; kk < kHd / 16; ++kk) {
              const uint32_t koff = (kk & 3) * 32;
              mma_bf16(acc, smem_desc_sw128(at + (kk >> 2) * kAtomBytes + koff),
                       smem_desc_sw128(b_base + (kk >> 2) * kRefAtom + koff), L::kIdesc, kk != 0 ? 1u : 0u);
            }
          } else {
#pragma unroll
            for (int sp = 0; sp < kParts; ++sp)
#pragma unroll
              for (int kk = 0; kk < kHd / 16; ++kk) {
                const uint32_t koff = (kk >> 2) * kAtomBytes + (kk & 3) * 32;
                mma_bf16(acc, smem_desc_sw128(at + koff), smem_desc_sw128(b_base + sp * kOpBytes + koff), L::kIdesc,
                         (sp | kk) != 0 ? 1u : 0u);
              }
          }
          if constexpr (!kStage) mma_commit(empty0 + 8 * s);  // the tile buffer is free once these MMAs are done
          mma_commit(tfull0 + 8 * x);
          committed = i;
        }
      }
      if (*abort && committed >= 0) {
        // MMAs complete in issue order: wait (bounded) for the last commit
        // before tensor memory is released.
        const long long c0 = clock64();
        while (!mbar_try_wait(tfull0 + 8 * (committed % kAcc), (committed / kAcc) & 1) &&
               clock64() - c0 < kWaitCycles) {
        }
      }
    }
    __syncwarp();
  } else {
    const int e = (warp - 2) >> 2;  // epilogue group
    const int q = warp & 3;         // the TMEM lane quadrant this warp may read
    const int et = tid - 64;
    if (!REFLECT && !prepared) {
      // Units u = (column n = u % 128, k-chunks 4 (u / 128) .. + 3) of M[h].
      for (int u = et; u < 4 * kHd; u += 128 * kEpi) {
        uint4 w[4][kParts];
        const int n = u & (kHd - 1), c0 = 4 * (u >> 7);
        split_column(a.rot + static_cast<int64_t>(h) * kHd * kHd, n, c0, w);
#pragma unroll
        for (int cc = 0; cc < 4; ++cc)
#pragma unroll
          for (int s = 0; s < kParts; ++s) sts128v(b_base + s * kOpBytes + sw_off(n, c0 + cc), w[cc][s]);
      }
      fence_proxy_async_smem();
      mbar_arrive(bar_b);
    }
    for (int i = e; i < n_local; i += kEpi) {
      const int x = i % kAcc;
      const bool waited = mbar_wait(tfull0 + 8 * x, (i / kAcc) & 1, abort);
      // The warp leaves together; with staged outputs (a group barrier per
      // tile) the whole group does.
      if (kStage ? wg_any(1 + e, !waited) : __any_sync(0xFFFFFFFFu, !waited)) break;
      tc_fence_after();
      const uint32_t row_tm = tmem + x * L::kAccCols + (static_cast<uint32_t>(q * 32) << 16);
      // y for columns (j, j + 1) of a 32-column chunk c: the accumulator, or
      // (structured) fma(acc, 1/sqrt(128), fl(-2 d w''_j)) with d = x . w.
      uint64_t nd2 = 0;
      if constexpr (REFLECT) {
        uint32_t dv[16];
        tmem_ld_16cols(row_tm + kHd, dv);
        tmem_ld_wait();
        const float d = (__uint_as_float(dv[0]) + __uint_as_float(dv[1])) + __uint_as_float(dv[2]);  // x . w
        nd2 = pack2(-2.f * d, -2.f * d);
      }
      const uint64_t* w2 = reinterpret_cast<const uint64_t*>(smem + kRefBBytes);  // w'' pairs (structured)
      auto ypair = [&](const uint32_t (&v)[32], int c, int j) -> uint64_t {
        const uint64_t acc2 = pack2(__uint_as_float(v[j]), __uint_as_float(v[j + 1]));
        if constexpr (REFLECT) {
          return fma2v(acc2, pack2(kInvSqrtHd, kInvSqrtHd), mul2v(nd2, w2[(c * 32 + j) >> 1]));
        } else {
          return acc2;
        }
      };
      // Thread (q, lane) owns token tile * 128 + 32 q + lane (TMEM lane 32 q + lane).
      const int64_t tok = (blockIdx.x + static_cast<int64_t>(i) * gridDim.x) * kTM + q * 32 + lane;
      const bool ok = tok < a.T;
      const int64_t th = tok * a.H + h;
      if (a.quantize) {
        // Pass 1: the offset (two fp32 partial sums, lanes of one f32x2 add)
        // and the extremes of y.
        uint64_t sum2 = pack2(0.f, 0.f);
        float ymax0 = -INFINITY, ymax1 = -INFINITY, ymin0 = INFINITY, ymin1 = INFINITY;
        tmem_row_pass(
            row_tm,
            [&](const uint32_t (&v)[32], int c) {
#pragma unroll
              for (int j = 0; j < 32; j += 2) {
                const uint64_t y2 = ypair(v, c, j);
                float y0, y1;
                unpack2(y2, y0, y1);
                sum2 = add2v(sum2, y2);
                ymax0 = fmaxf(ymax0, y0);
                ymax1 = fmaxf(ymax1, y1);
                ymin0 = fminf(ymin0, y0);
                ymin1 = fminf(ymin1, y1);
              }
            },
            [] {});
        float s0, s1;
        unpack2(sum2, s0, s1);
        const float o = a.offset ? (s0 + s1) * (1.0f / kHd) : 0.f;
        // max_j |fl(y_j - o)| from the extremes: rounding is monotone and
        // fl(o - y) = -fl(y - o), so the largest are fl(ymax - o) and fl(o - ymin).
        const float amax = fmaxf(fmaxf(ymax0, ymax1) - o, o - fminf(ymin0, ymin1));
        const float inv = amax > 0.f ? __fdiv_rn(7.0f, amax) : 0.f;
        // Pass 2: q = rne(fl(fl(y - o) * inv)). |fl(y - o)| <= amax and
        // inv <= (7 / amax)(1 + 2^-24), so |q| <= 7 and the clamp to [-7, 7]
        // never binds. Adding 1.5 * 2^23 + 8 rounds to the nearest even integer
        // (the float spacing there is 1) and leaves u = q + 8 in the low bits of
        // the sum; eight of them are packed with shifts and one bias subtraction.
        const uint64_t o2 = pack2(o, o), inv2 = pack2(inv, inv), magic2 = pack2(kRoundMagic, kRoundMagic);
        tmem_row_pass(
            row_tm,
            [&](const uint32_t (&v)[32], int c) {
              uint32_t pk[4];
#pragma unroll
              for (int w8 = 0; w8 < 4; ++w8) {
                uint32_t word = 0u;
#pragma unroll
                for (int j = 8 * w8 + 6; j >= 8 * w8; j -= 2) {
                  const uint64_t r2 = sub2v(ypair(v, c, j), o2);
                  float f0, f1;
                  unpack2(add2v(mul2v(r2, inv2), magic2), f0, f1);
                  word = (word << 4) + __float_as_uint(f1);
                  word = (word << 4) + __float_as_uint(f0);
                }
                pk[w8] = word - kRoundMagicBits * 0x11111111u;
              }
              if (ok)
                *reinterpret_cast<uint4*>(a.codes + th * (kHd / 2) + 16 * c) =
                    make_uint4(pk[0], pk[1], pk[2], pk[3]);
            },
            [&] {
              // The accumulator's last read: hand it back to the MMA warp.
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(tempty0 + 8 * x);
            });
        if (ok) {
          a.scale[th] = amax * (1.0f / 7.0f);
          if (a.off != nullptr) a.off[th] = o;
        }
      } else if constexpr (kStage) {
        // Row q * 32 + lane of the slot, in the swizzled layout of the
        // output tensor map's two 64-channel boxes.
        const int s = i % L::kSlots;
        const uint32_t st = ring + s * kOpBytes;
        tmem_row_pass(
            row_tm,
            [&](const uint32_t (&v)[32], int c) {
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                uint32_t pk[4];
#pragma unroll
                for (int p = 0; p < 4; ++p) {
                  float y0, y1;
                  unpack2(ypair(v, c, 8 * k + 2 * p), y0, y1);
                  pk[p] = pack16<OUT>(y0, y1);
                }
                sts128v(st + sw_off(q * 32 + lane, 4 * c + k), make_uint4(pk[0], pk[1], pk[2], pk[3]));
              }
            },
            [&] {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(tempty0 + 8 * x);
            });
        fence_proxy_async_smem();  // the staged rows, visible to the TMA unit
        wg_sync(1 + e);
        if (warp == 2 + 4 * e && lane == 0) {
          const int y0 = static_cast<int>((blockIdx.x + static_cast<int64_t>(i) * gridDim.x) * kTM);
          tma_store_2d(&omap, st, h * kHd, y0);
          tma_store_2d(&omap, st + kAtomBytes, h * kHd + 64, y0);
          bulk_commit();
          bulk_wait_read_all();
          mbar_arrive(empty0 + 8 * s);
        }
      } else {
        tmem_row_pass(
            row_tm,
            [&](const uint32_t (&v)[32], int c) {
              if (ok) {
#pragma unroll
                for (int j = 0; j < 32; j += 4) {
                  float y0, y1, y2, y3;
                  unpack2(ypair(v, c, j), y0, y1);
                  unpack2(ypair(v, c, j + 2), y2, y3);
                  store4<OUT>(a.out, tok * a.ld_out + static_cast<int64_t>(h) * kHd + c * 32 + j, y0, y1, y2, y3);
                }
              }
            },
            [&] {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(tempty0 + 8 * x);
            });
      }
    }
    if constexpr (kStage) {
      if (warp == 2 + 4 * e && lane == 0) bulk_wait_all();  // the stores are complete before the CTA exits
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
  if (tid == 0 && *abort && a.status != nullptr) atomicExch(a.status, kErrTimeout);
}

int rot_num_sms() {
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

template <typename Tin, int OUT>
int launch_rotate(const RotArgs& a, cudaStream_t s) {
  auto kern = rotate_heads_kernel<Tin, OUT>;
  if (!smem_optin<rotate_heads_kernel<Tin, OUT>>(kRotSmem)) return OFFQ_ERR_CUDA;
  // About two CTAs per SM (the shared-memory limit), spread over the heads;
  // each loops over its head's token tiles.
  const int sms = rot_num_sms();
  if (sms < 1) return OFFQ_ERR_CUDA;
  const int64_t tiles = (a.T + kTokTile - 1) / kTokTile;
  int64_t per_head = (2 * sms + a.H - 1) / a.H;
  if (per_head > tiles) per_head = tiles;
  const dim3 grid(static_cast<unsigned>(per_head), static_cast<unsigned>(a.H));
  return launch_pdl(kern, grid, dim3(kRotWarps * 32), kRotSmem, s, a);
}

// A [T][H * 128] tensor of 16-bit elements (row pitch ld elements) in boxes
// of 64 channels x 128 tokens with the 128-byte swizzle of the MMA operand:
// the bf16 keys read (rows past T read as zeros), or the 16-bit rotated
// outputs written (rows past T are not written).
int encode_heads_map(CUtensorMap* map, const void* x, int dtype, int64_t T, int H, int64_t ld) {
  const auto enc = tensor_map_encoder();
  if (enc == nullptr) return OFFQ_ERR_CUDA;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(H) * kHd, static_cast<cuuint64_t>(T)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld) * 2};
  const cuuint32_t box[2] = {64, kTM};
  const cuuint32_t elem_strides[2] = {1, 1};
  const CUresult r = enc(map, dtype == OFFQ_F16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                         const_cast<void*>(x), dims, strides, box,
                         elem_strides, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                         CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? OFFQ_OK : OFFQ_ERR_CUDA;
}

template <int OUT, bool REFLECT = false>
int launch_rotate_mma(const RotArgs& a, cudaStream_t s) {
  using L = RotLayout<REFLECT>;
  auto kern = rotate_heads_mma_kernel<OUT, REFLECT>;
  if (!smem_optin<rotate_heads_mma_kernel<OUT, REFLECT>>(L::kSmem)) return OFFQ_ERR_CUDA;
  CUtensorMap xmap, omap;
  if (encode_heads_map(&xmap, a.x, OFFQ_BF16, a.T, a.H, a.ld_token) != OFFQ_OK) return OFFQ_ERR_CUDA;
  if constexpr (OUT != OFFQ_F32) {
    if (encode_heads_map(&omap, a.out, OUT, a.T, a.H, a.ld_out) != OFFQ_OK) return OFFQ_ERR_CUDA;
  } else {
    omap = xmap;  // not used
  }
  // One CTA per SM (shared memory), spread over the heads; each takes every
  // gridDim.x-th of its head's 128-token tiles.
  const int sms = rot_num_sms();
  if (sms < 1) return OFFQ_ERR_CUDA;
  const int64_t tiles = (a.T + kTM - 1) / kTM;
  int64_t per_head = sms / a.H > 0 ? sms / a.H : 1;
  if (per_head > tiles) per_head = tiles;
  const dim3 grid(static_cast<unsigned>(per_head), static_cast<unsigned>(a.H));
  return launch_pdl(kern, grid, dim3(kMmaThreads), L::kSmem, s, xmap, omap, a);
}

template <int OUT>
int dispatch_in(int dtype, const RotArgs& a, cudaStream_t s) {
  switch (dtype) {
    case OFFQ_F32: return launch_rotate<float, OUT>(a, s);
    case OFFQ_BF16: return launch_rotate_mma<OUT>(a, s);
    case OFFQ_F16: return launch_rotate<__half, OUT>(a, s);
    default: return OFFQ_ERR_INVALID_ARG;
  }
}

int check_heads(const void* x, int dtype, int64_t T, int32_t H, int32_t head_dim, int64_t ld_token,
                const void* rot) {
  const int eb = elem_bytes(dtype);
  if (eb == 0 || T < 0 || H < 1 || head_dim <= 0 || ld_token < static_cast<int64_t>(H) * head_dim)
    return OFFQ_ERR_INVALID_ARG;
  if (head_dim != kHd) return OFFQ_ERR_UNSUPPORTED;
  if (T > 0x3FFFFFFF || H > 65535) return OFFQ_ERR_UNSUPPORTED;
  if (T > 0 && (x == nullptr || rot == nullptr)) return OFFQ_ERR_INVALID_ARG;
  if (T > 0 && (!aligned(x, 16) || (ld_token * eb) % 16 != 0 || !aligned(rot, 16))) return OFFQ_ERR_MISALIGNED;
  return OFFQ_OK;
}

}  // namespace

extern "C" int offq_kv4_quantize_rotated(const void* kv, int dtype, int64_t T, int32_t H, int32_t head_dim,
                                         int64_t ld_token, const float* rot, int32_t flags, uint8_t* codes,
                                         float* scale, float* offset, void* stream) {
  if ((flags & ~OFFQ_OFFSET) != 0) return OFFQ_ERR_INVALID_ARG;
  int st = check_heads(kv, dtype, T, H, head_dim, ld_token, rot);
  if (st != OFFQ_OK) return st;
  if (T == 0) return OFFQ_OK;
  if (codes == nullptr || scale == nullptr || ((flags & OFFQ_OFFSET) && offset == nullptr))
    return OFFQ_ERR_INVALID_ARG;
  if (!aligned(codes, 16) || !aligned(scale, 4) || (offset != nullptr && !aligned(offset, 4)))
    return OFFQ_ERR_MISALIGNED;
  RotArgs a{};
  a.x = kv;
  a.ld_token = ld_token;
  a.T = T;
  a.H = H;
  a.rot = rot;
  a.quantize = 1;
  a.offset = (flags & OFFQ_OFFSET) != 0;
  a.codes = codes;
  a.scale = scale;
  a.off = offset;
  a.status = device_status_ptr();
  return dispatch_in<OFFQ_F32>(dtype, a, static_cast<cudaStream_t>(stream));
}

extern "C" int offq_rotate_heads(const void* x, int dtype, int64_t T, int32_t H, int32_t head_dim, int64_t ld_token,
                                 const float* rot, void* out, int out_dtype, int64_t ld_out, void* stream) {
  const int ob = elem_bytes(out_dtype);
  if (ob == 0 || ld_out < static_cast<int64_t>(H) * head_dim) return OFFQ_ERR_INVALID_ARG;
  int st = check_heads(x, dtype, T, H, head_dim, ld_token, rot);
  if (st != OFFQ_OK) return st;
  if (T == 0) return OFFQ_OK;
  if (out == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(out, 16) || (ld_out * ob) % 16 != 0) return OFFQ_ERR_MISALIGNED;
  RotArgs a{};
  a.x = x;
  a.ld_token = ld_token;
  a.T = T;
  a.H = H;
  a.rot = rot;
  a.quantize = 0;
  a.out = out;
  a.ld_out = ld_out;
  a.status = device_status_ptr();
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  switch (out_dtype) {
    case OFFQ_F32: return dispatch_in<OFFQ_F32>(dtype, a, s);
    case OFFQ_BF16: return dispatch_in<OFFQ_BF16>(dtype, a, s);
    case OFFQ_F16: return dispatch_in<OFFQ_F16>(dtype, a, s);
    default: return OFFQ_ERR_INVALID_ARG;
  }
}

extern "C" int offq_prepare_key_rotation(const float* rot, int32_t H, int32_t head_dim, void* prepared,
                                         void* stream) {
  if (H < 1 || head_dim <= 0) return OFFQ_ERR_INVALID_ARG;
  if (head_dim != kHd) return OFFQ_ERR_UNSUPPORTED;
  if (H > 65535) return OFFQ_ERR_UNSUPPORTED;
  if (rot == nullptr || prepared == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(rot, 16) || !aligned(prepared, 16)) return OFFQ_ERR_MISALIGNED;
  return launch_pdl(prepare_rotation_kernel, dim3(kHd / 32, static_cast<unsigned>(H)), dim3(kHd),
                    0, static_cast<cudaStream_t>(stream), rot, static_cast<uint8_t*>(prepared));
}

extern "C" int offq_kv4_quantize_prepared(const void* kv, int dtype, int64_t T, int32_t H, int32_t head_dim,
                                          int64_t ld_token, const void* prepared, int32_t flags, uint8_t* codes,
                                          float* scale, float* offset, void* stream) {
  if ((flags & ~OFFQ_OFFSET) != 0) return OFFQ_ERR_INVALID_ARG;
  int st = check_heads(kv, dtype, T, H, head_dim, ld_token, prepared);
  if (st != OFFQ_OK) return st;
  if (dtype != OFFQ_BF16) return OFFQ_ERR_UNSUPPORTED;
  if (T == 0) return OFFQ_OK;
  if (codes == nullptr || scale == nullptr || ((flags & OFFQ_OFFSET) && offset == nullptr))
    return OFFQ_ERR_INVALID_ARG;
  if (!aligned(codes, 16) || !aligned(scale, 4) || (offset != nullptr && !aligned(offset, 4)))
    return OFFQ_ERR_MISALIGNED;
  RotArgs a{};
  a.x = kv;
  a.ld_token = ld_token;
  a.T = T;
  a.H = H;
  a.prep = prepared;
  a.quantize = 1;
  a.offset = (flags & OFFQ_OFFSET) != 0;
  a.codes = codes;
  a.scale = scale;
  a.off = offset;
  a.status = device_status_ptr();
  return launch_rotate_mma<OFFQ_F32>(a, static_cast<cudaStream_t>(stream));
}

extern "C" int offq_rotate_heads_prepared(const void* x, int dtype, int64_t T, int32_t H, int32_t head_dim,
                                          int64_t ld_token, const void* prepared, void* out, int out_dtype,
                                          int64_t ld_out, void* stream) {
  const int ob = elem_bytes(out_dtype);
  if (ob == 0 || ld_out < static_cast<int64_t>(H) * head_dim) return OFFQ_ERR_INVALID_ARG;
  int st = check_heads(x, dtype, T, H, head_dim, ld_token, prepared);
  if (st != OFFQ_OK) return st;
  if (dtype != OFFQ_BF16) return OFFQ_ERR_UNSUPPORTED;
  if (T == 0) return OFFQ_OK;
  if (out == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(out, 16) || (ld_out * ob) % 16 != 0) return OFFQ_ERR_MISALIGNED;
  RotArgs a{};
  a.x = x;
  a.ld_token = ld_token;
  a.T = T;
  a.H = H;
  a.prep = prepared;
  a.quantize = 0;
  a.out = out;
  a.ld_out = ld_out;
  a.status = device_status_ptr();
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  switch (out_dtype) {
    case OFFQ_F32: return launch_rotate_mma<OFFQ_F32>(a, s);
    case OFFQ_BF16: return launch_rotate_mma<OFFQ_BF16>(a, s);
    case OFFQ_F16: return launch_rotate_mma<OFFQ_F16>(a, s);
    default: return OFFQ_ERR_INVALID_ARG;
  }
}

namespace {

// Host round-to-nearest-even of a finite float to bf16 bits.
uint16_t host_bf16(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  return static_cast<uint16_t>((u + 0x7FFFu + ((u >> 16) & 1u)) >> 16);
}

float host_bf16_value(uint16_t b) {
  const uint32_t u = static_cast<uint32_t>(b) << 16;
  float f;
  std::memcpy(&f, &u, 4);
  return f;
}

}  // namespace

extern "C" int offq_prepare_key_reflection(const float* v, const int32_t* perm, int32_t H, int32_t head_dim,
                                           void* prepared) {
  if (H < 1 || head_dim <= 0) return OFFQ_ERR_INVALID_ARG;
  if (head_dim != kHd) return OFFQ_ERR_UNSUPPORTED;
  if (H > 65535) return OFFQ_ERR_UNSUPPORTED;
  if (v == nullptr || perm == nullptr || prepared == nullptr) return OFFQ_ERR_INVALID_ARG;
  for (int32_t h = 0; h < H; ++h) {
    bool seen[kHd] = {};
    double nv = 0.0;
    for (int c = 0; c < kHd; ++c) {
      const int32_t p = perm[static_cast<int64_t>(h) * kHd + c];
      if (p < 0 || p >= kHd || seen[p]) return OFFQ_ERR_INVALID_ARG;
      seen[p] = true;
      const double vc = v[static_cast<int64_t>(h) * kHd + c];
      if (!std::isfinite(vc)) return OFFQ_ERR_INVALID_ARG;
      nv += vc * vc;
    }
    if (!(nv > 0.0)) return OFFQ_ERR_INVALID_ARG;
  }
  uint8_t* out = static_cast<uint8_t*>(prepared);
  for (int32_t h = 0; h < H; ++h) {
    const float* vh = v + static_cast<int64_t>(h) * kHd;
    const int32_t* ph = perm + static_cast<int64_t>(h) * kHd;
    // The reflection taking e_0 to v / |v|: U3 = I - 2 w w^T, w = (v/|v| - e_0)
    // normalised (U3 = I when v / |v| = e_0), in float64.
    double nv = 0.0;
    for (int c = 0; c < kHd; ++c) nv += static_cast<double>(vh[c]) * vh[c];
    nv = std::sqrt(nv);
    double w[kHd];
    double nw = 0.0;
    for (int c = 0; c < kHd; ++c) {
      w[c] = vh[c] / nv - (c == 0 ? 1.0 : 0.0);
      nw += w[c] * w[c];
    }
    if (nw < 1e-30) {
      for (int c = 0; c < kHd; ++c) w[c] = 0.0;
    } else {
      nw = std::sqrt(nw);
      for (int c = 0; c < kHd; ++c) w[c] /= nw;
    }
    // (x P3)_c = x_perm[c], so (P3 H)[k][n] = H[inv[k]][n] with inv = perm^-1,
    // and H[i][n] = (-1)^popcount(i & n) (Sylvester).
    int inv[kHd];
    for (int c = 0; c < kHd; ++c) inv[ph[c]] = c;
    auto ph_entry = [&](int k, int n) { return (__builtin_popcount(static_cast<unsigned>(inv[k] & n)) & 1) ? -1 : 1; };
    uint8_t* img = out + static_cast<int64_t>(h) * kRefImgBytes;
    std::memset(img, 0, kRefImgBytes);
    // Rows 128..130: the three bf16 parts of fp32(w).
    uint16_t wp[3][kHd];
    for (int k = 0; k < kHd; ++k) {
      const float wf = static_cast<float>(w[k]);
      wp[0][k] = host_bf16(wf);
      const float r1 = wf - host_bf16_value(wp[0][k]);
      wp[1][k] = host_bf16(r1);
      const float r2 = r1 - host_bf16_value(wp[1][k]);
      wp[2][k] = host_bf16(r2);
    }
    for (int r = 0; r < kRefRows; ++r)
      for (int c = 0; c < kHd / 8; ++c) {
        uint16_t chunk[8] = {};
        for (int e = 0; e < 8; ++e) {
          const int k = 8 * c + e;
          if (r < kHd) chunk[e] = ph_entry(k, r) > 0 ? 0x3F80u : 0xBF80u;
          else if (r < kHd + 3) chunk[e] = wp[r - kHd][k];
        }
        std::memcpy(img + (c >> 3) * kRefAtom + r * 128 + (((c & 7) ^ (r & 7)) << 4), chunk, 16);
      }
    // w'' = (P3 H3)^T w, H3 = H / sqrt(128).
    float* wpp = reinterpret_cast<float*>(img + kRefBBytes);
    for (int n = 0; n < kHd; ++n) {
      double acc = 0.0;
      for (int k = 0; k < kHd; ++k) acc += ph_entry(k, n) * w[k];
      wpp[n] = static_cast<float>(acc / std::sqrt(static_cast<double>(kHd)));
    }
  }
  return OFFQ_OK;
}

extern "C" int offq_kv4_quantize_reflected(const void* kv, int dtype, int64_t T, int32_t H, int32_t head_dim,
                                           int64_t ld_token, const void* prepared, int32_t flags, uint8_t* codes,
                                           float* scale, float* offset, void* stream) {
  if ((flags & ~OFFQ_OFFSET) != 0) return OFFQ_ERR_INVALID_ARG;
  int st = check_heads(kv, dtype, T, H, head_dim, ld_token, prepared);
  if (st != OFFQ_OK) return st;
  if (dtype != OFFQ_BF16) return OFFQ_ERR_UNSUPPORTED;
  if (T == 0) return OFFQ_OK;
  if (codes == nullptr || scale == nullptr || ((flags & OFFQ_OFFSET) && offset == nullptr))
    return OFFQ_ERR_INVALID_ARG;
  if (!aligned(codes, 16) || !aligned(scale, 4) || (offset != nullptr && !aligned(offset, 4)))
    return OFFQ_ERR_MISALIGNED;
  RotArgs a{};
  a.x = kv;
  a.ld_token = ld_token;
  a.T = T;
  a.H = H;
  a.prep = prepared;
  a.quantize = 1;
  a.offset = (flags & OFFQ_OFFSET) != 0;
  a.codes = codes;
  a.scale = scale;
  a.off = offset;
  a.status = device_status_ptr();
  return launch_rotate_mma<OFFQ_F32, true>(a, static_cast<cudaStream_t>(stream));
}

extern "C" int offq_rotate_heads_reflected(const void* x, int dtype, int64_t T, int32_t H, int32_t head_dim,
                                           int64_t ld_token, const void* prepared, void* out, int out_dtype,
                                           int64_t ld_out, void* stream) {
  const int ob = elem_bytes(out_dtype);
  if (ob == 0 || ld_out < static_cast<int64_t>(H) * head_dim) return OFFQ_ERR_INVALID_ARG;
  int st = check_heads(x, dtype, T, H, head_dim, ld_token, prepared);
  if (st != OFFQ_OK) return st;
  if (dtype != OFFQ_BF16) return OFFQ_ERR_UNSUPPORTED;
  if (T == 0) return OFFQ_OK;
  if (out == nullptr) return OFFQ_ERR_INVALID_ARG;
  if (!aligned(out, 16) || (ld_out * ob) % 16 != 0) return OFFQ_ERR_MISALIGNED;
  RotArgs a{};
  a.x = x;
  a.ld_token = ld_token;
  a.T = T;
  a.H = H;
  a.prep = prepared;
  a.quantize = 0;
  a.out = out;
  a.ld_out = ld_out;
  a.status = device_status_ptr();
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  switch (out_dtype) {
    case OFFQ_F32: return launch_rotate_mma<OFFQ_F32, true>(a, s);
    case OFFQ_BF16: return launch_rotate_mma<OFFQ_BF16, true>(a, s);
    case OFFQ_F16: return launch_rotate_mma<OFFQ_F16, true>(a, s);
    default: return OFFQ_ERR_INVALID_ARG;
  }
}

namespace offq {

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

}  // namespace offq
