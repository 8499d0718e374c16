// The g = 1024 rotating activation quantizer (offq_quantize_act, bf16 rows of
// one head) with a 128-point factor of the transform on the tensor cores.
//
// Per row and block of 1024 channels (paper Sec. 3.2, Eq. 4-5; Sec. 3 Eq. 1):
// R = x H_1024 / 32 - o with o = x[0] / 32, s = max|R| / 7 over the row,
// q = rne(R / s), stored as q + 8. As in the register kernels, sqrt(1024) R is
// formed unnormalised (the first Hadamard row is all ones, so removing x[0]
// from the transform's input removes the offset) and 1/32 goes only into the
// stored scale and offset.
//
// The Sylvester matrix factors over channel bits, H_1024 = H_2 (x) H_4 (x) H_128
// for channel c = 512 h + 128 c + a (h: half block, c: 128-channel chunk of
// the half, a: channel in the chunk):
//  * bits a (H_128) on the tensor cores: tcgen05.mma kind::f16, A = the bf16
//    rows, B = H_128 (entries +-1, exact in bf16), so every product is exact
//    and the accumulator holds the fp32 sum of 128 of them. The A tile has
//    128 rows, (h, token, block) for 64 (token, block) pairs: row
//    64 h + t G + j holds channels 512 h .. 512 h + 511 of block j of the
//    tile's token t, loaded by TMA from a 4-D view [T][G][2][512] of the
//    activations (128-byte swizzle, 64-channel slabs). Per chunk c, MMAs of
//    N = 128 write columns 128 c .. 128 c + 127 of TMEM lane (h, t, j): the
//    tile fills all 512 columns.
//  * bits c (H_4) in registers: a thread owns one TMEM lane and, per pass,
//    16 output channels n of the 4 chunks (4 loads of 16 columns), and runs
//    2 butterfly stages on fp32x2 pairs.
//  * bit h (H_2) between the two lanes of a (token, block): threads h = 0 and
//    1 (warps w and w ^ 2, same lane) swap half their values through shared
//    memory; each forms both outputs of 2 chunks and writes them back to its
//    TMEM columns. The larger magnitude of each output pair is fl(|u| + |t|)
//    of its inputs, which gives the row's absmax.
// The absmax goes through shared memory (a per-warp maximum per row, then a
// 64-bit atomic max keyed by the tile), and a second sweep reads 32 output
// channels per TMEM load, rounds them (magic-number rounding) and writes one
// 16-byte chunk of codes. Each 32-column slot is handed to the next tile's
// MMAs as soon as it has been read.
//
// Roles (320 threads, one CTA per SM, persistent over tiles):
//   warp 8    TMA producer: per tile, 8 slabs of both halves; slab s of the
//             next tile is loaded as soon as the MMAs have read slab s;
//   warp 9    allocates TMEM (512 columns) and issues the MMAs;
//   warps 0-7 the register work, two warps per TMEM lane quarter (warps w and
//             w + 4): warp w takes output channels n in 64 (w / 4) ..
//             64 (w / 4) + 63 of every chunk in the first sweep and column
//             slots 8 (w / 4) .. 8 (w / 4) + 7 in the second.
// Every wait is bounded; a wait that runs out marks the CTA aborted, the
// copies and MMAs in flight are waited for (bounded) and TMEM is released.
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <climits>
#include <cstring>

#include "offq.h"
#include "offq_device.cuh"
#include "offq_host.h"

namespace {

using namespace offq;

constexpr int kSlabs = 8;                            // 64-channel slabs of a half block
constexpr int kHalfRows = 64;                        // (token, block) rows per half
constexpr int kSlabBytes = 2 * kHalfRows * 128;      // both halves of one slab
constexpr int kABytes = kSlabs * kSlabBytes;         // 128 KB
constexpr int kBSlab = 128 * 128;                    // H_128, channels 64 k .. 64 k + 63 of its 128 rows
constexpr int kBBytes = 2 * kBSlab;
constexpr int kRegWarps = 8;                         // two per TMEM lane quarter
constexpr int kXWarpBytes = 8 * 32 * 16;             // a warp's exchange area: 8 entries x 32 lanes x 16 B
constexpr int kXBufBytes = kRegWarps * kXWarpBytes;
constexpr int kXBytes = 2 * kXBufBytes;              // two buffers, alternating passes
constexpr int kCtrlOff = kABytes + kBBytes + kXBytes;
constexpr int kBars = 2 * kSlabs + 16 + 2;           // full[8], empty[8], tfull, tempty[16], done
constexpr int kKeysOff = kCtrlOff + 8 * kBars;
constexpr int kSmem = kKeysOff + kHalfRows * 8 + 16 + 1024;
constexpr int kProducerWarp = kRegWarps, kMmaWarp = kRegWarps + 1;
constexpr int kThreads = 32 * (kRegWarps + 2);
static_assert(kSmem <= 232448, "one CTA per SM");
// kind::f16: D f32 (bits 4-5 = 1), A and B bf16 (7-9, 10-12 = 1), both
// K-major, N = 128 (N >> 3 at bit 17), M = 128 (M >> 4 at bit 24).
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((128u >> 3) << 17) | ((128u >> 4) << 24);

// Named barriers: 0 is __syncthreads; 1-4 the four warp pairs (w, w ^ 2) of
// the register warps; 5 all register warps; 6 their per-tile vote.
constexpr int kBarAll = 5;
constexpr int kBarVote = 6;

struct Args {
  const __nv_bfloat16* x;
  int64_t ld_t;
  int64_t rows;
  int64_t tiles;
  int K, G, P;          // P tokens of G blocks per tile
  int offs;             // subtract the offset (OFFQ_OFFSET)
  uint8_t* codes;
  float* scale;
  float* offset;
  float inv_sqrt_g;
  float scale_mul;
  int* status;
  long long wait_cycles;
};

__device__ __forceinline__ void bar_sync(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Barrier `id` over `count` threads; true if `pred` held for any of them.
__device__ __forceinline__ bool bar_any(int id, int count, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n"
      ".reg .pred p, q;\n"
      "setp.ne.b32 p, %1, 0;\n"
      "bar.red.or.pred q, %2, %3, p;\n"
      "selp.u32 %0, 1, 0, q;\n"
      "}\n"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(pred)), "r"(id), "r"(count)
      : "memory");
  return r != 0;
}

// Columns col0 + 128 c + (0..15) of the thread's TMEM lane into
// r[16 c .. 16 c + 15], c = 0..3, with the wait in the same statement (no
// register is read before its data has arrived).
__device__ __forceinline__ void tmem_ld_chunks(uint32_t col0, uint32_t (&r)[64]) {
  asm volatile(
      "{\n"
      ".reg .b32 ta;\n"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%64];\n"
      "add.u32 ta, %64, 128;\n"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [ta];\n"
      "add.u32 ta, %64, 256;\n"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47}, [ta];\n"
      "add.u32 ta, %64, 384;\n"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [ta];\n"
      "tcgen05.wait::ld.sync.aligned;\n"
      "}\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
        "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
        "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
        "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
        "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
      : "r"(col0)
      : "memory");
}

// tmem_ld_chunks with the warp pair's barrier between the loads and their
// wait: the barrier's wait overlaps the loads' latency.
__device__ __forceinline__ void tmem_ld_chunks_pair_sync(uint32_t col0, int pair_bar, uint32_t (&r)[64]) {
  asm volatile(
      "{\n"
      ".reg .b32 ta;\n"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%64];\n"
      "add.u32 ta, %64, 128;\n"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [ta];\n"
      "add.u32 ta, %64, 256;\n"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47}, [ta];\n"
      "add.u32 ta, %64, 384;\n"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [ta];\n"
      "bar.sync %65, 64;\n"
      "tcgen05.wait::ld.sync.aligned;\n"
      "}\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
        "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
        "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
        "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
        "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
      : "r"(col0), "r"(pair_bar)
      : "memory");
}

// Columns col0 .. col0 + 31 and col1 .. col1 + 31 of the thread's TMEM lane,
// waited in the same statement.
__device__ __forceinline__ void tmem_ld_2x32_waited(uint32_t col0, uint32_t col1, uint32_t (&r)[64]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%64];\n"
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,"
      "%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%65];\n"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
        "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
        "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
        "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
        "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
      : "r"(col0), "r"(col1)
      : "memory");
}

// Sixteen consecutive columns of the thread's TMEM lane from eight fp32 pairs.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint64_t (&v)[8]) {
  asm volatile(
      "{\n"
      ".reg .b32 a<16>;\n"
      "mov.b64 {a0, a1}, %1;\n"
      "mov.b64 {a2, a3}, %2;\n"
      "mov.b64 {a4, a5}, %3;\n"
      "mov.b64 {a6, a7}, %4;\n"
      "mov.b64 {a8, a9}, %5;\n"
      "mov.b64 {a10, a11}, %6;\n"
      "mov.b64 {a12, a13}, %7;\n"
      "mov.b64 {a14, a15}, %8;\n"
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {a0, a1, a2, a3, a4, a5, a6, a7, a8, a9, a10, a11, a12, a13, "
      "a14, a15};\n"
      "}\n" ::"r"(taddr),
      "l"(v[0]), "l"(v[1]), "l"(v[2]), "l"(v[3]), "l"(v[4]), "l"(v[5]), "l"(v[6]), "l"(v[7])
      : "memory");
}

__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ void sts_pair(uint32_t addr, uint64_t a, uint64_t b) {
  asm volatile("st.shared.v2.b64 [%0], {%1, %2};" ::"r"(addr), "l"(a), "l"(b) : "memory");
}

__device__ __forceinline__ void lds_pair(uint32_t addr, uint64_t& a, uint64_t& b) {
  asm volatile("ld.shared.v2.b64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "r"(addr) : "memory");
}

__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

__device__ __forceinline__ uint64_t sub2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}

__device__ __forceinline__ float max3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// Running absmax of a thread's outputs, two independent chains. The outputs
// come in pairs fl(u + t), fl(u - t) (the H_2 stage); rounding is symmetric
// and monotone, so the larger magnitude of the two is exactly fl(|u| + |t|).
struct AbsMax {
  float m0 = 0.f, m1 = 0.f;
  __device__ __forceinline__ void add_a(uint64_t u, uint64_t t) {
    float a, b, c, d;
    unpack2(u, a, b);
    unpack2(t, c, d);
    m0 = max3(m0, fabsf(a) + fabsf(c), fabsf(b) + fabsf(d));
  }
  __device__ __forceinline__ void add_b(uint64_t u, uint64_t t) {
    float a, b, c, d;
    unpack2(u, a, b);
    unpack2(t, c, d);
    m1 = max3(m1, fabsf(a) + fabsf(c), fabsf(b) + fabsf(d));
  }
  __device__ __forceinline__ float value() const { return fmaxf(m0, m1); }
};

// fl(x * inv + 1.5 * 2^23 + 8) has rne(x * inv) + 8 in its low mantissa bits
// for |x * inv| <= 7 (the ulp there is 1); bits 4-21 of those words are zero.
constexpr float kMagic8 = 12582920.0f;

// The 32-bit word of 8 codes (channel 2k in the low nibble of byte k) from
// eight such words.
__device__ __forceinline__ uint32_t pack8(const uint32_t* u) {
  const uint32_t b0 = (u[1] << 4) + u[0], b1 = (u[3] << 4) + u[2], b2 = (u[5] << 4) + u[4], b3 = (u[7] << 4) + u[6];
  return __byte_perm(__byte_perm(b0, b1, 0x0040), __byte_perm(b2, b3, 0x0040), 0x5410);
}

// The first sweep of a thread of half H, in 4 passes of 16 output channels n
// of the 4 chunks (columns col + 16 i + 128 c of its TMEM lane, pass i): per
// pass the H_4 stages over the chunks, the H_2 stage with the partner thread
// (through xw / xr, two buffers alternating), and the results back in place:
// the thread keeps output chunks 2 H and 2 H + 1; output bit h = e of chunk
// c' lands in chunk position c' for e = 0 and c' ^ 2 for e = 1. The next
// pass's TMEM loads are issued before the pair barrier.
template <int H>
__device__ __forceinline__ void first_sweep(uint32_t col, uint32_t xw, uint32_t xr, int pair_bar, uint64_t x0x0,
                                            AbsMax& am) {
  uint32_t r[64];
  tmem_ld_chunks(col, r);
#pragma unroll 1
  for (int i = 0; i < 4; ++i) {
    const uint32_t buf = (i & 1) * kXBufBytes;
    uint64_t p[4][8];
#pragma unroll
    for (int c = 0; c < 4; ++c)
#pragma unroll
      for (int k = 0; k < 8; ++k) p[c][k] = pack2(__uint_as_float(r[16 * c + 2 * k]), __uint_as_float(r[16 * c + 2 * k + 1]));
    if (H == 0) {
      // Chunk 0 of the first half holds the block's leading channel: every
      // output of its H_128 includes x[0] once. Removing it is removing the
      // offset (x0x0 is zero without OFFQ_OFFSET).
#pragma unroll
      for (int k = 0; k < 8; ++k) p[0][k] = sub2(p[0][k], x0x0);
    }
#pragma unroll
    for (int d = 1; d < 4; d <<= 1) {
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        if ((c & d) == 0) {
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint64_t u = p[c][k], v = p[c + d][k];
            p[c][k] = add2(u, v);
            p[c + d][k] = sub2(u, v);
          }
        }
      }
    }
    // Send chunks 2 (1 - H), 2 (1 - H) + 1: entry k of the buffer is chunk
    // 2 (1 - H) + (k >> 2), pairs 2 (k & 3), 2 (k & 3) + 1.
#pragma unroll
    for (int k = 0; k < 8; ++k)
      sts_pair(xw + buf + k * 512, p[2 * (1 - H) + (k >> 2)][2 * (k & 3)], p[2 * (1 - H) + (k >> 2)][2 * (k & 3) + 1]);
    if (i < 3) {
      tmem_ld_chunks_pair_sync(col + 16 * (i + 1), pair_bar, r);
    } else {
      bar_sync(pair_bar, 64);
    }
    uint64_t sum[2][8], dif[2][8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      uint64_t t0, t1;
      lds_pair(xr + buf + k * 512, t0, t1);
      const int c = 2 * H + (k >> 2), j = 2 * (k & 3);
      const uint64_t u0 = p[c][j], u1 = p[c][j + 1];
      // Output bit 0 is (half 0) + (half 1), bit 1 is (half 0) - (half 1).
      sum[k >> 2][j] = add2(u0, t0);
      sum[k >> 2][j + 1] = add2(u1, t1);
      dif[k >> 2][j] = H == 0 ? sub2(u0, t0) : sub2(t0, u0);
      dif[k >> 2][j + 1] = H == 0 ? sub2(u1, t1) : sub2(t1, u1);
      am.add_a(u0, t0);
      am.add_b(u1, t1);
    }
    const uint32_t cc = col + 16 * i;
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
      tmem_st16(cc + 128 * (2 * H + kk), sum[kk]);
      tmem_st16(cc + 128 * (2 * (1 - H) + kk), dif[kk]);
    }
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    quantize_rows_mma_kernel(const __grid_constant__ CUtensorMap xmap, const Args a) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (base - raw);
  const uint32_t a_s = base, b_s = base + kABytes, x_s = b_s + kBBytes;
  const uint32_t full0 = base + kCtrlOff, empty0 = full0 + 8 * kSlabs;
  // tempty[q]: column slot q (32 columns) has been read by the second sweep.
  const uint32_t tfull = empty0 + 8 * kSlabs, tempty0 = tfull + 8, done = tempty0 + 8 * 16;
  unsigned long long* keys = reinterpret_cast<unsigned long long*>(smem + kKeysOff);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kKeysOff + kHalfRows * 8);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + kKeysOff + kHalfRows * 8 + 4);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  if (tid == 0) {
#pragma unroll
    for (int s = 0; s < kSlabs; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(tfull, 1);
#pragma unroll
    for (int q = 0; q < 16; ++q) mbar_init(tempty0 + 8 * q, 4);
    mbar_init(done, 1);
    *abort = 0;
    mbar_fence_init();
  }
  if (tid < kHalfRows) keys[tid] = 0ull;
  if (tid < 256) {
    // B = H_128 (B[n][k] = (-1)^popcount(n & k)), K-major in two slabs of 64
    // channels: row n of slab bs is 128 bytes, 16-byte chunk c (channels
    // 64 bs + 8 c .. + 7) at chunk c ^ (n & 7).
    const int n = tid >> 1, bs = tid & 1;
#pragma unroll 1
    for (int pc = 0; pc < 8; ++pc) {
      const int c = pc ^ (n & 7);
      uint32_t w[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int k = 64 * bs + 8 * c + 2 * i;
        const uint32_t lo = (__popc(n & k) & 1) ? 0xBF80u : 0x3F80u;
        const uint32_t hi = (__popc(n & (k + 1)) & 1) ? 0xBF80u : 0x3F80u;
        w[i] = lo | (hi << 16);
      }
      asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(b_s + bs * kBSlab + n * 128 + pc * 16),
                   "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3])
                   : "memory");
    }
    fence_proxy_async_smem();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(smem_u32(tmem_slot), 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  griddep_wait();
  griddep_launch_dependents();

  const int G = a.G, P = a.P, rows_t = G * P;
  const int n_local = static_cast<int>((a.tiles - blockIdx.x + gridDim.x - 1) / gridDim.x);  // >= 1

  if (warp == kProducerWarp) {
    if (lane == 0) {
      tma_prefetch_desc(&xmap);
      const uint32_t bytes = 2u * rows_t * 128u;
      int n = 0, s_stop = kSlabs;
      for (; n < n_local; ++n) {
        const int t0 = static_cast<int>((blockIdx.x + static_cast<int64_t>(n) * gridDim.x) * P);
        for (int s = 0; s < kSlabs; ++s) {
          if (n > 0 && !mbar_wait(empty0 + 8 * s, (n - 1) & 1, abort)) {
            s_stop = s;
            break;
          }
          const uint32_t dst = a_s + s * kSlabBytes;
          mbar_arrive_expect_tx(full0 + 8 * s, bytes);
          tma_load_4d(dst, &xmap, full0 + 8 * s, 64 * s, 0, 0, t0);
          tma_load_4d(dst + kSlabBytes / 2, &xmap, full0 + 8 * s, 64 * s, 1, 0, t0);
        }
        if (s_stop < kSlabs) break;
      }
      if (*abort) {
        // Slab s took n + (s < s_stop) loads (n_local each without a stop):
        // wait (bounded) for the last of them before shared memory is released.
        for (int s = 0; s < kSlabs; ++s) {
          const int cnt = n < n_local ? n + (s < s_stop ? 1 : 0) : n_local;
          if (cnt > 0) mbar_wait_teardown(full0 + 8 * s, (cnt - 1) & 1);
        }
      }
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    if (lane == 0) {
      bool issued = false;
      for (int n = 0; n < n_local; ++n) {
        bool ok = true;
        for (int c = 0; c < 4; ++c) {
          // Chunk c (slabs 2 c, 2 c + 1) writes column slots 4 c .. 4 c + 3: each
          // must have been read by the previous tile's second sweep.
          ok = mbar_wait(full0 + 16 * c, n & 1, abort) && mbar_wait(full0 + 16 * c + 8, n & 1, abort);
          for (int q = 4 * c; ok && n > 0 && q < 4 * c + 4; ++q) ok = mbar_wait(tempty0 + 8 * q, (n - 1) & 1, abort);
          if (!ok) break;
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < 8; ++kk)
            mma_bf16(tmem + 128 * c, smem_desc_sw128(a_s + (2 * c + (kk >> 2)) * kSlabBytes + 32 * (kk & 3)),
                     smem_desc_sw128(b_s + (kk >> 2) * kBSlab + 32 * (kk & 3)), kIdesc, kk);
          issued = true;
          mma_commit(empty0 + 16 * c);  // slabs 2 c and 2 c + 1 may take the next tile
          mma_commit(empty0 + 16 * c + 8);
        }
        if (!ok) break;
        mma_commit(tfull);
      }
      if (*abort && issued) {
        // MMAs complete in issue order: one more commit tracks them all.
        mma_commit(done);
        mbar_wait_teardown(done, 0);
      }
    }
    __syncwarp();
  } else {
    const int wg = warp >> 2, sp = warp & 3, h = sp >> 1;
    const int mp = 32 * (sp & 1) + lane;  // (token, block) row of the half
    const int t = mp / G, j = mp - t * G;
    const bool lane_ok = mp < rows_t;
    const uint32_t tl = tmem + (static_cast<uint32_t>(32 * sp) << 16);
    const int pair_bar = 1 + 2 * wg + (sp & 1);
    const uint32_t xw = x_s + warp * kXWarpBytes + lane * 16, xr = x_s + (warp ^ 2) * kXWarpBytes + lane * 16;
    const int t_lo = (32 * (sp & 1)) / G, t_hi = min(P - 1, (32 * (sp & 1) + 31) / G);
    const int cpr = a.K / 32;
    for (int n = 0; n < n_local; ++n) {
      const int64_t row = (blockIdx.x + static_cast<int64_t>(n) * gridDim.x) * P + t;
      const bool ok = lane_ok && row < a.rows;
      float x0 = 0.f;
      if (a.offs && h == 0 && ok)
        x0 = __uint_as_float(static_cast<uint32_t>(__ldg(reinterpret_cast<const unsigned short*>(
                                                   a.x + row * a.ld_t + 1024 * j)))
                             << 16);
      const bool waited = mbar_wait_for(tfull, n & 1, abort, a.wait_cycles);
      if (bar_any(kBarVote, 32 * kRegWarps, !waited)) break;
      tc_fence_after();
      const uint64_t x0x0 = pack2(x0, x0);
      AbsMax am;
      const uint32_t col = tl + 64 * wg;  // output channels n = 64 wg .. 64 wg + 63 of each chunk
      if (h == 0) {
        first_sweep<0>(col, xw, xr, pair_bar, x0x0, am);
      } else {
        first_sweep<1>(col, xw, xr, pair_bar, x0x0, am);
      }
      const float m = am.value();
      tmem_st_wait();
      // Row absmax: per row of this warp a warp maximum (non-negative floats
      // order as their bits), then a 64-bit atomic max keyed by the tile
      // (n + 1 in the high word), so older tiles' entries never win.
      for (int tt = t_lo; tt <= t_hi; ++tt) {
        const uint32_t wm = __reduce_max_sync(0xFFFFFFFFu, (ok && t == tt) ? __float_as_uint(m) : 0u);
        if (lane == 0) atomicMax(&keys[tt], (static_cast<unsigned long long>(n + 1) << 32) | wm);
      }
      tc_fence_before();
      bar_sync(kBarAll, 32 * kRegWarps);
      tc_fence_after();
      const unsigned long long key = keys[t];
      const float amax = (key >> 32) == static_cast<unsigned long long>(n + 1) ? __uint_as_float(static_cast<uint32_t>(key)) : 0.f;
      const float inv = amax > 0.f ? __fdiv_rn(7.0f, amax) : 0.f;
      const uint64_t inv2 = pack2(inv, inv), mag2 = pack2(kMagic8, kMagic8);
      // Second sweep: slot q = 8 wg + k holds output channels 32 b' .. 32 b' + 31
      // of group b' = 8 h + k, half e = wg ^ h of the block.
      const int kt0 = 32 * j + 16 * (wg ^ h) + 8 * h;
      uint8_t* dst0 = a.codes + ((row >> 5) * cpr + kt0) * 512 + (row & 31) * 16;  // the 32-row tiled layout
#pragma unroll 1
      for (int k = 0; k < 8; k += 2) {
        uint32_t v[64];
        const uint32_t q = 8 * wg + k;
        tmem_ld_2x32_waited(tl + 32 * q, tl + 32 * (q + 1), v);
        // Slots q and q + 1 are read in this lane quarter: the next tile's MMAs
        // may overwrite them once the four quarters have.
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(tempty0 + 8 * q);
          mbar_arrive(tempty0 + 8 * (q + 1));
        }
#pragma unroll
        for (int hk = 0; hk < 2; ++hk) {
          uint32_t u[32];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            float f0, f1;
            unpack2(fma2v(pack2(__uint_as_float(v[32 * hk + 2 * i]), __uint_as_float(v[32 * hk + 2 * i + 1])), inv2,
                          mag2),
                    f0, f1);
            u[2 * i] = __float_as_uint(f0);
            u[2 * i + 1] = __float_as_uint(f1);
          }
          if (ok)
            *reinterpret_cast<uint4*>(dst0 + (k + hk) * 512) =
                make_uint4(pack8(u), pack8(u + 8), pack8(u + 16), pack8(u + 24));
        }
      }
      if (wg == 0 && h == 0 && ok) {
        if (a.offset != nullptr) a.offset[row * G + j] = x0 * a.inv_sqrt_g;
        if (j == 0) a.scale[row] = amax * a.scale_mul;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
  if (tid == 0 && *abort && a.status != nullptr) atomicExch(a.status, kErrTimeout);
}

int mma_num_sms() {
  static int sms[kMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 0;
  if (sms[dev] == 0) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    sms[dev] = v;
  }
  return sms[dev];
}

}  // namespace

namespace offq {

int quantize_rows_mma(const MmaQuantRows& p, cudaStream_t stream) {
  constexpr int kNotSuitable = 1;
  if (p.K % 1024 != 0 || p.K < 1024 || p.K / 1024 > kHalfRows) return kNotSuitable;
  if (!p.tiled || !aligned(p.x, 16) || p.ld_t % 8 != 0 || p.ld_t < p.K) return kNotSuitable;
  const int G = p.K / 1024, P = kHalfRows / G;
  const int sms = mma_num_sms();
  if (sms < 1) return OFFQ_ERR_CUDA;
  const int64_t tiles = (p.rows + P - 1) / P;
  // Fewer tiles than SMs leave SMs idle: the warp-per-block kernel serves those.
  if (tiles < sms || p.rows > INT_MAX - kHalfRows) return kNotSuitable;
  const auto enc = tensor_map_encoder();
  if (enc == nullptr) return OFFQ_ERR_CUDA;
  // [T][G][2][512] bf16: channel within the half, half, block, token.
  CUtensorMap map;
  const cuuint64_t dims[4] = {512, 2, static_cast<cuuint64_t>(G), static_cast<cuuint64_t>(p.rows)};
  const cuuint64_t strides[3] = {1024, 2048, static_cast<cuuint64_t>(p.ld_t) * 2};
  const cuuint32_t box[4] = {64, 1, static_cast<cuuint32_t>(G), static_cast<cuuint32_t>(P)};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  if (enc(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(p.x), dims, strides, box, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return OFFQ_ERR_CUDA;
  if (!smem_optin<quantize_rows_mma_kernel>(kSmem)) return OFFQ_ERR_CUDA;
  Args a{};
  a.x = static_cast<const __nv_bfloat16*>(p.x);
  a.ld_t = p.ld_t;
  a.rows = p.rows;
  a.tiles = tiles;
  a.K = p.K;
  a.G = G;
  a.P = P;
  a.offs = (p.flags & OFFQ_OFFSET) != 0;
  a.codes = p.codes;
  a.scale = p.scale;
  a.offset = p.offset;
  a.inv_sqrt_g = p.inv_sqrt_g;
  a.scale_mul = p.scale_mul;
  a.status = p.status;
  a.wait_cycles = p.wait_cycles;
  const int64_t grid = tiles < sms ? tiles : sms;
  return launch_pdl(quantize_rows_mma_kernel, dim3(static_cast<unsigned>(grid)), dim3(kThreads), kSmem, stream, map, a);
}

}  // namespace offq
