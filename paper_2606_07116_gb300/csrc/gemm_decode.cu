// W4A4 GEMM of the OffQ path for few tokens (decode, T <= 64): the same
// product and epilogue as w4a4_gemm_kernel (paper Sec. 1: all matrix
// multiplications in uniform 4-bit execution; Eq. 5: the offsets meet the
// weight block row sums),
//
//   y[t][n] = s_w[n] * ( s_a[t] * (acc'[n][t] - 8 Rt[n]) + sum_b o[t][b] * R[b][n] ),
//   acc'[n][t] = sum_k q_w[n][k] * (q_a[t][k] + 8),   Rt[n] = sum_b R[b][n],
//
// laid out for the regime where the weights dominate the bytes: each weight
// code is read once and used by at most 64 tokens, so the time is the HBM
// stream of the weight codes.
//
// Design:
//  * The MMA's M side is the weights: a CTA owns whole 32-row blocks of the
//    weight codes (block counts differ by at most one between CTAs) over the
//    whole K, so every SM streams an equal share of the weight bytes with no
//    reduction across CTAs; up to 4 blocks (128 rows, one TMEM lane quarter
//    each) make one pass of the accumulator. The N side is the tokens, padded
//    to a multiple of 16 (tcgen05.mma.cta_group::1.kind::f8f6f4, M = 128,
//    N = 16..64, K = 32), both operands in shared memory: with N this small,
//    reading the 4 KB A operand of each instruction dominates the MMA, and the
//    shared-memory path reads it faster than tensor memory.
//  * In the tiled code layout a block's codes are contiguous along K (16-byte
//    chunk c of row r at ((block * K/32 + c) * 32 + r) * 16), so one plain bulk
//    copy (cp.async.bulk) moves 4 k-tiles of a block, 8 KB. The copies land in
//    a ring of packed slots (one slot: 4 k-tiles of the pass's blocks and of
//    the tokens), as many as shared memory holds; the converters release a slot
//    as soon as they have read it.
//  * Converter warps (four per 32-row quarter, taking turns by k-tile) widen
//    the weights (sign-magnitude nibbles -> E4M3) and the activation codes
//    (u = q + 8 -> E4M3 u * 2^-9) into the 128-byte-swizzled K-major operands,
//    through a ring of 4 operand stages that the MMAs release. The products are integers
//    times 2^-18, exact in the fp32 accumulator.
//  * Epilogue warps compute each row's offset correction sum_b o[t][b] R[b][n]
//    while the pass's MMAs run (into tensor memory), then drain the
//    accumulator: lane = weight row n, column = token t, so a warp writes 32
//    consecutive outputs of one token at a time.
// Warps: 0 bulk-copy producer (and TMEM allocation), 1-16 converters, 17 MMA
// issuer, 18-21 epilogue. Every wait is bounded; a wait that runs out aborts
// the CTA, which lets its copies and MMAs in flight finish before it exits and
// records OFFQ_ERR_TIMEOUT in the device status word.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "offq.h"
#include "offq_device.cuh"
#include "offq_host.h"
#include "pair_common.cuh"

namespace {

using namespace offq;

constexpr int kDecMaxT = 64;           // tokens handled (MMA N <= 64)
constexpr int kDecBK = 128;            // codes per k-tile
constexpr int kDecKtBytes = 32 * kDecBK / 2;  // 2 KB: one block's (or 32 tokens') codes of one k-tile
constexpr int kDecSlotKt = 4;          // k-tiles per packed slot (one bulk copy of 8 KB per block)
constexpr int kDecOpStages = 4;        // operand stages (A and B in shared memory)
constexpr int kDecAStage = 128 * kDecBK;  // 16 KB: E4M3 A operand, 128 weight rows x 128 B
constexpr int kDecMaxPk = 16;          // packed slots at most
constexpr int kDecPhases = 4;          // converter warps per TMEM lane quarter
constexpr int kDecConv0 = 1, kDecMma = kDecConv0 + 4 * kDecPhases, kDecEpi0 = kDecMma + 1;
constexpr int kDecThreads = (kDecEpi0 + 4) * 32;
// Tensor memory: accumulator (64 columns), offset correction (64).
constexpr int kDecAcc = 0, kDecCorr = 64, kDecTmemCols = 128;
constexpr int kDecSmemMax = 224 * 1024;  // dynamic shared memory of the kernel (opt-in)
constexpr int kDecNumBars = 2 * kDecMaxPk + 2 * kDecOpStages + 2;

// Shared memory, laid out at launch from the block and token counts:
//   [op stages x A operand (16 KB)] [op stages x B operand (n_mma rows x 128 B, 1024-aligned)]
//   [pk slots x (blocks x 4 k-tiles, token blocks x 4 k-tiles)] [s_a] [barriers] [misc]
struct DecLayout {
  int off_b;     // first B operand stage (after the A stages)
  int b_stage;   // bytes of one B operand stage
  int w_bytes;   // weight part of a packed slot: max blocks per pass x 4 k-tiles x 2 KB
  int pk_slot;   // bytes of one packed slot
  int n_pk;      // packed slots
  int off_pk, off_sa, off_bars, off_misc;
};

struct DecodeParams {
  DecLayout L;
  const uint8_t* a_codes;
  const uint8_t* w_codes;
  const float* a_scale;
  const float* a_offset;   // [T][G] or nullptr
  const float* w_scale;
  const float* rowsum;     // [G][N]
  void* out;
  int64_t ldo;
  int32_t* acc_debug;
  int* status;
  int T, N, K, G;
  int n_mma;               // tokens padded to a multiple of 16
  int nk;                  // k-tiles
  int kchunks;             // K / 32
  int a_blocks;            // 32-token blocks of the activation codes
  int blk_q, blk_r;        // blocks per CTA: blk_q, plus one for the first blk_r CTAs
};

__device__ __forceinline__ void mbar_arrive_n(uint32_t bar, uint32_t n) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(n) : "memory");
}

template <int OUT>
__global__ void __launch_bounds__(kDecThreads, 1) w4a4_decode_kernel(const DecodeParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (base - raw);
  const DecLayout& L = p.L;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int c = blockIdx.x;
  const int nblocks = p.blk_q + (c < p.blk_r ? 1 : 0);               // weight row blocks of this CTA
  const int first = c * p.blk_q + (c < p.blk_r ? c : p.blk_r);       // its first block
  const int passes = (nblocks + 3) / 4;
  const int groups = (p.nk + kDecSlotKt - 1) / kDecSlotKt;           // packed slots per pass
  const int npk = L.n_pk;
  const uint32_t bar0 = base + L.off_bars;
  auto pk_full = [&](int i) { return bar0 + 8u * i; };                               // copies landed
  auto pk_empty = [&](int i) { return bar0 + 8u * (kDecMaxPk + i); };                // converters read the slot
  auto op_full = [&](int s) { return bar0 + 8u * (2 * kDecMaxPk + s); };             // operands converted
  auto op_empty = [&](int s) { return bar0 + 8u * (2 * kDecMaxPk + kDecOpStages + s); };  // MMAs done
  const uint32_t acc_full = bar0 + 8u * (2 * kDecMaxPk + 2 * kDecOpStages);          // a pass's MMAs done
  const uint32_t acc_empty = acc_full + 8u;                                          // its accumulator read
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L.off_misc);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + L.off_misc + 16);

  if (threadIdx.x == 0) {
    for (int i = 0; i < npk; ++i) {
      mbar_init(pk_full(i), 1);
      mbar_init(pk_empty(i), 4 * kDecSlotKt);  // four warps per k-tile of the slot
    }
    for (int s = 0; s < kDecOpStages; ++s) {
      mbar_init(op_full(s), 4);
      mbar_init(op_empty(s), 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 4);
    *abort = 0;
    mbar_fence_init();
  }
  if (warp == 0) {
    tmem_alloc(smem_u32(tmem_slot), kDecTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  griddep_wait();
  griddep_launch_dependents();

  int steps_issued = 0;  // producer: packed slots filled
  int commits = 0;       // MMA issuer: passes committed to acc_full

  if (warp == 0) {
    // ---------------- bulk-copy producer ----------------
    if (lane == 0) {
      int st = 0;
      bool ok = true;
      for (int j = 0; j < passes && ok; ++j) {
        const int nbp = nblocks - 4 * j < 4 ? nblocks - 4 * j : 4;
        const int blk0 = first + 4 * j;
        for (int g = 0; g < groups; ++g, ++st) {
          const int i = st % npk;
          if (!mbar_wait(pk_empty(i), ((st / npk) & 1) ^ 1, abort)) {
            ok = false;
            break;
          }
          const int c0 = 4 * kDecSlotKt * g;  // first chunk of the slot
          const int nch = p.kchunks - c0 < 4 * kDecSlotKt ? p.kchunks - c0 : 4 * kDecSlotKt;
          const uint32_t bytes = static_cast<uint32_t>(nch) * 512u;
          mbar_arrive_expect_tx(pk_full(i), bytes * static_cast<uint32_t>(nbp + p.a_blocks));
          const uint32_t slot = base + L.off_pk + i * L.pk_slot;
          for (int jb = 0; jb < nbp; ++jb)
            bulk_load(slot + jb * kDecSlotKt * kDecKtBytes,
                      p.w_codes + (static_cast<int64_t>(blk0 + jb) * p.kchunks + c0) * 512, bytes, pk_full(i));
          for (int ab = 0; ab < p.a_blocks; ++ab)
            bulk_load(slot + L.w_bytes + ab * kDecSlotKt * kDecKtBytes,
                      p.a_codes + (static_cast<int64_t>(ab) * p.kchunks + c0) * 512, bytes, pk_full(i));
          steps_issued = st + 1;
        }
      }
    }
  } else if (warp < kDecMma) {
    // ---------------- converters ----------------
    const int q = warp & 3;                     // TMEM lane quarter = block within the pass
    const int phase = (warp - kDecConv0) / 4;   // this warp's k-tiles: u == phase mod kDecPhases
    const int t = 32 * q + lane;                // this lane's token row of B
    const bool b_row = t < p.n_mma;
    const int total = passes * p.nk;
    for (int u = phase; u < total; u += kDecPhases) {
      const int j = u / p.nk, kt = u - j * p.nk;
      const int g = kt / kDecSlotKt, i = kt - g * kDecSlotKt;
      const int st = j * groups + g;
      const int slot_i = st % npk;
      const int s = u % kDecOpStages;
      const int nbp = nblocks - 4 * j < 4 ? nblocks - 4 * j : 4;
      if (!__all_sync(0xFFFFFFFFu, mbar_wait(pk_full(slot_i), (st / npk) & 1, abort))) break;
      const uint32_t slot = base + L.off_pk + slot_i * L.pk_slot;
      uint4 wv[4], av[4];
#pragma unroll
      for (int cc = 0; cc < 4; ++cc) {
        const bool chunk_ok = 4 * kt + cc < p.kchunks;
        wv[cc] = q < nbp && chunk_ok ? lds128(slot + (q * kDecSlotKt + i) * kDecKtBytes + cc * 512 + lane * 16)
                                     : make_uint4(0u, 0u, 0u, 0u);
        av[cc] = b_row && chunk_ok
                     ? lds128(slot + L.w_bytes + ((t >> 5) * kDecSlotKt + i) * kDecKtBytes + cc * 512 + (t & 31) * 16)
                     : make_uint4(0u, 0u, 0u, 0u);
      }
      __syncwarp();
      if (lane == 0) {
        // The last k-tile of a short last slot also arrives for the k-tiles it lacks.
        const int in_slot = p.nk - g * kDecSlotKt < kDecSlotKt ? p.nk - g * kDecSlotKt : kDecSlotKt;
        mbar_arrive_n(pk_empty(slot_i), i == in_slot - 1 ? 1 + kDecSlotKt - in_slot : 1);
      }
      if (!__all_sync(0xFFFFFFFFu, mbar_wait(op_empty(s), ((u / kDecOpStages) & 1) ^ 1, abort))) break;
      {
        // A: this weight row's 128 codes -> one 128-byte row of the swizzled operand.
        const int jr = 32 * q + lane;
        const uint32_t dst = base + s * kDecAStage + (jr >> 3) * 1024 + (jr & 7) * 128;
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
          uint32_t a0, a1, a2, a3, b0, b1, b2, b3;
          widen_weight(wv[cc].x, a0, a1);
          widen_weight(wv[cc].y, a2, a3);
          widen_weight(wv[cc].z, b0, b1);
          widen_weight(wv[cc].w, b2, b3);
          sts128(dst + (((2 * cc) ^ (jr & 7)) << 4), a0, a1, a2, a3);
          sts128(dst + (((2 * cc + 1) ^ (jr & 7)) << 4), b0, b1, b2, b3);
        }
      }
      if (b_row) {
        const uint32_t dst = base + L.off_b + s * L.b_stage + (t >> 3) * 1024 + (t & 7) * 128;
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
          uint32_t a0, a1, a2, a3, b0, b1, b2, b3;
          widen_act(av[cc].x, a0, a1);
          widen_act(av[cc].y, a2, a3);
          widen_act(av[cc].z, b0, b1);
          widen_act(av[cc].w, b2, b3);
          sts128(dst + (((2 * cc) ^ (t & 7)) << 4), a0, a1, a2, a3);
          sts128(dst + (((2 * cc + 1) ^ (t & 7)) << 4), b0, b1, b2, b3);
        }
      }
      fence_proxy_async_smem();  // the operand rows, visible to the MMA's reads
      __syncwarp();
      if (lane == 0) mbar_arrive(op_full(s));
    }
  } else if (warp == kDecMma) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t idesc = idesc_e4m3_f32(128, p.n_mma);
      bool ok = true;
      for (int j = 0; j < passes && ok; ++j) {
        ok = mbar_wait(acc_empty, (j & 1) ^ 1, abort);  // the previous pass has been read out
        tc_fence_after();
        for (int kt = 0; kt < p.nk && ok; ++kt) {
          const int u = j * p.nk + kt;
          const int s = u % kDecOpStages;
          if (!mbar_wait(op_full(s), (u / kDecOpStages) & 1, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_addr = base + s * kDecAStage;
          const uint32_t b_addr = base + L.off_b + s * L.b_stage;
#pragma unroll
          for (int kk = 0; kk < kDecBK / 32; ++kk)
            mma_f8f6f4(tmem + kDecAcc, smem_desc_sw128(a_addr + 32 * kk), smem_desc_sw128(b_addr + 32 * kk), idesc,
                       (kt | kk) != 0 ? 1u : 0u);
          mma_commit(op_empty(s));
        }
        mma_commit(acc_full);  // also after an abort: its arrival tells teardown the MMAs are done
        ++commits;
      }
    }
  } else {
    // ---------------- epilogue ----------------
    const int q = warp & 3;
    float* Sa = reinterpret_cast<float*>(smem + L.off_sa);
    const int et = threadIdx.x - kDecEpi0 * 32;
    for (int i = et; i < kDecMaxT; i += 4 * 32) Sa[i] = i < p.T ? __ldg(p.a_scale + i) : 0.f;
    asm volatile("bar.sync 1, 128;" ::: "memory");  // Sa staged by the four epilogue warps
    const uint32_t lane_base = static_cast<uint32_t>(32 * q) << 16;
    for (int j = 0; j < passes; ++j) {
      const int n = (first + 4 * j + q) * 32 + lane;
      const bool row_ok = q < (nblocks - 4 * j < 4 ? nblocks - 4 * j : 4) && n < p.N;
      // Offset correction corr[t] = sum_b o[t][b] R[b][n] while the pass's MMAs run.
      for (int t0 = 0; t0 < p.n_mma; t0 += 16) {
        uint32_t cr[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) cr[i] = 0u;
        if (row_ok && p.a_offset != nullptr) {
          float cv[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) cv[i] = 0.f;
          for (int b = 0; b < p.G; ++b) {
            const float rv = __ldg(p.rowsum + static_cast<int64_t>(b) * p.N + n);
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const int tt = t0 + i;
              const float o = tt < p.T ? __ldg(p.a_offset + static_cast<int64_t>(tt) * p.G + b) : 0.f;
              cv[i] = b == 0 ? o * rv : fmaf(o, rv, cv[i]);
            }
          }
#pragma unroll
          for (int i = 0; i < 16; ++i) cr[i] = __float_as_uint(cv[i]);
        }
        tmem_st_16cols(tmem + lane_base + kDecCorr + t0, cr);
      }
      tmem_st_wait();
      // -8 Rt[n] 2^-18: integers, exact in fp32.
      float rt = 0.f, sw = 0.f;
      if (row_ok) {
        for (int b = 0; b < p.G; ++b) rt += __ldg(p.rowsum + static_cast<int64_t>(b) * p.N + n);
        sw = __ldg(p.w_scale + n);
      }
      const float m8r = rt * -0x1p-15f;
      const bool ok = __all_sync(0xFFFFFFFFu, mbar_wait(acc_full, j & 1, abort)) && !*abort;
      tc_fence_after();
      if (!ok) break;
      for (int t0 = 0; t0 < p.n_mma; t0 += 16) {
        uint32_t acc[16], cr[16];
        tmem_ld_16cols(tmem + lane_base + kDecAcc + t0, acc);
        tmem_ld_16cols(tmem + lane_base + kDecCorr + t0, cr);
        tmem_ld_wait();
        if (!row_ok) continue;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int tt = t0 + i;
          if (tt >= p.T) break;
          const float a = (__uint_as_float(acc[i]) + m8r) * 262144.0f;  // exact: the integer dot product
          const float y = sw * fmaf(Sa[tt], a, __uint_as_float(cr[i]));
          const int64_t off = static_cast<int64_t>(tt) * p.ldo + n;
          if (OUT == OFFQ_F32) {
            static_cast<float*>(p.out)[off] = y;
          } else if (OUT == OFFQ_BF16) {
            static_cast<__nv_bfloat16*>(p.out)[off] = __float2bfloat16_rn(y);
          } else {
            static_cast<__half*>(p.out)[off] = __float2half_rn(y);
          }
          if (p.acc_debug != nullptr)
            p.acc_debug[static_cast<int64_t>(tt) * p.N + n] = __float2int_rn(__uint_as_float(acc[i]) * 262144.0f);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty);
    }
  }

  // ---------------- teardown ----------------
  if (warp == 0 && lane == 0 && *abort) {
    // Copies of slots nobody consumed land before the CTA ends: the last use of
    // each slot (earlier uses of a slot completed before its reuse).
    for (int st = steps_issued > npk ? steps_issued - npk : 0; st < steps_issued; ++st)
      mbar_wait_teardown(pk_full(st % npk), (st / npk) & 1);
  }
  if (warp == kDecMma && lane == 0 && commits > 0)
    mbar_wait_teardown(acc_full, (commits - 1) & 1);  // the MMAs are done before TMEM is released
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kDecTmemCols);
  }
  if (threadIdx.x == 0 && *abort && p.status != nullptr) atomicExch(p.status, kErrTimeout);
}

int decode_num_sms() {
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

// Shared-memory layout for passes of up to `max_blocks` weight blocks and T
// tokens: the operand stages, then as many packed slots as fit.
DecLayout decode_layout(int max_blocks, int T) {
  DecLayout L{};
  const int n_mma = (T + 15) / 16 * 16;
  const int a_blocks = (T + 31) / 32;
  L.b_stage = (n_mma * kDecBK + 1023) / 1024 * 1024;
  L.off_b = kDecOpStages * kDecAStage;
  L.w_bytes = max_blocks * kDecSlotKt * kDecKtBytes;
  L.pk_slot = L.w_bytes + a_blocks * kDecSlotKt * kDecKtBytes;
  const int fixed = L.off_b + kDecOpStages * L.b_stage + kDecMaxT * 4 + kDecNumBars * 8 + 64 + 1024;
  const int n = (kDecSmemMax - fixed) / L.pk_slot;
  L.n_pk = n < kDecMaxPk ? n : kDecMaxPk;
  L.off_pk = L.off_b + kDecOpStages * L.b_stage;
  L.off_sa = L.off_pk + L.n_pk * L.pk_slot;
  L.off_bars = L.off_sa + kDecMaxT * 4;
  L.off_misc = L.off_bars + kDecNumBars * 8;
  return L;
}

template <int OUT>
int launch_decode(const DecodeParams& p, int grid, cudaStream_t s) {
  if (!smem_optin<w4a4_decode_kernel<OUT>>(kDecSmemMax)) return OFFQ_ERR_CUDA;
  const size_t bytes = static_cast<size_t>(p.L.off_misc) + 64 + 1024;
  return launch_pdl(w4a4_decode_kernel<OUT>, dim3(grid), dim3(kDecThreads), bytes, s, p);
}

// ---------------------------------------------------------------------------
// Few-token form (T <= 4): integer dot products on the CUDA cores.
//
// At T <= 4 every weight code meets at most 4 activations, so widening it for
// the tensor cores costs more than the products: the weights stream from HBM
// straight into registers and meet the activations in dp4a (four int8
// products per instruction, exact int32 sums). (Measured on 4096 -> 11008:
// 8.3 us at one token; at eight tokens 14.85 us, level with the tensor-core
// form's 14.9, so the tensor cores take T >= 5: the sign-magnitude unpacking
// and one dp4a per 4 codes and token make the cost grow with T.) A CTA owns one 32-row weight block: lane l of each of
// its 8 warps takes row l, warp w a contiguous eighth of the K chunks, 8
// chunks (128 B of codes per lane) in flight;
// the warps' partial sums meet in shared memory. The activation codes
// (u = q + 8 nibbles) are unpacked once per CTA into shared memory as the byte
// vectors dp4a takes, so the accumulator is acc' = sum (q_a + 8) q_w and the
// epilogue is the decode kernel's, term for term.
// ---------------------------------------------------------------------------
constexpr int kGemvWarps = 8;
constexpr int kGemvBatch = 8;  // chunks of weight codes in flight per lane (128 B)
constexpr int kGemvMaxT = 4;
constexpr int kGemvMaxActBytes = 96 * 1024;  // NT * K bytes of unpacked activations

struct GemvParams {
  const uint8_t* a_codes;
  const uint8_t* w_codes;
  const float* a_scale;
  const float* a_offset;
  const float* w_scale;
  const float* rowsum;   // [G][N]
  void* out;
  int64_t ldo;
  int32_t* acc_debug;
  int T, N, G, kchunks;
};

// Eight interleaved sign-magnitude weight codes (one 32-bit word, channels
// c0..c7) as two vectors of signed bytes: even = (c0, c2, c4, c6),
// odd = (c1, c3, c5, c7). Byte j holds |q(c2j)| in bits 0-2 and its sign in
// bit 7, |q(c2j+1)| in bits 4-6, and in bit 3 the sign of c(2j-1 mod 8), so
// the odd signs sit one byte up (rotate by 8). Negation is (m ^ 0xFF) + 1 per
// byte, with no carry out of a byte since a code of magnitude 0 has sign 0.
__device__ __forceinline__ void weight_bytes(uint32_t w, int& even, int& odd) {
  const uint32_t me = w & 0x07070707u;
  const uint32_t se = (w >> 7) & 0x01010101u;
  even = static_cast<int>((me ^ (se * 0xFFu)) + se);
  const uint32_t mo = (w >> 4) & 0x07070707u;
  const uint32_t so = (__funnelshift_r(w, w, 8) >> 3) & 0x01010101u;
  odd = static_cast<int>((mo ^ (so * 0xFFu)) + so);
}

template <int OUT, int NT>
__global__ void __launch_bounds__(kGemvWarps * 32, 3) w4a4_gemv_kernel(const GemvParams p) {
  extern __shared__ __align__(16) uint8_t smem[];
  // act: [NT][kchunks][8] words (E0 O0 E1 O1 E2 O2 E3 O3 of a 32-code chunk);
  // red: [kGemvWarps][NT][32] partial sums; then the epilogue constants.
  uint32_t* act = reinterpret_cast<uint32_t*>(smem);
  int* red = reinterpret_cast<int*>(smem + static_cast<size_t>(NT) * p.kchunks * 32);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rb = blockIdx.x;  // weight row block
  const int kc = p.kchunks;
  // This warp's K chunks and the first batch of weight loads. They are issued
  // before the wait for the kernel ahead in the stream (programmatic dependent
  // launch), which produces the activations, not the weights: no kernel of this
  // library that writes weight codes releases its dependents early.
  const int per = (kc + kGemvWarps - 1) / kGemvWarps;
  const int c0 = warp * per;
  const int c1 = c0 + per < kc ? c0 + per : kc;
  const uint8_t* wrow = p.w_codes + (static_cast<int64_t>(rb) * kc) * 512 + lane * 16;
  uint4 wv[kGemvBatch];
#pragma unroll
  for (int i = 0; i < kGemvBatch; ++i)
    wv[i] = c0 + i < c1 ? ldg_stream(wrow + static_cast<int64_t>(c0 + i) * 512) : make_uint4(0u, 0u, 0u, 0u);
  // The epilogue's weight-side constants (thread (t, lane) of warps t < NT), also
  // ahead of the wait: s_w[n] and Rt[n] = sum_b R[b][n].
  // They wait in shared memory (ec: [4][NT][32] = s_w, Rt, s_a, corr), not in
  // registers, which the loads in flight need.
  float* ec = reinterpret_cast<float*>(red + kGemvWarps * NT * 32);
  {
    const int et = warp, n = rb * 32 + lane;
    if (et < NT && n < p.N) {
      float rt = 0.f;
      for (int b = 0; b < p.G; ++b) rt += __ldg(p.rowsum + static_cast<int64_t>(b) * p.N + n);
      ec[(0 * NT + et) * 32 + lane] = __ldg(p.w_scale + n);
      ec[(1 * NT + et) * 32 + lane] = rt;
    }
  }
  griddep_wait();
  griddep_launch_dependents();

  // This warp unpacks the activation codes of its own chunks: token t, chunk c ->
  // 8 words of byte vectors (no CTA barrier; the warp reads only what it wrote).
  const int nw = c1 > c0 ? c1 - c0 : 0;
  for (int i = lane; i < NT * nw; i += 32) {
    const int t = i / nw, c = c0 + (i - t * nw);
    uint4 a = make_uint4(0u, 0u, 0u, 0u);
    if (t < p.T) a = __ldg(reinterpret_cast<const uint4*>(p.a_codes + ((t >> 5) * kc + c) * 512 + (t & 31) * 16));
    uint4* dst = reinterpret_cast<uint4*>(act + (static_cast<size_t>(t) * kc + c) * 8);
    dst[0] = make_uint4(a.x & 0x0F0F0F0Fu, (a.x >> 4) & 0x0F0F0F0Fu, a.y & 0x0F0F0F0Fu, (a.y >> 4) & 0x0F0F0F0Fu);
    dst[1] = make_uint4(a.z & 0x0F0F0F0Fu, (a.z >> 4) & 0x0F0F0F0Fu, a.w & 0x0F0F0F0Fu, (a.w >> 4) & 0x0F0F0F0Fu);
  }
  // The activation-side constants of the epilogue: s_a[t] and the offset term
  // corr = sum_b o[t][b] R[b][n] (block 0 multiplied, then FMAs in block order).
  {
    const int et = warp, n = rb * 32 + lane;
    if (et < NT && et < p.T && n < p.N) {
      float corr = 0.f;
      if (p.a_offset != nullptr) {
        for (int b = 0; b < p.G; ++b) {
          const float rv = __ldg(p.rowsum + static_cast<int64_t>(b) * p.N + n);
          const float o = __ldg(p.a_offset + static_cast<int64_t>(et) * p.G + b);
          corr = b == 0 ? o * rv : fmaf(o, rv, corr);
        }
      }
      ec[(2 * NT + et) * 32 + lane] = __ldg(p.a_scale + et);
      ec[(3 * NT + et) * 32 + lane] = corr;
    }
  }
  __syncwarp();

  int acc[NT];
#pragma unroll
  for (int t = 0; t < NT; ++t) acc[t] = 0;
  for (int cb = c0; cb < c1; cb += kGemvBatch) {
#pragma unroll
    for (int i = 0; i < kGemvBatch; ++i) {
      const int c = cb + i;
      if (c >= c1) break;
      const uint4 w = wv[i];
      // The load kGemvBatch chunks ahead takes this register.
      const int cn = c + kGemvBatch;
      wv[i] = cn < c1 ? ldg_stream(wrow + static_cast<int64_t>(cn) * 512) : make_uint4(0u, 0u, 0u, 0u);
      int e0, o0, e1, o1, e2, o2, e3, o3;
      weight_bytes(w.x, e0, o0);
      weight_bytes(w.y, e1, o1);
      weight_bytes(w.z, e2, o2);
      weight_bytes(w.w, e3, o3);
#pragma unroll
      for (int t = 0; t < NT; ++t) {
        const uint4* av = reinterpret_cast<const uint4*>(act + (static_cast<size_t>(t) * kc + c) * 8);
        const uint4 a0 = av[0], a1 = av[1];
        int s = acc[t];
        s = __dp4a(e0, static_cast<int>(a0.x), s);
        s = __dp4a(o0, static_cast<int>(a0.y), s);
        s = __dp4a(e1, static_cast<int>(a0.z), s);
        s = __dp4a(o1, static_cast<int>(a0.w), s);
        s = __dp4a(e2, static_cast<int>(a1.x), s);
        s = __dp4a(o2, static_cast<int>(a1.y), s);
        s = __dp4a(e3, static_cast<int>(a1.z), s);
        s = __dp4a(o3, static_cast<int>(a1.w), s);
        acc[t] = s;
      }
    }
  }
#pragma unroll
  for (int t = 0; t < NT; ++t) red[(warp * NT + t) * 32 + lane] = acc[t];
  __syncthreads();

  // Epilogue: thread (t, lane) for row n = 32 rb + lane, as the decode kernel's:
  // a = acc' - 8 Rt[n] (exact), y = s_w * fma(s_a, a, corr).
  const int et = warp, n = rb * 32 + lane;
  if (et < NT && et < p.T && n < p.N) {
    int accp = 0;
#pragma unroll
    for (int w = 0; w < kGemvWarps; ++w) accp += red[(w * NT + et) * 32 + lane];
    const float rt = ec[(1 * NT + et) * 32 + lane];
    const float a = static_cast<float>(accp - 8 * static_cast<int>(rt));
    const float y = ec[(0 * NT + et) * 32 + lane] * fmaf(ec[(2 * NT + et) * 32 + lane], a, ec[(3 * NT + et) * 32 + lane]);
    const int64_t off = static_cast<int64_t>(et) * p.ldo + n;
    if (OUT == OFFQ_F32) {
      static_cast<float*>(p.out)[off] = y;
    } else if (OUT == OFFQ_BF16) {
      static_cast<__nv_bfloat16*>(p.out)[off] = __float2bfloat16_rn(y);
    } else {
      static_cast<__half*>(p.out)[off] = __float2half_rn(y);
    }
    if (p.acc_debug != nullptr) p.acc_debug[static_cast<int64_t>(et) * p.N + n] = accp;
  }
}

template <int OUT, int NT>
int launch_gemv(const GemvParams& p, int blocks, cudaStream_t s) {
  const size_t bytes =
      static_cast<size_t>(NT) * p.kchunks * 32 + static_cast<size_t>(kGemvWarps + 4) * NT * 32 * 4;
  if (bytes > 48 * 1024 &&
      !smem_optin<w4a4_gemv_kernel<OUT, NT>>(kGemvMaxActBytes + (kGemvWarps + 4) * kGemvMaxT * 32 * 4))
    return OFFQ_ERR_CUDA;
  return launch_pdl(w4a4_gemv_kernel<OUT, NT>, dim3(blocks), dim3(kGemvWarps * 32), bytes, s, p);
}

template <int OUT>
int dispatch_gemv(const GemvParams& p, int nt, int blocks, cudaStream_t s) {
  switch (nt) {
    case 1: return launch_gemv<OUT, 1>(p, blocks, s);
    case 2: return launch_gemv<OUT, 2>(p, blocks, s);
    default: return launch_gemv<OUT, 4>(p, blocks, s);
  }
}

}  // namespace

namespace offq {

int decode_max_tokens() { return kDecMaxT; }

// The decode form of offq_w4a4_linear (arguments checked by the caller; T in 1..64).
int w4a4_linear_decode(const uint8_t* a_codes, const float* a_scale, const float* a_offset, int64_t T, int64_t N,
                       int64_t K, int32_t g, const uint8_t* w_codes, const float* w_scale, const float* w_offsum,
                       void* out, int out_dtype, int64_t ldo, int32_t* acc_debug, cudaStream_t stream) {
  const int nt = T <= 1 ? 1 : (T <= 2 ? 2 : 4);
  if (T <= kGemvMaxT && static_cast<int64_t>(nt) * K <= kGemvMaxActBytes) {
    GemvParams q{};
    q.a_codes = a_codes;
    q.w_codes = w_codes;
    q.a_scale = a_scale;
    q.a_offset = a_offset;
    q.w_scale = w_scale;
    q.rowsum = w_offsum;
    q.out = out;
    q.ldo = ldo;
    q.acc_debug = acc_debug;
    q.T = static_cast<int>(T);
    q.N = static_cast<int>(N);
    q.G = static_cast<int>(K / g);
    q.kchunks = static_cast<int>(K / 32);
    const int64_t blocks = (N + 31) / 32;
    if (blocks > 0x7FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
    switch (out_dtype) {
      case OFFQ_F32: return dispatch_gemv<OFFQ_F32>(q, nt, static_cast<int>(blocks), stream);
      case OFFQ_BF16: return dispatch_gemv<OFFQ_BF16>(q, nt, static_cast<int>(blocks), stream);
      case OFFQ_F16: return dispatch_gemv<OFFQ_F16>(q, nt, static_cast<int>(blocks), stream);
      default: return OFFQ_ERR_INVALID_ARG;
    }
  }
  const int sms = decode_num_sms();
  if (sms < 1) return OFFQ_ERR_CUDA;
  const int64_t nblk = (N + 31) / 32;
  const int64_t grid = nblk < sms ? nblk : sms;
  DecodeParams p{};
  p.a_codes = a_codes;
  p.w_codes = w_codes;
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
  p.n_mma = static_cast<int>((T + 15) / 16 * 16);
  p.nk = static_cast<int>((K + kDecBK - 1) / kDecBK);
  p.kchunks = static_cast<int>(K / 32);
  p.a_blocks = static_cast<int>((T + 31) / 32);
  p.blk_q = static_cast<int>(nblk / grid);
  p.blk_r = static_cast<int>(nblk % grid);
  const int max_blocks = p.blk_q + (p.blk_r > 0 ? 1 : 0);
  p.L = decode_layout(max_blocks < 4 ? max_blocks : 4, p.T);
  if (p.L.n_pk < 2) return OFFQ_ERR_UNSUPPORTED;
  const int gr = static_cast<int>(grid);
  switch (out_dtype) {
    case OFFQ_F32: return launch_decode<OFFQ_F32>(p, gr, stream);
    case OFFQ_BF16: return launch_decode<OFFQ_BF16>(p, gr, stream);
    case OFFQ_F16: return launch_decode<OFFQ_F16>(p, gr, stream);
    default: return OFFQ_ERR_INVALID_ARG;
  }
}

}  // namespace offq
