// W4A4 GEMM of the OffQ path (offq_w4a4_linear) on the 5th-generation tensor
// cores of sm_103a, with the dequant + offset epilogue fused.
//
//   y[t][n] = s_w[n] * ( s_a[t] * (acc'[t][n] - 8 Rt[n]) + sum_b o[t][b] * R[b][n] )
//   acc'[t][n] = sum_k (q_a[t][k] + 8) * q_w[n][k],   Rt[n] = sum_b R[b][n]
//
// acc' is what the tensor cores accumulate: activation codes are stored as
// u = q + 8 (1..15) and weight codes as sign-magnitude q (-7..7). Both widen to
// E4M3 bytes whose values are exact integers times 2^-9: bytes 0x00..0x0F are
// the values 0..15 * 2^-9 (subnormals and the first binade share one step), and
// the sign bit negates. Every product and partial sum is then an integer times
// 2^-18 below 2^24 * 2^-18 for K <= 65536, exact in the fp32 accumulator. The
// "+8" is removed in the epilogue, still exactly: acc' - 8 Rt[n] is the integer
// dot product times 2^-18, with the weight row sum Rt = sum_k q_w[n][k] (the
// block row sums R added up). Only then is it scaled, so an output near zero
// is not the small difference of two large rounded terms.
//
// Design. Widening 4-bit codes to fp8 operands costs shared-memory bandwidth,
// which the tensor core's operand reads share. So:
//  * two SMs form a pair (cluster of 2, tcgen05 cta_group::2) computing a
//    256 x 256 tile; each SM holds 128 rows of A and half (128 rows) of B, and
//    the pair's MMA reads each half of B once for both SMs;
//  * A never touches shared memory: converter warps load its packed codes with
//    coalesced 16-byte loads, widen them in registers and write the E4M3
//    operand straight into tensor memory (tcgen05.st), where the MMA reads it;
//  * B is loaded the same way, widened, and stored once into the 128-byte-
//    swizzled K-major shared-memory layout the MMA reads;
//  * both code matrices use a 32-row tiled layout, so each 16-byte load of a
//    warp covers 512 contiguous bytes and lane i receives row i.
// Per SM and 128-code k-tile this moves 16 KB of shared memory for the MMA's B
// reads and 16 KB of B stores, against 512 cycles of MMA work.
//
// Warp roles per CTA (21 warps):
//   warp 0       TMEM allocation; in the leader CTA, lane 0 issues the MMAs
//   warps 1-8    A converters: two per 32-lane quarter of TMEM, alternating k-tiles
//   warps 9-16   B converters: two per 32-row group, alternating k-tiles
//   warps 17-20  epilogue (one per TMEM quarter, all 256 columns)
// Every wait is bounded; a wait that runs out aborts the CTA and records
// OFFQ_ERR_TIMEOUT in the device status word.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <mutex>

#include "offq.h"
#include "offq_device.cuh"
#include "offq_host.h"
#include "pair_common.cuh"

namespace {

using namespace offq;

constexpr int BM = 128;            // rows of A per CTA (256 per pair)
constexpr int BN = 256;            // output channels per pair tile (128 rows of B per CTA)
constexpr int BNH = BN / 2;        // rows of B held by one CTA
constexpr int BK = 128;            // codes per k-tile
constexpr int kChunksPerKt = BK / 32;  // 16-byte packed chunks per row per k-tile
// Warp roles of one instantiation. kSplitA / kSplitB converter warps serve each
// 32-row group of A / B, taking turns by k-tile; kEpiWarps drain the
// accumulator (one or two per 32-lane TMEM quarter). 21 warps put 6 on one SM
// sub-partition: 80 registers per thread. (Trading B converters for epilogue
// warps in the several-block kernel left one B warp per group too slow.)
template <bool kOneBlock>
struct Roles {
  // Stages of the operand ring. Several offset blocks take 4, so 128 TMEM columns
  // stay free for half of the precomputed offset correction.
  static constexpr int kStages = kOneBlock ? 6 : 4;
  static constexpr int kSplitA = 2;
  static constexpr int kSplitB = 2;
  static constexpr int kAWarps = 4 * kSplitA, kBWarps = 4 * kSplitB;
  static constexpr int kEpiWarps = 4;
  static constexpr int kEpiCols = BN / (kEpiWarps / 4);  // accumulator columns per epilogue warp
  static constexpr int kFirstA = 1, kFirstB = kFirstA + kAWarps, kFirstEpi = kFirstB + kBWarps;
  static constexpr int kThreads = (kFirstEpi + kEpiWarps) * 32;
  static_assert(kSplitA <= kStages && kSplitB <= kStages, "a converter's next stage is at most one ring turn ahead");
};
constexpr int kConvWarpsPerCta = 8;  // arrivals per stage and CTA: one per 32-row group of A and of B
// k-tiles of loads in flight per converter thread. With one, a warp's loads
// are issued right after its barrier arrival and have its next turn (two k-tiles
// later) to land, and no load is outstanding when the arrival's release orders
// the warp's earlier memory operations.
constexpr int kPrefetch = 1;
constexpr int kMaxStageG = 48;                       // offset blocks staged in shared memory
constexpr int kAccCols = BN;       // fp32 accumulator columns (TMEM lanes = rows)
constexpr int kACol0 = kAccCols;   // A operand stages live in TMEM after the accumulator
constexpr int kAColsPerStage = BK / 4;  // 4 E4M3 values per 32-bit column
constexpr int kTmemCols = 512;
static_assert(kACol0 + Roles<true>::kStages * kAColsPerStage <= kTmemCols, "TMEM budget");
// Several offset blocks: the correction sum_b (o_b - 8 s_a) R[b][n] of a tile is
// computed while its MMAs run; accumulator columns 0..127 keep theirs in TMEM
// after the A stages, columns 128..255 in shared memory.
constexpr int kCorrCol0 = kACol0 + Roles<false>::kStages * kAColsPerStage;
constexpr int kCorrTmemCols = 128;
static_assert(kCorrCol0 + kCorrTmemCols <= kTmemCols, "TMEM budget with the correction");
constexpr int kCorrPitch = (BN - kCorrTmemCols) * 4 + 16;  // bytes per row of the shared half, padded

constexpr int kBStage = BNH * BK;  // 16 KB of E4M3 per stage
// Output rows staged by the one-block epilogue (16-bit outputs): pitch padded
// by 16 bytes, so the 32 rows a warp writes at once fall in distinct bank groups.
constexpr int kOutPitch = BN * 2 + 16;

// Shared memory of one instantiation: B stages; the tile's epilogue constants
// (row sums R[b][256 columns], channel scales, per row o[t][b] - 8 s_a[t] with
// an odd pitch for conflict-free per-lane reads, s_a); for one offset block the
// staged output rows; barriers.
template <bool kOneBlock>
struct Smem {
  static constexpr int kStages = Roles<kOneBlock>::kStages;
  static constexpr int kNumBars = 2 * kStages + 2;
  static constexpr int kMaxG = kOneBlock ? 1 : kMaxStageG;
  static constexpr int kGp = kOneBlock ? 1 : kMaxStageG + 1;
  static constexpr int kOffB = 0;
  static constexpr int kOffR = kOffB + kStages * kBStage;
  static constexpr int kOffW = kOffR + kMaxG * BN * 4;
  static constexpr int kOffO = kOffW + BN * 4;
  static constexpr int kOffSa = kOffO + BM * kGp * 4;
  static constexpr int kOffRt = kOffSa + BM * 4;    // several blocks: -8 Rt[n] 2^-18 per column
  static constexpr int kOffOut = kOffRt + BN * 4;   // one block: staged output rows; several: the correction half
  static constexpr int kOffBars = kOffOut + (kOneBlock ? BM * kOutPitch : BM * kCorrPitch);
  static constexpr int kOffMisc = kOffBars + kNumBars * 8;
  static constexpr int kBytes = kOffMisc + 64 + 1024;  // + slack to align the base to 1024
  static_assert(kBytes <= 227 * 1024, "shared memory budget");
  static_assert(kOffOut % 16 == 0, "bulk copies need 16-byte aligned rows");
};

constexpr uint32_t kIdesc = idesc_e4m3_f32(2 * BM, BN);  // pair MMA: M = 256, N = 256

struct GemmParams {
  const uint8_t* a_codes;  // tiled [ceil(T/32)*32][K/2]
  const uint8_t* w_codes;  // tiled [ceil(N/32)*32][K/2]
  const float* a_scale;
  const float* a_offset;  // [T][G] or nullptr
  const float* w_scale;
  const float* rowsum;    // [G][N]
  void* out;
  int64_t ldo;
  int32_t* acc_debug;
  int* status;
  int T, N, K, G;
  int m_pairs, n_tiles;    // pair tiles: m_pairs x n_tiles
  int raster_m;            // m-pairs per raster group (see tile_mn)
  int t_blocks, n_blocks;  // 32-row tiles present in the code buffers
  int kchunks;             // K / 32
  int vec_ok;              // rowsum and w_scale rows are 16-byte aligned
  int async_out;           // 16-bit output and N % 8 == 0: one-block rows leave by bulk copy
  // MXFP4 operands (kFmtMx): per row and 32-channel block a shift 0..6, tiled as
  // ((row/32 * K/128 + k-tile) * 32 + row%32) * 4 + block%4.
  const uint8_t* a_shifts;
  const uint8_t* w_shifts;
  int nkt;                 // K / 128
};

// Operand formats of the pair kernel: 4-bit integers (activations u = q + 8,
// weights sign-magnitude), or MXFP4 E2M1 codes whose block shifts place each
// code times its block's power of two on the E4M3 grid.
constexpr int kFmtInt4 = 0, kFmtMx = 1;

// Loads the four 16-byte chunks of k-tile kt of one row of a tiled code matrix
// (zeros where the row block or the chunk does not exist).
// blk: this lane's first byte of the row block (nullptr if the block does not
// exist); the block's chunk c starts 512 * c bytes further.
// pol: the L2 policy of the loads.
__device__ __forceinline__ void load_kt(const uint8_t* blk, int kchunks, int kt, uint4 (&v)[kChunksPerKt],
                                        uint64_t pol) {
#pragma unroll
  for (int j = 0; j < kChunksPerKt; ++j) {
    const int c = kt * kChunksPerKt + j;
    if (blk != nullptr && c < kchunks)
      v[j] = ldg_stream_hint(blk + c * 512, pol);
    else
      v[j] = make_uint4(0u, 0u, 0u, 0u);
  }
}

// Pair tile index -> (m-pair, n-tile). Tiles are taken in groups of raster_m
// m-pairs; within a group the m-pair runs fastest. The clusters running at one
// time then share a few weight tiles across all m-pairs of the group, so each
// weight tile comes from DRAM about once per group while the group's
// activation rows (at most ~32 MB, chosen on the host) stay in L2.
__device__ __forceinline__ void tile_mn(const GemmParams& p, int tile, int& mp, int& nt) {
  const int per_group = p.raster_m * p.n_tiles;
  const int grp = tile / per_group;
  const int local = tile - grp * per_group;
  const int m_left = p.m_pairs - grp * p.raster_m;
  const int gm = m_left < p.raster_m ? m_left : p.raster_m;
  nt = local / gm;
  mp = grp * p.raster_m + (local - nt * gm);
}

// Row block (of 32 rows) of this CTA's A rows / B rows for a pair tile.
__device__ __forceinline__ int a_block(const GemmParams& p, int tile, uint32_t rank, int quarter) {
  int mp, nt;
  tile_mn(p, tile, mp, nt);
  return (mp * 2 * BM + static_cast<int>(rank) * BM + quarter * 32) >> 5;
}

__device__ __forceinline__ int b_block(const GemmParams& p, int tile, uint32_t rank, int wb) {
  int mp, nt;
  tile_mn(p, tile, mp, nt);
  return (nt * BN + static_cast<int>(rank) * BNH + wb * 32) >> 5;
}

// Persistent pair kernel: cluster c processes pair tiles c, c + clusters, ...
// (pair tile index mapped to (m-pair, n-tile) by tile_mn). The k-tile counter g runs
// across tiles so the stage ring never drains between tiles.
// kOneBlock: the offsets span the whole row (G == 1). kUnstaged: more than
// kMaxStageG offset blocks, whose constants are read from global memory at the
// tile end. Layers with several
// offset blocks run a separate instantiation, so the register allocation of
// the common one-block kernel does not carry the G-term epilogue loop.
template <int OUT, bool kOneBlock, bool kUnstaged, int FMT>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(Roles<kOneBlock>::kThreads, 1)
    w4a4_gemm_kernel(const GemmParams p) {
  // Integer operands are integers times 2^-9 (the accumulator carries 2^-18) and
  // the activations carry +8; MXFP4 operands are the values themselves.
  constexpr bool kPlus8 = FMT == kFmtInt4;
  constexpr float kAccScale = FMT == kFmtInt4 ? 262144.0f : 1.0f;
  extern __shared__ uint8_t smem_raw[];
  using SL = Smem<kOneBlock>;
  using RL = Roles<kOneBlock>;
  constexpr int kStages = RL::kStages;
  constexpr int kFirstA = RL::kFirstA, kFirstB = RL::kFirstB, kFirstEpi = RL::kFirstEpi;
  constexpr int kEpiWarps = RL::kEpiWarps, kEpiCols = RL::kEpiCols;
  constexpr int kOffB = SL::kOffB, kOffR = SL::kOffR, kOffW = SL::kOffW, kOffO = SL::kOffO, kOffSa = SL::kOffSa;
  constexpr int kOffBars = SL::kOffBars, kOffMisc = SL::kOffMisc, kStageGp = SL::kGp;
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (base - raw);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const int cluster = blockIdx.x >> 1;
  const int clusters = gridDim.x >> 1;
  const int nk = (p.K + BK - 1) / BK;
  const int num_tiles = p.m_pairs * p.n_tiles;

  const uint32_t bar0 = base + kOffBars;
  auto full = [&](int s) { return bar0 + 8u * s; };                // leader: operands of stage s ready
  auto empty = [&](int s) { return bar0 + 8u * (kStages + s); };   // both: stage s consumed
  const uint32_t acc_full = bar0 + 8u * (2 * kStages);             // both: accumulator complete
  const uint32_t acc_empty = bar0 + 8u * (2 * kStages + 1);        // leader: accumulator drained
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kOffMisc);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + kOffMisc + 16);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full(s), 2 * kConvWarpsPerCta);
      mbar_init(empty(s), 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 2 * kEpiWarps);
    *abort = 0;
    mbar_fence_init();
  }
  if (warp == 0) {
    tmem_alloc2(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish2();
  }
  tc_fence_before();
  cluster_sync();  // barriers initialised and TMEM allocated in both CTAs
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // Setup above touches no global memory; from here on, the inputs of the
  // previous kernel in the stream must be complete.
  griddep_wait();
  griddep_launch_dependents();
  int mma_tiles = 0;

  if (warp == 0) {
    // ---------------- MMA issuer (leader CTA) ----------------
    if (rank == 0 && lane == 0) {
      int s = 0, phase = 0, lt = 0;  // stage and phase parity of the next k-tile
      for (int tile = cluster; tile < num_tiles && !*abort; tile += clusters, ++lt) {
        if (!wait_cluster(acc_empty, (lt & 1) ^ 1, abort)) break;
        tc_fence_after();
        bool ok = true;
        for (int kt = 0; kt < nk; ++kt) {
          if (!wait_cluster(full(s), phase, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t b_addr = base + kOffB + s * kBStage;
#pragma unroll
          for (int kk = 0; kk < BK / 32; ++kk) {
            mma2_ts(tmem, tmem + kACol0 + s * kAColsPerStage + 8 * kk, smem_desc_sw128(b_addr + 32 * kk), kIdesc,
                    (kt | kk) != 0 ? 1u : 0u);
          }
          mma2_commit_both(empty(s));
          if (++s == kStages) {
            s = 0;
            phase ^= 1;
          }
        }
        mma2_commit_both(acc_full);
        mma_tiles = lt + 1;
        if (!ok) break;
      }
    }
  } else if (warp < kFirstEpi) {
    // ---------------- converters: packed codes -> E4M3 operands ----------------
    // A warps write 32 TMEM lanes (their quarter); B warps write 32 rows of the
    // shared-memory stage. Each thread keeps kPrefetch k-tiles of loads in
    // flight in a register ring.
    const bool is_a = warp < kFirstB;
    const int quarter = warp & 3;
    const int wb = (warp - kFirstB) & 3;
    const int part = is_a ? (warp - kFirstA) >> 2 : (warp - kFirstB) >> 2;  // k-tiles g == part mod split
    static_assert(RL::kSplitA == RL::kSplitB, "one k-tile stride for both converter kinds");
    constexpr int split = RL::kSplitA;
    const uint32_t full_l = leader_addr(full(0));
    const uint8_t* codes = is_a ? p.a_codes : p.w_codes;
    // The raster keeps a group of m-pairs' activation codes for every n-tile, so
    // they are kept in L2 ahead of the weight tiles streaming past them.
    const uint64_t pol = is_a ? l2_evict_last() : l2_evict_normal();
    const int rb_count = is_a ? p.t_blocks : p.n_blocks;
    // This lane's first byte of the row block a tile needs (nullptr: the block
    // lies past the buffer's rows). Computed once per tile, not per load.
    const uint8_t* shifts = is_a ? p.a_shifts : p.w_shifts;
    auto block_ptr = [&](int tile) -> const uint8_t* {
      const int rb = is_a ? a_block(p, tile, rank, quarter) : b_block(p, tile, rank, wb);
      return rb < rb_count ? codes + static_cast<int64_t>(rb) * p.kchunks * 512 + lane * 16 : nullptr;
    };
    // MXFP4: this lane's shift words of the row block a tile needs (nullptr as above).
    auto shift_ptr = [&](int tile) -> const uint8_t* {
      if constexpr (FMT == kFmtMx) {
        const int rb = is_a ? a_block(p, tile, rank, quarter) : b_block(p, tile, rank, wb);
        return rb < rb_count ? shifts + (static_cast<int64_t>(rb) * p.nkt * 32 + lane) * 4 : nullptr;
      } else {
        (void)tile;
        return nullptr;
      }
    };
    auto load_shift = [&](const uint8_t* sblk, int kt) -> uint32_t {
      if constexpr (FMT == kFmtMx) {
        return sblk != nullptr ? __ldg(reinterpret_cast<const uint32_t*>(sblk + kt * 128)) : 0u;
      } else {
        (void)sblk;
        (void)kt;
        return 0u;
      }
    };
    uint4 ring[kPrefetch][kChunksPerKt];
    uint32_t sring[kPrefetch];
    int ld_tile = cluster, ld_kt = 0;  // next k-tile to load
    auto advance1 = [&](int& tile, int& kt) {
      if (++kt == nk) {
        kt = 0;
        tile += clusters;
      }
    };
    auto advance = [&](int& tile, int& kt) {
#pragma unroll
      for (int i = 0; i < split; ++i) advance1(tile, kt);
    };
#pragma unroll
    for (int i = 0; i < split; ++i)
      if (i < part) advance1(ld_tile, ld_kt);
    const int start_tile = ld_tile, start_kt = ld_kt;
#pragma unroll
    for (int i = 0; i < kPrefetch; ++i) {
      sring[i] = 0u;
      if (ld_tile < num_tiles) {
        load_kt(block_ptr(ld_tile), p.kchunks, ld_kt, ring[i], pol);
        sring[i] = load_shift(shift_ptr(ld_tile), ld_kt);
      }
      advance(ld_tile, ld_kt);
    }
    int tile = start_tile, kt = start_kt;
    int s = part, phase = 0;  // stage and phase parity of this warp's k-tile g (g == part mod split)
    int blk_tile = ld_tile;  // the tile whose row block blk (and sblk) points into
    const uint8_t* blk = ld_tile < num_tiles ? block_ptr(ld_tile) : nullptr;
    const uint8_t* sblk = ld_tile < num_tiles ? shift_ptr(ld_tile) : nullptr;
    bool run = tile < num_tiles;
    while (run) {
#pragma unroll
      for (int slot = 0; slot < kPrefetch; ++slot) {
        if (!run) break;
        // Warp-uniform outcome, so the __syncwarp below is reached by all lanes. After
        // an abort no stage frees up again, so this wait is where a converter stops.
        if (!__all_sync(0xFFFFFFFFu, wait_cluster(empty(s), phase ^ 1, abort))) {
          run = false;
          break;
        }
        if (is_a) {
          tc_fence_after();
          uint32_t f8[32];
#pragma unroll
          for (int j = 0; j < kChunksPerKt; ++j) {
            if constexpr (FMT == kFmtMx) {
              uint32_t llo, lhi;
              mx_lut((sring[slot] >> (8 * j)) & 0xFFu, llo, lhi);
              widen_mx(ring[slot][j].x, llo, lhi, f8[8 * j + 0], f8[8 * j + 1]);
              widen_mx(ring[slot][j].y, llo, lhi, f8[8 * j + 2], f8[8 * j + 3]);
              widen_mx(ring[slot][j].z, llo, lhi, f8[8 * j + 4], f8[8 * j + 5]);
              widen_mx(ring[slot][j].w, llo, lhi, f8[8 * j + 6], f8[8 * j + 7]);
            } else {
              widen_act(ring[slot][j].x, f8[8 * j + 0], f8[8 * j + 1]);
              widen_act(ring[slot][j].y, f8[8 * j + 2], f8[8 * j + 3]);
              widen_act(ring[slot][j].z, f8[8 * j + 4], f8[8 * j + 5]);
              widen_act(ring[slot][j].w, f8[8 * j + 6], f8[8 * j + 7]);
            }
          }
          tmem_st_32cols(tmem + (static_cast<uint32_t>(quarter * 32) << 16) + kACol0 + s * kAColsPerStage, f8);
          tmem_st_wait();
          tc_fence_before();
        } else {
          const int r = wb * 32 + lane;
          const uint32_t st = base + kOffB + s * kBStage + r * 128;
#pragma unroll
          for (int j = 0; j < kChunksPerKt; ++j) {
            uint32_t a0, a1, a2, a3, b0, b1, b2, b3;
            if constexpr (FMT == kFmtMx) {
              uint32_t llo, lhi;
              mx_lut((sring[slot] >> (8 * j)) & 0xFFu, llo, lhi);
              widen_mx(ring[slot][j].x, llo, lhi, a0, a1);
              widen_mx(ring[slot][j].y, llo, lhi, a2, a3);
              widen_mx(ring[slot][j].z, llo, lhi, b0, b1);
              widen_mx(ring[slot][j].w, llo, lhi, b2, b3);
            } else {
              widen_weight(ring[slot][j].x, a0, a1);
              widen_weight(ring[slot][j].y, a2, a3);
              widen_weight(ring[slot][j].z, b0, b1);
              widen_weight(ring[slot][j].w, b2, b3);
            }
            sts128(st + (((2 * j) ^ (r & 7)) << 4), a0, a1, a2, a3);
            sts128(st + (((2 * j + 1) ^ (r & 7)) << 4), b0, b1, b2, b3);
          }
          fence_proxy_async_smem();
        }
        __syncwarp();
        if (lane == 0) arrive_cluster(full_l + 8u * s);
        // Refill this slot kPrefetch k-tiles ahead.
        if (ld_tile < num_tiles) {
          if (ld_tile != blk_tile) {
            blk_tile = ld_tile;
            blk = block_ptr(ld_tile);
            sblk = shift_ptr(ld_tile);
          }
          load_kt(blk, p.kchunks, ld_kt, ring[slot], pol);
          sring[slot] = load_shift(sblk, ld_kt);
        }
        advance(ld_tile, ld_kt);
        advance(tile, kt);
        s += split;
        if (s >= kStages) {
          s -= kStages;
          phase ^= 1;
        }
        run = tile < num_tiles;  // warp-uniform
      }
    }
  } else {
    // ---------------- epilogue ----------------
    const uint64_t out_pol = l2_evict_first();  // outputs: nothing here reads them again
    const int quarter = warp & 3;              // TMEM lanes this warp may read
    const int half = (warp - kFirstEpi) / 4;   // which kEpiCols accumulator columns
    const int et = threadIdx.x - kFirstEpi * 32;
    const int G = kOneBlock ? 1 : p.G;
    // More offset blocks than the staging area holds take their own
    // instantiation, so its register needs stay out of the staged kernels.
    constexpr bool staged = !kUnstaged;
    float* Rs = reinterpret_cast<float*>(smem + kOffR);
    float* Ws = reinterpret_cast<float*>(smem + kOffW);
    float* Os = reinterpret_cast<float*>(smem + kOffO);
    float* Sa = reinterpret_cast<float*>(smem + kOffSa);
    float* Rt = reinterpret_cast<float*>(smem + SL::kOffRt);
    const uint32_t acc_empty_l = leader_addr(acc_empty);
    // Loop exit decided only from a flag the epilogue warps write before their
    // own barrier, so all eight warps leave together (bar.sync has no timeout).
    volatile int* epi_stop = reinterpret_cast<volatile int*>(smem + kOffMisc + 32);
    if (et == 0) *epi_stop = 0;
    epi_sync<kEpiWarps>();
    int lt = 0;
    for (int tile = cluster; tile < num_tiles; tile += clusters, ++lt) {
      int mp, nt;
      tile_mn(p, tile, mp, nt);
      const int m0 = mp * 2 * BM + static_cast<int>(rank) * BM;
      const int nt0 = nt * BN;
      // Stage this tile's constants while the main loop runs.
      if (staged) {
        for (int i = et; i < G * BN; i += kEpiWarps * 32) {
          const int b = i / BN, j = i - b * BN, n = nt0 + j;
          Rs[i] = n < p.N ? __ldg(p.rowsum + static_cast<int64_t>(b) * p.N + n) : 0.f;
        }
        for (int i = et; i < BN; i += kEpiWarps * 32) Ws[i] = nt0 + i < p.N ? __ldg(p.w_scale + nt0 + i) : 0.f;
        for (int i = et; i < BM; i += kEpiWarps * 32) Sa[i] = m0 + i < p.T ? __ldg(p.a_scale + m0 + i) : 0.f;
        for (int i = et; i < BM * G; i += kEpiWarps * 32) {
          const int r = i / G, b = i - r * G, t = m0 + r;
          float v = 0.f;
          if (t < p.T && p.a_offset != nullptr) v = __ldg(p.a_offset + static_cast<int64_t>(t) * G + b);
          Os[r * kStageGp + b] = v;
        }
      }
      epi_sync<kEpiWarps>();
      if (!kOneBlock && staged && kPlus8) {
        // Rt[n] * 8 * 2^-18 = sum_b R[b][n] * 2^-15: integers, exact in fp32.
        for (int i = et; i < BN; i += kEpiWarps * 32) {
          float r = 0.f;
          for (int b = 0; b < G; ++b) r += Rs[b * BN + i];
          Rt[i] = r * -0x1p-15f;
        }
        epi_sync<kEpiWarps>();
      }
      if constexpr (!kOneBlock) {
        if (staged) {
          // While this tile's MMAs run: its offset correction, per element the same
          // chain as at the tile end (block 0 multiplied, then FMAs in block order).
          constexpr int CW = 16;
          const int rl = quarter * 32 + lane;
          const float* orow = Os + rl * kStageGp;
          const uint32_t corr_tm = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + kCorrCol0;
          const uint32_t corr_s = base + SL::kOffOut + rl * kCorrPitch;
          for (int c = 0; c < kEpiCols / CW; ++c) {
            const int jc = half * kEpiCols + c * CW;  // column within the tile
            float y[CW];
            {
              const float ob = orow[0];
              const float4* r4 = reinterpret_cast<const float4*>(Rs + jc);
#pragma unroll
              for (int q4 = 0; q4 < CW / 4; ++q4) {
                const float4 rv = r4[q4];
                y[4 * q4] = ob * rv.x; y[4 * q4 + 1] = ob * rv.y; y[4 * q4 + 2] = ob * rv.z; y[4 * q4 + 3] = ob * rv.w;
              }
            }
            for (int b = 1; b < G; ++b) {
              const float ob = orow[b];
              const float4* r4 = reinterpret_cast<const float4*>(Rs + b * BN + jc);
#pragma unroll
              for (int q4 = 0; q4 < CW / 4; ++q4) {
                const float4 rv = r4[q4];
                y[4 * q4] = fmaf(ob, rv.x, y[4 * q4]);
                y[4 * q4 + 1] = fmaf(ob, rv.y, y[4 * q4 + 1]);
                y[4 * q4 + 2] = fmaf(ob, rv.z, y[4 * q4 + 2]);
                y[4 * q4 + 3] = fmaf(ob, rv.w, y[4 * q4 + 3]);
              }
            }
            if (jc < kCorrTmemCols) {
              uint32_t u[CW];
#pragma unroll
              for (int jj = 0; jj < CW; ++jj) u[jj] = __float_as_uint(y[jj]);
              tmem_st_16cols(corr_tm + jc, u);
            } else {
              const uint32_t a = corr_s + (jc - kCorrTmemCols) * 4;
#pragma unroll
              for (int q4 = 0; q4 < CW / 4; ++q4)
                sts128(a + 16 * q4, __float_as_uint(y[4 * q4]), __float_as_uint(y[4 * q4 + 1]),
                       __float_as_uint(y[4 * q4 + 2]), __float_as_uint(y[4 * q4 + 3]));
            }
          }
          tmem_st_wait();
        }
      }
      const bool ok = __all_sync(0xFFFFFFFFu, wait_cluster(acc_full, lt & 1, abort));
      if (!ok && lane == 0) *epi_stop = 1;
      tc_fence_after();
      const int rl = quarter * 32 + lane;
      const int t = m0 + rl;
      const bool row_ok = t < p.T;
      const int n0 = nt0 + half * kEpiCols;
      const uint32_t acc_tm = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + half * kEpiCols;
      constexpr int CW = 16;  // accumulator columns per TMEM load
      if (!ok) {
        // Aborted: nothing to drain.
      } else if (!kOneBlock && staged) {
        // Several offset blocks: the correction was computed during the main loop.
        const float sa = Sa[rl];
        const uint32_t corr_tm = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + kCorrCol0;
        const uint32_t corr_s = base + SL::kOffOut + rl * kCorrPitch;
        for (int c = 0; c < kEpiCols / CW; ++c) {
          const int jc = half * kEpiCols + c * CW;  // column within the tile
          uint32_t acc[CW], cr[CW];
          tmem_ld_16cols(acc_tm + c * CW, acc);
          if (jc < kCorrTmemCols) tmem_ld_16cols(corr_tm + jc, cr);
          tmem_ld_wait();
          const int nb = n0 + c * CW;
          if (!row_ok || nb >= p.N) continue;
          if (jc >= kCorrTmemCols) {
            const uint32_t a = corr_s + (jc - kCorrTmemCols) * 4;
#pragma unroll
            for (int q4 = 0; q4 < CW / 4; ++q4) {
              const uint4 v = lds128(a + 16 * q4);
              cr[4 * q4] = v.x; cr[4 * q4 + 1] = v.y; cr[4 * q4 + 2] = v.z; cr[4 * q4 + 3] = v.w;
            }
          }
          const int nvalid = p.N - nb < CW ? p.N - nb : CW;
          float z[CW];
#pragma unroll
          for (int jj = 0; jj < CW; ++jj) {
            // (acc' - 8 Rt) 2^-18, then * 2^18: both steps exact.
            const float accf = kPlus8 ? (__uint_as_float(acc[jj]) + Rt[jc + jj]) * kAccScale : __uint_as_float(acc[jj]);
            z[jj] = Ws[jc + jj] * fmaf(sa, accf, __uint_as_float(cr[jj]));
          }
          store_out<OUT, CW>(p.out, static_cast<int64_t>(t) * p.ldo + nb, z, nvalid, out_pol);
          if (p.acc_debug != nullptr) {
            int32_t* d = p.acc_debug + static_cast<int64_t>(t) * p.N + nb;
#pragma unroll
            for (int jj = 0; jj < CW; ++jj)
              if (jj < nvalid) d[jj] = __float2int_rn(__uint_as_float(acc[jj]) * 262144.0f);
          }
        }
      } else if (kOneBlock) {
        // Packed fp32 pairs; each lane rounds as y = s_w * fma(s_a, acc * 2^18, o R)
        // does, with acc = (acc' - 8 R) 2^-18 formed exactly first (s_a * 2^18 and
        // its product with acc are exact). 16-bit rows go to shared memory and
        // leave by one bulk copy per row once the accumulator is read, so the
        // tile's output write overlaps the next tile's MMAs.
        const float sa2 = Sa[rl] * kAccScale;
        const float ob = Os[rl * kStageGp];
        const uint64_t SA2 = pack2(sa2, sa2), OB = pack2(ob, ob);
        const uint64_t M8 = pack2(-0x1p-15f, -0x1p-15f);  // -8 * 2^-18
        const bool async_out = OUT != OFFQ_F32 && p.async_out != 0;
        const uint32_t orow_s = base + SL::kOffOut + rl * kOutPitch;
        if (async_out) bulk_wait_read_all();  // this row's previous copy has read the buffer
        for (int c = 0; c < kEpiCols / CW; c += 2) {
          uint32_t acc2[2 * CW];
          tmem_ld_32cols_waited(acc_tm + c * CW, acc2);
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const uint32_t* acc = &acc2[h * CW];
            const int nb = n0 + (c + h) * CW;
            const int jc = half * kEpiCols + (c + h) * CW;
            if (!row_ok || nb >= p.N) continue;
            const int nvalid = p.N - nb < CW ? p.N - nb : CW;
            const float4* r4 = reinterpret_cast<const float4*>(Rs + jc);
            const float4* w4 = reinterpret_cast<const float4*>(Ws + jc);
            float y[CW];
#pragma unroll
            for (int q4 = 0; q4 < CW / 4; ++q4) {
              const float4 rv = r4[q4], wv = w4[q4];
              const uint64_t R0 = pack2(rv.x, rv.y), R1 = pack2(rv.z, rv.w);
              uint64_t A0 = pack2(__uint_as_float(acc[4 * q4]), __uint_as_float(acc[4 * q4 + 1]));
              uint64_t A1 = pack2(__uint_as_float(acc[4 * q4 + 2]), __uint_as_float(acc[4 * q4 + 3]));
              if constexpr (kPlus8) {
                A0 = fma2v(R0, M8, A0);
                A1 = fma2v(R1, M8, A1);
              }
              unpack2(mul2v(pack2(wv.x, wv.y), fma2v(SA2, A0, mul2v(OB, R0))), y[4 * q4], y[4 * q4 + 1]);
              unpack2(mul2v(pack2(wv.z, wv.w), fma2v(SA2, A1, mul2v(OB, R1))), y[4 * q4 + 2], y[4 * q4 + 3]);
            }
            if (async_out) {
              uint32_t hv[CW / 2];
#pragma unroll
              for (int i = 0; i < CW / 2; ++i) {
                if (OUT == OFFQ_BF16) {
                  const __nv_bfloat162 v = __floats2bfloat162_rn(y[2 * i], y[2 * i + 1]);
                  hv[i] = *reinterpret_cast<const uint32_t*>(&v);
                } else {
                  const __half2 v = __floats2half2_rn(y[2 * i], y[2 * i + 1]);
                  hv[i] = *reinterpret_cast<const uint32_t*>(&v);
                }
              }
              sts128(orow_s + (c + h) * CW * 2, hv[0], hv[1], hv[2], hv[3]);
              sts128(orow_s + (c + h) * CW * 2 + 16, hv[4], hv[5], hv[6], hv[7]);
            } else {
              store_out<OUT, CW>(p.out, static_cast<int64_t>(t) * p.ldo + nb, y, nvalid, out_pol);
            }
            if (p.acc_debug != nullptr) {
              int32_t* d = p.acc_debug + static_cast<int64_t>(t) * p.N + nb;
#pragma unroll
              for (int jj = 0; jj < CW; ++jj)
                if (jj < nvalid) d[jj] = __float2int_rn(__uint_as_float(acc[jj]) * 262144.0f);
            }
          }
        }
        if (async_out && row_ok && n0 < p.N) {
          const int ncols = p.N - n0 < kEpiCols ? p.N - n0 : kEpiCols;
          fence_proxy_async_smem();  // the row's shared stores, visible to the bulk copy
          bulk_store(static_cast<uint16_t*>(p.out) + static_cast<int64_t>(t) * p.ldo + n0, orow_s,
                     static_cast<uint32_t>(ncols) * 2, out_pol);
          bulk_commit();
        }
      } else {
        // More offset blocks than the staging area holds: read the constants directly.
        const float sa = row_ok ? __ldg(p.a_scale + t) : 0.f;
        const bool has_off = p.a_offset != nullptr && row_ok;
        const float* orow = has_off ? p.a_offset + static_cast<int64_t>(t) * G : p.a_scale;
        for (int c = 0; c < kEpiCols / CW; ++c) {
          uint32_t acc[CW];
          tmem_ld_16cols(acc_tm + c * CW, acc);
          tmem_ld_wait();
          const int nb = n0 + c * CW;
          if (!row_ok || nb >= p.N) continue;
          const int nvalid = p.N - nb < CW ? p.N - nb : CW;
          float y[CW], a[CW];
#pragma unroll
          for (int jj = 0; jj < CW; ++jj) {
            y[jj] = 0.f;
            a[jj] = __uint_as_float(acc[jj]);
          }
          for (int b = 0; b < G; ++b) {
            const float ob = has_off ? __ldg(orow + b) : 0.f;
            const float* rb = p.rowsum + static_cast<int64_t>(b) * p.N + nb;
#pragma unroll
            for (int jj = 0; jj < CW; ++jj)
              if (jj < nvalid) {
                const float r = __ldg(rb + jj);
                y[jj] = fmaf(ob, r, y[jj]);
                if (kPlus8) a[jj] = fmaf(r, -0x1p-15f, a[jj]);  // acc' - 8 R, in units of 2^-18: exact
              }
          }
#pragma unroll
          for (int jj = 0; jj < CW; ++jj) {
            const float accf = a[jj] * kAccScale;
            y[jj] = jj < nvalid ? __ldg(p.w_scale + nb + jj) * fmaf(sa, accf, y[jj]) : 0.f;
          }
          store_out<OUT, CW>(p.out, static_cast<int64_t>(t) * p.ldo + nb, y, nvalid, out_pol);
          if (p.acc_debug != nullptr) {
            int32_t* d = p.acc_debug + static_cast<int64_t>(t) * p.N + nb;
#pragma unroll
            for (int jj = 0; jj < CW; ++jj)
              if (jj < nvalid) d[jj] = __float2int_rn(__uint_as_float(acc[jj]) * 262144.0f);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (ok && lane == 0) arrive_cluster(acc_empty_l);
      epi_sync<kEpiWarps>();  // the staged constants are reused for the next tile
      if (*epi_stop) break;
    }
    if (kOneBlock) bulk_wait_all();  // output rows in flight are written before the CTA ends
  }

  // ---------------- teardown ----------------
  if (*abort && warp == 0 && lane == 0 && rank == 0 && mma_tiles > 0) {
    // Let the MMAs already issued finish before tensor memory is released.
    wait_teardown(acc_full, (mma_tiles - 1) & 1);
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the pair's MMAs read both CTAs' memory: leave together
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc2(tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && *abort && p.status != nullptr) atomicExch(p.status, kErrTimeout);
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

template <int OUT, bool kOneBlock, bool kUnstaged, int FMT>
int launch_gemm(const GemmParams& p, cudaStream_t s) {
  auto kern = w4a4_gemm_kernel<OUT, kOneBlock, kUnstaged, FMT>;
  constexpr int kThreads = Roles<kOneBlock>::kThreads;
  constexpr int kSmemBytes = Smem<kOneBlock>::kBytes;
  if (!smem_optin<w4a4_gemm_kernel<OUT, kOneBlock, kUnstaged, FMT>>(kSmemBytes)) return OFFQ_ERR_CUDA;
  const int sms = num_sms();
  if (sms < 2) return OFFQ_ERR_CUDA;
  const int tiles = p.m_pairs * p.n_tiles;
  const int clusters = tiles < sms / 2 ? tiles : sms / 2;
  return launch_pdl(kern, dim3(2 * clusters), dim3(kThreads), kSmemBytes, s, p);
}

template <int FMT>
int dispatch_gemm(const GemmParams& p, int out_dtype, cudaStream_t s) {
  const bool unstaged = p.G > kMaxStageG;
  switch (out_dtype) {
    case OFFQ_F32:
      return p.G == 1 ? launch_gemm<OFFQ_F32, true, false, FMT>(p, s)
                      : unstaged ? launch_gemm<OFFQ_F32, false, true, FMT>(p, s)
                                 : launch_gemm<OFFQ_F32, false, false, FMT>(p, s);
    case OFFQ_BF16:
      return p.G == 1 ? launch_gemm<OFFQ_BF16, true, false, FMT>(p, s)
                      : unstaged ? launch_gemm<OFFQ_BF16, false, true, FMT>(p, s)
                                 : launch_gemm<OFFQ_BF16, false, false, FMT>(p, s);
    case OFFQ_F16:
      return p.G == 1 ? launch_gemm<OFFQ_F16, true, false, FMT>(p, s)
                      : unstaged ? launch_gemm<OFFQ_F16, false, true, FMT>(p, s)
                                 : launch_gemm<OFFQ_F16, false, false, FMT>(p, s);
    default: return OFFQ_ERR_INVALID_ARG;
  }
}

// The shapes, tile counts and raster of one launch (arguments already checked).
GemmParams gemm_params(const uint8_t* a_codes, const float* a_scale, const float* a_offset, int64_t T, int64_t N,
                       int64_t K, int32_t g, const uint8_t* w_codes, const float* w_scale, const float* w_offsum,
                       void* out, int out_dtype, int64_t ldo, int32_t* acc_debug) {
  GemmParams p{};
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
  p.m_pairs = static_cast<int>((T + 2 * BM - 1) / (2 * BM));
  p.n_tiles = static_cast<int>((N + BN - 1) / BN);
  // Raster groups of m-pairs whose activation codes total at most ~32 MB.
  const int64_t pair_bytes = 2 * BM * (K / 2);
  int64_t rm = (int64_t{32} << 20) / pair_bytes;
  if (rm < 1) rm = 1;
  p.raster_m = static_cast<int>(rm < p.m_pairs ? rm : p.m_pairs);
  p.t_blocks = static_cast<int>((T + 31) / 32);
  p.n_blocks = static_cast<int>((N + 31) / 32);
  p.kchunks = static_cast<int>(K / 32);
  p.nkt = static_cast<int>(K / 128);
  p.vec_ok = aligned(w_offsum, 16) && aligned(w_scale, 16) && (N % 4 == 0);
  p.async_out = out_dtype != OFFQ_F32 && N % 8 == 0;
  return p;
}

}  // namespace

extern "C" int offq_w4a4_linear(const uint8_t* a_codes, const float* a_scale, const float* a_offset, int64_t T,
                                int64_t N, int64_t K, int32_t g, const uint8_t* w_codes, const float* w_scale,
                                const float* w_offsum, void* out, int out_dtype, int64_t ldo, int32_t* acc_debug,
                                void* stream) {
  const int ob = elem_bytes(out_dtype);
  if (ob == 0 || T < 0 || N < 1 || !is_pow2(g) || g < 32 || g > 8192) return OFFQ_ERR_INVALID_ARG;
  if (K <= 0 || K % g != 0 || K % 32 != 0 || ldo < N) return OFFQ_ERR_INVALID_ARG;
  if (K > kMaxGemmK || T > 0x3FFFFFFF || N > 0x3FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  if (T == 0) return OFFQ_OK;
  if (a_codes == nullptr || a_scale == nullptr || w_codes == nullptr || w_scale == nullptr || w_offsum == nullptr ||
      out == nullptr)
    return OFFQ_ERR_INVALID_ARG;
  if (!aligned(a_codes, 16) || !aligned(w_codes, 16) || !aligned(out, 16) || (ldo * ob) % 16 != 0 ||
      !aligned(a_scale, 4) || !aligned(w_scale, 4) || !aligned(w_offsum, 4) ||
      (a_offset != nullptr && !aligned(a_offset, 4)) || (acc_debug != nullptr && !aligned(acc_debug, 4)))
    return OFFQ_ERR_MISALIGNED;

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (T <= decode_max_tokens())
    return w4a4_linear_decode(a_codes, a_scale, a_offset, T, N, K, g, w_codes, w_scale, w_offsum, out, out_dtype, ldo,
                              acc_debug, s);
  const GemmParams p = gemm_params(a_codes, a_scale, a_offset, T, N, K, g, w_codes, w_scale, w_offsum, out, out_dtype,
                                   ldo, acc_debug);
  return dispatch_gemm<kFmtInt4>(p, out_dtype, s);
}

extern "C" int offq_mx_linear(const uint8_t* a_codes, const uint8_t* a_shifts, const float* a_scale,
                              const float* a_offset, int64_t T, int64_t N, int64_t K, int32_t g,
                              const uint8_t* w_codes, const uint8_t* w_shifts, const float* w_scale,
                              const float* w_offsum, void* out, int out_dtype, int64_t ldo, void* stream) {
  const int ob = elem_bytes(out_dtype);
  if (ob == 0 || T < 0 || N < 1 || !is_pow2(g) || g < 32 || g > 8192) return OFFQ_ERR_INVALID_ARG;
  if (K <= 0 || K % g != 0 || K % 128 != 0 || ldo < N) return OFFQ_ERR_INVALID_ARG;
  if (K > kMaxGemmK || T > 0x3FFFFFFF || N > 0x3FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  if (T == 0) return OFFQ_OK;
  if (a_codes == nullptr || a_shifts == nullptr || a_scale == nullptr || w_codes == nullptr || w_shifts == nullptr ||
      w_scale == nullptr || w_offsum == nullptr || out == nullptr)
    return OFFQ_ERR_INVALID_ARG;
  if (!aligned(a_codes, 16) || !aligned(w_codes, 16) || !aligned(out, 16) || (ldo * ob) % 16 != 0 ||
      !aligned(a_shifts, 4) || !aligned(w_shifts, 4) || !aligned(a_scale, 4) || !aligned(w_scale, 4) ||
      !aligned(w_offsum, 4) || (a_offset != nullptr && !aligned(a_offset, 4)))
    return OFFQ_ERR_MISALIGNED;
  GemmParams p = gemm_params(a_codes, a_scale, a_offset, T, N, K, g, w_codes, w_scale, w_offsum, out, out_dtype, ldo,
                             nullptr);
  p.a_shifts = a_shifts;
  p.w_shifts = w_shifts;
  return dispatch_gemm<kFmtMx>(p, out_dtype, static_cast<cudaStream_t>(stream));
}
