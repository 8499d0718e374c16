// W4A4 GEMM with per-group activation scales and zero-points
// (offq_w4a4_linear_group): the paper's evaluated activation setting, groups
// of 128 channels quantized asymmetrically (Sec. 3 Eq. 1 with its zero-point,
// Sec. 4 settings), against per-channel symmetric 4-bit weights.
//
//   y[t][n] = s_w[n] * sum_j s[t][j] * (P_j[t][n] - z[t][j] * R[j][n])
//   P_j[t][n] = sum_{k in group j} u[t][k] * q_w[n][k]
//
// u in [0, 15] is the stored code (Eq. 1's x_q), q_w in [-7, 7], and R[j][n]
// the integer row sum of the weight codes over group j. Both codes widen to
// exact E4M3 operands (bytes 0x00..0x0F are 0..15 * 2^-9), so P_j, an integer
// times 2^-18 below 2^24 * 2^-18, is exact in the fp32 accumulator.
//
// One 128-code k-tile is one group, so the per-(token, group) scale cannot sit
// in the operands, but the zero-point can: P_j - z R_j = sum (u - z) q_w. The A
// converters widen u - zc with zc = clamp(z, 0, 15) (|u - zc| <= 15 is exact
// in E4M3), the pair MMA (M 256, N 128) writes each group's P_j - zc R_j into
// one of two TMEM partial buffers, and eight scaler warps fold it into a
// running fp32 sum held in their registers,
//   d = fma(-(z - zc), R, acc)   (only in a warp with a row whose group does
//                                 not straddle zero; exact while |z R| < 2^24),
//   S = fma(s, d, S),
// (on the accumulator's values * 2^-18, with the factors scaled to match),
// while the MMA fills the other buffer. After a tile's last group the scalers
// multiply by s_w and store y, rounding once to the output type. d equals
// P_j - z R_j exactly either way, so the result does not depend on zc.
//
// TMEM (512 columns per CTA): P0 [0, 128), P1 [128, 256), 6 A stages of 32
// columns [256, 448). The N = 128 pair tile keeps both partials next to the
// A stages, and each scaler thread's 64 running sums in its registers.
//
// Warp roles per CTA (15 warps, so up to 128 registers per thread):
//   warp 0       TMEM allocation; in the leader CTA, lane 0 issues the MMAs
//   warps 1-4    A converters: one per 32-lane TMEM quarter, every k-tile
//   warps 5-6    B converters: one per 32-row group (64 rows of B per CTA)
//   warps 7-14   scalers and epilogue, two per TMEM quarter (64 columns each);
//                they prefetch the row sums R and s_w into shared memory
//                two groups ahead (cp.async)
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

constexpr int GBM = 128;         // rows of A per CTA (256 per pair)
constexpr int GBN = 128;         // output channels per pair tile
constexpr int GBNH = GBN / 2;    // rows of B held by one CTA
constexpr int GBK = 128;         // codes per k-tile = one activation group
constexpr int kGroup = GBK;
constexpr int kGChunks = GBK / 32;  // 16-byte packed chunks per row per k-tile
constexpr int kGStages = 6;
constexpr int kGRing = 3;           // k-tiles of loads in flight per converter thread
constexpr int kGAWarps = 4;         // one per 32-lane TMEM quarter, every k-tile
constexpr int kGBWarps = GBNH / 32; // one per 32-row group of B
constexpr int kGScWarps = 8;            // two per TMEM quarter
constexpr int kGScCols = GBN / (kGScWarps / 4);  // columns per scaler warp
constexpr int kGFirstA = 1, kGFirstB = kGFirstA + kGAWarps, kGFirstSc = kGFirstB + kGBWarps;
constexpr int kGThreads = (kGFirstSc + kGScWarps) * 32;
constexpr int kGArrivals = 4 + GBNH / 32;  // per stage and CTA: one per A quarter and per B row group
constexpr int kPCol0 = 0;                  // two partial buffers of GBN columns
constexpr int kGACol0 = 2 * GBN;           // A stages
constexpr int kGAColsPerStage = GBK / 4;
constexpr int kGTmemCols = 512;
static_assert(kGACol0 + kGStages * kGAColsPerStage <= kGTmemCols, "TMEM budget");
constexpr int kGBStage = GBNH * GBK;  // 8 KB of E4M3 per stage
constexpr uint32_t kGIdesc = idesc_e4m3_f32(2 * GBM, GBN);  // pair MMA: M = 256, N = 128

// Each scaler warp prefetches, two groups ahead, its columns of the row sums
// R[j] into a ring of kRSlots rows, and each tile's s_w into a ring of kWSlots
// rows (three, so that with one group per tile the copy two tiles ahead does
// not land on the row in use).
constexpr int kRSlots = 3;
constexpr int kWSlots = 3;
constexpr int kScRowBytes = kGScCols * 4;
constexpr int kScBytes = (kRSlots + kWSlots) * kScRowBytes;  // per scaler warp

// Shared memory: B stages, the scalers' rows, barriers (full/empty per stage,
// partial full/empty per buffer), misc. The request is padded so that one CTA
// holds an SM: the pair allocates all 512 TMEM columns.
constexpr int kGOffSc = kGStages * kGBStage;
constexpr int kGOffBars = kGOffSc + kGScWarps * kScBytes;
constexpr int kGNumBars = 2 * kGStages + 4;
constexpr int kGOffMisc = kGOffBars + kGNumBars * 8;
constexpr int kGUsed = kGOffMisc + 64 + 1024;
constexpr int kGBytes = kGUsed < 120 * 1024 ? 120 * 1024 : kGUsed;

struct GroupParams {
  const uint8_t* a_codes;  // tiled [ceil(T/32)*32][K/2], unsigned codes
  const uint8_t* w_codes;  // tiled [ceil(N/32)*32][K/2]
  const float* a_scale;    // [T][Gq]
  const float* a_zero;     // [T][Gq]
  const float* w_scale;    // [N]
  const float* gsum;       // [Gq][N]
  void* out;
  int64_t ldo;
  int* status;
  int T, N, K, Gq;
  int m_pairs, n_tiles;
  int t_blocks, n_blocks;
  int kchunks;  // K / 32
};

__device__ __forceinline__ void load_group_kt(const uint8_t* blk, int kchunks, int kt, uint4 (&v)[kGChunks]) {
#pragma unroll
  for (int j = 0; j < kGChunks; ++j) {
    const int c = kt * kGChunks + j;
    if (blk != nullptr && c < kchunks)
      v[j] = ldg_stream(blk + c * 512);
    else
      v[j] = make_uint4(0u, 0u, 0u, 0u);
  }
}

// Eight activation codes u (nibbles) minus a zero-point zc in [0, 15], as eight
// E4M3 bytes of (u - zc) * 2^-9 in widen_act's order: sign at bit 7, |u - zc|
// in bits 0-3 (exact, like the plain codes). c4 = 0x80808080 - zc * 0x01010101,
// z4 = zc * 0x01010101. Byte-wise, u + c4 = 0x80 + u - zc never borrows from
// the next byte, and its bit 7 is clear exactly when u < zc.
__device__ __forceinline__ void widen_act_zp(uint32_t w, uint32_t c4, uint32_t z4, uint32_t& lo, uint32_t& hi) {
  const uint32_t u0 = w & 0x0F0F0F0Fu, u1 = (w >> 4) & 0x0F0F0F0Fu;
  lo = (~(u0 + c4) & 0x80808080u) | __vabsdiffu4(u0, z4);
  hi = (~(u1 + c4) & 0x80808080u) | __vabsdiffu4(u1, z4);
}

// Two 64-bit shared-memory words (four floats as two packed pairs).
__device__ __forceinline__ void lds_2x64(uint32_t addr, uint64_t& a, uint64_t& b) {
  asm volatile("ld.shared.v2.b64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "r"(addr) : "memory");
}

__device__ __forceinline__ void cp_async4(uint32_t dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit_group() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait_groups() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Copies row[n0 .. n0 + kGScCols) (entries past N skipped) into shared memory
// at dst: lanes 0-15 four entries each.
__device__ __forceinline__ void copy_cols(uint32_t dst, const float* row, int n0, int N, int lane) {
  if (lane < kGScCols / 4) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int n = n0 + 4 * lane + i;
      if (n < N) cp_async4(dst + (4 * lane + i) * 4, row + n);
    }
  }
}

// Persistent pair kernel over pair tiles (m_pair * n_tiles + n_tile), cluster c
// taking tiles c, c + clusters, ... The global k-tile counter j runs across
// tiles: operand stage j mod 6, partial buffer j mod 2.
template <int OUT>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGThreads, 1)
    w4a4_group_gemm_kernel(const GroupParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* smem = smem_raw + (base - raw);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const int cluster = blockIdx.x >> 1;
  const int clusters = gridDim.x >> 1;
  const int nk = p.Gq;
  const int num_tiles = p.m_pairs * p.n_tiles;

  const uint32_t bar0 = base + kGOffBars;
  auto full = [&](int s) { return bar0 + 8u * s; };                  // leader: operands of stage s ready
  auto empty = [&](int s) { return bar0 + 8u * (kGStages + s); };    // both: stage s consumed
  auto pfull = [&](int b) { return bar0 + 8u * (2 * kGStages + b); };      // both: partial b written
  auto pempty = [&](int b) { return bar0 + 8u * (2 * kGStages + 2 + b); }; // leader: partial b read
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kGOffMisc);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + kGOffMisc + 16);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kGStages; ++s) {
      mbar_init(full(s), 2 * kGArrivals);
      mbar_init(empty(s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(pfull(b), 1);
      mbar_init(pempty(b), 2 * kGScWarps);
    }
    *abort = 0;
    mbar_fence_init();
  }
  if (warp == 0) {
    tmem_alloc2(smem_u32(tmem_slot), kGTmemCols);
    tmem_relinquish2();
  }
  tc_fence_before();
  cluster_sync();  // barriers initialised and TMEM allocated in both CTAs
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  griddep_wait();
  griddep_launch_dependents();
  uint32_t mma_groups = 0;

  if (warp == 0) {
    // ---------------- MMA issuer (leader CTA) ----------------
    if (rank == 0 && lane == 0) {
      int s = 0, phase = 0;
      uint32_t j = 0;
      for (int tile = cluster; tile < num_tiles && !*abort; tile += clusters) {
        bool ok = true;
        for (int kt = 0; kt < nk; ++kt, ++j) {
          const uint32_t b = j & 1u, use = j >> 1;
          if (!wait_cluster(pempty(b), (use & 1u) ^ 1u, abort) || !wait_cluster(full(s), phase, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t b_addr = base + s * kGBStage;
#pragma unroll
          for (int kk = 0; kk < GBK / 32; ++kk)
            mma2_ts(tmem + kPCol0 + b * GBN, tmem + kGACol0 + s * kGAColsPerStage + 8 * kk,
                    smem_desc_sw128(b_addr + 32 * kk), kGIdesc, kk != 0 ? 1u : 0u);
          mma2_commit_both(empty(s));
          mma2_commit_both(pfull(b));
          mma_groups = j + 1;
          if (++s == kGStages) {
            s = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
      }
    }
  } else if (warp < kGFirstSc) {
    // ---------------- converters: packed codes -> E4M3 operands ----------------
    // One warp per 32-row group converts every k-tile, with kGRing k-tiles of
    // loads in flight (a register ring), which covers the load latency over
    // three MMA k-tiles.
    const bool is_a = warp < kGFirstB;
    const int quarter = warp & 3;
    const int wb = warp - kGFirstB;
    const uint32_t full_l = leader_addr(full(0));
    const uint8_t* codes = is_a ? p.a_codes : p.w_codes;
    const int rb_count = is_a ? p.t_blocks : p.n_blocks;
    auto block_ptr = [&](int tile) -> const uint8_t* {
      const int rb = is_a ? ((tile / p.n_tiles) * 2 * GBM + static_cast<int>(rank) * GBM + quarter * 32) >> 5
                          : ((tile % p.n_tiles) * GBN + static_cast<int>(rank) * GBNH + wb * 32) >> 5;
      return rb < rb_count ? codes + static_cast<int64_t>(rb) * p.kchunks * 512 + lane * 16 : nullptr;
    };
    auto advance = [&](int& tile, int& kt) {
      if (++kt == nk) {
        kt = 0;
        tile += clusters;
      }
    };
    // A warps: this lane's row's zero-point of each loaded k-tile (group),
    // clamped to [0, 15], to subtract in the operand.
    auto load_zc = [&](int tile, int kt) -> uint32_t {
      const int t = (tile / p.n_tiles) * 2 * GBM + static_cast<int>(rank) * GBM + quarter * 32 + lane;
      const float z = t < p.T ? __ldg(p.a_zero + static_cast<int64_t>(t) * p.Gq + kt) : 0.f;
      return static_cast<uint32_t>(fminf(fmaxf(z, 0.f), 15.f));
    };
    uint4 ring[kGRing][kGChunks];
    uint32_t zring[kGRing];
    int ld_tile = cluster, ld_kt = 0;
    int blk_tile = ld_tile;
    const uint8_t* blk = block_ptr(ld_tile);
#pragma unroll
    for (int r = 0; r < kGRing; ++r) {
      zring[r] = 0u;
      if (ld_tile < num_tiles) {
        if (ld_tile != blk_tile) {
          blk_tile = ld_tile;
          blk = block_ptr(ld_tile);
        }
        load_group_kt(blk, p.kchunks, ld_kt, ring[r]);
        if (is_a) zring[r] = load_zc(ld_tile, ld_kt);
      }
      advance(ld_tile, ld_kt);
    }
    int tile = cluster, kt = 0, s = 0, phase = 0;
    bool run = true;
    while (run) {
#pragma unroll
      for (int r = 0; r < kGRing; ++r) {
        if (tile >= num_tiles) {
          run = false;
          break;
        }
        if (!__all_sync(0xFFFFFFFFu, wait_cluster(empty(s), phase ^ 1, abort))) {
          run = false;
          break;
        }
        if (is_a) {
          tc_fence_after();
          const uint32_t z4 = zring[r] * 0x01010101u, c4 = 0x80808080u - z4;
          uint32_t f8[32];
#pragma unroll
          for (int c = 0; c < kGChunks; ++c) {
            widen_act_zp(ring[r][c].x, c4, z4, f8[8 * c + 0], f8[8 * c + 1]);
            widen_act_zp(ring[r][c].y, c4, z4, f8[8 * c + 2], f8[8 * c + 3]);
            widen_act_zp(ring[r][c].z, c4, z4, f8[8 * c + 4], f8[8 * c + 5]);
            widen_act_zp(ring[r][c].w, c4, z4, f8[8 * c + 6], f8[8 * c + 7]);
          }
          tmem_st_32cols(tmem + (static_cast<uint32_t>(quarter * 32) << 16) + kGACol0 + s * kGAColsPerStage, f8);
          tmem_st_wait();
          tc_fence_before();
        } else {
          const int rr = wb * 32 + lane;
          const uint32_t st = base + s * kGBStage + rr * 128;
#pragma unroll
          for (int c = 0; c < kGChunks; ++c) {
            uint32_t a0, a1, a2, a3, b0, b1, b2, b3;
            widen_weight(ring[r][c].x, a0, a1);
            widen_weight(ring[r][c].y, a2, a3);
            widen_weight(ring[r][c].z, b0, b1);
            widen_weight(ring[r][c].w, b2, b3);
            sts128(st + (((2 * c) ^ (rr & 7)) << 4), a0, a1, a2, a3);
            sts128(st + (((2 * c + 1) ^ (rr & 7)) << 4), b0, b1, b2, b3);
          }
          fence_proxy_async_smem();
        }
        __syncwarp();
        if (lane == 0) arrive_cluster(full_l + 8u * s);
        // Refill this ring slot kGRing k-tiles ahead.
        if (ld_tile < num_tiles) {
          if (ld_tile != blk_tile) {
            blk_tile = ld_tile;
            blk = block_ptr(ld_tile);
          }
          load_group_kt(blk, p.kchunks, ld_kt, ring[r]);
          if (is_a) zring[r] = load_zc(ld_tile, ld_kt);
        }
        advance(ld_tile, ld_kt);
        advance(tile, kt);
        if (++s == kGStages) {
          s = 0;
          phase ^= 1;
        }
      }
    }
  } else {
    // ---------------- scalers and epilogue ----------------
    const int sw = warp - kGFirstSc;
    const int quarter = warp & 3;
    const int c0 = (sw >> 2) * kGScCols;  // this warp's first column of the tile
    const int rl = quarter * 32 + lane;   // TMEM lane = row within the CTA
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16) + c0;
    const uint32_t pempty_l = leader_addr(pempty(0));
    const uint32_t rbuf = base + kGOffSc + sw * kScBytes;  // kRSlots rows of R, then kWSlots rows of s_w
    const uint32_t wbuf = rbuf + kRSlots * kScRowBytes;
    // Prefetch position: two groups ahead of the one being scaled.
    int pf_tile = cluster, pf_kt = 0, pf_slot = 0, pf_wslot = 0;
    auto prefetch = [&]() {
      if (pf_tile < num_tiles) {
        const int n0 = (pf_tile % p.n_tiles) * GBN + c0;
        copy_cols(rbuf + pf_slot * kScRowBytes, p.gsum + static_cast<int64_t>(pf_kt) * p.N, n0, p.N, lane);
        if (pf_kt == 0) copy_cols(wbuf + pf_wslot * kScRowBytes, p.w_scale, n0, p.N, lane);
      }
      cp_async_commit_group();
      if (++pf_slot == kRSlots) pf_slot = 0;
      if (++pf_kt == nk) {
        pf_kt = 0;
        pf_tile += clusters;
        if (++pf_wslot == kWSlots) pf_wslot = 0;
      }
    };
    prefetch();
    prefetch();
    uint32_t j = 0;
    int slot = 0, wslot = 0;
    bool ok = true;
    for (int tile = cluster; tile < num_tiles && ok; tile += clusters, wslot = wslot + 1 == kWSlots ? 0 : wslot + 1) {
      const int t = (tile / p.n_tiles) * 2 * GBM + static_cast<int>(rank) * GBM + rl;
      const int n0 = (tile % p.n_tiles) * GBN + c0;
      const bool row_ok = t < p.T;
      const float* srow = p.a_scale + static_cast<int64_t>(row_ok ? t : 0) * p.Gq;
      const float* zrow = p.a_zero + static_cast<int64_t>(row_ok ? t : 0) * p.Gq;
      uint64_t S2[kGScCols / 2];  // running sums of this row's columns c0 .. c0 + kGScCols, packed in pairs
      // This row's scale and zero-point of the group being scaled, loaded one group ahead.
      float s_next = row_ok ? __ldg(srow) : 0.f, z_next = row_ok ? __ldg(zrow) : 0.f;
      for (int kt = 0; kt < nk; ++kt, ++j) {
        const uint32_t b = j & 1u, use = j >> 1;
        const bool last = kt == nk - 1;
        // The accumulator holds (P - zc R) * 2^-18: the A operand already carries
        // u - zc with zc = clamp(z, 0, 15), and each E4M3 operand 2^-9. What is
        // left of the zero-point, (z - zc) R, is nonzero only for a group that
        // does not straddle zero; a warp with such a row adds it here:
        // d' = acc - (z - zc) R 2^-18 and s 2^18 d' = s (P - z R), all exact.
        const float sg = s_next * 262144.0f;
        const float dz = z_next - fminf(fmaxf(z_next, 0.f), 15.f);
        const float nz = dz * -3.814697265625e-06f;
        const bool fix = __any_sync(0xFFFFFFFFu, dz != 0.f);
        if (row_ok && kt + 1 < nk) {
          s_next = __ldg(srow + kt + 1);
          z_next = __ldg(zrow + kt + 1);
        }
        __syncwarp();  // every lane is done with the ring slot the next copy overwrites
        prefetch();
        if (last)
          cp_async_wait_groups<0>();  // this tile's s_w as well
        else
          cp_async_wait_groups<2>();  // R of this group has landed (own copies)
        __syncwarp();                 // ... and the other lanes' copies are visible
        ok = __all_sync(0xFFFFFFFFu, wait_cluster(pfull(b), use & 1u, abort));
        if (!ok) break;
        tc_fence_after();
        const uint32_t rrow = rbuf + slot * kScRowBytes;
        const uint32_t wrow = wbuf + wslot * kScRowBytes;
        const uint64_t SG = pack2(sg, sg), NZ = pack2(nz, nz);
#pragma unroll
        for (int c = 0; c < kGScCols / 32; ++c) {
          uint32_t pv[32];
          tmem_ld_32cols(lane_base + kPCol0 + b * GBN + c * 32, pv);
          tmem_ld_wait();
          if (c == kGScCols / 32 - 1) {
            // The partial is in registers: its buffer may take the group after next.
            tc_fence_before();
            __syncwarp();
            if (lane == 0) arrive_cluster(pempty_l + 8u * b);
          }
          if (fix) {
            // The zero-point's remainder, in place: d = fma(-(z - zc) 2^-18, R, acc).
#pragma unroll
            for (int q4 = 0; q4 < 8; ++q4) {
              uint64_t r01, r23;
              lds_2x64(rrow + (c * 32 + 4 * q4) * 4, r01, r23);
              float f0, f1, f2, f3;
              unpack2(fma2v(NZ, r01, pack2(__uint_as_float(pv[4 * q4]), __uint_as_float(pv[4 * q4 + 1]))), f0, f1);
              unpack2(fma2v(NZ, r23, pack2(__uint_as_float(pv[4 * q4 + 2]), __uint_as_float(pv[4 * q4 + 3]))), f2, f3);
              pv[4 * q4] = __float_as_uint(f0);
              pv[4 * q4 + 1] = __float_as_uint(f1);
              pv[4 * q4 + 2] = __float_as_uint(f2);
              pv[4 * q4 + 3] = __float_as_uint(f3);
            }
          }
#pragma unroll
          for (int q4 = 0; q4 < 8; ++q4) {
            const uint64_t d0 = pack2(__uint_as_float(pv[4 * q4]), __uint_as_float(pv[4 * q4 + 1]));
            const uint64_t d1 = pack2(__uint_as_float(pv[4 * q4 + 2]), __uint_as_float(pv[4 * q4 + 3]));
            uint64_t& a0 = S2[c * 16 + 2 * q4];
            uint64_t& a1 = S2[c * 16 + 2 * q4 + 1];
            if (kt == 0) {
              a0 = mul2v(SG, d0);
              a1 = mul2v(SG, d1);
            } else {
              a0 = fma2v(SG, d0, a0);
              a1 = fma2v(SG, d1, a1);
            }
          }
          const int nc = n0 + c * 32;
          if (last && row_ok && nc < p.N) {
            float y[32];
#pragma unroll
            for (int q4 = 0; q4 < 8; ++q4) {
              uint64_t w01, w23;
              lds_2x64(wrow + (c * 32 + 4 * q4) * 4, w01, w23);
              unpack2(mul2v(w01, S2[c * 16 + 2 * q4]), y[4 * q4], y[4 * q4 + 1]);
              unpack2(mul2v(w23, S2[c * 16 + 2 * q4 + 1]), y[4 * q4 + 2], y[4 * q4 + 3]);
            }
            const int nvalid = p.N - nc < 32 ? p.N - nc : 32;
            store_out<OUT, 32>(p.out, static_cast<int64_t>(t) * p.ldo + nc, y, nvalid);
          }
        }
        if (++slot == kRSlots) slot = 0;
      }
    }
    cp_async_wait_groups<0>();  // no copy into shared memory outlives the CTA
  }

  // ---------------- teardown ----------------
  if (*abort && warp == 0 && lane == 0 && rank == 0 && mma_groups > 0) {
    // Let the MMAs already issued finish before tensor memory is released.
    const uint32_t last = mma_groups - 1;
    wait_teardown(pfull(last & 1u), (last >> 1) & 1u);
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc2(tmem, kGTmemCols);
  }
  if (threadIdx.x == 0 && *abort && p.status != nullptr) atomicExch(p.status, kErrTimeout);
}

int group_num_sms() {
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
int launch_group_gemm(const GroupParams& p, cudaStream_t s) {
  auto kern = w4a4_group_gemm_kernel<OUT>;
  if (!smem_optin<w4a4_group_gemm_kernel<OUT>>(kGBytes)) return OFFQ_ERR_CUDA;
  const int sms = group_num_sms();
  if (sms < 2) return OFFQ_ERR_CUDA;
  const int tiles = p.m_pairs * p.n_tiles;
  const int clusters = tiles < sms / 2 ? tiles : sms / 2;
  return launch_pdl(kern, dim3(2 * clusters), dim3(kGThreads), kGBytes, s, p);
}

}  // namespace

extern "C" int offq_w4a4_linear_group(const uint8_t* a_codes, const float* a_scale, const float* a_zero, int64_t T,
                                      int64_t N, int64_t K, int32_t group, const uint8_t* w_codes,
                                      const float* w_scale, const float* w_groupsum, void* out, int out_dtype,
                                      int64_t ldo, void* stream) {
  const int ob = elem_bytes(out_dtype);
  if (ob == 0 || T < 0 || N < 1 || K <= 0 || ldo < N) return OFFQ_ERR_INVALID_ARG;
  if (group != kGroup) return group > 0 ? OFFQ_ERR_UNSUPPORTED : OFFQ_ERR_INVALID_ARG;
  if (K % kGroup != 0) return OFFQ_ERR_INVALID_ARG;
  if (K > kMaxGemmK || T > 0x3FFFFFFF || N > 0x3FFFFFFF) return OFFQ_ERR_UNSUPPORTED;
  if (T == 0) return OFFQ_OK;
  if (a_codes == nullptr || a_scale == nullptr || a_zero == nullptr || w_codes == nullptr || w_scale == nullptr ||
      w_groupsum == nullptr || out == nullptr)
    return OFFQ_ERR_INVALID_ARG;
  if (!aligned(a_codes, 16) || !aligned(w_codes, 16) || !aligned(out, 16) || (ldo * ob) % 16 != 0 ||
      !aligned(a_scale, 4) || !aligned(a_zero, 4) || !aligned(w_scale, 4) || !aligned(w_groupsum, 4))
    return OFFQ_ERR_MISALIGNED;
  GroupParams p{};
  p.a_codes = a_codes;
  p.w_codes = w_codes;
  p.a_scale = a_scale;
  p.a_zero = a_zero;
  p.w_scale = w_scale;
  p.gsum = w_groupsum;
  p.out = out;
  p.ldo = ldo;
  p.status = device_status_ptr();
  p.T = static_cast<int>(T);
  p.N = static_cast<int>(N);
  p.K = static_cast<int>(K);
  p.Gq = static_cast<int>(K / kGroup);
  p.m_pairs = static_cast<int>((T + 2 * GBM - 1) / (2 * GBM));
  p.n_tiles = static_cast<int>((N + GBN - 1) / GBN);
  p.t_blocks = static_cast<int>((T + 31) / 32);
  p.n_blocks = static_cast<int>((N + 31) / 32);
  p.kchunks = static_cast<int>(K / 32);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  switch (out_dtype) {
    case OFFQ_F32: return launch_group_gemm<OFFQ_F32>(p, s);
    case OFFQ_BF16: return launch_group_gemm<OFFQ_BF16>(p, s);
    case OFFQ_F16: return launch_group_gemm<OFFQ_F16>(p, s);
    default: return OFFQ_ERR_INVALID_ARG;
  }
}
