// Device helpers of the pair (cluster of 2) tensor-core GEMMs: cluster
// barriers, pair TMEM allocation and MMA issue, shared-memory and bulk-copy
// access, and the widening of packed 4-bit codes to fp8 operands.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "offq.h"
#include "offq_device.cuh"

namespace {

using namespace offq;

// Arrivals on the leader's barriers use the default (CTA-scope) release. Each
// producing thread has already completed its own writes for the consumer (the
// MMA reads them through the async proxy): fence.proxy.async after shared-memory
// stores, tcgen05.wait::st after tensor-memory stores, tcgen05.wait::ld before
// releasing the accumulator. A cluster-scope release would add a fence that
// also waits for the converters' prefetch loads still in flight.
constexpr bool kArriveClusterScope = false;

// ---------------------------------------------------------------------------
// Cluster / pair helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Address of the same shared-memory offset in the leader CTA (rank 0).
__device__ __forceinline__ uint32_t leader_addr(uint32_t local) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(0u));
  return r;
}

__device__ __forceinline__ void arrive_cluster(uint32_t cluster_addr) {
  if constexpr (kArriveClusterScope)
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
  else
    asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

__device__ __forceinline__ bool try_wait_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n"
      ".reg .pred p;\n"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
      "selp.u32 %0, 1, 0, p;\n"
      "}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool wait_cluster(uint32_t bar, uint32_t parity, volatile int* abort) {
  if (try_wait_cluster(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (try_wait_cluster(bar, parity)) return true;
    if (*abort) return false;
    if (clock64() - t0 > kWaitCycles) {
      *abort = 1;
      return false;
    }
  }
}

__device__ __forceinline__ bool wait_teardown(uint32_t bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!try_wait_cluster(bar, parity)) {
    if (clock64() - t0 > kWaitCycles) return false;
  }
  return true;
}

__device__ __forceinline__ void tmem_alloc2(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish2() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc2(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem]^T over the CTA pair, E4M3 operands, fp32 accumulate.
__device__ __forceinline__ void mma2_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n"
      ".reg .pred p;\n"
      "setp.ne.b32 p, %4, 0;\n"
      "tcgen05.mma.cta_group::2.kind::f8f6f4 [%0], [%1], %2, %3, p;\n"
      "}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrives on the barrier at this offset in both CTAs of the pair once every
// MMA issued so far by this thread is done.
__device__ __forceinline__ void mma2_commit_both(uint32_t bar) {
  const uint16_t mask = 0x3;
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
          bar),
      "h"(mask)
      : "memory");
}

__device__ __forceinline__ void tmem_st_32cols(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]),
      "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]),
      "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

// Named barrier among the epilogue warps only.
template <int kEpiWarps>
__device__ __forceinline__ void epi_sync() {
  asm volatile("bar.sync 1, %0;" ::"r"(kEpiWarps * 32) : "memory");
}

__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ uint4 ldg_stream(const uint8_t* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

// L2 eviction policies (createpolicy): evict_last for operand codes that later
// tiles read again, evict_first for outputs, which nothing in the kernel reads.
__device__ __forceinline__ uint64_t l2_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_evict_normal() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// ldg_stream with an L2 eviction policy.
__device__ __forceinline__ uint4 ldg_stream_hint(const uint8_t* p, uint64_t pol) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p), "l"(pol));
  return r;
}

// A 16-byte global store with an L2 eviction policy.
__device__ __forceinline__ void stg_hint(void* p, uint4 v, uint64_t pol) {
  asm volatile("st.global.L2::cache_hint.v4.b32 [%0], {%1,%2,%3,%4}, %5;" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w), "l"(pol)
               : "memory");
}

// Bulk copy global -> this CTA's shared memory, completing `bytes` on the
// mbarrier at `bar` (both addresses 16-byte aligned, bytes a multiple of 16).
__device__ __forceinline__ void bulk_load(uint32_t sdst, const void* gsrc, uint32_t bytes, uint32_t bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   sdst),
               "l"(gsrc), "r"(bytes), "r"(bar)
               : "memory");
}

// Bulk copy shared -> global (async proxy), tracked per thread in bulk groups,
// with an L2 eviction policy for the written lines.
__device__ __forceinline__ void bulk_store(void* gdst, uint32_t ssrc, uint32_t bytes, uint64_t pol) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group.L2::cache_hint [%0], [%1], %2, %3;" ::"l"(gdst),
               "r"(ssrc), "r"(bytes), "l"(pol)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// This thread's bulk copies have read their shared-memory source.
__device__ __forceinline__ void bulk_wait_read_all() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// This thread's bulk copies are complete.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
  uint4 r;
  asm volatile("ld.shared.v4.b32 {%0,%1,%2,%3}, [%4];" : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "r"(addr) : "memory");
  return r;
}

__device__ __forceinline__ void sts128(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
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

// E4M3 bytes of four E2M1 codes, one per byte of x (sign in bit 3, magnitude
// code in bits 0-2), with the byte table lut_lo:lut_hi (magnitude code -> E4M3
// byte of the magnitude times the block's power of two).
__device__ __forceinline__ uint32_t mx_bytes(uint32_t x, uint32_t lut_lo, uint32_t lut_hi) {
  const uint32_t m = x & 0x07070707u;
  const uint32_t t = m | (m >> 4);                  // byte 0: m0 | m1 << 4, byte 2: m2 | m3 << 4
  const uint32_t sel = __byte_perm(t, 0u, 0x0020);  // the four magnitude codes as byte selectors
  return __byte_perm(lut_lo, lut_hi, sel) | ((x & 0x08080808u) << 4);
}

// Byte table of the E2M1 magnitudes 0, .5, 1, 1.5, 2, 3, 4, 6 times 2^sh as E4M3
// (exponent field 6 + sh .. 9 + sh, sh in 0..6; zero stays zero).
__device__ __forceinline__ void mx_lut(uint32_t sh, uint32_t& lut_lo, uint32_t& lut_hi) {
  lut_lo = 0x3C383000u + sh * 0x08080800u;
  lut_hi = 0x4C484440u + sh * 0x08080808u;
}

// Eight MXFP4 codes (two per byte, even channel low) -> eight E4M3 bytes in the
// channel order of widen_act / widen_weight: [c0 c2 c4 c6 | c1 c3 c5 c7].
__device__ __forceinline__ void widen_mx(uint32_t w, uint32_t lut_lo, uint32_t lut_hi, uint32_t& lo, uint32_t& hi) {
  lo = mx_bytes(w & 0x0F0F0F0Fu, lut_lo, lut_hi);
  hi = mx_bytes((w >> 4) & 0x0F0F0F0Fu, lut_lo, lut_hi);
}

// A 16-byte store, with the L2 policy pol unless pol is 0.
__device__ __forceinline__ void stg_maybe_hint(void* p, uint4 v, uint64_t pol) {
  if (pol != 0)
    stg_hint(p, v, pol);
  else
    *reinterpret_cast<uint4*>(p) = v;
}

// Outputs of CW consecutive columns (nvalid of them inside the matrix); whole
// runs leave by 16-byte stores, with the L2 policy pol unless pol is 0.
template <int OUT, int CW>
__device__ __forceinline__ void store_out(void* out, int64_t off, const float* y, int nvalid, uint64_t pol = 0) {
  if (OUT == OFFQ_F32) {
    float* o = static_cast<float*>(out) + off;
    if (nvalid == CW) {
#pragma unroll
      for (int i = 0; i < CW / 4; ++i)
        stg_maybe_hint(o + 4 * i, make_uint4(__float_as_uint(y[4 * i]), __float_as_uint(y[4 * i + 1]),
                                             __float_as_uint(y[4 * i + 2]), __float_as_uint(y[4 * i + 3])),
                       pol);
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
        stg_maybe_hint(o + 8 * i, make_uint4(p[4 * i], p[4 * i + 1], p[4 * i + 2], p[4 * i + 3]), pol);
    } else {
#pragma unroll
      for (int i = 0; i < CW; ++i)
        if (i < nvalid) o[i] = static_cast<uint16_t>(p[i >> 1] >> (16 * (i & 1)));
    }
  }
}

}  // namespace
