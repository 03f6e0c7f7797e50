// tc_common.cuh -- tcgen05 / tensor-memory helpers shared by the tensor-core
// scoring kernels: allocation, fences, the kind::f16 MMA with its shared-memory
// descriptor, commits, TMEM loads, bounded warp waits and the score formula
// on the raw accumulator.  Inline PTX from the public PTX ISA (sm_100a family).
#pragma once

#include "lam_internal.cuh"

namespace lam {
namespace {

// ---------------------------------------------------------- tcgen05 PTX --
__device__ __forceinline__ void tmem_alloc(uint32_t *slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// D[tmem] (+)= A[smem] * B[smem]^T, fp16 inputs, fp32 accumulate.
__device__ __forceinline__ void umma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on `bar` once every MMA this thread issued so far has completed.
__device__ __forceinline__ void umma_commit(uint64_t *bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}
// 32 consecutive fp32 columns of this warp's 32 TMEM lanes.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t *v) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]),
        "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]),
        "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
        "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]),
        "=r"(v[31])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ __half2 u32_as_h2(uint32_t u) {
  __half2 h;
  *reinterpret_cast<uint32_t *>(&h) = u;
  return h;
}
__device__ __forceinline__ uint32_t h2_as_u32(__half2 h) { return *reinterpret_cast<uint32_t *>(&h); }

// Shared-memory matrix descriptor: K-major operand, rows of 64 bytes in the
// 64-byte swizzle, 8-row groups 512 bytes apart (SBO); LBO unused.
__device__ __forceinline__ uint64_t desc_sw64(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);  // start address
  d |= (uint64_t)1 << 16;                     // leading byte offset (unused)
  d |= (uint64_t)(512 >> 4) << 32;            // stride byte offset
  d |= (uint64_t)1 << 46;                     // descriptor version
  d |= (uint64_t)4 << 61;                     // 64-byte swizzle
  return d;
}
// Instruction descriptor, kind::f16: fp32 accumulate, fp16 A and B, both
// K-major, dense, no negation; N in bits 17-22 (N / 8), M in bits 24-28 (M / 16).
__host__ __device__ constexpr uint32_t idesc_f16(int m, int n) {
  return (1u << 4) | (0u << 7) | (0u << 10) | ((uint32_t)(n >> 3) << 17) |
         ((uint32_t)(m >> 4) << 24);
}

// Warp-uniform bounded wait: lane 0 waits, the verdict is broadcast, and every
// lane then observes the completed phase itself.
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, volatile int *abort,
                                          uint32_t *gflags) {
  int ok = 0;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, abort, gflags) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  if (ok)
    while (!mbar_try_wait(bar, parity)) {
    }
  return ok != 0;
}

__device__ __forceinline__ void drain_wait_tc(uint64_t *bar, uint32_t parity) {
  long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > kWaitCycles) break;
}


// Score from the raw accumulator (2^e q.c), a per-query factor fq and a
// per-row factor rowf (written by the converters at the end of each tile):
//   inner product  fq acc                 fq = s 2^-e
//   cosine         fq acc rowf            fq = 2^-e / ||q||, rowf = 1/||c||
//   squared L2     fq acc + ||q||^2 + rowf    fq = -2 s 2^-e, rowf = s^2 ||c||^2
// (the k L2 survivors are rescored in the direct form by the merge).
__device__ __forceinline__ float tile_score(int metric, float acc, float fq, float qq,
                                            float rowf) {
  if (metric == LAM_METRIC_IP) return fq * acc;
  if (metric == LAM_METRIC_COSINE) return (fq * acc) * rowf;
  return fmaf(fq, acc, qq + rowf);
}


// v[j] for a run-time j, by a tree of selects (no local-memory indexing).
__device__ __forceinline__ uint32_t select32(const uint32_t (&v)[32], int j) {
  uint32_t t16[16], t8[8], t4[4], t2[2];
#pragma unroll
  for (int i = 0; i < 16; ++i) t16[i] = (j & 1) ? v[2 * i + 1] : v[2 * i];
#pragma unroll
  for (int i = 0; i < 8; ++i) t8[i] = (j & 2) ? t16[2 * i + 1] : t16[2 * i];
#pragma unroll
  for (int i = 0; i < 4; ++i) t4[i] = (j & 4) ? t8[2 * i + 1] : t8[2 * i];
#pragma unroll
  for (int i = 0; i < 2; ++i) t2[i] = (j & 8) ? t4[2 * i + 1] : t4[2 * i];
  return (j & 16) ? t2[1] : t2[0];
}

}  // namespace
}  // namespace lam

namespace lam {
namespace {

// MMA instruction text per CTA group: 1, this SM; 2, the CTA pair of a
// 2-CTA cluster, issued by its even CTA (M = 256 split 128 / 128 over the
// pair's accumulators, B's N rows split half / half over the pair's shared
// memories, both at the same offsets).
#define LAM_MMA1 "tcgen05.mma.cta_group::1.kind::f16 "
#define LAM_MMA2 "tcgen05.mma.cta_group::2.kind::f16 "

// Back-to-back MMAs into one accumulator, issued from one asm block.  An
// issued tcgen05.mma keeps its source registers (descriptors and the
// enable-input predicate) for about 200 cycles; an instruction that rewrites
// one of them waits for that, so a loop that recomputes a descriptor or
// re-sets the predicate before every MMA issues one MMA per ~200 cycles
// (measured on this part: 197 cycles for any M, N and operand source,
// against 64 cycles of tensor work at M = 128, N = 128).  Here every operand
// is computed before the block, only the first MMA reads the predicate
// (`accumulate`: 0 overwrites the accumulator), the others always accumulate.
// MMA i multiplies a[i] by b[i].
#define LAM_UMMA_X2(I)                                                               \
  asm volatile("{\n\t.reg .pred p;\n\t"                                              \
               "setp.ne.b32 p, %6, 0;\n\t" I "[%0], %1, %3, %5, p;\n\t" I            \
               "[%0], %2, %4, %5, 1;\n\t}" ::"r"(d),                                 \
               "l"(a[0]), "l"(a[1]), "l"(b[0]), "l"(b[1]), "r"(idesc), "r"(accumulate) \
               : "memory")
#define LAM_UMMA_X4(I)                                                                  \
  asm volatile("{\n\t.reg .pred p;\n\t"                                                 \
               "setp.ne.b32 p, %10, 0;\n\t" I "[%0], %1, %5, %9, p;\n\t" I              \
               "[%0], %2, %6, %9, 1;\n\t" I "[%0], %3, %7, %9, 1;\n\t" I                \
               "[%0], %4, %8, %9, 1;\n\t}" ::"r"(d),                                    \
               "l"(a[0]), "l"(a[1]), "l"(a[2]), "l"(a[3]), "l"(b[0]), "l"(b[1]),        \
               "l"(b[2]), "l"(b[3]), "r"(idesc), "r"(accumulate)                        \
               : "memory")
#define LAM_UMMA_X8(I)                                                                   \
  asm volatile("{\n\t.reg .pred p;\n\t"                                                  \
               "setp.ne.b32 p, %18, 0;\n\t" I "[%0], %1, %9, %17, p;\n\t" I              \
               "[%0], %2, %10, %17, 1;\n\t" I "[%0], %3, %11, %17, 1;\n\t" I             \
               "[%0], %4, %12, %17, 1;\n\t" I "[%0], %5, %13, %17, 1;\n\t" I             \
               "[%0], %6, %14, %17, 1;\n\t" I "[%0], %7, %15, %17, 1;\n\t" I             \
               "[%0], %8, %16, %17, 1;\n\t}" ::"r"(d),                                   \
               "l"(a[0]), "l"(a[1]), "l"(a[2]), "l"(a[3]), "l"(a[4]), "l"(a[5]),         \
               "l"(a[6]), "l"(a[7]), "l"(b[0]), "l"(b[1]), "l"(b[2]), "l"(b[3]),         \
               "l"(b[4]), "l"(b[5]), "l"(b[6]), "l"(b[7]), "r"(idesc), "r"(accumulate)   \
               : "memory")
template <int CG = 1>
__device__ __forceinline__ void umma_f16_x2(uint32_t d, const uint64_t (&a)[2],
                                            const uint64_t (&b)[2], uint32_t idesc,
                                            uint32_t accumulate) {
  if constexpr (CG == 2) LAM_UMMA_X2(LAM_MMA2);
  else LAM_UMMA_X2(LAM_MMA1);
}
template <int CG = 1>
__device__ __forceinline__ void umma_f16_x4(uint32_t d, const uint64_t (&a)[4],
                                            const uint64_t (&b)[4], uint32_t idesc,
                                            uint32_t accumulate) {
  if constexpr (CG == 2) LAM_UMMA_X4(LAM_MMA2);
  else LAM_UMMA_X4(LAM_MMA1);
}
template <int CG = 1>
__device__ __forceinline__ void umma_f16_x8(uint32_t d, const uint64_t (&a)[8],
                                            const uint64_t (&b)[8], uint32_t idesc,
                                            uint32_t accumulate) {
  if constexpr (CG == 2) LAM_UMMA_X8(LAM_MMA2);
  else LAM_UMMA_X8(LAM_MMA1);
}

// The MMAs of `nc` (1 or 2) 32-wide K chunks of the query-block x code-tile
// product: per chunk c and K step j (two of 16), hi * codes then (unless
// hi-only) lo * codes.  ahi / alo / bd: the chunks' operand descriptors.
template <int CG = 1>
__device__ __forceinline__ void umma_chunks(uint32_t d, int nc, const uint64_t (&ahi)[2],
                                            const uint64_t (&alo)[2], const uint64_t (&bd)[2],
                                            bool hi_only, uint32_t idesc, uint32_t accumulate) {
  constexpr uint64_t k1 = (16 * 2) >> 4;  // second K16 step: 32 bytes further
  if (hi_only) {
    if (nc == 2) {
      const uint64_t a[4] = {ahi[0], ahi[0] + k1, ahi[1], ahi[1] + k1};
      const uint64_t b[4] = {bd[0], bd[0] + k1, bd[1], bd[1] + k1};
      umma_f16_x4<CG>(d, a, b, idesc, accumulate);
    } else {
      const uint64_t a[2] = {ahi[0], ahi[0] + k1};
      const uint64_t b[2] = {bd[0], bd[0] + k1};
      umma_f16_x2<CG>(d, a, b, idesc, accumulate);
    }
  } else if (nc == 2) {
    const uint64_t a[8] = {ahi[0], alo[0], ahi[0] + k1, alo[0] + k1,
                           ahi[1], alo[1], ahi[1] + k1, alo[1] + k1};
    const uint64_t b[8] = {bd[0], bd[0], bd[0] + k1, bd[0] + k1,
                           bd[1], bd[1], bd[1] + k1, bd[1] + k1};
    umma_f16_x8<CG>(d, a, b, idesc, accumulate);
  } else {
    const uint64_t a[4] = {ahi[0], alo[0], ahi[0] + k1, alo[0] + k1};
    const uint64_t b[4] = {bd[0], bd[0], bd[0] + k1, bd[0] + k1};
    umma_f16_x4<CG>(d, a, b, idesc, accumulate);
  }
}

// ------------------------------------------- CTA pairs (cta_group::2) --
// A 2-CTA cluster whose even CTA issues M = 256 MMAs for both.  Tensor memory
// is allocated and freed collectively by one warp of each CTA; the commits of
// the issuing CTA arrive on the barrier at the same offset in each CTA of
// `mask`.  Every tcgen05 instruction of such a kernel names the pair.
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// All threads of both CTAs (also orders this CTA's threads, as __syncthreads).
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t *slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
// Arrive on `bar` in every CTA of `mask` once the pair MMAs issued so far completed.
__device__ __forceinline__ void umma_commit_pair(uint64_t *bar, uint16_t mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 "
      "[%0], %1;" ::"r"(smem_u32(bar)),
      "h"(mask)
      : "memory");
}
// Arrive (release, cluster scope) on the barrier at this barrier's offset in CTA `rank`.
__device__ __forceinline__ void mbar_arrive_peer(uint64_t *bar, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(bar)), "r"(rank));
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_cl(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(1000000u)
      : "memory");
  return ok != 0;
}
// mbar_wait for a barrier the other CTA of the pair arrives on (acquire at
// cluster scope); the same budget, abort flag and timeout report.
__device__ __forceinline__ bool mbar_wait_cl(uint64_t *bar, uint32_t parity,
                                             volatile int *abort, uint32_t *gflags) {
  long long t0 = clock64();
  long long budget = -1;
  while (true) {
    if (mbar_try_wait_cl(bar, parity)) return true;
    if (*abort) return false;
    if (budget < 0) budget = wait_budget(gflags);
    if (clock64() - t0 > budget) {
      *abort = 1;
      if (gflags) atomicOr(gflags, kFlagTimeout);
      return false;
    }
  }
}

}  // namespace
}  // namespace lam
