// scan.cuh -- exclusive prefix sums of uint32 arrays on the device (three
// phases: per-block sums, one block scanning them, per-block scans plus
// offsets), shared by the admission and the byte-codec kernels.  Everything
// here has internal linkage: each translation unit that includes it gets its
// own copy.
#pragma once

#include "lam_internal.cuh"

namespace lam {
namespace {

constexpr int kSortThreads = 256;
constexpr int kSortItems = 16;                    // per thread
constexpr int kTile = kSortThreads * kSortItems;  // values per block
constexpr int kScanThreads = 1024;

inline int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Exclusive scan of n uint32 values (in place), totals wrapped mod 2^32 (the
// callers' totals stay below 2^32).  Three phases over blocks of kTile values.
__device__ __forceinline__ uint32_t block_exclusive_scan_256(uint32_t v, uint32_t *total) {
  __shared__ uint32_t warp_tot[kSortThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) warp_tot[warp] = x;
  __syncthreads();
  uint32_t base = 0, tot = 0;
  for (int w = 0; w < kSortThreads / 32; ++w) {
    if (w < warp) base += warp_tot[w];
    tot += warp_tot[w];
  }
  __syncthreads();
  *total = tot;
  return base + x - v;
}

// Phase 1: the sum of each block of kTile values.  VEC: the array is 16-byte
// aligned, so a thread's 16 values load as four 16-byte vectors.
template <bool VEC>
__global__ void __launch_bounds__(kSortThreads) scan_reduce_kernel(const uint32_t *in, int64_t n,
                                                                   uint32_t *block_sums) {
  const int64_t base = (int64_t)blockIdx.x * kTile + (int64_t)threadIdx.x * kSortItems;
  uint32_t s = 0;
  if (VEC && base + kSortItems <= n) {
    const uint4 *p = reinterpret_cast<const uint4 *>(in + base);
#pragma unroll
    for (int k = 0; k < kSortItems / 4; ++k) {
      const uint4 t = p[k];
      s += t.x + t.y + t.z + t.w;
    }
  } else {
#pragma unroll
    for (int k = 0; k < kSortItems; ++k)
      if (base + k < n) s += in[base + k];
  }
  uint32_t tot;
  block_exclusive_scan_256(s, &tot);
  if (threadIdx.x == 0) block_sums[blockIdx.x] = tot;
}

// Phase 2, one block: exclusive scan of the nb block sums in place (each
// thread a run of them, a warp-shuffle scan of the 1,024 runs' totals); the
// total to *total.
__global__ void __launch_bounds__(kScanThreads) scan_sums_kernel(uint32_t *sums, int64_t nb,
                                                                 uint32_t *total) {
  __shared__ uint32_t wt[kScanThreads / 32];
  const int64_t per = (nb + kScanThreads - 1) / kScanThreads;
  const int64_t lo = (int64_t)threadIdx.x * per, hi = lo + per < nb ? lo + per : nb;
  uint32_t s = 0;
  for (int64_t i = lo; i < hi; ++i) s += sums[i];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t x = s;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) wt[warp] = x;
  __syncthreads();
  if (warp == 0) {
    const uint32_t t = wt[lane];
    uint32_t u = t;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, u, off);
      if (lane >= off) u += y;
    }
    wt[lane] = u - t;
    if (lane == 31 && total) *total = u;
  }
  __syncthreads();
  uint32_t run = wt[warp] + x - s;
  for (int64_t i = lo; i < hi; ++i) {
    const uint32_t v = sums[i];
    sums[i] = run;
    run += v;
  }
}

// Phase 3: each block scans its values and adds its block's offset.
template <bool VEC>
__global__ void __launch_bounds__(kSortThreads) scan_apply_kernel(uint32_t *data, int64_t n,
                                                                  const uint32_t *block_base) {
  const int64_t base = (int64_t)blockIdx.x * kTile + (int64_t)threadIdx.x * kSortItems;
  const bool full = VEC && base + kSortItems <= n;
  uint32_t v[kSortItems], s = 0;
  if (full) {
    const uint4 *p = reinterpret_cast<const uint4 *>(data + base);
#pragma unroll
    for (int k = 0; k < kSortItems / 4; ++k) {
      const uint4 t = p[k];
      v[4 * k] = t.x;
      v[4 * k + 1] = t.y;
      v[4 * k + 2] = t.z;
      v[4 * k + 3] = t.w;
    }
  } else {
#pragma unroll
    for (int k = 0; k < kSortItems; ++k) v[k] = base + k < n ? data[base + k] : 0u;
  }
#pragma unroll
  for (int k = 0; k < kSortItems; ++k) s += v[k];
  uint32_t tot;
  uint32_t run = block_exclusive_scan_256(s, &tot) + block_base[blockIdx.x];
  uint32_t o[kSortItems];
#pragma unroll
  for (int k = 0; k < kSortItems; ++k) {
    o[k] = run;
    run += v[k];
  }
  if (full) {
    uint4 *p = reinterpret_cast<uint4 *>(data + base);
#pragma unroll
    for (int k = 0; k < kSortItems / 4; ++k)
      p[k] = make_uint4(o[4 * k], o[4 * k + 1], o[4 * k + 2], o[4 * k + 3]);
  } else {
#pragma unroll
    for (int k = 0; k < kSortItems; ++k)
      if (base + k < n) data[base + k] = o[k];
  }
}

// Exclusive scan of n values in place (sums: >= cdiv(n, kTile) + 1 words);
// the total goes to *total (device).
cudaError_t scan_u32(uint32_t *data, int64_t n, uint32_t *sums, uint32_t *total,
                     cudaStream_t st) {
  const int64_t nblk = cdiv(n, kTile);
  if (nblk == 0) return total ? cudaMemsetAsync(total, 0, 4, st) : cudaSuccess;
  const bool vec = (reinterpret_cast<uintptr_t>(data) & 15u) == 0;
  if (vec)
    scan_reduce_kernel<true><<<(unsigned)nblk, kSortThreads, 0, st>>>(data, n, sums);
  else
    scan_reduce_kernel<false><<<(unsigned)nblk, kSortThreads, 0, st>>>(data, n, sums);
  scan_sums_kernel<<<1, kScanThreads, 0, st>>>(sums, nblk, total);
  if (vec)
    scan_apply_kernel<true><<<(unsigned)nblk, kSortThreads, 0, st>>>(data, n, sums);
  else
    scan_apply_kernel<false><<<(unsigned)nblk, kSortThreads, 0, st>>>(data, n, sums);
  return cudaGetLastError();
}

}  // namespace
}  // namespace lam
