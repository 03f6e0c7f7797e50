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

__global__ void __launch_bounds__(kSortThreads) scan_reduce_kernel(const uint32_t *in, int64_t n,
                                                                   uint32_t *block_sums) {
  const int64_t base = (int64_t)blockIdx.x * kTile + (int64_t)threadIdx.x * kSortItems;
  uint32_t s = 0;
#pragma unroll
  for (int k = 0; k < kSortItems; ++k)
    if (base + k < n) s += in[base + k];
  uint32_t tot;
  block_exclusive_scan_256(s, &tot);
  if (threadIdx.x == 0) block_sums[blockIdx.x] = tot;
}

// Single block: exclusive scan of nb block sums, in place; total to *total.
__global__ void __launch_bounds__(kScanThreads) scan_sums_kernel(uint32_t *sums, int64_t nb,
                                                                 uint32_t *total) {
  __shared__ uint32_t part[kScanThreads];
  const int64_t per = (nb + kScanThreads - 1) / kScanThreads;
  const int64_t lo = (int64_t)threadIdx.x * per, hi = lo + per < nb ? lo + per : nb;
  uint32_t s = 0;
  for (int64_t i = lo; i < hi; ++i) s += sums[i];
  part[threadIdx.x] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t run = 0;
    for (int i = 0; i < kScanThreads; ++i) {
      const uint32_t v = part[i];
      part[i] = run;
      run += v;
    }
    if (total) *total = run;
  }
  __syncthreads();
  uint32_t run = part[threadIdx.x];
  for (int64_t i = lo; i < hi; ++i) {
    const uint32_t v = sums[i];
    sums[i] = run;
    run += v;
  }
}

__global__ void __launch_bounds__(kSortThreads) scan_apply_kernel(uint32_t *data, int64_t n,
                                                                  const uint32_t *block_base) {
  const int64_t base = (int64_t)blockIdx.x * kTile + (int64_t)threadIdx.x * kSortItems;
  uint32_t v[kSortItems], s = 0;
#pragma unroll
  for (int k = 0; k < kSortItems; ++k) {
    v[k] = base + k < n ? data[base + k] : 0u;
    s += v[k];
  }
  uint32_t tot;
  uint32_t run = block_exclusive_scan_256(s, &tot) + block_base[blockIdx.x];
#pragma unroll
  for (int k = 0; k < kSortItems; ++k)
    if (base + k < n) {
      data[base + k] = run;
      run += v[k];
    }
}

// Exclusive scan of n values in place (sums: >= cdiv(n, kTile) + 1 words);
// the total goes to *total (device).
cudaError_t scan_u32(uint32_t *data, int64_t n, uint32_t *sums, uint32_t *total,
                     cudaStream_t st) {
  const int64_t nblk = cdiv(n, kTile);
  if (nblk == 0) return total ? cudaMemsetAsync(total, 0, 4, st) : cudaSuccess;
  scan_reduce_kernel<<<(unsigned)nblk, kSortThreads, 0, st>>>(data, n, sums);
  scan_sums_kernel<<<1, kScanThreads, 0, st>>>(sums, nblk, total);
  scan_apply_kernel<<<(unsigned)nblk, kSortThreads, 0, st>>>(data, n, sums);
  return cudaGetLastError();
}

}  // namespace
}  // namespace lam
