// bands.cu -- Q_eps fused with the band digests of the quantized rows
// (Sec. 3.2, layer L1: quantize each coordinate, divide the vector into bands
// and hash each band; records sharing a band digest are candidates;
// Algorithm 1: B <- BandHash(Q_eps(e_j))).
//
// One pass over x: each thread takes whole bands of r consecutive values of a
// row, quantizes them exactly as the quantize kernels do (the IEEE-rounded
// quotient by s = 2 eps, round half to even), writes the codes (optional) and the 64-bit
// FNV-1a digest of the band: the band's index within its row as 2
// little-endian bytes, then the band's codes as their `width` little-endian
// bytes.  The range is tracked for the width decision, as in Q_eps alone.
#include "lam_internal.cuh"

#include <map>
#include <mutex>

namespace lam {

namespace {

constexpr int kThreads = 256;
constexpr int kBlocksPerSm = 8;
constexpr uint64_t kFnvOffset = 14695981039346656037ULL;
constexpr uint64_t kFnvPrime = 1099511628211ULL;


__device__ __forceinline__ uint64_t fnv_byte(uint64_t h, uint32_t byte) {
  return (h ^ (uint64_t)(byte & 0xffu)) * kFnvPrime;
}
// The digest state after a band's index (its two little-endian bytes): the
// same for band b of every row, so a block tabulates it once per launch for
// rows of up to kTab bands (8 KB of shared memory) instead of two 64-bit
// multiplies per band.
constexpr int kTab = 1024;
__device__ __forceinline__ uint64_t band_prefix(uint32_t b) {
  return fnv_byte(fnv_byte(kFnvOffset, b), b >> 8);
}
// Fills tab[0, nb) (every thread of the block calls this); the table, or
// nullptr when rows have more than kTab bands.
__device__ __forceinline__ const uint64_t *fill_prefix(uint64_t *tab, int nb) {
  if (nb > kTab) return nullptr;
  for (int i = threadIdx.x; i < nb; i += blockDim.x) tab[i] = band_prefix((uint32_t)i);
  __syncthreads();
  return tab;
}

// Running range of the finite inputs; non-finite inputs raise a flag.
struct BRange {
  float vmin = INFINITY, vmax = -INFINITY;
  uint32_t nonfinite = 0;
  __device__ __forceinline__ void add(float x) {
    if (fabsf(x) <= 3.402823466e38f) {
      vmin = fminf(vmin, x);
      vmax = fmaxf(vmax, x);
    } else {
      nonfinite = 1;
    }
  }
  // Block reduction into thread 0 (every thread of the block calls this).
  __device__ __forceinline__ void block_reduce() {
    __shared__ float s_min[kThreads / 32], s_max[kThreads / 32];
    __shared__ uint32_t s_nf[kThreads / 32];
    for (int off = 16; off > 0; off >>= 1) {
      vmin = fminf(vmin, __shfl_xor_sync(0xffffffffu, vmin, off));
      vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, off));
      nonfinite |= __shfl_xor_sync(0xffffffffu, nonfinite, off);
    }
    if ((threadIdx.x & 31) == 0) {
      s_min[threadIdx.x >> 5] = vmin;
      s_max[threadIdx.x >> 5] = vmax;
      s_nf[threadIdx.x >> 5] = nonfinite;
    }
    __syncthreads();
    if (threadIdx.x == 0)
      for (int i = 1; i < (int)(blockDim.x >> 5); ++i) {
        vmin = fminf(vmin, s_min[i]);
        vmax = fmaxf(vmax, s_max[i]);
        nonfinite |= s_nf[i];
      }
    __syncthreads();
  }
  // Folds the block's range into the status block (guarded atomics).
  __device__ __forceinline__ void flush(QuantStatus *st) {
    block_reduce();
    if (threadIdx.x != 0) return;
    if (vmin <= vmax) {
      const uint32_t a = ~ord_f32(vmin), b = ord_f32(vmax);
      if (a > *(volatile uint32_t *)&st->neg_min) atomicMax(&st->neg_min, a);
      if (b > *(volatile uint32_t *)&st->max) atomicMax(&st->max, b);
    }
    if (nonfinite) atomicOr(&st->flags, kFlagNonfinite);
  }
};

__device__ __forceinline__ int width_of_range(uint32_t neg_min, uint32_t mx, float s) {
  if (neg_min == 0) return 1;
  const float xmin = unord_f32(~neg_min), xmax = unord_f32(mx);
  const float rmin = rintf(__fdiv_rn(xmin, s)), rmax = rintf(__fdiv_rn(xmax, s));
  if (rmin >= -128.0f && rmax <= 127.0f) return 1;
  if (rmin >= -32768.0f && rmax <= 32767.0f) return 2;
  if (rmin >= -2147483648.0f && rmax < 2147483648.0f) return 4;
  return 0;
}

// Stores the V codes c[0..V) of positions i .. i+V-1 as one V*W-byte word
// (the caller guarantees that alignment).
template <int W, int V>
__device__ __forceinline__ void put_codes(void *codes, int64_t i, const int32_t *c) {
  if (V * W == 1) {
    reinterpret_cast<uint8_t *>(codes)[i] = (uint8_t)c[0];
  } else if (V * W == 2) {
    uint32_t u = W == 1 ? __byte_perm(c[0], c[V - 1], 0x0040) : (uint32_t)c[0];
    reinterpret_cast<uint16_t *>(codes)[i * W / 2] = (uint16_t)u;
  } else if (V * W == 4) {
    uint32_t u;
    if (W == 1) u = __byte_perm(__byte_perm(c[0], c[1 % V], 0x0040),
                                __byte_perm(c[2 % V], c[3 % V], 0x0040), 0x5410);
    else if (W == 2) u = __byte_perm(c[0], c[1 % V], 0x5410);
    else u = (uint32_t)c[0];
    reinterpret_cast<uint32_t *>(codes)[i * W / 4] = u;
  } else if (V * W == 8) {
    uint2 u;
    if (W == 2) u = make_uint2(__byte_perm(c[0], c[1 % V], 0x5410), __byte_perm(c[2 % V], c[3 % V], 0x5410));
    else u = make_uint2((uint32_t)c[0], (uint32_t)c[1 % V]);
    reinterpret_cast<uint2 *>(codes)[i * W / 8] = u;
  } else {  // V = 4, W = 4
    reinterpret_cast<uint4 *>(codes)[i / 4] =
        make_uint4((uint32_t)c[0], (uint32_t)c[1 % V], (uint32_t)c[2 % V], (uint32_t)c[3 % V]);
  }
}

// Quantizes and hashes every band of x (nbands_total = N * D / r bands, band j
// covering x[j r, j r + r)); V values per load (r a multiple of V, x 4V-byte
// aligned).  Codes are written when `codes` is not NULL.
// Bands of exactly LB loads of V values (r = LB V), U bands per thread and
// iteration (bands j, j + stride, ...): every load of the U bands is issued
// before any of them is quantized, so a thread keeps U LB loads in flight.
template <int W, int V, bool TRACK, int U, int LB>
__device__ __forceinline__ void bands_body_u(const float *__restrict__ x, int64_t nbands_total,
                                             int nb, float s, void *__restrict__ codes,
                                             uint64_t *__restrict__ digests, QuantStatus *st,
                                             const uint64_t *__restrict__ pre) {
  constexpr int r = LB * V;
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int step_b = (int)(stride % nb);  // band index advance per grid stride
  int b = (int)(tid % nb);
  const QDiv qd = QDiv::of(s);
  BRange rg;
  for (int64_t j0 = tid; j0 < nbands_total; j0 += (int64_t)U * stride) {
    float f[U][r];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t j = j0 + (int64_t)u * stride;
#pragma unroll
      for (int l = 0; l < LB; ++l) {
        const int64_t i = j * r + l * V;
        if (j < nbands_total) {
          if (V == 4) {
            const float4 t = __ldg(reinterpret_cast<const float4 *>(x + i));
            f[u][l * V] = t.x;
            f[u][(l * V + 1) % r] = t.y;
            f[u][(l * V + 2) % r] = t.z;
            f[u][(l * V + 3) % r] = t.w;
          } else if (V == 2) {
            const float2 t = __ldg(reinterpret_cast<const float2 *>(x + i));
            f[u][l * V] = t.x;
            f[u][(l * V + 1) % r] = t.y;
          } else {
            f[u][l * V] = __ldg(x + i);
          }
        }
      }
    }
    int bu = b;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t j = j0 + (int64_t)u * stride;
      if (j < nbands_total) {
        uint64_t h = pre != nullptr ? pre[bu] : band_prefix((uint32_t)bu);
#pragma unroll
        for (int l = 0; l < LB; ++l) {
          int32_t c[V];
#pragma unroll
          for (int e = 0; e < V; ++e) {
            const float fe = f[u][l * V + e];
            if (TRACK) rg.add(fe);
            c[e] = qd.code(fe);
#pragma unroll
            for (int t = 0; t < W; ++t) h = fnv_byte(h, (uint32_t)c[e] >> (8 * t));
          }
          if (codes != nullptr) put_codes<W, V>(codes, j * r + l * V, c);
        }
        digests[j] = h;
      }
      bu += step_b;
      if (bu >= nb) bu -= nb;
    }
    b = bu;
  }
  if (TRACK) rg.flush(st);
}

template <int W, int V, bool TRACK>
__device__ __forceinline__ void bands_body(const float *__restrict__ x, int64_t nbands_total,
                                           int r, int nb, float s, void *__restrict__ codes,
                                           uint64_t *__restrict__ digests, QuantStatus *st,
                                           const uint64_t *__restrict__ pre) {
  // one load per band: four bands per thread and iteration; two loads per band:
  // two bands (measured best of 1 / 2 / 4 / 8 bands on one box: 329 and 299 us
  // for r = 4 and 8 over 361,802 x 768 values, against 373 and 322 us)
  if (r == V) return bands_body_u<W, V, TRACK, 4, 1>(x, nbands_total, nb, s, codes, digests, st, pre);
  if (r == 2 * V)
    return bands_body_u<W, V, TRACK, 2, 2>(x, nbands_total, nb, s, codes, digests, st, pre);
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int step_b = (int)(stride % nb);  // band index advance per grid stride
  int b = (int)(tid % nb);
  const QDiv qd = QDiv::of(s);
  BRange rg;
  for (int64_t j = tid; j < nbands_total; j += stride) {
    uint64_t h = pre != nullptr ? pre[b] : band_prefix((uint32_t)b);
    const int64_t base = j * r;
    for (int v = 0; v < r; v += V) {
      float f[V];
      if (V == 4) {
        const float4 t = __ldg(reinterpret_cast<const float4 *>(x + base + v));
        f[0] = t.x;
        f[1 % V] = t.y;
        f[2 % V] = t.z;
        f[3 % V] = t.w;
      } else if (V == 2) {
        const float2 t = __ldg(reinterpret_cast<const float2 *>(x + base + v));
        f[0] = t.x;
        f[1 % V] = t.y;
      } else {
        f[0] = __ldg(x + base + v);
      }
      int32_t c[V];
#pragma unroll
      for (int e = 0; e < V; ++e) {
        if (TRACK) rg.add(f[e]);
        c[e] = qd.code(f[e]);
#pragma unroll
        for (int t = 0; t < W; ++t) h = fnv_byte(h, (uint32_t)c[e] >> (8 * t));
      }
      if (codes != nullptr) put_codes<W, V>(codes, base + v, c);
    }
    digests[j] = h;
    b += step_b;
    if (b >= nb) b -= nb;
  }
  if (TRACK) rg.flush(st);
}

template <int W, int V>
__global__ void __launch_bounds__(kThreads) bands_forced_kernel(
    const float *__restrict__ x, int64_t nbands_total, int r, int nb, float s,
    void *__restrict__ codes, uint64_t *__restrict__ digests, QuantStatus *st) {
  __shared__ uint64_t s_pre[kTab];
  const uint64_t *pre = fill_prefix(s_pre, nb);
  bands_body<W, V, true>(x, nbands_total, r, nb, s, codes, digests, st, pre);
}

// AUTO width as in Q_eps alone: every block speculates the same width from
// the same 64-position sample, hashes at it while tracking the exact range;
// the last block resolves the exact width (passes = 2 asks the host for a
// second, forced pass when the sample missed a wider extreme).
constexpr int kSample = 64;

template <int V>
__global__ void __launch_bounds__(kThreads) bands_auto_kernel(
    const float *__restrict__ x, int64_t nbands_total, int r, int nb, float s,
    void *__restrict__ codes, unsigned long long codes_bytes, uint64_t *__restrict__ digests,
    QuantStatus *st) {
  __shared__ int s_ws;
  __shared__ bool s_last;
  __shared__ uint64_t s_pre[kTab];
  const uint64_t *pre = fill_prefix(s_pre, nb);
  const int64_t n = nbands_total * r;
  {
    BRange rg;
    const int64_t groups = n / 4;
    for (int j = threadIdx.x; j < kSample; j += blockDim.x) {
      const int64_t i = 4 * (int64_t)((unsigned long long)j * (unsigned long long)groups / kSample);
      for (int64_t k = i; k < i + 4 && k < n; ++k) rg.add(__ldg(x + k));
    }
    rg.block_reduce();
    if (threadIdx.x == 0)
      s_ws = rg.vmin <= rg.vmax ? width_of_range(~ord_f32(rg.vmin), ord_f32(rg.vmax), s) : 1;
    __syncthreads();
  }
  const int ws = s_ws;
  const bool fits = ws != 0 && (codes == nullptr ||
                                (unsigned long long)n * (unsigned long long)ws <= codes_bytes);
  const int wrun = fits ? ws : 4;  // a range-only pass still needs some width to run at
  void *cw = fits ? codes : nullptr;
  if (wrun == 1) bands_body<1, V, true>(x, nbands_total, r, nb, s, cw, digests, st, pre);
  else if (wrun == 2) bands_body<2, V, true>(x, nbands_total, r, nb, s, cw, digests, st, pre);
  else bands_body<4, V, true>(x, nbands_total, r, nb, s, cw, digests, st, pre);
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(&st->bar, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last || threadIdx.x != 0) return;
  __threadfence();
  const uint32_t nm = *(volatile uint32_t *)&st->neg_min, mx = *(volatile uint32_t *)&st->max;
  st->s_max = (uint32_t)ws;
  if (*(volatile uint32_t *)&st->flags & kFlagNonfinite) return;
  const int w = width_of_range(nm, mx, s);
  st->width = (uint32_t)w;
  st->passes = (fits && w == ws) ? 1u : 2u;
  if (w == 0) atomicOr(&st->flags, kFlagRange);
  else if (codes != nullptr && (unsigned long long)n * (unsigned long long)w > codes_bytes)
    atomicOr(&st->flags, kFlagWorkspace);
}

int resident_blocks(const void *kern) {
  static std::mutex mu;
  static std::map<const void *, int> cache;
  std::lock_guard<std::mutex> lk(mu);
  auto it = cache.find(kern);
  if (it != cache.end()) return it->second;
  int b = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, kern, kThreads, 0) != cudaSuccess || b < 1)
    b = 1;
  if (b > kBlocksPerSm) b = kBlocksPerSm;
  cache[kern] = b;
  return b;
}

template <typename K>
int grid_for(K kern, int64_t work, int sms) {
  int64_t blocks = (work + kThreads - 1) / kThreads;
  const int64_t cap = (int64_t)sms * resident_blocks(reinterpret_cast<const void *>(kern));
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  return (int)blocks;
}

// Widest group of values that divides r and keeps every band start aligned,
// for the fp32 loads and for the V*W-byte code stores (width w; 4 for AUTO,
// whose codes pointer is 4-byte aligned and may end at any width).
int vec_for(const float *x, const void *codes, int r, int w) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(x), c = reinterpret_cast<uintptr_t>(codes);
  if (r % 4 == 0 && (a & 15u) == 0 && (c & (uintptr_t)(4 * w - 1)) == 0) return 4;
  if (r % 2 == 0 && (a & 7u) == 0 && (c & (uintptr_t)(2 * w - 1)) == 0) return 2;
  return 1;
}

template <int W>
cudaError_t launch_forced_w(const float *x, int64_t nbt, int r, int nb, float s, void *codes,
                            uint64_t *dig, QuantStatus *st, int sms, cudaStream_t stream) {
  const int v = vec_for(x, codes, r, W);
  auto kern = v == 4 ? bands_forced_kernel<W, 4> : v == 2 ? bands_forced_kernel<W, 2>
                                                          : bands_forced_kernel<W, 1>;
  kern<<<grid_for(kern, nbt, sms), kThreads, 0, stream>>>(x, nbt, r, nb, s, codes, dig, st);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_quantize_bands(const float *x, int64_t N, int D, int r, float s,
                                  int width_req, void *codes, size_t codes_bytes,
                                  uint64_t *digests, QuantStatus *st, int sms,
                                  cudaStream_t stream) {
  const int nb = D / r;
  const int64_t nbt = N * nb;
  if (width_req == 1) return launch_forced_w<1>(x, nbt, r, nb, s, codes, digests, st, sms, stream);
  if (width_req == 2) return launch_forced_w<2>(x, nbt, r, nb, s, codes, digests, st, sms, stream);
  if (width_req == 4) return launch_forced_w<4>(x, nbt, r, nb, s, codes, digests, st, sms, stream);
  const int v = vec_for(x, codes, r, 4);
  auto kern = v == 4 ? bands_auto_kernel<4> : v == 2 ? bands_auto_kernel<2> : bands_auto_kernel<1>;
  const unsigned long long cb = codes_bytes;
  kern<<<grid_for(kern, nbt, sms), kThreads, 0, stream>>>(x, nbt, r, nb, s, codes, cb, digests, st);
  return cudaGetLastError();
}

}  // namespace lam
