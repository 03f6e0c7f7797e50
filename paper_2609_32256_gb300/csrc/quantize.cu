// quantize.cu -- Q_eps streaming kernels (Sec. 3.2, layer L1:
// Q_eps(x) = round(x / 2 eps)) and dequantisation xhat = 2 eps * code.
//
// One pass reads fp32 with 128-bit loads and writes codes with 128-bit
// stores; it is HBM-bound at (4 + width) bytes per element.  The quotient is
// the IEEE-rounded x / s (QDiv: a reciprocal and two FMA steps, equal to the
// division) and the rounding is half-to-even (__float2int_rn), the same
// operations the host uses to resolve the width.
#include "lam_internal.cuh"

#include <map>
#include <mutex>

namespace lam {

namespace {

constexpr int kThreads = 256;
constexpr int kBlocksPerSm = 8;


struct Range {
  float vmin, vmax;
  uint32_t nonfinite;
  __device__ __forceinline__ Range() : vmin(INFINITY), vmax(-INFINITY), nonfinite(0) {}
  __device__ __forceinline__ void add(float x) {
    if (fabsf(x) <= 3.402823466e38f) {
      vmin = fminf(vmin, x);
      vmax = fmaxf(vmax, x);
    } else {
      nonfinite = 1;
    }
  }
  // Block-reduce (every thread of the block calls this), then one thread
  // folds the block's range into the status block, with an atomic only where
  // it would change it: thousands of blocks otherwise queue on two words.
  __device__ __forceinline__ void flush(QuantStatus *st) { flush_to(&st->neg_min, &st->max, &st->flags); }
  // The block's range, in thread 0 (every thread of the block calls this).
  __device__ __forceinline__ void block_reduce() {
    __shared__ float s_min[kThreads / 32], s_max[kThreads / 32];
    __shared__ uint32_t s_nf[kThreads / 32];
    for (int off = 16; off > 0; off >>= 1) {
      vmin = fminf(vmin, __shfl_xor_sync(0xffffffffu, vmin, off));
      vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, off));
      nonfinite |= __shfl_xor_sync(0xffffffffu, nonfinite, off);
    }
    const int w = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) {
      s_min[w] = vmin;
      s_max[w] = vmax;
      s_nf[w] = nonfinite;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      for (int i = 1; i < (int)(blockDim.x >> 5); ++i) {
        vmin = fminf(vmin, s_min[i]);
        vmax = fmaxf(vmax, s_max[i]);
        nonfinite |= s_nf[i];
      }
    }
    __syncthreads();
  }
  __device__ __forceinline__ void flush_to(uint32_t *neg_min, uint32_t *mx, uint32_t *flags) {
    block_reduce();
    if (threadIdx.x == 0) {
      if (vmin <= vmax) {
        const uint32_t a = ~ord_f32(vmin), b = ord_f32(vmax);
        if (a > *(volatile uint32_t *)neg_min) atomicMax(neg_min, a);
        if (b > *(volatile uint32_t *)mx) atomicMax(mx, b);
      }
      if (nonfinite) atomicOr(flags, kFlagNonfinite);
    }
  }
};

template <int W>
__device__ __forceinline__ void store_code(void *codes, int64_t i, int32_t c) {
  if (W == 1) reinterpret_cast<int8_t *>(codes)[i] = static_cast<int8_t>(c);
  if (W == 2) reinterpret_cast<int16_t *>(codes)[i] = static_cast<int16_t>(c);
  if (W == 4) reinterpret_cast<int32_t *>(codes)[i] = c;
}

// Four codes of width W packed into one W*4-byte word (two's complement).
template <int W>
struct Pack4;
template <>
struct Pack4<1> {
  using T = uint32_t;
  __device__ __forceinline__ static T pack(const int32_t *c) {
    return __byte_perm(__byte_perm(c[0], c[1], 0x0040), __byte_perm(c[2], c[3], 0x0040), 0x5410);
  }
  __device__ __forceinline__ static void unpack(T u, int32_t *c) {
#pragma unroll
    for (int e = 0; e < 4; ++e) c[e] = (int32_t)(int8_t)(u >> (8 * e));
  }
};
template <>
struct Pack4<2> {
  using T = uint2;
  __device__ __forceinline__ static T pack(const int32_t *c) {
    return make_uint2(__byte_perm(c[0], c[1], 0x5410), __byte_perm(c[2], c[3], 0x5410));
  }
  __device__ __forceinline__ static void unpack(T u, int32_t *c) {
    c[0] = (int32_t)(int16_t)u.x;
    c[1] = (int32_t)(int16_t)(u.x >> 16);
    c[2] = (int32_t)(int16_t)u.y;
    c[3] = (int32_t)(int16_t)(u.y >> 16);
  }
};
template <>
struct Pack4<4> {
  using T = uint4;
  __device__ __forceinline__ static T pack(const int32_t *c) {
    return make_uint4((uint32_t)c[0], (uint32_t)c[1], (uint32_t)c[2], (uint32_t)c[3]);
  }
  __device__ __forceinline__ static void unpack(T u, int32_t *c) {
    c[0] = (int32_t)u.x;
    c[1] = (int32_t)u.y;
    c[2] = (int32_t)u.z;
    c[3] = (int32_t)u.w;
  }
};

constexpr int kUnroll = 4;  // independent 4-value groups in flight per thread

// Quantizes x[0, n) into codes of width W.  VEC: x and codes 16-byte aligned.
// Each thread takes groups of four values (one 16-byte load, one 4W-byte
// store) and a warp kUnroll * 32 consecutive groups per iteration, so every
// warp access is contiguous.
template <int W, bool TRACK, bool VEC>
__device__ __forceinline__ void quantize_body(const float *__restrict__ x, int64_t n, float s,
                                              void *__restrict__ codes, QuantStatus *st) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const QDiv qd = QDiv::of(s);
  Range rg;
  int64_t done = 0;
  if (VEC) {
    using T = typename Pack4<W>::T;
    const int64_t ng = n / 4;
    const float4 *xv = reinterpret_cast<const float4 *>(x);
    T *cv = reinterpret_cast<T *>(codes);
    // a warp takes kUnroll * 32 consecutive groups per iteration
    const int lane = threadIdx.x & 31;
    const int64_t gw = tid >> 5, nw = stride >> 5;
    for (int64_t g0 = gw * (32 * kUnroll) + lane; g0 < ng; g0 += nw * (32 * kUnroll)) {
      float4 t[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u)
        if (g0 + u * 32 < ng) t[u] = __ldg(xv + g0 + u * 32);
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t g = g0 + u * 32;
        if (g < ng) {
          const float f[4] = {t[u].x, t[u].y, t[u].z, t[u].w};
          int32_t c[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            c[e] = qd.code(f[e]);
            if (TRACK) rg.add(f[e]);
          }
          cv[g] = Pack4<W>::pack(c);
        }
      }
    }
    done = ng * 4;
  }
  for (int64_t i = done + tid; i < n; i += stride) {
    float f = x[i];
    if (TRACK) rg.add(f);
    store_code<W>(codes, i, qd.code(f));
  }
  if (TRACK) rg.flush(st);
}

// The AUTO kernel reaches each width's body through a call: inlining all
// three left it at 60 registers (4 blocks per SM) against the forced kernel's
// 48 (5 blocks), 2-5% slower.
template <int W, bool VEC>
__device__ __noinline__ void quantize_body_call(const float *__restrict__ x, int64_t n, float s,
                                                void *__restrict__ codes, QuantStatus *st) {
  quantize_body<W, true, VEC>(x, n, s, codes, st);
}

template <int W, bool VEC>
__global__ void __launch_bounds__(kThreads) quantize_forced_kernel(const float *__restrict__ x,
                                                                   int64_t n, float s,
                                                                   void *__restrict__ codes,
                                                                   QuantStatus *st) {
  quantize_body<W, true, VEC>(x, n, s, codes, st);
}

// Range pass for width resolution: min/max of the finite inputs and a
// non-finite flag (Q_eps is monotone, so the code range is Q_eps of it).
template <bool VEC>
__global__ void __launch_bounds__(kThreads) range_kernel(const float *__restrict__ x, int64_t n,
                                                         QuantStatus *st) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  Range rg;
  int64_t done = 0;
  if (VEC) {
    const int64_t nvec = n / 16;
    const float4 *xv = reinterpret_cast<const float4 *>(x);
    for (int64_t v = tid; v < nvec; v += stride) {
      float4 t[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) t[j] = __ldg(xv + v * 4 + j);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        rg.add(t[j].x);
        rg.add(t[j].y);
        rg.add(t[j].z);
        rg.add(t[j].w);
      }
    }
    done = nvec * 16;
  }
  for (int64_t i = done + tid; i < n; i += stride) rg.add(x[i]);
  rg.flush(st);
}

// Narrowest code width for the range (neg_min, mx) of the status block
// (neg_min == 0: nothing finite seen); 0 if not even int32 holds it.
__device__ __forceinline__ int width_of_range(uint32_t neg_min, uint32_t mx, float s) {
  if (neg_min == 0) return 1;
  const float xmin = unord_f32(~neg_min), xmax = unord_f32(mx);
  const float rmin = rintf(__fdiv_rn(xmin, s)), rmax = rintf(__fdiv_rn(xmax, s));
  if (rmin >= -128.0f && rmax <= 127.0f) return 1;
  if (rmin >= -32768.0f && rmax <= 32767.0f) return 2;
  if (rmin >= -2147483648.0f && rmax < 2147483648.0f) return 4;
  return 0;
}

// Narrowest-width Q_eps in one launch with no grid-wide wait.  Every block
// first takes the range of the same fixed sample of x (kSample groups of four
// values spread evenly over the array; small, because every block reads the
// same lines), so all blocks speculate the same width; each then quantizes its share at that width while tracking the exact
// range, and the last block to finish resolves the exact width.  The sample's
// range lies inside the exact one, so the guess is never too wide; when it is
// too narrow (the sample missed an extreme) the status says so (passes = 2)
// and the host quantizes again at the exact width.
constexpr int kSample = 64;

template <bool VEC>
__global__ void __launch_bounds__(kThreads) quantize_auto_kernel(
    const float *__restrict__ x, int64_t n, float s, void *__restrict__ codes,
    unsigned long long codes_bytes, QuantStatus *st) {
  __shared__ int s_ws;
  __shared__ bool s_last;
  {
    Range rg;
    const int64_t groups = n / 4;
    for (int j = threadIdx.x; j < kSample; j += blockDim.x) {
      const int64_t i = 4 * (int64_t)((unsigned long long)j * (unsigned long long)groups / kSample);
      if (VEC && i + 3 < n) {
        const float4 t = __ldg(reinterpret_cast<const float4 *>(x + i));
        rg.add(t.x);
        rg.add(t.y);
        rg.add(t.z);
        rg.add(t.w);
      } else {
        for (int64_t k = i; k < i + 4 && k < n; ++k) rg.add(x[k]);
      }
    }
    rg.block_reduce();
    if (threadIdx.x == 0)
      s_ws = rg.vmin <= rg.vmax ? width_of_range(~ord_f32(rg.vmin), ord_f32(rg.vmax), s) : 1;
    __syncthreads();
  }
  const int ws = s_ws;
  const bool write1 = codes != nullptr && ws != 0 &&
                      (unsigned long long)n * (unsigned long long)ws <= codes_bytes;
  if (write1) {
    if (ws == 1) quantize_body_call<1, VEC>(x, n, s, codes, st);
    else if (ws == 2) quantize_body_call<2, VEC>(x, n, s, codes, st);
    else quantize_body_call<4, VEC>(x, n, s, codes, st);
  } else {
    Range rg;
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = tid; i < n; i += stride) rg.add(x[i]);
    rg.flush(st);
  }
  // the block's range updates are in; count it, and let the last block resolve
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
  st->passes = (write1 && w == ws) ? 1u : 2u;
  if (w == 0) atomicOr(&st->flags, kFlagRange);
  else if (codes != nullptr && (unsigned long long)n * (unsigned long long)w > codes_bytes)
    atomicOr(&st->flags, kFlagWorkspace);
}

template <int W, bool VEC>
__device__ __forceinline__ void dequantize_body(const void *__restrict__ codes, int64_t n, float s,
                                                float *__restrict__ out) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t done = 0;
  if (VEC) {
    using T = typename Pack4<W>::T;
    const int64_t ng = n / 4;
    const T *cv = reinterpret_cast<const T *>(codes);
    float4 *ov = reinterpret_cast<float4 *>(out);
    // a warp takes kUnroll * 32 consecutive groups per iteration
    const int lane = threadIdx.x & 31;
    const int64_t gw = tid >> 5, nw = stride >> 5;
    for (int64_t g0 = gw * (32 * kUnroll) + lane; g0 < ng; g0 += nw * (32 * kUnroll)) {
      T u4[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u)
        if (g0 + u * 32 < ng) u4[u] = __ldg(cv + g0 + u * 32);
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t g = g0 + u * 32;
        if (g < ng) {
          int32_t c[4];
          Pack4<W>::unpack(u4[u], c);
          ov[g] = make_float4(__fmul_rn(s, (float)c[0]), __fmul_rn(s, (float)c[1]),
                              __fmul_rn(s, (float)c[2]), __fmul_rn(s, (float)c[3]));
        }
      }
    }
    done = ng * 4;
  }
  for (int64_t i = done + tid; i < n; i += stride) {
    int32_t c;
    if (W == 1) c = reinterpret_cast<const int8_t *>(codes)[i];
    else if (W == 2) c = reinterpret_cast<const int16_t *>(codes)[i];
    else c = reinterpret_cast<const int32_t *>(codes)[i];
    out[i] = __fmul_rn(s, (float)c);
  }
}

template <int W, bool VEC>
__global__ void __launch_bounds__(kThreads) dequantize_kernel(const void *__restrict__ codes,
                                                              int64_t n, float s,
                                                              float *__restrict__ out) {
  dequantize_body<W, VEC>(codes, n, s, out);
}

// Status-driven forms (lam_quantize_async and its consumers): the width comes
// from the quantize status block on the device, so no host round trip sits
// between quantizing and using the codes.
template <bool VEC>
__global__ void __launch_bounds__(kThreads) dequantize_from_kernel(const void *__restrict__ codes,
                                                                   int64_t n, float s,
                                                                   const QuantStatus *st,
                                                                   float *__restrict__ out) {
  if (!status_ok(st)) return;
  const uint32_t w = status_width(st);
  if (w == 1) dequantize_body<1, VEC>(codes, n, s, out);
  else if (w == 2) dequantize_body<2, VEC>(codes, n, s, out);
  else if (w == 4) dequantize_body<4, VEC>(codes, n, s, out);
}

// Settles an asynchronous quantization on the device.  Forced width: one
// thread records the width and flags a range error when the exact range
// needs a wider type.  AUTO:
// the AUTO kernel resolved the width; when its speculation was too narrow
// (passes == 2) every block quantizes again at the resolved width.
template <bool VEC>
__global__ void __launch_bounds__(kThreads) quantize_settle_kernel(
    const float *__restrict__ x, int64_t n, float s, void *__restrict__ codes,
    unsigned long long codes_bytes, int width_req, QuantStatus *st) {
  if (n == 0) {  // nothing was quantized: the width alone
    if (blockIdx.x == 0 && threadIdx.x == 0)
      st->width = width_req != LAM_WIDTH_AUTO ? (uint32_t)width_req : 1u;
    return;
  }
  // (the block is read as the earlier kernels left it: in AUTO mode the
  // second pass only re-adds the same range, in forced mode one thread reads
  // and writes it)
  const uint32_t f = width_req == LAM_WIDTH_AUTO ? __ldg(&st->flags)
                                                 : *(volatile const uint32_t *)&st->flags;
  if (width_req != LAM_WIDTH_AUTO) {
    if (blockIdx.x == 0 && threadIdx.x == 0) st->width = (uint32_t)width_req;
    if (blockIdx.x == 0 && threadIdx.x == 0 && !(f & (kFlagNonfinite | kFlagTimeout))) {
      const int need = width_of_range(*(volatile const uint32_t *)&st->neg_min,
                                      *(volatile const uint32_t *)&st->max, s);
      if (need == 0 || need > width_req) atomicOr(&st->flags, kFlagRange);
    }
    return;
  }
  if (f & (kFlagNonfinite | kFlagRange | kFlagWorkspace | kFlagTimeout)) return;
  if (__ldg(&st->passes) != 2u || codes == nullptr) return;
  const uint32_t w = __ldg(&st->width);
  if ((unsigned long long)n * w > codes_bytes) return;
  if (w == 1) quantize_body<1, true, VEC>(x, n, s, codes, st);
  else if (w == 2) quantize_body<2, true, VEC>(x, n, s, codes, st);
  else if (w == 4) quantize_body<4, true, VEC>(x, n, s, codes, st);
}

// One warp per code row: exact int64 sum of squares, rounded once to fp32.
template <int W>
__global__ void __launch_bounds__(kThreads) code_sqnorms_kernel(const void *__restrict__ codes,
                                                                int64_t N, int D,
                                                                float *__restrict__ out) {
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t r = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < N;
       r += nwarps) {
    long long acc = 0;
    if (W == 1) {
      const int8_t *row = static_cast<const int8_t *>(codes) + r * (int64_t)D;
      for (int d = lane; d < D; d += 32) acc += (int)row[d] * (int)row[d];
    } else {
      const int16_t *row = static_cast<const int16_t *>(codes) + r * (int64_t)D;
      for (int d = lane; d < D; d += 32) acc += (long long)((int)row[d] * (int)row[d]);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    if (lane == 0) out[r] = __ll2float_rn(acc);
  }
}

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Resident blocks per SM of a kernel at kThreads threads (registers decide
// it), looked up once per kernel.
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

// One wave of resident blocks (or fewer, for little work): the grid-stride
// loops then split the array evenly with no second wave.
template <typename K>
int grid_for(K kern, int64_t work_items, int sms) {
  int64_t blocks = (work_items + kThreads - 1) / kThreads;
  const int64_t cap = (int64_t)sms * resident_blocks(reinterpret_cast<const void *>(kern));
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  return (int)blocks;
}

}  // namespace

cudaError_t launch_quant_range(const float *x, int64_t n, QuantStatus *status, int sms,
                               cudaStream_t st) {
  const bool vec = aligned16(x);
  auto kern = vec ? range_kernel<true> : range_kernel<false>;
  kern<<<grid_for(kern, vec ? n / 16 + 1 : n, sms), kThreads, 0, st>>>(x, n, status);
  return cudaGetLastError();
}

cudaError_t launch_quantize(const float *x, int64_t n, float s, int width_req, void *codes,
                            size_t codes_bytes, QuantStatus *status, int sms,
                            cudaStream_t st) {
  const bool vec = aligned16(x) && (codes == nullptr || aligned16(codes));
  if (width_req == LAM_WIDTH_AUTO) return cudaErrorInvalidValue;  // AUTO: launch_quantize_auto
  auto kern = width_req == 1 ? (vec ? quantize_forced_kernel<1, true> : quantize_forced_kernel<1, false>)
              : width_req == 2 ? (vec ? quantize_forced_kernel<2, true> : quantize_forced_kernel<2, false>)
                               : (vec ? quantize_forced_kernel<4, true> : quantize_forced_kernel<4, false>);
  kern<<<grid_for(kern, vec ? n / 4 + 1 : n, sms), kThreads, 0, st>>>(x, n, s, codes, status);
  return cudaGetLastError();
}

cudaError_t launch_quantize_auto(const float *x, int64_t n, float s, void *codes,
                                 size_t codes_bytes, QuantStatus *status, int sms,
                                 cudaStream_t st) {
  const bool vec = aligned16(x) && (codes == nullptr || aligned16(codes));
  auto kern = vec ? quantize_auto_kernel<true> : quantize_auto_kernel<false>;
  const unsigned long long cb = codes_bytes;
  kern<<<grid_for(kern, vec ? n / 4 + 1 : n, sms), kThreads, 0, st>>>(x, n, s, codes, cb, status);
  return cudaGetLastError();
}

cudaError_t launch_quantize_settle(const float *x, int64_t n, float s, int width_req, void *codes,
                                   size_t codes_bytes, QuantStatus *status, int sms,
                                   cudaStream_t st) {
  const bool vec = aligned16(x) && (codes == nullptr || aligned16(codes));
  auto kern = vec ? quantize_settle_kernel<true> : quantize_settle_kernel<false>;
  // (AUTO rarely needs the second pass: one block per SM keeps the idle
  // launch short and still streams when it does)
  unsigned grid = width_req == LAM_WIDTH_AUTO && n > 0 ? grid_for(kern, vec ? n / 4 + 1 : n, sms) : 1;
  if (grid > (unsigned)sms) grid = (unsigned)sms;
  if (grid < 1) grid = 1;
  kern<<<grid, kThreads, 0, st>>>(x, n, s, codes, (unsigned long long)codes_bytes, width_req,
                                  status);
  return cudaGetLastError();
}

cudaError_t launch_dequantize_from(const void *codes, const QuantStatus *status, int64_t n,
                                   float s, float *out, int sms, cudaStream_t st) {
  const bool vec = aligned16(codes) && aligned16(out);
  auto kern = vec ? dequantize_from_kernel<true> : dequantize_from_kernel<false>;
  kern<<<grid_for(kern, vec ? n / 4 + 1 : n, sms), kThreads, 0, st>>>(codes, n, s, status, out);
  return cudaGetLastError();
}

cudaError_t launch_dequantize(const void *codes, int width, int64_t n, float s, float *out,
                              int sms, cudaStream_t st) {
  const bool vec = aligned16(codes) && aligned16(out);
  auto kern = width == 1 ? (vec ? dequantize_kernel<1, true> : dequantize_kernel<1, false>)
              : width == 2 ? (vec ? dequantize_kernel<2, true> : dequantize_kernel<2, false>)
                           : (vec ? dequantize_kernel<4, true> : dequantize_kernel<4, false>);
  kern<<<grid_for(kern, vec ? n / 4 + 1 : n, sms), kThreads, 0, st>>>(codes, n, s, out);
  return cudaGetLastError();
}

cudaError_t launch_code_sqnorms(const void *codes, int width, int64_t N, int D, float *out,
                                int sms, cudaStream_t st) {
  auto kern = width == 1 ? code_sqnorms_kernel<1> : code_sqnorms_kernel<2>;
  const int g = grid_for(kern, N * 32, sms);
  kern<<<g, kThreads, 0, st>>>(codes, N, D, out);
  return cudaGetLastError();
}

}  // namespace lam
