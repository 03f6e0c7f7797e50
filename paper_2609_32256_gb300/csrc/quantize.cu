// quantize.cu -- Q_eps streaming kernels (Sec. 3.2, layer L1:
// Q_eps(x) = round(x / 2 eps)) and dequantisation xhat = 2 eps * code.
//
// One pass reads fp32 with 128-bit loads and writes codes with 128-bit
// stores; it is HBM-bound at (4 + width) bytes per element.  The quotient is
// one IEEE division (__fdiv_rn) and the rounding is half-to-even
// (__float2int_rn), the same operations the host uses to resolve the width.
#include "lam_internal.cuh"

namespace lam {

namespace {

constexpr int kThreads = 256;
constexpr int kBlocksPerSm = 8;

__device__ __forceinline__ int32_t q_code(float x, float s) {
  return __float2int_rn(__fdiv_rn(x, s));
}

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
  // Warp-reduce, then one atomic per warp into the status block.
  __device__ __forceinline__ void flush(QuantStatus *st) {
    for (int off = 16; off > 0; off >>= 1) {
      vmin = fminf(vmin, __shfl_xor_sync(0xffffffffu, vmin, off));
      vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, off));
      nonfinite |= __shfl_xor_sync(0xffffffffu, nonfinite, off);
    }
    if ((threadIdx.x & 31) == 0) {
      if (vmin <= vmax) {
        atomicMax(&st->neg_min, ~ord_f32(vmin));
        atomicMax(&st->max, ord_f32(vmax));
      }
      if (nonfinite) atomicOr(&st->flags, kFlagNonfinite);
    }
  }
};

template <int W>
__device__ __forceinline__ void store_code(void *codes, int64_t i, int32_t c) {
  if (W == 1) reinterpret_cast<int8_t *>(codes)[i] = static_cast<int8_t>(c);
  if (W == 2) reinterpret_cast<int16_t *>(codes)[i] = static_cast<int16_t>(c);
  if (W == 4) reinterpret_cast<int32_t *>(codes)[i] = c;
}

// Packs 16/W codes into one 16-byte word (two's-complement truncation).
template <int W>
__device__ __forceinline__ uint4 pack(const int32_t *c) {
  uint4 o;
  if (W == 1) {
    uint32_t w[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      uint32_t lo = __byte_perm(c[4 * j], c[4 * j + 1], 0x0040);
      uint32_t hi = __byte_perm(c[4 * j + 2], c[4 * j + 3], 0x0040);
      w[j] = __byte_perm(lo, hi, 0x5410);
    }
    o = make_uint4(w[0], w[1], w[2], w[3]);
  } else if (W == 2) {
    o = make_uint4(__byte_perm(c[0], c[1], 0x5410), __byte_perm(c[2], c[3], 0x5410),
                   __byte_perm(c[4], c[5], 0x5410), __byte_perm(c[6], c[7], 0x5410));
  } else {
    o = make_uint4(c[0], c[1], c[2], c[3]);
  }
  return o;
}

// Quantizes x[0, n) into codes of width W.  VEC: x and codes 16-byte aligned.
template <int W, bool TRACK, bool VEC>
__device__ __forceinline__ void quantize_body(const float *__restrict__ x, int64_t n, float s,
                                              void *__restrict__ codes, QuantStatus *st) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  Range rg;
  int64_t done = 0;
  if (VEC) {
    constexpr int EPT = 16 / W;  // elements per 16-byte store
    const int64_t nvec = n / EPT;
    const float4 *xv = reinterpret_cast<const float4 *>(x);
    uint4 *cv = reinterpret_cast<uint4 *>(codes);
    for (int64_t v = tid; v < nvec; v += stride) {
      float f[EPT];
#pragma unroll
      for (int j = 0; j < EPT / 4; ++j) {
        float4 t = __ldg(xv + v * (EPT / 4) + j);
        f[4 * j] = t.x;
        f[4 * j + 1] = t.y;
        f[4 * j + 2] = t.z;
        f[4 * j + 3] = t.w;
      }
      int32_t c[EPT];
#pragma unroll
      for (int e = 0; e < EPT; ++e) {
        c[e] = q_code(f[e], s);
        if (TRACK) rg.add(f[e]);
      }
      cv[v] = pack<W>(c);
    }
    done = nvec * EPT;
  }
  for (int64_t i = done + tid; i < n; i += stride) {
    float f = x[i];
    if (TRACK) rg.add(f);
    store_code<W>(codes, i, q_code(f, s));
  }
  if (TRACK) rg.flush(st);
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

// Narrowest width from the range the range pass left in *st; 0 if not int32.
__device__ __forceinline__ int resolve_width(const QuantStatus *st, float s) {
  if (st->neg_min == 0) return 1;  // no finite value
  float xmin = unord_f32(~st->neg_min), xmax = unord_f32(st->max);
  float rmin = rintf(__fdiv_rn(xmin, s)), rmax = rintf(__fdiv_rn(xmax, s));
  if (rmin >= -128.0f && rmax <= 127.0f) return 1;
  if (rmin >= -32768.0f && rmax <= 32767.0f) return 2;
  if (rmin >= -2147483648.0f && rmax < 2147483648.0f) return 4;
  return 0;
}

template <bool VEC>
__global__ void __launch_bounds__(kThreads) quantize_auto_kernel(const float *__restrict__ x,
                                                                 int64_t n, float s,
                                                                 void *__restrict__ codes,
                                                                 unsigned long long codes_bytes,
                                                                 QuantStatus *st) {
  if (st->flags & kFlagNonfinite) return;
  const int w = resolve_width(st, s);
  const bool fits = w != 0 && (unsigned long long)n * (unsigned long long)w <= codes_bytes;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    st->width = (uint32_t)w;
    if (w == 0) atomicOr(&st->flags, kFlagRange);
    else if (codes != nullptr && !fits) atomicOr(&st->flags, kFlagWorkspace);
  }
  if (codes == nullptr || !fits) return;
  if (w == 1) quantize_body<1, false, VEC>(x, n, s, codes, st);
  else if (w == 2) quantize_body<2, false, VEC>(x, n, s, codes, st);
  else quantize_body<4, false, VEC>(x, n, s, codes, st);
}

// Bounded grid barrier for a cooperative launch (every block resident):
// block leaders count arrivals up to `target`; a wait longer than
// kWaitCycles records a timeout and lets the block go on.
__device__ __forceinline__ void grid_barrier(uint32_t *count, uint32_t target, uint32_t *flags) {
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    atomicAdd(count, 1u);
    const long long t0 = clock64();
    while (*(volatile uint32_t *)count < target) {
      if (clock64() - t0 > kWaitCycles) {
        atomicOr(flags, kFlagTimeout);
        break;
      }
      __nanosleep(64);
    }
    __threadfence();
  }
  __syncthreads();
}

__device__ __forceinline__ int width_of_range(uint32_t neg_min, uint32_t mx, float s) {
  if (neg_min == 0) return 1;
  const float xmin = unord_f32(~neg_min), xmax = unord_f32(mx);
  const float rmin = rintf(__fdiv_rn(xmin, s)), rmax = rintf(__fdiv_rn(xmax, s));
  if (rmin >= -128.0f && rmax <= 127.0f) return 1;
  if (rmin >= -32768.0f && rmax <= 32767.0f) return 2;
  if (rmin >= -2147483648.0f && rmax < 2147483648.0f) return 4;
  return 0;
}

// Narrowest-width Q_eps in one cooperative launch.  Phase 1 takes the range
// of a strided 1/64 sample and speculates the width from it; phase 2
// quantizes at that width while tracking the exact range; if the exact range
// needs a wider type (the sample missed an extreme), phase 3 quantizes again
// at the exact width.  The sample's range lies inside the exact one, so the
// speculation is never wider than needed and the result is always the
// narrowest width.
template <bool VEC>
__global__ void __launch_bounds__(kThreads) quantize_auto_coop_kernel(
    const float *__restrict__ x, int64_t n, float s, void *__restrict__ codes,
    unsigned long long codes_bytes, QuantStatus *st) {
  const uint32_t G = gridDim.x;
  {  // phase 1: sample range
    Range rg;
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t nsamp = (n + 255) / 256;  // one 4-value group per 256 values
    for (int64_t v = tid; v < nsamp; v += stride) {
      const int64_t i = v * 256;
      if (VEC && i + 3 < n) {
        const float4 t = __ldg(reinterpret_cast<const float4 *>(x + i));
        rg.add(t.x);
        rg.add(t.y);
        rg.add(t.z);
        rg.add(t.w);
      } else {
        for (int64_t j = i; j < i + 4 && j < n; ++j) rg.add(x[j]);
      }
    }
    for (int off = 16; off > 0; off >>= 1) {
      rg.vmin = fminf(rg.vmin, __shfl_xor_sync(0xffffffffu, rg.vmin, off));
      rg.vmax = fmaxf(rg.vmax, __shfl_xor_sync(0xffffffffu, rg.vmax, off));
    }
    if ((threadIdx.x & 31) == 0 && rg.vmin <= rg.vmax) {
      atomicMax(&st->s_neg_min, ~ord_f32(rg.vmin));
      atomicMax(&st->s_max, ord_f32(rg.vmax));
    }
  }
  grid_barrier(&st->bar, G, &st->flags);
  const int ws = width_of_range(*(volatile uint32_t *)&st->s_neg_min,
                                *(volatile uint32_t *)&st->s_max, s);
  const bool write1 = codes != nullptr && ws != 0 &&
                      (unsigned long long)n * (unsigned long long)ws <= codes_bytes;
  // phase 2: quantize at the speculated width, tracking the exact range
  if (write1) {
    if (ws == 1) quantize_body<1, true, VEC>(x, n, s, codes, st);
    else if (ws == 2) quantize_body<2, true, VEC>(x, n, s, codes, st);
    else quantize_body<4, true, VEC>(x, n, s, codes, st);
  } else {
    Range rg;
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = tid; i < n; i += stride) rg.add(x[i]);
    rg.flush(st);
  }
  grid_barrier(&st->bar, 2 * G, &st->flags);
  if (*(volatile uint32_t *)&st->flags & kFlagNonfinite) return;
  const int w = width_of_range(*(volatile uint32_t *)&st->neg_min, *(volatile uint32_t *)&st->max, s);
  const bool fits = w != 0 && (unsigned long long)n * (unsigned long long)w <= codes_bytes;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    st->width = (uint32_t)w;
    st->passes = (write1 && w == ws) ? 1u : 2u;
    if (w == 0) atomicOr(&st->flags, kFlagRange);
    else if (codes != nullptr && !fits) atomicOr(&st->flags, kFlagWorkspace);
  }
  // phase 3 (rare): the exact range needs a wider type than the sample said
  if (codes == nullptr || !fits || (write1 && w == ws)) return;
  if (w == 1) quantize_body<1, false, VEC>(x, n, s, codes, st);
  else if (w == 2) quantize_body<2, false, VEC>(x, n, s, codes, st);
  else quantize_body<4, false, VEC>(x, n, s, codes, st);
}

template <int W, bool VEC>
__global__ void __launch_bounds__(kThreads) dequantize_kernel(const void *__restrict__ codes,
                                                              int64_t n, float s,
                                                              float *__restrict__ out) {
  const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t done = 0;
  if (VEC) {
    constexpr int EPT = 16 / W;
    const int64_t nvec = n / EPT;
    const uint4 *cv = reinterpret_cast<const uint4 *>(codes);
    float4 *ov = reinterpret_cast<float4 *>(out);
    for (int64_t v = tid; v < nvec; v += stride) {
      const uint4 u = __ldg(cv + v);
      float f[EPT];
#pragma unroll
      for (int e = 0; e < EPT; ++e) {
        constexpr int PER = 4 / W;  // codes per 32-bit word
        const int j = e / PER;
        const uint32_t wj = j == 0 ? u.x : (j == 1 ? u.y : (j == 2 ? u.z : u.w));
        const int sh = (e % PER) * 8 * W;
        int32_t c;
        if (W == 1) c = (int32_t)(int8_t)(wj >> sh);
        else if (W == 2) c = (int32_t)(int16_t)(wj >> sh);
        else c = (int32_t)wj;
        f[e] = __fmul_rn(s, (float)c);
      }
#pragma unroll
      for (int j = 0; j < EPT / 4; ++j)
        ov[v * (EPT / 4) + j] = make_float4(f[4 * j], f[4 * j + 1], f[4 * j + 2], f[4 * j + 3]);
    }
    done = nvec * EPT;
  }
  for (int64_t i = done + tid; i < n; i += stride) {
    int32_t c;
    if (W == 1) c = reinterpret_cast<const int8_t *>(codes)[i];
    else if (W == 2) c = reinterpret_cast<const int16_t *>(codes)[i];
    else c = reinterpret_cast<const int32_t *>(codes)[i];
    out[i] = __fmul_rn(s, (float)c);
  }
}

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

inline int grid_for(int64_t work_items, int sms) {
  int64_t blocks = (work_items + kThreads - 1) / kThreads;
  int64_t cap = (int64_t)sms * kBlocksPerSm;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  return (int)blocks;
}

}  // namespace

cudaError_t launch_quant_range(const float *x, int64_t n, QuantStatus *status, int sms,
                               cudaStream_t st) {
  const bool vec = aligned16(x);
  const int g = grid_for(vec ? n / 16 + 1 : n, sms);
  if (vec) range_kernel<true><<<g, kThreads, 0, st>>>(x, n, status);
  else range_kernel<false><<<g, kThreads, 0, st>>>(x, n, status);
  return cudaGetLastError();
}

cudaError_t launch_quantize(const float *x, int64_t n, float s, int width_req, void *codes,
                            size_t codes_bytes, QuantStatus *status, int sms,
                            cudaStream_t st) {
  const bool vec = aligned16(x) && (codes == nullptr || aligned16(codes));
  if (width_req == LAM_WIDTH_AUTO) {
    const int g = grid_for(vec ? n / 4 + 1 : n, sms);
    if (vec) quantize_auto_kernel<true><<<g, kThreads, 0, st>>>(x, n, s, codes, codes_bytes, status);
    else quantize_auto_kernel<false><<<g, kThreads, 0, st>>>(x, n, s, codes, codes_bytes, status);
    return cudaGetLastError();
  }
  const int g = grid_for(vec ? n / (16 / width_req) + 1 : n, sms);
#define LAM_Q(W)                                                                      \
  if (vec) quantize_forced_kernel<W, true><<<g, kThreads, 0, st>>>(x, n, s, codes, status); \
  else quantize_forced_kernel<W, false><<<g, kThreads, 0, st>>>(x, n, s, codes, status);
  if (width_req == 1) { LAM_Q(1) }
  else if (width_req == 2) { LAM_Q(2) }
  else { LAM_Q(4) }
#undef LAM_Q
  return cudaGetLastError();
}

cudaError_t launch_quantize_auto_coop(const float *x, int64_t n, float s, void *codes,
                                      size_t codes_bytes, QuantStatus *status, int sms,
                                      cudaStream_t st) {
  const bool vec = aligned16(x) && (codes == nullptr || aligned16(codes));
  const void *kern = vec ? (const void *)quantize_auto_coop_kernel<true>
                         : (const void *)quantize_auto_coop_kernel<false>;
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, 0);
  if (e != cudaSuccess) return e;
  if (per_sm > kBlocksPerSm) per_sm = kBlocksPerSm;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  int64_t g = (int64_t)sms * per_sm;
  const int64_t need = (n / 4 + kThreads - 1) / kThreads + 1;
  if (g > need) g = need;
  unsigned long long cb = codes_bytes;
  void *args[] = {(void *)&x, (void *)&n, (void *)&s, (void *)&codes, (void *)&cb,
                  (void *)&status};
  return cudaLaunchCooperativeKernel(kern, dim3((unsigned)g), dim3(kThreads), args, 0, st);
}

cudaError_t launch_dequantize(const void *codes, int width, int64_t n, float s, float *out,
                              int sms, cudaStream_t st) {
  const bool vec = aligned16(codes) && aligned16(out);
  const int g = grid_for(vec ? n / (16 / width) + 1 : n, sms);
#define LAM_D(W)                                                                   \
  if (vec) dequantize_kernel<W, true><<<g, kThreads, 0, st>>>(codes, n, s, out);   \
  else dequantize_kernel<W, false><<<g, kThreads, 0, st>>>(codes, n, s, out);
  if (width == 1) { LAM_D(1) }
  else if (width == 2) { LAM_D(2) }
  else { LAM_D(4) }
#undef LAM_D
  return cudaGetLastError();
}

}  // namespace lam
