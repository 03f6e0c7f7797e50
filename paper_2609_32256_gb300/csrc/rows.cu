// rows.cu -- encoders and decoder of the per-vector byte codecs of the
// composite-reduction experiment (Sec. "Composite reduction", Table
// "composite": fp16, per-vector int8, sign-binary).  The definitions are the
// ones lam.h states; the arithmetic is IEEE round-to-nearest with no
// contraction (every step written with the _rn intrinsics).
#include "lam_internal.cuh"

namespace lam {
namespace {

constexpr int kRowWarps = 8;

__device__ __forceinline__ float warp_min(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}
__device__ __forceinline__ double warp_sum_f64(double v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = __dadd_rn(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}

// Per-vector int8: one warp per row.  The row's min and max, the step
// (hi - lo)/255, then codes rint((x - lo)/step) - 128 and the offset.
__global__ void __launch_bounds__(kRowWarps * 32)
    encode_int8_rows_kernel(const float *__restrict__ x, int64_t N, int D,
                            int8_t *__restrict__ codes, float *__restrict__ scale,
                            float *__restrict__ offset) {
  const int lane = threadIdx.x & 31;
  const int64_t nw = (int64_t)gridDim.x * kRowWarps;
  for (int64_t r = (int64_t)blockIdx.x * kRowWarps + (threadIdx.x >> 5); r < N; r += nw) {
    const float *xr = x + r * D;
    float lo = INFINITY, hi = -INFINITY;
    for (int d = lane; d < D; d += 32) {
      const float v = xr[d];
      lo = fminf(lo, v);
      hi = fmaxf(hi, v);
    }
    lo = warp_min(lo);
    hi = warp_max(hi);
    const float sc = __fdiv_rn(__fsub_rn(hi, lo), 255.0f);
    int8_t *cr = codes + r * D;
    for (int d = lane; d < D; d += 32) {
      int c = -128;
      if (sc > 0.0f) {
        c = __float2int_rn(__fdiv_rn(__fsub_rn(xr[d], lo), sc)) - 128;
        c = c < -128 ? -128 : (c > 127 ? 127 : c);
      }
      cr[d] = (int8_t)c;
    }
    if (lane == 0) {
      scale[r] = sc;
      offset[r] = __fadd_rn(lo, __fmul_rn(128.0f, sc));
    }
  }
}

// Sign-binary: one warp per row.  alpha = sum |x| / D in fp64; lane t packs
// the signs of x[8t .. 8t + 7] into byte t (bit i for x[8t + i] >= 0).
__global__ void __launch_bounds__(kRowWarps * 32)
    encode_sign_rows_kernel(const float *__restrict__ x, int64_t N, int D,
                            uint8_t *__restrict__ bits, float *__restrict__ alpha) {
  const int lane = threadIdx.x & 31;
  const int64_t nw = (int64_t)gridDim.x * kRowWarps;
  const int nb = D / 8;
  for (int64_t r = (int64_t)blockIdx.x * kRowWarps + (threadIdx.x >> 5); r < N; r += nw) {
    const float *xr = x + r * D;
    double acc = 0.0;
    uint8_t *br = bits + r * nb;
    for (int t = lane; t < nb; t += 32) {
      unsigned byte = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float v = xr[8 * t + i];
        acc = __dadd_rn(acc, fabs((double)v));
        byte |= (v >= 0.0f ? 1u : 0u) << i;
      }
      br[t] = (uint8_t)byte;
    }
    acc = warp_sum_f64(acc);
    if (lane == 0) alpha[r] = __double2float_rn(__ddiv_rn(acc, (double)D));
  }
}

__global__ void __launch_bounds__(256) encode_fp16_kernel(const float *__restrict__ x, int64_t n,
                                                          __half *__restrict__ out) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
    out[i] = __float2half_rn(x[i]);
}

// Decoder: one warp per row, xhat as row_value() evaluates it.
__global__ void __launch_bounds__(kRowWarps * 32)
    decode_rows_kernel(ScoreArgs a, float *__restrict__ out) {
  const int lane = threadIdx.x & 31;
  const int64_t nw = (int64_t)gridDim.x * kRowWarps;
  for (int64_t r = (int64_t)blockIdx.x * kRowWarps + (threadIdx.x >> 5); r < a.N; r += nw)
    for (int d = lane; d < a.D; d += 32) out[r * a.D + d] = row_value(a, r, d);
}

unsigned row_grid(int64_t N, int sms) {
  const int64_t want = (N + kRowWarps - 1) / kRowWarps;
  const int64_t cap = (int64_t)sms * 8;
  return (unsigned)(want < cap ? want : cap);
}

}  // namespace

cudaError_t launch_encode_rows(const float *x, int64_t N, int D, int fmt, void *codes,
                               float *scale, float *offset, int sms, cudaStream_t st) {
  if (fmt == LAM_ROWS_INT8) {
    encode_int8_rows_kernel<<<row_grid(N, sms), kRowWarps * 32, 0, st>>>(
        x, N, D, static_cast<int8_t *>(codes), scale, offset);
  } else if (fmt == LAM_ROWS_SIGN) {
    encode_sign_rows_kernel<<<row_grid(N, sms), kRowWarps * 32, 0, st>>>(
        x, N, D, static_cast<uint8_t *>(codes), scale);
  } else {
    const int64_t n = N * D;
    int64_t g = (n + 255) / 256;
    if (g > (int64_t)sms * 16) g = (int64_t)sms * 16;
    encode_fp16_kernel<<<(unsigned)g, 256, 0, st>>>(x, n, static_cast<__half *>(codes));
  }
  return cudaGetLastError();
}

cudaError_t launch_decode_rows(const void *codes, int fmt, int64_t N, int D, const float *scale,
                               const float *offset, float *out, int sms, cudaStream_t st) {
  ScoreArgs a{};
  a.codes = codes;
  a.N = N;
  a.D = D;
  a.fmt = fmt;
  a.row_scale = scale;
  a.row_offset = offset;
  decode_rows_kernel<<<row_grid(N, sms), kRowWarps * 32, 0, st>>>(a, out);
  return cudaGetLastError();
}

}  // namespace lam
