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
    const QDiv qd = QDiv::of(sc);  // the IEEE quotient by sc, as a division gives it
    int8_t *cr = codes + r * D;
    for (int d = lane; d < D; d += 32) {
      int c = -128;
      if (sc > 0.0f) {
        c = qd.code(__fsub_rn(xr[d], lo)) - 128;
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

// The same with 16-byte loads and 4-byte code stores, the row held in
// registers (D a multiple of 4, at most 128 NCH; 16-byte aligned x rows).
template <int NCH>
__global__ void __launch_bounds__(kRowWarps * 32)
    encode_int8_rows_vec_kernel(const float *__restrict__ x, int64_t N, int D,
                                int8_t *__restrict__ codes, float *__restrict__ scale,
                                float *__restrict__ offset) {
  const int lane = threadIdx.x & 31;
  const int64_t nw = (int64_t)gridDim.x * kRowWarps;
  for (int64_t r = (int64_t)blockIdx.x * kRowWarps + (threadIdx.x >> 5); r < N; r += nw) {
    const float4 *xr = reinterpret_cast<const float4 *>(x + r * D);
    float4 v[NCH];
    float lo = INFINITY, hi = -INFINITY;
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
      const int g = lane + 32 * j;
      v[j] = 4 * g < D ? xr[g] : make_float4(0.f, 0.f, 0.f, 0.f);
      if (4 * g < D) {
        lo = fminf(lo, fminf(fminf(v[j].x, v[j].y), fminf(v[j].z, v[j].w)));
        hi = fmaxf(hi, fmaxf(fmaxf(v[j].x, v[j].y), fmaxf(v[j].z, v[j].w)));
      }
    }
    lo = warp_min(lo);
    hi = warp_max(hi);
    const float sc = __fdiv_rn(__fsub_rn(hi, lo), 255.0f);
    const QDiv qd = QDiv::of(sc);
    uint32_t *cr = reinterpret_cast<uint32_t *>(codes + r * D);
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
      const int g = lane + 32 * j;
      if (4 * g >= D) break;
      const float e[4] = {v[j].x, v[j].y, v[j].z, v[j].w};
      uint32_t packed = 0;
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        int c = -128;
        if (sc > 0.0f) {
          c = qd.code(__fsub_rn(e[t], lo)) - 128;
          c = c < -128 ? -128 : (c > 127 ? 127 : c);
        }
        packed |= ((uint32_t)c & 0xffu) << (8 * t);
      }
      cr[g] = packed;
    }
    if (lane == 0) {
      scale[r] = sc;
      offset[r] = __fadd_rn(lo, __fmul_rn(128.0f, sc));
    }
  }
}

// Sign-binary: one warp per row.  alpha = sum |x| / D; lane t packs the
// signs of x[8t .. 8t + 7] into byte t (bit i for x[8t + i] >= 0).  With a
// 16-byte aligned x (vec) the eight values come as two 16-byte loads.
__global__ void __launch_bounds__(kRowWarps * 32)
    encode_sign_rows_kernel(const float *__restrict__ x, int64_t N, int D,
                            uint8_t *__restrict__ bits, float *__restrict__ alpha, bool vec) {
  const int lane = threadIdx.x & 31;
  const int64_t nw = (int64_t)gridDim.x * kRowWarps;
  const int nb = D / 8;
  for (int64_t r = (int64_t)blockIdx.x * kRowWarps + (threadIdx.x >> 5); r < N; r += nw) {
    const float *xr = x + r * D;
    // sum |x| per lane as an unevaluated fp32 pair (hi + lo, Knuth's TwoSum
    // for every addition), then in fp64 across lanes: far below half an fp32
    // ulp of error, without the slow fp64 pipe in the loop
    float shi = 0.0f, slo = 0.0f;
    uint8_t *br = bits + r * nb;
    for (int t = lane; t < nb; t += 32) {
      float e[8];
      if (vec) {
        const float4 a = reinterpret_cast<const float4 *>(xr)[2 * t];
        const float4 b = reinterpret_cast<const float4 *>(xr)[2 * t + 1];
        e[0] = a.x; e[1] = a.y; e[2] = a.z; e[3] = a.w;
        e[4] = b.x; e[5] = b.y; e[6] = b.z; e[7] = b.w;
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) e[i] = xr[8 * t + i];
      }
      unsigned byte = 0;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float a = fabsf(e[i]);
        const float sn = __fadd_rn(shi, a);
        const float bv = __fsub_rn(sn, shi);
        const float err = __fadd_rn(__fsub_rn(shi, __fsub_rn(sn, bv)), __fsub_rn(a, bv));
        shi = sn;
        slo = __fadd_rn(slo, err);
        byte |= (e[i] >= 0.0f ? 1u : 0u) << i;
      }
      br[t] = (uint8_t)byte;
    }
    double acc = __dadd_rn((double)shi, (double)slo);
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
    decode_rows_kernel(ScoreArgs a, RowPtrs rp, float *__restrict__ out) {
  const int lane = threadIdx.x & 31;
  const int64_t nw = (int64_t)gridDim.x * kRowWarps;
  for (int64_t r = (int64_t)blockIdx.x * kRowWarps + (threadIdx.x >> 5); r < a.N; r += nw)
    for (int d = lane; d < a.D; d += 32) out[r * a.D + d] = row_value(a, rp, r, d);
}

unsigned row_grid(int64_t N, int sms) {
  const int64_t want = (N + kRowWarps - 1) / kRowWarps;
  const int64_t cap = (int64_t)sms * 8;
  return (unsigned)(want < cap ? want : cap);
}

}  // namespace

cudaError_t launch_encode_rows(const float *x, int64_t N, int D, int fmt, void *codes,
                               float *scale, float *offset, int sms, cudaStream_t st) {
  const bool x16 = (reinterpret_cast<uintptr_t>(x) & 15u) == 0;
  if (fmt == LAM_ROWS_INT8) {
    int8_t *c = static_cast<int8_t *>(codes);
    const bool vec = x16 && (reinterpret_cast<uintptr_t>(codes) & 3u) == 0 && D % 4 == 0;
    const unsigned g = row_grid(N, sms);
    if (vec && D <= 256)
      encode_int8_rows_vec_kernel<2><<<g, kRowWarps * 32, 0, st>>>(x, N, D, c, scale, offset);
    else if (vec && D <= 512)
      encode_int8_rows_vec_kernel<4><<<g, kRowWarps * 32, 0, st>>>(x, N, D, c, scale, offset);
    else if (vec && D <= 1024)
      encode_int8_rows_vec_kernel<8><<<g, kRowWarps * 32, 0, st>>>(x, N, D, c, scale, offset);
    else
      encode_int8_rows_kernel<<<g, kRowWarps * 32, 0, st>>>(x, N, D, c, scale, offset);
  } else if (fmt == LAM_ROWS_SIGN) {
    encode_sign_rows_kernel<<<row_grid(N, sms), kRowWarps * 32, 0, st>>>(
        x, N, D, static_cast<uint8_t *>(codes), scale, x16);
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
  RowPtrs rp;
  rp.scale = scale;
  rp.offset = offset;
  decode_rows_kernel<<<row_grid(N, sms), kRowWarps * 32, 0, st>>>(a, rp, out);
  return cudaGetLastError();
}

}  // namespace lam
