// lamz.cu -- error-bounded byte codec for retained embeddings (Sec. 3.2,
// layer L2: error-bounded byte compression under a relative codec bound, 1%
// of max|x| when deployed).  Format (little-endian):
//   "LAMZ" | n (int64) | s (fp32) | one byte L per block of 32 values, zero
//   padded to a multiple of 4 | for each block with L > 0: a sign word and L
//   bit planes of the block's |deltas| (32-bit words).
// s = fl32(2 eb) with eb = fl32(rel * max|x|) (s = 1 when all x are 0); the
// codes are Q_eps at eps = eb (one IEEE division, round half to even); inside
// a block the deltas are d_0 = q_0, d_j = q_j - q_{j-1} (a tail block repeats
// its last code); L = bit length of the block's largest |d|.  Decoding sums the
// deltas (a warp prefix sum) and returns fl32(s * q).
//
// A warp owns a block: lane j holds value j, the sign word is one ballot and
// bit plane p another (bit p of every |d_j|).  Compression runs a sizing pass
// (L bytes straight into the header), a scan of the payload sizes, then the
// writing pass.
#include "lam_internal.cuh"
#include "scan.cuh"

#include <string.h>

namespace lam {

namespace {

constexpr int kCodecThreads = 256;  // 8 blocks of 32 values per CTA

struct CodecStatus {
  uint32_t amax;   // bit pattern of max|x| (non-negative floats order as uints)
  uint32_t flags;  // kFlagNonfinite
  uint32_t total;  // payload bytes
  uint32_t bad;    // malformed stream (decoder)
};

__global__ void amax_kernel(const float *__restrict__ x, int64_t n, CodecStatus *st) {
  float m = 0.0f;
  uint32_t nf = 0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const float a = fabsf(__ldg(x + i));
    if (a <= 3.402823466e38f) m = fmaxf(m, a);
    else nf = 1;
  }
  for (int off = 16; off > 0; off >>= 1) {
    m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    nf |= __shfl_xor_sync(0xffffffffu, nf, off);
  }
  if ((threadIdx.x & 31) == 0) {
    const uint32_t u = __float_as_uint(m);
    if (u > *(volatile uint32_t *)&st->amax) atomicMax(&st->amax, u);
    if (nf) atomicOr(&st->flags, kFlagNonfinite);
  }
}

__device__ __forceinline__ float codec_step(const CodecStatus *st, float rel) {
  const float mx = __uint_as_float(st->amax);
  return mx > 0.0f ? 2.0f * __fmul_rn(rel, mx) : 1.0f;
}

constexpr int kUnrollBlocks = 8;  // blocks a warp loads ahead (memory-level parallelism)

// Codes, deltas and |deltas| of the warp's block b from its value xv (lane's
// element, loaded by the caller); returns L (0..31).
__device__ __forceinline__ int block_deltas(float xv, int64_t n, int64_t b, const QDiv &qd, int lane,
                                            int32_t &d, uint32_t &m) {
  const int64_t i = b * 32 + lane;
  const int valid = (int)min((int64_t)32, n - b * 32);
  int32_t q = i < n ? qd.code(xv) : 0;
  q = __shfl_sync(0xffffffffu, q, lane < valid ? lane : valid - 1);  // pad: repeat the last code
  const int32_t prev = __shfl_up_sync(0xffffffffu, q, 1);
  d = lane == 0 ? q : q - prev;
  m = d < 0 ? (uint32_t)(-(int64_t)d) : (uint32_t)d;
  const uint32_t mx = __reduce_max_sync(0xffffffffu, m);
  return 32 - __clz(mx);
}

__global__ void __launch_bounds__(kCodecThreads) lamz_size_kernel(const float *__restrict__ x,
                                                                 int64_t n, float rel,
                                                                 const CodecStatus *st,
                                                                 uint8_t *hdr, uint32_t *sizes,
                                                                 int64_t nb) {
  const float s = codec_step(st, rel);
  const QDiv qd = QDiv::of(s);
  const int lane = threadIdx.x & 31;
  const int64_t gw = (int64_t)blockIdx.x * (kCodecThreads / 32) + (threadIdx.x >> 5);
  const int64_t nw = (int64_t)gridDim.x * (kCodecThreads / 32);
  for (int64_t b0 = gw * kUnrollBlocks; b0 < nb; b0 += nw * kUnrollBlocks) {
    float xv[kUnrollBlocks];
#pragma unroll
    for (int u = 0; u < kUnrollBlocks; ++u) {
      const int64_t i = (b0 + u) * 32 + lane;
      xv[u] = i < n ? __ldg(x + i) : 0.0f;
    }
#pragma unroll
    for (int u = 0; u < kUnrollBlocks; ++u) {
      const int64_t b = b0 + u;
      if (b >= nb) break;
      int32_t d;
      uint32_t m;
      const int L = block_deltas(xv[u], n, b, qd, lane, d, m);
      if (lane == 0) {
        hdr[b] = (uint8_t)L;
        sizes[b] = L > 0 ? 4u + 4u * (uint32_t)L : 0u;
      }
    }
  }
}

// Writes the stream when the sizing pass found it finite and within `cap`
// bytes: block 0 the fixed header (magic, n, step s), every warp its blocks'
// sign words and planes.  (The decision is read from the status on the device,
// so the host waits once, after this kernel.)
__global__ void __launch_bounds__(kCodecThreads) lamz_write_kernel(
    const float *__restrict__ x, int64_t n, float rel, const CodecStatus *st,
    const uint32_t *offs, int64_t nb, uint32_t *payload, uint32_t *out, uint64_t head,
    uint64_t cap) {
  if ((__ldg(&st->flags) & kFlagNonfinite) || head + __ldg(&st->total) > cap) return;
  const float s = codec_step(st, rel);
  const QDiv qd = QDiv::of(s);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    out[0] = 0x5A4D414Cu;  // "LAMZ" little-endian
    out[1] = (uint32_t)((uint64_t)n & 0xffffffffu);
    out[2] = (uint32_t)((uint64_t)n >> 32);
    out[3] = __float_as_uint(s);
  }
  const int lane = threadIdx.x & 31;
  const int64_t gw = (int64_t)blockIdx.x * (kCodecThreads / 32) + (threadIdx.x >> 5);
  const int64_t nw = (int64_t)gridDim.x * (kCodecThreads / 32);
  for (int64_t b0 = gw * kUnrollBlocks; b0 < nb; b0 += nw * kUnrollBlocks) {
   float xv[kUnrollBlocks];
#pragma unroll
   for (int u = 0; u < kUnrollBlocks; ++u) {
     const int64_t i = (b0 + u) * 32 + lane;
     xv[u] = i < n ? __ldg(x + i) : 0.0f;
   }
#pragma unroll
   for (int u = 0; u < kUnrollBlocks; ++u) {
    const int64_t b = b0 + u;
    if (b >= nb) break;
    int32_t d;
    uint32_t m;
    const int L = block_deltas(xv[u], n, b, qd, lane, d, m);
    if (L == 0) continue;
    uint32_t *w = payload + offs[b] / 4;
    const uint32_t sign = __ballot_sync(0xffffffffu, d < 0);
    uint32_t mine = 0;  // lane p keeps plane p
#pragma unroll 1
    for (int p = 0; p < L; ++p) {
      const uint32_t plane = __ballot_sync(0xffffffffu, (m >> p) & 1u);
      if (lane == p) mine = plane;
    }
    if (lane == 0) w[0] = sign;
    if (lane < L) w[1 + lane] = mine;
   }
  }
}

__global__ void lamz_dsize_kernel(const uint8_t *hdr, int64_t nb, uint32_t *sizes,
                                  CodecStatus *st) {
  for (int64_t b = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; b < nb;
       b += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t L = hdr[b];
    if (L > 31) atomicOr(&st->bad, 1u);
    sizes[b] = L > 0 && L <= 31 ? 4u + 4u * L : 0u;
  }
}

__global__ void __launch_bounds__(kCodecThreads) lamz_decode_kernel(
    const uint8_t *hdr, const uint32_t *payload, const uint32_t *offs, int64_t nb, int64_t n,
    float s, float *__restrict__ out) {
  const int lane = threadIdx.x & 31;
  const int64_t gw = (int64_t)blockIdx.x * (kCodecThreads / 32) + (threadIdx.x >> 5);
  const int64_t nw = (int64_t)gridDim.x * (kCodecThreads / 32);
  for (int64_t b0 = gw * kUnrollBlocks; b0 < nb; b0 += nw * kUnrollBlocks) {
   int Ls[kUnrollBlocks];
   uint32_t words[kUnrollBlocks];
#pragma unroll
   for (int u = 0; u < kUnrollBlocks; ++u) {  // every block's words in flight at once
     const int64_t b = b0 + u;
     Ls[u] = b < nb ? min((int)hdr[b], 31) : 0;
     words[u] = (b < nb && Ls[u] > 0 && lane <= Ls[u]) ? payload[offs[b] / 4 + lane] : 0u;
   }
#pragma unroll
   for (int u = 0; u < kUnrollBlocks; ++u) {
    const int64_t b = b0 + u;
    if (b >= nb) break;
    const int L = Ls[u];
    int32_t q = 0;
    if (L > 0) {
      const uint32_t word = words[u];  // lane 0: sign, lane p+1: plane p
      const uint32_t sign = __shfl_sync(0xffffffffu, word, 0);
      uint32_t m = 0;
#pragma unroll 1
      for (int p = 0; p < L; ++p) m |= ((__shfl_sync(0xffffffffu, word, p + 1) >> lane) & 1u) << p;
      q = ((sign >> lane) & 1u) ? -(int32_t)m : (int32_t)m;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {  // inclusive prefix sum of the deltas
        const int32_t t = __shfl_up_sync(0xffffffffu, q, off);
        if (lane >= off) q += t;
      }
    }
    const int64_t i = b * 32 + lane;
    if (i < n) out[i] = __fmul_rn(s, (float)q);
   }
  }
}

unsigned codec_grid(int64_t nb, int sms) {
  int64_t g = cdiv(nb, (int64_t)(kCodecThreads / 32) * kUnrollBlocks);
  if (g > (int64_t)sms * 8) g = (int64_t)sms * 8;
  return (unsigned)(g < 1 ? 1 : g);
}

inline size_t al256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace

size_t lamz_head_bytes(int64_t n) {
  const int64_t nb = (n + 31) / 32;
  return 16 + (size_t)((nb + 3) / 4 * 4);
}

size_t lamz_bound_bytes(int64_t n) {
  const int64_t nb = (n + 31) / 32;
  return lamz_head_bytes(n) + (size_t)nb * (4 + 4 * 31);
}

size_t lamz_workspace_bytes(int64_t n) {
  const int64_t nb = (n + 31) / 32;
  return al256(sizeof(CodecStatus)) + al256(4 * (size_t)(nb + 1)) +
         al256(4 * (size_t)(cdiv(nb, kTile) + 2));
}

// Compression: returns the stream size in *bytes (host); *fits false when it
// exceeds cap (nothing past the header region is written then).
cudaError_t launch_lamz_compress(const float *x, int64_t n, float rel, uint8_t *out, size_t cap,
                                 void *ws, int sms, cudaStream_t stream, size_t *bytes,
                                 bool *fits, bool *nonfinite) {
  const int64_t nb = (n + 31) / 32;
  uint8_t *w = static_cast<uint8_t *>(ws);
  CodecStatus *st = reinterpret_cast<CodecStatus *>(w);
  uint32_t *sizes = reinterpret_cast<uint32_t *>(w + al256(sizeof(CodecStatus)));
  uint32_t *sums = reinterpret_cast<uint32_t *>(w + al256(sizeof(CodecStatus)) +
                                                al256(4 * (size_t)(nb + 1)));
  const size_t head = lamz_head_bytes(n);
  cudaError_t e = cudaMemsetAsync(st, 0, sizeof(CodecStatus), stream);
  if (e != cudaSuccess) return e;
  int64_t g = cdiv(n, 256);
  if (g > (int64_t)sms * 8) g = (int64_t)sms * 8;
  amax_kernel<<<(unsigned)(g < 1 ? 1 : g), 256, 0, stream>>>(x, n, st);
  e = cudaMemsetAsync(out + 16, 0, head - 16, stream);  // header padding
  if (e != cudaSuccess) return e;
  lamz_size_kernel<<<codec_grid(nb, sms), kCodecThreads, 0, stream>>>(x, n, rel, st, out + 16,
                                                                      sizes, nb);
  e = scan_u32(sizes, nb, sums, &st->total, stream);
  if (e != cudaSuccess) return e;
  lamz_write_kernel<<<codec_grid(nb, sms), kCodecThreads, 0, stream>>>(
      x, n, rel, st, sizes, nb, reinterpret_cast<uint32_t *>(out + head),
      reinterpret_cast<uint32_t *>(out), (uint64_t)head, (uint64_t)cap);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  CodecStatus h;  // one wait, after the stream is written
  e = read_back(&h, st, sizeof(h), stream);
  if (e != cudaSuccess) return e;
  *nonfinite = (h.flags & kFlagNonfinite) != 0;
  *bytes = head + h.total;
  *fits = *bytes <= cap;
  return cudaSuccess;
}

cudaError_t launch_lamz_decompress(const uint8_t *in, size_t in_bytes, float *out, int64_t n,
                                   void *ws, int sms, cudaStream_t stream, bool *bad) {
  const int64_t nb = (n + 31) / 32;
  uint8_t *w = static_cast<uint8_t *>(ws);
  CodecStatus *st = reinterpret_cast<CodecStatus *>(w);
  uint32_t *sizes = reinterpret_cast<uint32_t *>(w + al256(sizeof(CodecStatus)));
  uint32_t *sums = reinterpret_cast<uint32_t *>(w + al256(sizeof(CodecStatus)) +
                                                al256(4 * (size_t)(nb + 1)));
  const size_t head = lamz_head_bytes(n);
  *bad = true;
  if (in_bytes < head) return cudaSuccess;
  uint8_t fixed[16];
  cudaError_t e = read_back(fixed, in, 16, stream);
  if (e != cudaSuccess) return e;
  e = cudaMemsetAsync(st, 0, sizeof(CodecStatus), stream);
  if (e != cudaSuccess) return e;
  lamz_dsize_kernel<<<codec_grid(nb * 32, sms), 256, 0, stream>>>(in + 16, nb, sizes, st);
  e = scan_u32(sizes, nb, sums, &st->total, stream);
  if (e != cudaSuccess) return e;
  CodecStatus h;
  e = read_back(&h, st, sizeof(h), stream);
  if (e != cudaSuccess) return e;
  uint64_t nn = 0;
  for (int k = 0; k < 8; ++k) nn |= (uint64_t)fixed[4 + k] << (8 * k);
  if (memcmp(fixed, "LAMZ", 4) != 0 || (int64_t)nn != n || h.bad || head + h.total > in_bytes)
    return cudaSuccess;
  float s;
  memcpy(&s, fixed + 12, 4);
  *bad = false;
  lamz_decode_kernel<<<codec_grid(nb, sms), kCodecThreads, 0, stream>>>(
      in + 16, reinterpret_cast<const uint32_t *>(in + head), sizes, nb, n, s, out);
  return cudaGetLastError();
}

}  // namespace lam
