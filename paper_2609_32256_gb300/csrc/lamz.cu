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

#include <cstdlib>
#include <cstring>

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

// Transpose of the 8 x 8 bit matrix held in x, bit (r, c) at position 8 r + c
// (row r in byte r, column c from the least significant bit): three rounds of
// swaps between the bits 7, 14 and 28 positions apart (the recursive 2 x 2
// block transpose; Hacker's Delight, section 7-3).  Its own inverse.
__device__ __forceinline__ uint64_t transpose8x8(uint64_t x) {
  x = (x & 0xAA55AA55AA55AA55ull) | ((x & 0x00AA00AA00AA00AAull) << 7) |
      ((x >> 7) & 0x00AA00AA00AA00AAull);
  x = (x & 0xCCCC3333CCCC3333ull) | ((x & 0x0000CCCC0000CCCCull) << 14) |
      ((x >> 14) & 0x0000CCCC0000CCCCull);
  x = (x & 0xF0F0F0F00F0F0F0Full) | ((x & 0x00000000F0F0F0F0ull) << 28) |
      ((x >> 28) & 0x00000000F0F0F0F0ull);
  return x;
}

// Byte k of each of a, b, c, d, as one word (a's byte lowest).
__device__ __forceinline__ uint32_t gather_bytes(uint32_t a, uint32_t b, uint32_t c, uint32_t d,
                                                 int k) {
  const uint32_t sel = (uint32_t)k | ((uint32_t)(4 + k) << 4);
  return __byte_perm(__byte_perm(a, b, sel), __byte_perm(c, d, sel), 0x5410);
}

constexpr int kWarps = kCodecThreads / 32;

// One lane, one block b: the block's codes (a tail block repeats its last
// code), the magnitudes m of its deltas, their sign word, and L.  VEC: x is
// 16-byte aligned, so a full block loads as eight 16-byte vectors.
template <bool VEC>
__device__ __forceinline__ int lane_block(const float *__restrict__ x, int64_t n, int64_t b,
                                          const QDiv &qd, uint32_t (&m)[32], uint32_t &sign) {
  const int64_t base = b * 32;
  const int valid = (int)min((int64_t)32, n - base);
  float v[32];
  if (VEC && valid == 32) {
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const float4 t = __ldg(reinterpret_cast<const float4 *>(x + base) + k);
      v[4 * k] = t.x;
      v[4 * k + 1] = t.y;
      v[4 * k + 2] = t.z;
      v[4 * k + 3] = t.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = i < valid ? __ldg(x + base + i) : 0.0f;
  }
  int32_t prev = 0;
  uint32_t mx = 0;
  sign = 0;
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const int32_t q = i < valid ? qd.code(v[i]) : prev;
    const int32_t d = i == 0 ? q : (int32_t)((uint32_t)q - (uint32_t)prev);
    m[i] = d < 0 ? (uint32_t)(-(int64_t)d) : (uint32_t)d;
    sign |= (uint32_t)(d < 0) << i;
    mx = max(mx, m[i]);
    prev = q;
  }
  return 32 - __clz(mx);
}

// Tile states of the single-pass writer: bits 62-63 of a tile's 64-bit word
// (0: not yet published), the rest the payload words of the tile alone (AGG)
// or of every tile up to it (PRE).
constexpr uint64_t kTileAgg = 1ull << 62, kTilePre = 2ull << 62;
constexpr uint64_t kTileValue = (1ull << 62) - 1;
constexpr long long kLookBackCycles = 2000000000LL;  // ~1 s: a bounded wait
constexpr int kCompWarps = 4;  // warps per compression CTA: a tile of 128 blocks (2: slower, 8: slower)

// Compression in one pass over x (after amax_kernel): block 0 writes the
// fixed header (magic, n, step s); a CTA of NW warps claims tiles of 32 NW blocks in order
// (an atomic ticket, so every earlier tile belongs to a CTA already running),
// lane j of warp w computes block 32 w + j of the tile (codes, deltas, L into
// the stream header), the CTA adds up the tile's payload words, and warp 0
// publishes them and finds the words of all earlier tiles by looking back
// over their published states, 32 at a time (a tile that also published its
// running total ends the look-back: decoupled look-back).  Then each warp's
// blocks' sign words and planes, built by 8 x 8 bit transposes (byte g of the
// values 8q .. 8q + 7 transposed into byte q of planes 8g .. 8g + 7) and
// staged in shared memory, leave in coalesced rows, unless the tile would
// end past `cap` (the stream then reports only its size).  The look-back spin
// is bounded: it gives up after `budget` SM cycles (~1 s), raising
// kFlagTimeout, and so do all later look-backs.  (stall: tile 0 publishes
// nothing, so that the look-backs run out: the timeout path under test.)
template <bool VEC, int NW>
__global__ void __launch_bounds__(NW * 32) lamz_compress_kernel(
    const float *__restrict__ x, int64_t n, float rel, CodecStatus *st, uint8_t *hdr, int64_t nb,
    uint32_t *payload, uint32_t *out, uint64_t head, uint64_t cap,
    unsigned long long *tiles, unsigned int *ticket, int64_t ntiles, long long budget, int stall) {
  // (a block takes 1 + L <= 33 words: L = 32 only when a delta reaches 2^31)
  __shared__ uint32_t stage[NW][32 * 33];
  __shared__ uint32_t s_words[NW];  // per warp: its words, then its offset in the tile
  __shared__ unsigned long long s_before;
  __shared__ int64_t s_tile;
  __shared__ int s_write;
  if (*(volatile uint32_t *)&st->flags & kFlagNonfinite) return;
  const float s = codec_step(st, rel);
  const QDiv qd = QDiv::of(s);
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    out[0] = 0x5A4D414Cu;  // "LAMZ" little-endian
    out[1] = (uint32_t)((uint64_t)n & 0xffffffffu);
    out[2] = (uint32_t)((uint64_t)n >> 32);
    out[3] = __float_as_uint(s);
  }
  const int lane = threadIdx.x & 31, wi = threadIdx.x >> 5;
  uint32_t *U = stage[wi];
  while (true) {
    if (threadIdx.x == 0) s_tile = (int64_t)atomicAdd(ticket, 1u);
    __syncthreads();
    const int64_t t = s_tile;
    if (t >= ntiles) break;
    const int64_t b = (t * NW + wi) * 32 + lane;
    const bool has = b < nb;
    uint32_t m[32], sign = 0;
    int L = 0;
    if (has) {
      L = lane_block<VEC>(x, n, b, qd, m, sign);
      hdr[b] = (uint8_t)L;
    }
    const uint32_t words = L > 0 ? 1u + (uint32_t)L : 0u;
    uint32_t incl = words;  // the blocks' word offsets within the warp's stretch
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    const uint32_t mw = incl - words;
    const uint32_t warp_words = __shfl_sync(0xffffffffu, incl, 31);
    if (lane == 0) s_words[wi] = warp_words;
    __syncthreads();
    if (wi == 0) {
      // the warps' offsets within the tile, the tile's words
      const uint32_t ww = lane < NW ? s_words[lane] : 0u;
      uint32_t wincl = ww;
#pragma unroll
      for (int off = 1; off < NW; off <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, wincl, off);
        if (lane >= off) wincl += y;
      }
      const uint32_t tile_words = __shfl_sync(0xffffffffu, wincl, NW - 1);
      // payload words of the earlier tiles: lane i reads the state of tile
      // j - i; wait until every state up to the nearest running total is
      // published, and add them up
      unsigned long long before = 0;
      bool gave_up = false;
      if (t == 0) {
        if (lane == 0 && !stall) atomicExch(tiles, kTilePre | tile_words);
      } else {
        if (lane == 0) atomicExch(tiles + t, kTileAgg | tile_words);
        const long long c0 = clock64();
        for (int64_t jh = t - 1;;) {
          const int64_t j = jh - lane;
          // (before tile 0: a running total of 0)
          const unsigned long long f =
              j >= 0 ? *(volatile unsigned long long *)(tiles + j) : kTilePre;
          const unsigned pre = __ballot_sync(0xffffffffu, (f & kTilePre) != 0);
          const unsigned unset = __ballot_sync(0xffffffffu, f == 0);
          const int near = pre ? __ffs(pre) - 1 : 31;  // the last lane needed
          const unsigned need = near == 31 ? 0xffffffffu : (2u << near) - 1u;
          if (unset & need) {
            // (one decision for the whole warp: every lane stays in the ballots)
            if (__any_sync(0xffffffffu, (*(volatile uint32_t *)&st->flags & kFlagTimeout) ||
                                            clock64() - c0 > budget)) {
              if (lane == 0) atomicOr(&st->flags, kFlagTimeout);
              gave_up = true;
              break;
            }
            continue;
          }
          unsigned long long v = lane <= near ? (f & kTileValue) : 0ull;
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
          before += v;
          if (pre) break;
          jh -= 32;
        }
        if (lane == 0 && !gave_up) atomicExch(tiles + t, kTilePre | (before + tile_words));
      }
      if (lane < NW) s_words[lane] = wincl - ww;
      if (lane == 0) {
        s_before = before;
        if (t == ntiles - 1) st->total = (uint32_t)(4 * (before + tile_words));
        // the tile's words, if they end within cap (and every look-back held)
        s_write = !gave_up && head + 4 * (before + tile_words) <= cap &&
                  !(*(volatile uint32_t *)&st->flags & kFlagTimeout);
      }
    }
    __syncthreads();
    const bool write = s_write != 0;
    const unsigned long long w0 = s_before + s_words[wi];  // this warp's first word
    if (write) {
      if (L > 0) {
        U[mw] = sign;
        for (int g = 0; 8 * g < L; ++g) {
          uint32_t P[8];
#pragma unroll
          for (int p = 0; p < 8; ++p) P[p] = 0u;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint32_t lo =
                gather_bytes(m[8 * q], m[8 * q + 1], m[8 * q + 2], m[8 * q + 3], g);
            const uint32_t hi =
                gather_bytes(m[8 * q + 4], m[8 * q + 5], m[8 * q + 6], m[8 * q + 7], g);
            const uint64_t tx = transpose8x8(((uint64_t)hi << 32) | lo);
#pragma unroll
            for (int p = 0; p < 8; ++p) P[p] |= (uint32_t)((tx >> (8 * p)) & 0xffu) << (8 * q);
          }
#pragma unroll
          for (int p = 0; p < 8; ++p)
            if (8 * g + p < L) U[mw + 1 + 8 * g + p] = P[p];
        }
      }
      __syncwarp();
      for (uint32_t k = lane; k < warp_words; k += 32) payload[w0 + k] = U[k];
    }
    __syncthreads();  // (s_tile, s_words, s_before and the stage are reused)
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

// Lane j of a warp decodes block b0 + j on its own: the sign word and the L
// bit planes (plane p holds bit p of the block's 32 |deltas|) become the 32
// |deltas| by 8 x 8 bit transposes (planes 8g .. 8g + 7 of values 8t ..
// 8t + 7 in one 64-bit word, one byte per plane, transposed into one byte per
// value), the signs are applied and the deltas summed in order (the codes), and
// the values fl32(s q) leave through a shared-memory tile as coalesced rows of
// the warp's 32 blocks.  No cross-lane traffic besides the tile.
//
// The stream is checked here, before any payload word is read, so that the
// host waits only once, after this kernel: the magic, n, every L <= 31 (the
// size pass) and the payload within in_bytes; otherwise block 0 marks the
// stream malformed and nothing is written.  Every block reads the same words,
// so all of them take the same decision.
__global__ void __launch_bounds__(kCodecThreads) lamz_decode_kernel(
    const uint8_t *in, uint64_t in_bytes, uint64_t head, const uint32_t *offs, int64_t nb,
    int64_t n, CodecStatus *st, float *__restrict__ out) {
  __shared__ float tile[kWarps][32][33];
  uint64_t nn = 0;
  for (int k = 0; k < 8; ++k) nn |= (uint64_t)__ldg(in + 4 + k) << (8 * k);
  const bool magic = __ldg(in) == 'L' && __ldg(in + 1) == 'A' && __ldg(in + 2) == 'M' &&
                     __ldg(in + 3) == 'Z';
  if (!magic || (int64_t)nn != n || *(volatile uint32_t *)&st->bad != 0u ||
      head + *(volatile uint32_t *)&st->total > in_bytes) {
    if (blockIdx.x == 0 && threadIdx.x == 0) atomicOr(&st->bad, 2u);
    return;
  }
  uint32_t sbits = 0;
  for (int k = 0; k < 4; ++k) sbits |= (uint32_t)__ldg(in + 12 + k) << (8 * k);
  const float s = __uint_as_float(sbits);
  const uint8_t *hdr = in + 16;
  const uint32_t *payload = reinterpret_cast<const uint32_t *>(in + head);
  const int lane = threadIdx.x & 31, wi = threadIdx.x >> 5;
  float(*T)[33] = tile[wi];
  const int64_t gw = (int64_t)blockIdx.x * kWarps + wi;
  const int64_t nw = (int64_t)gridDim.x * kWarps;
  for (int64_t b0 = gw * 32; b0 < nb; b0 += nw * 32) {
    const int64_t b = b0 + lane;
    const bool has = b < nb;
    const int L = has ? min((int)hdr[b], 31) : 0;
    const uint32_t *w = payload + (has ? offs[b] / 4 : 0);
    uint32_t m[32];
    uint32_t sign = 0u;
    if (L > 0) {
      sign = __ldg(w);
      {  // planes 0 .. 7 give the low byte of every magnitude
        uint32_t P[8];
#pragma unroll
        for (int p = 0; p < 8; ++p) P[p] = p < L ? __ldg(w + 1 + p) : 0u;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const uint32_t sel = (uint32_t)t | ((uint32_t)(4 + t) << 4);
          const uint32_t lo = __byte_perm(__byte_perm(P[0], P[1], sel),
                                          __byte_perm(P[2], P[3], sel), 0x5410);
          const uint32_t hi = __byte_perm(__byte_perm(P[4], P[5], sel),
                                          __byte_perm(P[6], P[7], sel), 0x5410);
          const uint64_t x = transpose8x8(((uint64_t)hi << 32) | lo);
          const uint32_t vlo = (uint32_t)x, vhi = (uint32_t)(x >> 32);
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            m[8 * t + c] = __byte_perm(vlo, 0u, 0x4440u | (uint32_t)c);
            m[8 * t + 4 + c] = __byte_perm(vhi, 0u, 0x4440u | (uint32_t)c);
          }
        }
      }
      for (int g = 1; 8 * g < L; ++g) {  // planes 8 g .. 8 g + 7: byte g
        uint32_t P[8];
#pragma unroll
        for (int p = 0; p < 8; ++p) P[p] = 8 * g + p < L ? __ldg(w + 1 + 8 * g + p) : 0u;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          // byte t of planes (0, 1), (2, 3), ... side by side, then four to a word
          const uint32_t sel = (uint32_t)t | ((uint32_t)(4 + t) << 4);
          const uint32_t lo = __byte_perm(__byte_perm(P[0], P[1], sel),
                                          __byte_perm(P[2], P[3], sel), 0x5410);
          const uint32_t hi = __byte_perm(__byte_perm(P[4], P[5], sel),
                                          __byte_perm(P[6], P[7], sel), 0x5410);
          const uint64_t x = transpose8x8(((uint64_t)hi << 32) | lo);
          const uint32_t vlo = (uint32_t)x, vhi = (uint32_t)(x >> 32);
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            m[8 * t + c] |= ((vlo >> (8 * c)) & 0xffu) << (8 * g);
            m[8 * t + 4 + c] |= ((vhi >> (8 * c)) & 0xffu) << (8 * g);
          }
        }
      }
    } else {
#pragma unroll
      for (int i = 0; i < 32; ++i) m[i] = 0u;
    }
    int32_t q = 0;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      q += ((sign >> i) & 1u) ? -(int32_t)m[i] : (int32_t)m[i];
      T[lane][i] = __fmul_rn(s, (float)q);
    }
    __syncwarp();
#pragma unroll 4
    for (int k = 0; k < 32; ++k) {
      const int64_t i = (b0 + k) * 32 + lane;
      if (b0 + k < nb && i < n) out[i] = T[k][lane];
    }
    __syncwarp();
  }
}

unsigned decode_grid(int64_t nb, int sms) {
  int64_t g = cdiv(nb, (int64_t)kWarps * 32);
  if (g > (int64_t)sms * 4) g = (int64_t)sms * 4;  // (4 resident per SM: 63 registers)
  return (unsigned)(g < 1 ? 1 : g);
}

// A thread per block (sizing pass, header check).
unsigned codec_grid(int64_t nb, int sms) {
  int64_t g = cdiv(nb, (int64_t)kCodecThreads);
  if (g > (int64_t)sms * 4) g = (int64_t)sms * 4;
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
                                 bool *fits, bool *nonfinite, bool *timed_out) {
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
  // tile states and the ticket, in the sizes region (4 (nb + 1) bytes, at
  // least 8 per tile of 256 blocks plus 4)
  const int64_t ntiles = cdiv(nb, (int64_t)kCompWarps * 32);
  unsigned long long *tiles = reinterpret_cast<unsigned long long *>(sizes);
  unsigned int *ticket = reinterpret_cast<unsigned int *>(tiles + ntiles);
  (void)sums;
  e = cudaMemsetAsync(tiles, 0, (size_t)ntiles * 8 + 4, stream);
  if (e != cudaSuccess) return e;
  // test hooks (unset in normal use): LAM_TEST_WAIT_CYCLES=<n> gives the
  // look-backs a budget of n SM cycles, LAM_TEST_STALL=1 keeps tile 0 from
  // publishing, so that they run out
  const char *hw = getenv("LAM_TEST_WAIT_CYCLES");
  const char *hs = getenv("LAM_TEST_STALL");
  const long long budget = (hw && *hw) ? (long long)strtoull(hw, nullptr, 10) : 0;
  const int stall = (hs && strcmp(hs, "1") == 0) ? 1 : 0;
  const bool vec = (reinterpret_cast<uintptr_t>(x) & 15u) == 0;
  auto kern = vec ? lamz_compress_kernel<true, kCompWarps> : lamz_compress_kernel<false, kCompWarps>;
  int64_t grid = ntiles < (int64_t)sms * 8 ? ntiles : (int64_t)sms * 8;
  kern<<<(unsigned)(grid < 1 ? 1 : grid), kCompWarps * 32, 0, stream>>>(
      x, n, rel, st, out + 16, nb, reinterpret_cast<uint32_t *>(out + head),
      reinterpret_cast<uint32_t *>(out), (uint64_t)head, (uint64_t)cap, tiles, ticket, ntiles,
      budget > 0 ? budget : kLookBackCycles, stall);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  CodecStatus h;  // one wait, after the stream is written
  e = read_back(&h, st, sizeof(h), stream);
  if (e != cudaSuccess) return e;
  *nonfinite = (h.flags & kFlagNonfinite) != 0;
  *timed_out = (h.flags & kFlagTimeout) != 0;
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
  cudaError_t e = cudaMemsetAsync(st, 0, sizeof(CodecStatus), stream);
  if (e != cudaSuccess) return e;
  lamz_dsize_kernel<<<codec_grid(nb, sms), 256, 0, stream>>>(in + 16, nb, sizes, st);
  e = scan_u32(sizes, nb, sums, &st->total, stream);
  if (e != cudaSuccess) return e;
  lamz_decode_kernel<<<decode_grid(nb, sms), kCodecThreads, 0, stream>>>(
      in, (uint64_t)in_bytes, (uint64_t)head, sizes, nb, n, st, out);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  CodecStatus h;  // one wait, after the decode
  e = read_back(&h, st, sizeof(h), stream);
  if (e != cudaSuccess) return e;
  *bad = h.bad != 0;
  return cudaSuccess;
}

}  // namespace lam
