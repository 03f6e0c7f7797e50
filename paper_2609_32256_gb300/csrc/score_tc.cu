// score_tc.cu -- exact search on the codes for query batches large enough to
// make the score a dense contraction (Sec. "Brute-force scan crossover": the
// scan is a matrix product once several queries share it), on the 5th-gen
// tensor cores (tcgen05) with accumulators in tensor memory.
//
// Exactness.  Codes are integers with |c| <= 2048, exact in fp16.  Each query
// is scaled by a power of two 2^e (max|q| 2^e in [2^14, 2^15)) and split into
// two fp16 terms hi + lo with |q 2^e - hi - lo| <= 2^-22 |q 2^e|.  Both terms
// are multiplied by the same fp16 code tile and accumulated in fp32 in TMEM:
//   acc = sum_d (hi_d + lo_d) c_d  ~=  2^e sum_d q_d c_d,
// every product being exact in fp32.  The score is then formed from acc*2^-e
// exactly as the CUDA-core paths form it.
//
// CTA: 128 queries (MMA M) x a contiguous range of 256-row tiles (MMA N),
// K = 32 fp16 per pipeline stage.  Warp roles (320 threads):
//   warp 0      TMA producer: query hi/lo tiles (64B swizzle) and raw codes;
//   warp 1      TMEM allocation; one lane issues tcgen05.mma (2 K-steps x
//               hi/lo per stage) and commits stage/accumulator barriers;
//   warps 2-5   convert raw int8/int16 codes to fp16 in the UMMA K-major
//               64B-swizzled layout, and sum c^2 per row for cosine / L2;
//   warps 6-9   epilogue: tcgen05.ld of the 128x256 fp32 accumulator (double
//               buffered, 2 x 256 TMEM columns), scores, per-query top-k.
// Every wait is bounded; a timeout records LAM_ERR_TIMEOUT and unwinds.
#include "score_common.cuh"

#include <cstring>

namespace lam {

namespace {

constexpr int kBM = 128;        // queries per CTA (MMA M)
constexpr int kBN = 256;        // code rows per tile (MMA N)
constexpr int kBK = 32;         // fp16 per stage along D (64-byte rows)
constexpr int kUmmaK = 16;      // K of one kind::f16 MMA
constexpr int kTcThreads = 320;
constexpr int kABytes = kBM * kBK * 2;    // one of hi / lo: 8 KB
constexpr int kB16Bytes = kBN * kBK * 2;  // converted codes: 16 KB
constexpr uint32_t kTmemCols = 512;       // two 256-column accumulators
constexpr int kMaxDynSmem = 232448;       // 227 KB
constexpr int kTcMaxK = 128;

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
// K-major, N = 256, M = 128.
constexpr uint32_t kIdesc = (1u << 4) | (0u << 7) | (0u << 10) | ((uint32_t)(kBN >> 3) << 17) |
                            ((uint32_t)(kBM >> 4) << 24);

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

struct TcLayout {
  int ns;
  int stage_bytes;
  int raw_bytes;
  size_t lists_off, cc_off, bar_off, smem_bytes;
};

inline TcLayout tc_layout(int width, int k) {
  TcLayout L;
  L.raw_bytes = kBN * kBK * width;
  L.stage_bytes = 2 * kABytes + kB16Bytes + L.raw_bytes;
  const size_t lists = (size_t)kBM * k * 8;
  const size_t cc = 2 * kBN * 4;
  const size_t fixed = lists + cc + 8 * 64 + 1024;  // barriers, slots, alignment slack
  int ns = (int)((kMaxDynSmem - fixed) / L.stage_bytes);
  if (ns > 6) ns = 6;
  L.ns = ns;
  L.lists_off = (size_t)ns * L.stage_bytes;
  L.cc_off = L.lists_off + lists;
  L.bar_off = L.cc_off + cc;
  L.smem_bytes = L.bar_off + 8 * 64 + 1024;
  return L;
}

template <int W>
__global__ void __launch_bounds__(kTcThreads, 1)
    score_tc_kernel(const __grid_constant__ CUtensorMap qmap,
                    const __grid_constant__ CUtensorMap cmap, ScoreArgs a, int ns,
                    int stage_bytes, int lists_off, int cc_off, int bar_off) {
  extern __shared__ uint8_t tc_smem_raw[];
  // 1024-byte alignment for the swizzled tiles (address bits drive the swizzle)
  const uint32_t base_u32 = smem_u32(tc_smem_raw);
  uint8_t *smem = tc_smem_raw + (((base_u32 + 1023u) & ~1023u) - base_u32);
  uint64_t *lists = reinterpret_cast<uint64_t *>(smem + lists_off);
  float *ccbuf = reinterpret_cast<float *>(smem + cc_off);
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + bar_off);
  uint64_t *conv = full + ns;
  uint64_t *empty = conv + ns;
  uint64_t *accf = empty + ns;
  uint64_t *acce = accf + 2;
  uint64_t *ccf = acce + 2;
  uint64_t *cce = ccf + 2;
  uint64_t *done = cce + 2;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qb = blockIdx.y;
  const int64_t n_tiles = (a.N + kBN - 1) / kBN;
  const int64_t tb = (int64_t)blockIdx.x * n_tiles / gridDim.x;
  const int64_t te = (int64_t)(blockIdx.x + 1) * n_tiles / gridDim.x;
  const int ntl = (int)(te - tb);
  const int nk = (a.D + kBK - 1) / kBK;
  const bool need_cc = a.metric != LAM_METRIC_IP;
  const int raw_off = 2 * kABytes + kB16Bytes;

  if (threadIdx.x == 0) {
    for (int s = 0; s < ns; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&conv[s], 128);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], 128);
      mbar_init(&ccf[b], 128);
      mbar_init(&cce[b], 128);
    }
    mbar_init(done, 1);
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 1) tmem_alloc(tmem_slot, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------ TMA producer -------
    if (lane == 0) {
      int it = 0, issued = 0;
      bool ok = true;
      for (int lt = 0; lt < ntl && ok; ++lt) {
        const int tile = (int)(tb + lt);
        for (int kc = 0; kc < nk; ++kc, ++it) {
          const int s = it % ns, r = it / ns;
          if (r > 0 && !mbar_wait(&empty[s], (r - 1) & 1, abort_flag, a.gflags)) {
            ok = false;
            break;
          }
          uint8_t *st = smem + (size_t)s * stage_bytes;
          mbar_arrive_expect_tx(&full[s], 2 * kABytes + kBN * kBK * W);
          tma_load_2d(st, &qmap, kc * kBK, qb * kBM, &full[s]);
          tma_load_2d(st + kABytes, &qmap, kc * kBK, (int)a.Bpad + qb * kBM, &full[s]);
          tma_load_2d(st + raw_off, &cmap, kc * kBK, tile * kBN, &full[s]);
          issued = it + 1;
        }
      }
      for (int t = max(0, issued - ns); t < issued; ++t) drain_wait_tc(&full[t % ns], (t / ns) & 1);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer ---------
    if (lane == 0) {
      int it = 0;
      bool ok = true;
      for (int lt = 0; lt < ntl && ok; ++lt) {
        const int buf = lt & 1, u = lt >> 1;
        if (u > 0 && !mbar_wait(&acce[buf], (u - 1) & 1, abort_flag, a.gflags)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(buf * kBN);
        for (int kc = 0; kc < nk; ++kc, ++it) {
          const int s = it % ns, r = it / ns;
          if (!mbar_wait(&conv[s], r & 1, abort_flag, a.gflags) ||
              !mbar_wait(&full[s], r & 1, abort_flag, a.gflags)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = smem_u32(smem + (size_t)s * stage_bytes);
          const uint64_t ahi = desc_sw64(st), alo = desc_sw64(st + kABytes),
                         bd = desc_sw64(st + 2 * kABytes);
#pragma unroll
          for (int j = 0; j < kBK / kUmmaK; ++j) {
            const uint64_t koff = (uint64_t)((j * kUmmaK * 2) >> 4);
            umma_f16(d_tmem, ahi + koff, bd + koff, kIdesc, (kc > 0 || j > 0) ? 1u : 0u);
            umma_f16(d_tmem, alo + koff, bd + koff, kIdesc, 1u);
          }
          umma_commit(&empty[s]);
        }
        if (ok) umma_commit(&accf[buf]);
      }
      umma_commit(done);
      drain_wait_tc(done, 0);
    }
  } else if (warp < 6) {
    // ------------------------------------------------ converters ---------
    const int ct = threadIdx.x - 64;  // 0..127
    constexpr int kTasks = (W == 1) ? 4 : 8;
    const __half2 bias = __float2half2_rn(1152.0f);
    int it = 0;
    bool ok = true;
    float amax = 0.0f;
    for (int lt = 0; lt < ntl && ok; ++lt) {
      const int buf = lt & 1, u = lt >> 1;
      float ccp[kTasks];
#pragma unroll
      for (int i = 0; i < kTasks; ++i) ccp[i] = 0.0f;
      for (int kc = 0; kc < nk; ++kc, ++it) {
        const int s = it % ns, r = it / ns;
        if (!mbar_wait(&full[s], r & 1, abort_flag, a.gflags)) {
          ok = false;
          break;
        }
        uint8_t *st = smem + (size_t)s * stage_bytes;
        const uint8_t *raw = st + raw_off;
        uint8_t *b16 = st + 2 * kABytes;
#pragma unroll
        for (int i = 0; i < kTasks; ++i) {
          const int task = ct + 128 * i;
          if (W == 1) {
            const int row = task >> 1, h = task & 1;
            const uint4 v = *reinterpret_cast<const uint4 *>(raw + row * 32 + h * 16);
            const uint32_t w[4] = {v.x, v.y, v.z, v.w};
            uint32_t o[8];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const uint32_t x = w[j] ^ 0x80808080u;
              // fp16 bits 0x64uu = 1024 + u with u = code + 128; minus 1152 = code
              o[2 * j] = h2_as_u32(__hsub2(u32_as_h2(__byte_perm(x, 0x64646464u, 0x5140)), bias));
              o[2 * j + 1] = h2_as_u32(__hsub2(u32_as_h2(__byte_perm(x, 0x64646464u, 0x7362)), bias));
            }
            const int sw = (row >> 1) & 3;
            uint8_t *rowp = b16 + row * 64;
            *reinterpret_cast<uint4 *>(rowp + (((2 * h) ^ sw) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
            *reinterpret_cast<uint4 *>(rowp + (((2 * h + 1) ^ sw) << 4)) = make_uint4(o[4], o[5], o[6], o[7]);
            if (need_cc) {
              int c2 = 0;
#pragma unroll
              for (int j = 0; j < 4; ++j) c2 = __dp4a((int)w[j], (int)w[j], c2);
              ccp[i] += (float)c2;
            }
          } else {
            const int row = task >> 2, qt = task & 3;
            const uint4 v = *reinterpret_cast<const uint4 *>(raw + row * 64 + qt * 16);
            const uint32_t w[4] = {v.x ^ 0x80008000u, v.y ^ 0x80008000u, v.z ^ 0x80008000u,
                                   v.w ^ 0x80008000u};
            uint32_t o[4];
            float c2 = 0.0f;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const float f0 = __int_as_float(__byte_perm(w[j], 0x4B000000u, 0x7410)) - 8421376.0f;
              const float f1 = __int_as_float(__byte_perm(w[j], 0x4B000000u, 0x7432)) - 8421376.0f;
              amax = fmaxf(amax, fmaxf(fabsf(f0), fabsf(f1)));
              c2 = fmaf(f0, f0, fmaf(f1, f1, c2));
              o[j] = h2_as_u32(__floats2half2_rn(f0, f1));
            }
            const int sw = (row >> 1) & 3;
            *reinterpret_cast<uint4 *>(b16 + row * 64 + ((qt ^ sw) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
            if (need_cc) ccp[i] += c2;
          }
        }
        fence_proxy_async_smem();
        mbar_arrive(&conv[s]);
      }
      if (!ok) break;
      if (need_cc) {
        if (u > 0 && !mbar_wait(&cce[buf], (u - 1) & 1, abort_flag, a.gflags)) break;
#pragma unroll
        for (int i = 0; i < kTasks; ++i) {
          const int task = ct + 128 * i;
          float t = ccp[i] + __shfl_xor_sync(0xffffffffu, ccp[i], 1);
          if (W == 2) t += __shfl_xor_sync(0xffffffffu, t, 2);
          const bool writer = (W == 1) ? ((task & 1) == 0) : ((task & 3) == 0);
          if (writer) ccbuf[buf * kBN + (W == 1 ? task >> 1 : task >> 2)] = t;
        }
        mbar_arrive(&ccf[buf]);
      }
    }
    if (W == 2 && amax > 2048.0f) atomicOr(a.gflags, kFlagRange);
  } else {
    // ------------------------------------------------ epilogue -----------
    const int quad = warp & 3;
    const int m = quad * 32 + lane;  // TMEM lane = query within the block
    const int64_t qidx = (int64_t)qb * kBM + m;
    const bool qvalid = qidx < a.B;
    const int k = a.k;
    const bool desc = a.metric != LAM_METRIC_L2;
    const float s = a.s, s2 = a.s * a.s;
    float pw = 0.0f, qn = 0.0f, qq = 0.0f;
    if (qvalid) {
      const float4 qi = reinterpret_cast<const float4 *>(
          static_cast<const uint8_t *>(a.qprep) + (size_t)2 * a.Bpad * a.D * 2)[qidx];
      pw = qi.x;
      qn = qi.y;
      qq = qi.z;
    }
    for (int i = 0; i < k; ++i) lists[(size_t)i * kBM + m] = kSentinel;
    uint64_t thr = kSentinel;
    for (int lt = 0; lt < ntl; ++lt) {
      const int buf = lt & 1, u = lt >> 1;
      if (!warp_wait(&accf[buf], u & 1, abort_flag, a.gflags)) break;
      if (need_cc && !warp_wait(&ccf[buf], u & 1, abort_flag, a.gflags)) break;
      tc_fence_after();
      const int64_t row0 = (tb + lt) * kBN;
      const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(buf * kBN);
#pragma unroll 1
      for (int c = 0; c < kBN / 32; ++c) {
        uint32_t v[32];
        tmem_ld32(taddr + c * 32, v);
        if (qvalid) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int64_t row = row0 + c * 32 + j;
            if (row < a.N) {
              const float acc = __uint_as_float(v[j]) * pw;
              const float cc = need_cc ? ccbuf[buf * kBN + c * 32 + j] : 0.0f;
              const float sc = finish_score(a.metric, acc, cc, s, s2, qq, qn);
              const uint64_t key = make_key(sc, (uint32_t)row, desc);
              if (key < thr) {
                int p = k - 1;
                while (p > 0) {
                  const uint64_t prev = lists[(size_t)(p - 1) * kBM + m];
                  if (prev <= key) break;
                  lists[(size_t)p * kBM + m] = prev;
                  --p;
                }
                lists[(size_t)p * kBM + m] = key;
                thr = lists[(size_t)(k - 1) * kBM + m];
              }
            }
          }
        }
      }
      tc_fence_before();
      mbar_arrive(&acce[buf]);
      if (need_cc) mbar_arrive(&cce[buf]);
    }
    if (qvalid) {
      uint64_t *out = a.partial + ((size_t)blockIdx.x * a.B + qidx) * k;
      for (int i = 0; i < k; ++i) out[i] = lists[(size_t)i * kBM + m];
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// Query preparation: per query the power-of-two scale, the fp16 hi/lo split
// (rows [0, Bpad) hold hi, rows [Bpad, 2 Bpad) hold lo; padding rows are zero)
// and (2^-e, ||q||, ||q||^2).  One warp per query.
__global__ void __launch_bounds__(256) qprep_kernel(const float *__restrict__ q, int64_t B, int D,
                                                    int64_t Bpad, __half *__restrict__ qh,
                                                    float4 *__restrict__ qinfo) {
  const int64_t b = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (b >= Bpad) return;
  __half *hi = qh + b * D;
  __half *lo = qh + (Bpad + b) * D;
  if (b >= B) {
    for (int d = lane; d < D; d += 32) {
      hi[d] = __float2half_rn(0.0f);
      lo[d] = __float2half_rn(0.0f);
    }
    if (lane == 0) qinfo[b] = make_float4(0.f, 0.f, 0.f, 0.f);
    return;
  }
  const float *qr = q + b * D;
  float mx = 0.0f, qq = 0.0f;
  for (int d = lane; d < D; d += 32) {
    const float v = qr[d];
    mx = fmaxf(mx, fabsf(v));
    qq = fmaf(v, v, qq);
  }
  for (int off = 16; off > 0; off >>= 1) {
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    qq += __shfl_xor_sync(0xffffffffu, qq, off);
  }
  int e = 0;
  if (mx > 0.0f) {
    int ex;
    frexpf(mx, &ex);  // mx = f * 2^ex, f in [0.5, 1)
    e = 15 - ex;      // mx * 2^e in [2^14, 2^15)
    e = max(-126, min(126, e));
  }
  const float sc = ldexpf(1.0f, e);
  for (int d = lane; d < D; d += 32) {
    const float v = qr[d] * sc;
    const __half h = __float2half_rn(v);
    hi[d] = h;
    lo[d] = __float2half_rn(v - __half2float(h));
  }
  if (lane == 0) qinfo[b] = make_float4(ldexpf(1.0f, -e), sqrtf(qq), qq, 0.0f);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (fn == nullptr) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult qr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &qr) == cudaSuccess &&
        qr == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

bool make_map_2d(CUtensorMap *map, CUtensorMapDataType dt, const void *base, uint64_t inner,
                 uint64_t rows, uint64_t row_bytes, uint32_t box_inner, uint32_t box_rows,
                 CUtensorMapSwizzle swz) {
  EncodeTiledFn fn = encode_fn();
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, dt, 2, const_cast<void *>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

int gcd_i(int x, int y) {
  while (y) {
    int t = x % y;
    x = y;
    y = t;
  }
  return x;
}

}  // namespace

bool tensor_fits(int width, int k) {
  if (k > kTcMaxK || (width != 1 && width != 2)) return false;
  return tc_layout(width, k).ns >= 2;
}

int tensor_splits(int64_t B, int64_t N, int sms) {
  const int64_t nqb = (B + kBM - 1) / kBM;
  const int64_t n_tiles = (N + kBN - 1) / kBN;
  // splits x query blocks a multiple of the SM count: whole waves of CTAs
  int64_t ns = sms / gcd_i(sms, (int)(nqb % (1 << 30)));
  if (ns > n_tiles) ns = n_tiles;
  if (ns < 1) ns = 1;
  return (int)ns;
}

size_t tensor_qprep_bytes(int64_t Bpad, int D) {
  return (size_t)2 * Bpad * D * 2 + (size_t)Bpad * 16;
}

cudaError_t launch_score_tensor(const ScoreArgs &a, cudaStream_t st) {
  if (a.k > kTcMaxK || (a.width != 1 && a.width != 2)) return cudaErrorInvalidValue;
  const TcLayout L = tc_layout(a.width, a.k);
  if (L.ns < 2) return cudaErrorInvalidValue;
  __half *qh = static_cast<__half *>(a.qprep);
  float4 *qinfo = reinterpret_cast<float4 *>(static_cast<uint8_t *>(a.qprep) +
                                             (size_t)2 * a.Bpad * a.D * 2);
  qprep_kernel<<<(unsigned)((a.Bpad + 7) / 8), 256, 0, st>>>(a.queries, a.B, a.D, a.Bpad, qh,
                                                             qinfo);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;

  CUtensorMap qmap, cmap;
  if (!make_map_2d(&qmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, qh, (uint64_t)a.D,
                   (uint64_t)(2 * a.Bpad), (uint64_t)a.D * 2, kBK, kBM,
                   CU_TENSOR_MAP_SWIZZLE_64B))
    return cudaErrorInvalidValue;
  if (!make_map_2d(&cmap,
                   a.width == 1 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_UINT16,
                   a.codes, (uint64_t)a.D, (uint64_t)a.N, (uint64_t)a.D * a.width, kBK, kBN,
                   CU_TENSOR_MAP_SWIZZLE_NONE))
    return cudaErrorInvalidValue;

  const dim3 grid((unsigned)a.n_lists, (unsigned)(a.Bpad / kBM));
  if (a.width == 1) {
    e = cudaFuncSetAttribute(score_tc_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)L.smem_bytes);
    if (e != cudaSuccess) return e;
    score_tc_kernel<1><<<grid, kTcThreads, L.smem_bytes, st>>>(
        qmap, cmap, a, L.ns, L.stage_bytes, (int)L.lists_off, (int)L.cc_off, (int)L.bar_off);
  } else {
    e = cudaFuncSetAttribute(score_tc_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)L.smem_bytes);
    if (e != cudaSuccess) return e;
    score_tc_kernel<2><<<grid, kTcThreads, L.smem_bytes, st>>>(
        qmap, cmap, a, L.ns, L.stage_bytes, (int)L.lists_off, (int)L.cc_off, (int)L.bar_off);
  }
  return cudaGetLastError();
}

}  // namespace lam
