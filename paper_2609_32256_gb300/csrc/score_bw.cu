// score_bw.cu -- exact search on the codes for small query batches (the
// matrix-vector regime of Sec. "Brute-force scan crossover"), the generic
// fallback for any shape, and the final top-k merge.
//
// Bandwidth kernel: one persistent CTA per SM streams a contiguous range of
// code rows through a ring of shared-memory stages filled by 1-D bulk copies
// (cp.async.bulk, completion on mbarriers).  Eight consumer warps each score
// whole rows: a lane owns eight consecutive coordinates per 256-coordinate
// chunk, converts the codes to fp32 exactly (byte-permute into the mantissa of
// 2^23, then one subtraction), multiplies by the query held in registers, and
// the warp sums with shuffles.  Each warp keeps its top-k in registers (one
// key per lane per 32 entries); the CTA merges its eight lists by rank and
// writes one partial list per query.  Work per element: a few integer/FP
// instructions, so the kernel is bound by HBM at width bytes per element.
#include "score_common.cuh"

#include <type_traits>

namespace lam {

namespace {

constexpr int kBwWarps = 16;  // consumer warps; each scores two rows at a time
constexpr int kBwThreads = (kBwWarps + 1) * 32;
constexpr int kNchMax = 4;  // 8-coordinate vectors per lane per row: D <= 1024
constexpr int kRg = 4;      // rows per warp pass of the int8 single-query consumer
constexpr int kBwStageTarget = 48 * 1024;
constexpr int kBwSmemBudget = 200 * 1024;

// 8 codes -> 8 exact fp32 values as 4 packed pairs (element 2i in .x, 2i+1 in
// .y): the byte-permute places a biased code in the mantissa of 2^23, one
// packed subtraction removes 2^23 and the bias.
template <int W>
__device__ __forceinline__ void decode8x2(const uint8_t *p, float2 *f) {
  if (W == 1) {
    const uint2 v = *reinterpret_cast<const uint2 *>(p);
    const uint32_t a = v.x ^ 0x80808080u, b = v.y ^ 0x80808080u;
    // bits 0x4B0000uu = 2^23 + u with u = code + 128
    const float2 bias = make_float2(-8388736.0f, -8388736.0f);
    f[0] = __fadd2_rn(make_float2(__int_as_float(__byte_perm(a, 0x4B000000u, 0x7540)),
                                  __int_as_float(__byte_perm(a, 0x4B000000u, 0x7541))), bias);
    f[1] = __fadd2_rn(make_float2(__int_as_float(__byte_perm(a, 0x4B000000u, 0x7542)),
                                  __int_as_float(__byte_perm(a, 0x4B000000u, 0x7543))), bias);
    f[2] = __fadd2_rn(make_float2(__int_as_float(__byte_perm(b, 0x4B000000u, 0x7540)),
                                  __int_as_float(__byte_perm(b, 0x4B000000u, 0x7541))), bias);
    f[3] = __fadd2_rn(make_float2(__int_as_float(__byte_perm(b, 0x4B000000u, 0x7542)),
                                  __int_as_float(__byte_perm(b, 0x4B000000u, 0x7543))), bias);
  } else {
    const uint4 v = *reinterpret_cast<const uint4 *>(p);
    const uint32_t w[4] = {v.x ^ 0x80008000u, v.y ^ 0x80008000u, v.z ^ 0x80008000u,
                           v.w ^ 0x80008000u};
    // bits 0x4B00uuuu = 2^23 + u with u = code + 32768
    const float2 bias = make_float2(-8421376.0f, -8421376.0f);
#pragma unroll
    for (int j = 0; j < 4; ++j)
      f[j] = __fadd2_rn(make_float2(__int_as_float(__byte_perm(w[j], 0x4B000000u, 0x7410)),
                                    __int_as_float(__byte_perm(w[j], 0x4B000000u, 0x7432))), bias);
  }
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}

// Power of two that brings the largest |q| near 1, so that a query's squared
// norm neither underflows nor overflows in fp32 while it is summed (the norm
// itself is then rescaled exactly).
__device__ __forceinline__ float norm_scale(float mx) {
  if (!(mx > 0.0f) || !isfinite(mx)) return 1.0f;
  int ex;
  frexpf(mx, &ex);
  return ldexpf(1.0f, max(-126, min(126, -ex)));
}

// Sums a over the lanes 0-15 and b over the lanes 16-31 with one shared
// butterfly: lanes 0-15 end with sum(a), lanes 16-31 with sum(b).
__device__ __forceinline__ float pair_sum(float a, float b, int lane) {
  const bool lo = lane < 16;
  float keep = lo ? a : b;
  keep += __shfl_xor_sync(0xffffffffu, lo ? b : a, 16);
#pragma unroll
  for (int off = 8; off > 0; off >>= 1) keep += __shfl_xor_sync(0xffffffffu, keep, off);
  return keep;
}

// Warp sums of V values at once (V a power of two, <= 32): at each butterfly
// step a lane keeps one half of its values and sends the other half, so the
// V sums cost V - 1 + (5 - log2 V) shuffles instead of 5 V.  Afterwards lane L
// holds the warp total of value L >> (5 - log2 V).
template <int V>
__device__ __forceinline__ float warp_sums_transposed(float (&v)[V], int lane) {
  int n = V;
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    if (n > 1) {
      const int h = n / 2;
      const bool up = (lane & o) != 0;
#pragma unroll
      for (int i = 0; i < V / 2; ++i) {
        if (i < h) {
          const float send = up ? v[i] : v[i + h];
          const float keep = up ? v[i + h] : v[i];
          v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
      }
      n = h;
    } else {
      v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
    }
  }
  return v[0];
}

// Waits (bounded, ignoring the abort flag) until a phase that is known to be
// in flight completes; used only to drain copies before the CTA exits.
__device__ __forceinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
  long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > kWaitCycles) break;
}

struct BwShape {
  int tr;           // rows per stage (multiple of the consumer warp count)
  int ns;           // stages
  int stage_bytes;  // tr * D * width, a multiple of 16
};

inline BwShape bw_shape(int D, int width) {
  const int row = D * width;
  int tr = (kBwStageTarget / (row * 2 * kBwWarps)) * 2 * kBwWarps;
  if (tr < 2 * kBwWarps) tr = 2 * kBwWarps;
  BwShape sh;
  sh.tr = tr;
  sh.stage_bytes = tr * row;
  sh.ns = kBwSmemBudget / sh.stage_bytes;
  if (sh.ns > 8) sh.ns = 8;
  if (sh.ns < 2) sh.ns = 2;
  return sh;
}

template <int W, int QB, int KPL, bool CC>
__global__ void __launch_bounds__(kBwThreads, 1)
    score_bw_kernel(ScoreArgs a, int tr, int ns, int stage_bytes, const QuantStatus *qst) {
  // status-driven call: only the variant of the codes' width runs
  if (qst != nullptr && (!status_ok(qst) || status_width(qst) != (uint32_t)W)) return;
  extern __shared__ __align__(1024) uint8_t smem[];
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + (size_t)ns * stage_bytes);
  uint64_t *empty = full + ns;
  volatile int *abort_flag = reinterpret_cast<volatile int *>(empty + ns);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t N = a.N;
  const int D = a.D;
  const int64_t r0 = (int64_t)blockIdx.x * N / gridDim.x;
  const int64_t r1 = (int64_t)(blockIdx.x + 1) * N / gridDim.x;
  const int64_t nrows = r1 - r0;
  const int ntiles = (int)((nrows + tr - 1) / tr);
  const size_t row_bytes = (size_t)D * W;

  if (threadIdx.x == 0) {
    for (int s = 0; s < ns; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kBwWarps);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();

  WarpList<KPL> lists[QB];
#pragma unroll
  for (int q = 0; q < QB; ++q) lists[q].init();

  if (warp == kBwWarps) {
    // ---------------- producer: one lane issues the bulk copies ----------
    if (lane == 0) {
      int issued = 0;
      const int nt = producers_stalled(a.gflags) ? 0 : ntiles;
      for (int t = 0; t < nt; ++t) {
        const int s = t % ns, r = t / ns;
        if (r > 0 && !mbar_wait(&empty[s], (r - 1) & 1, abort_flag, a.gflags)) break;
        const int64_t nr = min((int64_t)tr, nrows - (int64_t)t * tr);
        const uint32_t bytes = (uint32_t)(nr * row_bytes);
        mbar_arrive_expect_tx(&full[s], bytes);
        bulk_g2s(smem + (size_t)s * stage_bytes,
                 static_cast<const uint8_t *>(a.codes) + (r0 + (int64_t)t * tr) * row_bytes,
                 bytes, &full[s]);
        issued = t + 1;
      }
      for (int t = max(0, issued - ns); t < issued; ++t) drain_wait(&full[t % ns], (t / ns) & 1);
    }
  } else {
    // ---------------- consumers: two rows per warp at a time -------------
    const int nch = (D + 255) / 256;
    float2 qreg[QB][kNchMax][4];
    float qq[QB], qn[QB];
#pragma unroll
    for (int q = 0; q < QB; ++q) {
      const bool qv = q < a.B;
      float part = 0.0f;
#pragma unroll
      for (int j = 0; j < kNchMax; ++j) {
        const int e0 = (j * 32 + lane) * 8;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int d = e0 + 2 * t;
          const float v0 = (qv && j < nch && d < D) ? a.queries[(int64_t)q * D + d] : 0.0f;
          const float v1 = (qv && j < nch && d + 1 < D) ? a.queries[(int64_t)q * D + d + 1] : 0.0f;
          qreg[q][j][t] = make_float2(v0, v1);
          part = fmaf(v0, v0, fmaf(v1, v1, part));
        }
      }
      // the norm from the scaled query (range-safe), then ||q||^2
      float mx = 0.0f;
#pragma unroll
      for (int j = 0; j < kNchMax; ++j)
#pragma unroll
        for (int t = 0; t < 4; ++t)
          mx = fmaxf(mx, fmaxf(fabsf(qreg[q][j][t].x), fabsf(qreg[q][j][t].y)));
      const float ns = norm_scale(warp_max(mx));
      part = 0.0f;
#pragma unroll
      for (int j = 0; j < kNchMax; ++j)
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const float u0 = qreg[q][j][t].x * ns, u1 = qreg[q][j][t].y * ns;
          part = fmaf(u0, u0, fmaf(u1, u1, part));
        }
      qn[q] = sqrtf(warp_sum(part)) / ns;
      qq[q] = qn[q] * qn[q];
    }
    // int8 codes: the query as signed base-256 digits of round(q 2^e) with
    // max|q| 2^e in [2^21, 2^22), so that the products with the codes are
    // integer dot products (__dp4a) summed exactly per digit plane; the
    // query's rounding, |q 2^e - round(q 2^e)| <= 1/2, is the only error
    // besides the final fp32 sums (the tensor path's hi/lo split has 2^-22)
    uint32_t qdig[W == 1 ? QB : 1][W == 1 ? kNchMax : 1][3][2];
    float qinv[QB];
#pragma unroll
    for (int q = 0; q < QB; ++q) qinv[q] = 1.0f;
    if constexpr (W == 1) {
#pragma unroll
      for (int q = 0; q < QB; ++q) {
        float mx = 0.0f;
#pragma unroll
        for (int j = 0; j < kNchMax; ++j)
#pragma unroll
          for (int t = 0; t < 4; ++t)
            mx = fmaxf(mx, fmaxf(fabsf(qreg[q][j][t].x), fabsf(qreg[q][j][t].y)));
        mx = warp_max(mx);
        int e = 0;
        if (mx > 0.0f) {
          int ex;
          frexpf(mx, &ex);  // mx = f 2^ex, f in [0.5, 1)
          e = max(-126, min(126, 22 - ex));
        }
        const float sc = ldexpf(1.0f, e);
        qinv[q] = ldexpf(1.0f, -e);
#pragma unroll
        for (int j = 0; j < kNchMax; ++j)
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            uint32_t w0 = 0, w1 = 0, w2 = 0;
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              const float2 pr = qreg[q][j][2 * h + (t >> 1)];
              const int qi = __float2int_rn((t & 1) ? pr.y * sc : pr.x * sc);
              const int d2 = ((qi + 128) & 255) - 128;
              const int r1 = (qi - d2) >> 8;
              const int d1 = ((r1 + 128) & 255) - 128;
              const int d0 = (r1 - d1) >> 8;
              w0 |= ((uint32_t)d0 & 0xffu) << (8 * t);
              w1 |= ((uint32_t)d1 & 0xffu) << (8 * t);
              w2 |= ((uint32_t)d2 & 0xffu) << (8 * t);
            }
            qdig[q][j][0][h] = w0;
            qdig[q][j][1][h] = w1;
            qdig[q][j][2][h] = w2;
          }
      }
    }
    const bool desc = a.metric != LAM_METRIC_L2;
    const float s = a.s, s2 = a.s * a.s;
    float thr_s[QB];  // score of each list's k-th entry; rows come in increasing
                      // order, so only a strictly better score can enter
#pragma unroll
    for (int q = 0; q < QB; ++q) thr_s[q] = desc ? -INFINITY : INFINITY;

    for (int t = 0; t < ntiles; ++t) {
      const int st = t % ns, r = t / ns;
      if (!mbar_wait(&full[st], r & 1, abort_flag, a.gflags)) break;
      const int nr = (int)min((int64_t)tr, nrows - (int64_t)t * tr);
      const uint8_t *stage = smem + (size_t)st * stage_bytes;
      if constexpr (W == 1 && QB == 1) {
        // int8 codes, one query: kRg consecutive rows per warp pass.  All
        // their code words are loaded first, each lane sums its integer dot
        // products per row, and one transposed butterfly gives every row's
        // totals (and sum c^2) to its own lanes, which finish the scores in
        // parallel; one ballot then admits rows into the warp's list in row
        // order.
        constexpr int V = CC ? 2 * kRg : kRg;
        constexpr int lsh = CC ? 2 : 3;  // lane L ends with value L >> lsh
        for (int g0 = warp * kRg; g0 < nr; g0 += kBwWarps * kRg) {
          uint2 cw[kRg][kNchMax];
#pragma unroll
          for (int i = 0; i < kRg; ++i) {
            const uint8_t *pr = stage + (size_t)min(g0 + i, nr - 1) * row_bytes;
#pragma unroll
            for (int j = 0; j < kNchMax; ++j) {
              const int e0 = (j * 32 + lane) * 8;
              cw[i][j] = (j < nch && e0 < D) ? *reinterpret_cast<const uint2 *>(pr + e0)
                                             : make_uint2(0u, 0u);
            }
          }
          float v[V];
#pragma unroll
          for (int i = 0; i < kRg; ++i) {
            int d0 = 0, d1 = 0, d2 = 0, cc = 0;
#pragma unroll
            for (int j = 0; j < kNchMax; ++j) {
              if (j < nch) {  // (warp-uniform)
                const int wx = (int)cw[i][j].x, wy = (int)cw[i][j].y;
                d0 = __dp4a(wx, (int)qdig[0][j][0][0], __dp4a(wy, (int)qdig[0][j][0][1], d0));
                d1 = __dp4a(wx, (int)qdig[0][j][1][0], __dp4a(wy, (int)qdig[0][j][1][1], d1));
                d2 = __dp4a(wx, (int)qdig[0][j][2][0], __dp4a(wy, (int)qdig[0][j][2][1], d2));
                if constexpr (CC) cc = __dp4a(wx, wx, __dp4a(wy, wy, cc));
              }
            }
            v[i] = fmaf((float)d0, 65536.0f, fmaf((float)d1, 256.0f, (float)d2));
            if constexpr (CC) v[kRg + i] = (float)cc;
          }
          const float tot = warp_sums_transposed<V>(v, lane);
          const int i_row = (lane >> lsh) & (kRg - 1);
          const float cc = CC ? __shfl_xor_sync(0xffffffffu, tot, 16) : 0.0f;
          const float sc = finish_score(a.metric, tot * qinv[0], cc, s, s2, qq[0], qn[0]);
          const bool leader = (lane & ((1 << lsh) - 1)) == 0 && (!CC || lane < 16);
          unsigned pass = __ballot_sync(0xffffffffu, leader && g0 + i_row < nr &&
                                                         (desc ? sc > thr_s[0] : sc < thr_s[0]));
          while (pass) {
            const int l = __ffs(pass) - 1;
            pass &= pass - 1;
            const float sl = __shfl_sync(0xffffffffu, sc, l);
            if (!(desc ? sl > thr_s[0] : sl < thr_s[0])) continue;  // the list moved on
            const int64_t row = r0 + (int64_t)t * tr + g0 + ((l >> lsh) & (kRg - 1));
            lists[0].insert(make_key(sl, (uint32_t)row, desc), lane);
            const uint64_t kk = lists[0].kth(a.k);
            thr_s[0] = kk == kSentinel ? (desc ? -INFINITY : INFINITY)
                                       : rank_key32_score((uint32_t)(kk >> 32), desc);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[st]);
        continue;
      }
      for (int rr = warp; rr < nr; rr += 2 * kBwWarps) {
        const int rb = rr + kBwWarps;
        const bool has_b = rb < nr;
        const uint8_t *pa = stage + (size_t)rr * row_bytes;
        const uint8_t *pb = stage + (size_t)(has_b ? rb : rr) * row_bytes;
        // packed pairs: two partial sums per lane, FFMA2 / FADD2
        float2 acc_a[QB], acc_b[QB];
#pragma unroll
        for (int q = 0; q < QB; ++q) acc_a[q] = acc_b[q] = make_float2(0.0f, 0.0f);
        float2 cc_a = make_float2(0.0f, 0.0f), cc_b = make_float2(0.0f, 0.0f);
        if constexpr (W == 1) {
          // integer dot products per digit plane, exact in int32
          int ia[QB][3], ib[QB][3], ca = 0, cb = 0;
#pragma unroll
          for (int q = 0; q < QB; ++q)
#pragma unroll
            for (int p = 0; p < 3; ++p) ia[q][p] = ib[q][p] = 0;
#pragma unroll
          for (int j = 0; j < kNchMax; ++j) {
            const int e0 = (j * 32 + lane) * 8;
            if (j < nch && e0 < D) {
              const uint2 wa = *reinterpret_cast<const uint2 *>(pa + e0);
              const uint2 wb = *reinterpret_cast<const uint2 *>(pb + e0);
#pragma unroll
              for (int q = 0; q < QB; ++q)
#pragma unroll
                for (int p = 0; p < 3; ++p) {
                  ia[q][p] = __dp4a((int)wa.x, (int)qdig[q][j][p][0], ia[q][p]);
                  ia[q][p] = __dp4a((int)wa.y, (int)qdig[q][j][p][1], ia[q][p]);
                  ib[q][p] = __dp4a((int)wb.x, (int)qdig[q][j][p][0], ib[q][p]);
                  ib[q][p] = __dp4a((int)wb.y, (int)qdig[q][j][p][1], ib[q][p]);
                }
              if (CC) {
                ca = __dp4a((int)wa.x, (int)wa.x, ca);
                ca = __dp4a((int)wa.y, (int)wa.y, ca);
                cb = __dp4a((int)wb.x, (int)wb.x, cb);
                cb = __dp4a((int)wb.y, (int)wb.y, cb);
              }
            }
          }
#pragma unroll
          for (int q = 0; q < QB; ++q) {
            acc_a[q].x = fmaf((float)ia[q][0], 65536.0f, fmaf((float)ia[q][1], 256.0f,
                                                              (float)ia[q][2]));
            acc_b[q].x = fmaf((float)ib[q][0], 65536.0f, fmaf((float)ib[q][1], 256.0f,
                                                              (float)ib[q][2]));
          }
          cc_a.x = (float)ca;
          cc_b.x = (float)cb;
        }
#pragma unroll
        for (int j = 0; j < (W == 1 ? 0 : kNchMax); ++j) {
          const int e0 = (j * 32 + lane) * 8;
          if (j < nch && e0 < D) {
            float2 fa[4], fb[4];
            decode8x2<W>(pa + (size_t)e0 * W, fa);
            decode8x2<W>(pb + (size_t)e0 * W, fb);
#pragma unroll
            for (int q = 0; q < QB; ++q)
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                acc_a[q] = __ffma2_rn(qreg[q][j][u], fa[u], acc_a[q]);
                acc_b[q] = __ffma2_rn(qreg[q][j][u], fb[u], acc_b[q]);
              }
            if (CC)
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                cc_a = __ffma2_rn(fa[u], fa[u], cc_a);
                cc_b = __ffma2_rn(fb[u], fb[u], cc_b);
              }
          }
        }
        const float cc = CC ? pair_sum(cc_a.x + cc_a.y, cc_b.x + cc_b.y, lane) : 0.0f;
#pragma unroll
        for (int q = 0; q < QB; ++q) {
          const float acc =
              pair_sum(acc_a[q].x + acc_a[q].y, acc_b[q].x + acc_b[q].y, lane) * qinv[q];
          // lanes 0-15 hold row rr, lanes 16-31 row rb
          const float sc = finish_score(a.metric, acc, cc, s, s2, qq[q], qn[q]);
          const float sa = __shfl_sync(0xffffffffu, sc, 0);
          const float sb = __shfl_sync(0xffffffffu, sc, 16);
          if (q >= a.B) continue;
          if (desc ? sa > thr_s[q] : sa < thr_s[q]) {
            lists[q].insert(make_key(sa, (uint32_t)(r0 + (int64_t)t * tr + rr), desc), lane);
            const uint64_t kk = lists[q].kth(a.k);
            thr_s[q] = kk == kSentinel ? (desc ? -INFINITY : INFINITY)
                                       : rank_key32_score((uint32_t)(kk >> 32), desc);
          }
          if (has_b && (desc ? sb > thr_s[q] : sb < thr_s[q])) {
            lists[q].insert(make_key(sb, (uint32_t)(r0 + (int64_t)t * tr + rb), desc), lane);
            const uint64_t kk = lists[q].kth(a.k);
            thr_s[q] = kk == kSentinel ? (desc ? -INFINITY : INFINITY)
                                       : rank_key32_score((uint32_t)(kk >> 32), desc);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }
  }
  __syncthreads();  // every stage consumed and every copy drained: reuse them
  uint64_t *cand = reinterpret_cast<uint64_t *>(smem);
  if (warp < kBwWarps) {
#pragma unroll
    for (int q = 0; q < QB; ++q)
      lists[q].store(cand + ((size_t)q * kBwWarps + warp) * a.k, a.k, lane);
  }
  __syncthreads();
  // ---------------- CTA merge of the warp lists, per query -----------------
  for (int q = 0; q < QB && q < a.B; ++q)
    rank_merge(cand + (size_t)q * kBwWarps * a.k, kBwWarps, a.k,
               a.partial + ((size_t)blockIdx.x * a.B + q) * a.k, threadIdx.x, kBwThreads);
}

// ---------------------------------------------------------------------------
// Per-vector codecs for B <= 2: the same pipeline over the stored rows (int8
// codes with a scale and an offset per row, fp16 values, or sign bits with a
// scale per row).  The decoding moves into the per-row finish:
//   int8   q.xhat = scale (q.c) + offset sum(q),
//          ||xhat||^2 = D offset^2 + 2 scale offset sum(c) + scale^2 sum(c^2)
//          (q.c by __dp4a against the query's base-256 digits, as for Q_eps
//          int8 codes; sum(c) and sum(c^2) by __dp4a as well)
//   fp16   q.xhat with the values widened to fp32, ||xhat||^2 summed alongside
//   sign   q.xhat = alpha (2 sum_{bit set} q - sum(q)), ||xhat||^2 = D alpha^2
template <int FMT>
__host__ __device__ constexpr int rows_bytes_per_dim8() {  // bytes per 8 coordinates
  return FMT == LAM_ROWS_INT8 ? 8 : FMT == LAM_ROWS_FP16 ? 16 : 1;
}

template <int FMT, int QB, int KPL, bool CC>
__global__ void __launch_bounds__(kBwThreads, 1)
    score_bw_rows_kernel(ScoreArgs a, RowPtrs rp, int tr, int ns, int stage_bytes) {
  extern __shared__ __align__(1024) uint8_t smem[];
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + (size_t)ns * stage_bytes);
  uint64_t *empty = full + ns;
  volatile int *abort_flag = reinterpret_cast<volatile int *>(empty + ns);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t N = a.N;
  const int D = a.D;
  const int64_t r0 = (int64_t)blockIdx.x * N / gridDim.x;
  const int64_t r1 = (int64_t)(blockIdx.x + 1) * N / gridDim.x;
  const int64_t nrows = r1 - r0;
  const int ntiles = (int)((nrows + tr - 1) / tr);
  constexpr int B8 = rows_bytes_per_dim8<FMT>();
  const size_t row_bytes = (size_t)(D / 8) * B8;

  if (threadIdx.x == 0) {
    for (int s = 0; s < ns; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kBwWarps);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();

  WarpList<KPL> lists[QB];
#pragma unroll
  for (int q = 0; q < QB; ++q) lists[q].init();

  if (warp == kBwWarps) {
    if (lane == 0) {
      int issued = 0;
      const int nt = producers_stalled(a.gflags) ? 0 : ntiles;
      for (int t = 0; t < nt; ++t) {
        const int s = t % ns, r = t / ns;
        if (r > 0 && !mbar_wait(&empty[s], (r - 1) & 1, abort_flag, a.gflags)) break;
        const int64_t nr = min((int64_t)tr, nrows - (int64_t)t * tr);
        const uint32_t bytes = (uint32_t)(nr * row_bytes);
        mbar_arrive_expect_tx(&full[s], bytes);
        bulk_g2s(smem + (size_t)s * stage_bytes,
                 static_cast<const uint8_t *>(a.codes) + (r0 + (int64_t)t * tr) * row_bytes,
                 bytes, &full[s]);
        issued = t + 1;
      }
      for (int t = max(0, issued - ns); t < issued; ++t) drain_wait(&full[t % ns], (t / ns) & 1);
    }
  } else {
    const int nch = (D + 255) / 256;
    float2 qreg[QB][kNchMax][4];
    float qq[QB], qn[QB], qs[QB];
#pragma unroll
    for (int q = 0; q < QB; ++q) {
      const bool qv = q < a.B;
      float part = 0.0f, sum = 0.0f;
#pragma unroll
      for (int j = 0; j < kNchMax; ++j) {
        const int e0 = (j * 32 + lane) * 8;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int d = e0 + 2 * t;
          const float v0 = (qv && j < nch && d < D) ? a.queries[(int64_t)q * D + d] : 0.0f;
          const float v1 = (qv && j < nch && d + 1 < D) ? a.queries[(int64_t)q * D + d + 1] : 0.0f;
          qreg[q][j][t] = make_float2(v0, v1);
          part = fmaf(v0, v0, fmaf(v1, v1, part));
          sum += v0 + v1;
        }
      }
      // the norm from the scaled query (range-safe), then ||q||^2
      float mx = 0.0f;
#pragma unroll
      for (int j = 0; j < kNchMax; ++j)
#pragma unroll
        for (int t = 0; t < 4; ++t)
          mx = fmaxf(mx, fmaxf(fabsf(qreg[q][j][t].x), fabsf(qreg[q][j][t].y)));
      const float ns = norm_scale(warp_max(mx));
      part = 0.0f;
#pragma unroll
      for (int j = 0; j < kNchMax; ++j)
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const float u0 = qreg[q][j][t].x * ns, u1 = qreg[q][j][t].y * ns;
          part = fmaf(u0, u0, fmaf(u1, u1, part));
        }
      qn[q] = sqrtf(warp_sum(part)) / ns;
      qq[q] = qn[q] * qn[q];
      qs[q] = warp_sum(sum);
    }
    uint32_t qdig[FMT == LAM_ROWS_INT8 ? QB : 1][FMT == LAM_ROWS_INT8 ? kNchMax : 1][3][2];
    float qinv[QB];
#pragma unroll
    for (int q = 0; q < QB; ++q) qinv[q] = 1.0f;
    if constexpr (FMT == LAM_ROWS_INT8) {
#pragma unroll
      for (int q = 0; q < QB; ++q) {
        float mx = 0.0f;
#pragma unroll
        for (int j = 0; j < kNchMax; ++j)
#pragma unroll
          for (int t = 0; t < 4; ++t)
            mx = fmaxf(mx, fmaxf(fabsf(qreg[q][j][t].x), fabsf(qreg[q][j][t].y)));
        mx = warp_max(mx);
        int e = 0;
        if (mx > 0.0f) {
          int ex;
          frexpf(mx, &ex);
          e = max(-126, min(126, 22 - ex));
        }
        const float sc = ldexpf(1.0f, e);
        qinv[q] = ldexpf(1.0f, -e);
#pragma unroll
        for (int j = 0; j < kNchMax; ++j)
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            uint32_t w0 = 0, w1 = 0, w2 = 0;
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              const float2 pr = qreg[q][j][2 * h + (t >> 1)];
              const int qi = __float2int_rn((t & 1) ? pr.y * sc : pr.x * sc);
              const int d2 = ((qi + 128) & 255) - 128;
              const int r1 = (qi - d2) >> 8;
              const int d1 = ((r1 + 128) & 255) - 128;
              const int d0 = (r1 - d1) >> 8;
              w0 |= ((uint32_t)d0 & 0xffu) << (8 * t);
              w1 |= ((uint32_t)d1 & 0xffu) << (8 * t);
              w2 |= ((uint32_t)d2 & 0xffu) << (8 * t);
            }
            qdig[q][j][0][h] = w0;
            qdig[q][j][1][h] = w1;
            qdig[q][j][2][h] = w2;
          }
      }
    }
    const bool desc = a.metric != LAM_METRIC_L2;
    float thr_s[QB];
#pragma unroll
    for (int q = 0; q < QB; ++q) thr_s[q] = desc ? -INFINITY : INFINITY;
    // Per-row factors one row pair ahead: lanes 0-15 finish rows r0 + warp +
    // 32 i, lanes 16-31 rows r0 + warp + 16 + 32 i (tiles hold a multiple of
    // 32 rows), so the next factors are those of the row 32 further on.
    int64_t frow = r0 + warp + (lane >= 16 ? kBwWarps : 0);
    float f_sr = 1.0f, f_or = 0.0f;
    if (FMT != LAM_ROWS_FP16 && frow < r1) f_sr = rp.scale[frow];
    if (FMT == LAM_ROWS_INT8 && frow < r1) f_or = rp.offset[frow];
    // int8 rows, one query: the factors of the row this lane finishes in its
    // warp's next group of kRg rows (lane L finishes row (L >> lsh) % kRg)
    constexpr int kLsh = CC ? 1 : 3;
    const int g_row = (lane >> kLsh) & (kRg - 1);
    float p_sr = 1.0f, p_or = 0.0f;
    if (FMT == LAM_ROWS_INT8 && QB == 1) {
      const int64_t row = r0 + warp * kRg + g_row;
      if (row < r1) {
        p_sr = rp.scale[row];
        p_or = rp.offset[row];
      }
    }

    for (int t = 0; t < ntiles; ++t) {
      const int st = t % ns, r = t / ns;
      if (!mbar_wait(&full[st], r & 1, abort_flag, a.gflags)) break;
      const int nr = (int)min((int64_t)tr, nrows - (int64_t)t * tr);
      const uint8_t *stage = smem + (size_t)st * stage_bytes;
      if constexpr (FMT == LAM_ROWS_INT8 && QB == 1) {
        // As the Q_eps int8 single-query consumer: kRg consecutive rows per
        // warp pass, all code words loaded first, per lane the integer dot
        // products against the query's digit planes (and sum c, sum c^2 for
        // cosine / L2), one transposed butterfly for every row's totals, the
        // rows' scale and offset prefetched one group ahead, one ballot.
        constexpr int V = CC ? 4 * kRg : kRg;  // dot, sum c, sum c^2, padding
        for (int g0 = warp * kRg; g0 < nr; g0 += kBwWarps * kRg) {
          const float sr = p_sr, orr = p_or;
          {
            const int ng = g0 + kBwWarps * kRg;
            const int64_t nrow = ng < nr ? r0 + (int64_t)t * tr + ng + g_row
                                         : r0 + (int64_t)(t + 1) * tr + warp * kRg + g_row;
            if (nrow < r1) {
              p_sr = rp.scale[nrow];
              p_or = rp.offset[nrow];
            }
          }
          uint2 cw[kRg][kNchMax];
#pragma unroll
          for (int i = 0; i < kRg; ++i) {
            const uint8_t *pr = stage + (size_t)min(g0 + i, nr - 1) * row_bytes;
#pragma unroll
            for (int j = 0; j < kNchMax; ++j) {
              const int e0 = (j * 32 + lane) * 8;
              cw[i][j] = (j < nch && e0 < D) ? *reinterpret_cast<const uint2 *>(pr + e0)
                                             : make_uint2(0u, 0u);
            }
          }
          float v[V];
#pragma unroll
          for (int i = 0; i < kRg; ++i) {
            int d0 = 0, d1 = 0, d2 = 0, c1 = 0, c2 = 0;
#pragma unroll
            for (int j = 0; j < kNchMax; ++j) {
              if (j < nch) {  // (warp-uniform)
                const int wx = (int)cw[i][j].x, wy = (int)cw[i][j].y;
                d0 = __dp4a(wx, (int)qdig[0][j][0][0], __dp4a(wy, (int)qdig[0][j][0][1], d0));
                d1 = __dp4a(wx, (int)qdig[0][j][1][0], __dp4a(wy, (int)qdig[0][j][1][1], d1));
                d2 = __dp4a(wx, (int)qdig[0][j][2][0], __dp4a(wy, (int)qdig[0][j][2][1], d2));
                if constexpr (CC) {
                  c1 = __dp4a(wx, 0x01010101, __dp4a(wy, 0x01010101, c1));
                  c2 = __dp4a(wx, wx, __dp4a(wy, wy, c2));
                }
              }
            }
            v[i] = fmaf((float)d0, 65536.0f, fmaf((float)d1, 256.0f, (float)d2));
            if constexpr (CC) {
              v[kRg + i] = (float)c1;
              v[2 * kRg + i] = (float)c2;
              v[3 * kRg + i] = 0.0f;
            }
          }
          // lane L: the total of value L >> kLsh (CC: dot of row L / 2 on lanes
          // 0-7, its sum c 8 lanes and its sum c^2 16 lanes further on)
          const float tot = warp_sums_transposed<V>(v, lane);
          const float c1 = CC ? __shfl_down_sync(0xffffffffu, tot, 8) : 0.0f;
          const float c2 = CC ? __shfl_down_sync(0xffffffffu, tot, 16) : 0.0f;
          const float acc = tot * qinv[0];
          const float dot = fmaf(sr, acc, orr * qs[0]);
          const float xx = CC ? fmaf(sr * sr, c2, fmaf(2.0f * sr * orr, c1, (float)D * orr * orr))
                              : 0.0f;
          float sc;
          if (a.metric == LAM_METRIC_IP) sc = dot;
          else if (a.metric == LAM_METRIC_COSINE)
            sc = (qn[0] == 0.0f || xx == 0.0f) ? 0.0f : dot / (qn[0] * sqrtf(xx));
          else sc = fmaf(-2.0f, dot, qq[0] + xx);
          const bool leader = CC ? (lane < 2 * kRg && (lane & 1) == 0) : (lane & 7) == 0;
          unsigned pass = __ballot_sync(0xffffffffu, leader && g0 + g_row < nr &&
                                                         (desc ? sc > thr_s[0] : sc < thr_s[0]));
          while (pass) {
            const int l = __ffs(pass) - 1;
            pass &= pass - 1;
            const float sl = __shfl_sync(0xffffffffu, sc, l);
            if (!(desc ? sl > thr_s[0] : sl < thr_s[0])) continue;  // the list moved on
            const int64_t row = r0 + (int64_t)t * tr + g0 + ((l >> kLsh) & (kRg - 1));
            lists[0].insert(make_key(sl, (uint32_t)row, desc), lane);
            const uint64_t kk = lists[0].kth(a.k);
            thr_s[0] = kk == kSentinel ? (desc ? -INFINITY : INFINITY)
                                       : rank_key32_score((uint32_t)(kk >> 32), desc);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[st]);
        continue;
      }
      for (int rr = warp; rr < nr; rr += 2 * kBwWarps) {
        const int rb = rr + kBwWarps;
        const bool has_b = rb < nr;
        const uint8_t *pa = stage + (size_t)rr * row_bytes;
        const uint8_t *pb = stage + (size_t)(has_b ? rb : rr) * row_bytes;
        const float sr = f_sr, orr = f_or;
        frow += 2 * kBwWarps;
        if (FMT != LAM_ROWS_FP16 && frow < r1) f_sr = rp.scale[frow];
        if (FMT == LAM_ROWS_INT8 && frow < r1) f_or = rp.offset[frow];
        float pa_acc[QB], pb_acc[QB], pa_c1 = 0.0f, pb_c1 = 0.0f, pa_c2 = 0.0f, pb_c2 = 0.0f;
        if constexpr (FMT == LAM_ROWS_INT8) {
          int ia[QB][3], ib[QB][3], sa1 = 0, sb1 = 0, sa2 = 0, sb2 = 0;
#pragma unroll
          for (int q = 0; q < QB; ++q)
#pragma unroll
            for (int p = 0; p < 3; ++p) ia[q][p] = ib[q][p] = 0;
#pragma unroll
          for (int j = 0; j < kNchMax; ++j) {
            const int e0 = (j * 32 + lane) * 8;
            if (j < nch && e0 < D) {
              const uint2 wa = *reinterpret_cast<const uint2 *>(pa + e0);
              const uint2 wb = *reinterpret_cast<const uint2 *>(pb + e0);
#pragma unroll
              for (int q = 0; q < QB; ++q)
#pragma unroll
                for (int p = 0; p < 3; ++p) {
                  ia[q][p] = __dp4a((int)wa.x, (int)qdig[q][j][p][0], ia[q][p]);
                  ia[q][p] = __dp4a((int)wa.y, (int)qdig[q][j][p][1], ia[q][p]);
                  ib[q][p] = __dp4a((int)wb.x, (int)qdig[q][j][p][0], ib[q][p]);
                  ib[q][p] = __dp4a((int)wb.y, (int)qdig[q][j][p][1], ib[q][p]);
                }
              if (CC) {
                sa1 = __dp4a((int)wa.x, 0x01010101, __dp4a((int)wa.y, 0x01010101, sa1));
                sb1 = __dp4a((int)wb.x, 0x01010101, __dp4a((int)wb.y, 0x01010101, sb1));
                sa2 = __dp4a((int)wa.x, (int)wa.x, __dp4a((int)wa.y, (int)wa.y, sa2));
                sb2 = __dp4a((int)wb.x, (int)wb.x, __dp4a((int)wb.y, (int)wb.y, sb2));
              }
            }
          }
#pragma unroll
          for (int q = 0; q < QB; ++q) {
            pa_acc[q] = fmaf((float)ia[q][0], 65536.0f, fmaf((float)ia[q][1], 256.0f,
                                                              (float)ia[q][2]));
            pb_acc[q] = fmaf((float)ib[q][0], 65536.0f, fmaf((float)ib[q][1], 256.0f,
                                                              (float)ib[q][2]));
          }
          pa_c1 = (float)sa1;
          pb_c1 = (float)sb1;
          pa_c2 = (float)sa2;
          pb_c2 = (float)sb2;
        } else if constexpr (FMT == LAM_ROWS_FP16) {
          float2 aa[QB], ab[QB], ca = make_float2(0.f, 0.f), cb = make_float2(0.f, 0.f);
#pragma unroll
          for (int q = 0; q < QB; ++q) aa[q] = ab[q] = make_float2(0.f, 0.f);
#pragma unroll
          for (int j = 0; j < kNchMax; ++j) {
            const int e0 = (j * 32 + lane) * 8;
            if (j < nch && e0 < D) {
              const uint4 va = *reinterpret_cast<const uint4 *>(pa + (size_t)e0 * 2);
              const uint4 vb = *reinterpret_cast<const uint4 *>(pb + (size_t)e0 * 2);
              const uint32_t wa[4] = {va.x, va.y, va.z, va.w}, wb[4] = {vb.x, vb.y, vb.z, vb.w};
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                __half2 ha, hb;
                memcpy(&ha, &wa[u], 4);
                memcpy(&hb, &wb[u], 4);
                const float2 fa = __half22float2(ha), fb = __half22float2(hb);
#pragma unroll
                for (int q = 0; q < QB; ++q) {
                  aa[q] = __ffma2_rn(qreg[q][j][u], fa, aa[q]);
                  ab[q] = __ffma2_rn(qreg[q][j][u], fb, ab[q]);
                }
                if (CC) {
                  ca = __ffma2_rn(fa, fa, ca);
                  cb = __ffma2_rn(fb, fb, cb);
                }
              }
            }
          }
#pragma unroll
          for (int q = 0; q < QB; ++q) {
            pa_acc[q] = aa[q].x + aa[q].y;
            pb_acc[q] = ab[q].x + ab[q].y;
          }
          pa_c2 = ca.x + ca.y;
          pb_c2 = cb.x + cb.y;
        } else {
          // sign bits: the sum of q over the set bits
          float2 aa[QB], ab[QB];
#pragma unroll
          for (int q = 0; q < QB; ++q) aa[q] = ab[q] = make_float2(0.f, 0.f);
#pragma unroll
          for (int j = 0; j < kNchMax; ++j) {
            const int e0 = (j * 32 + lane) * 8;
            if (j < nch && e0 < D) {
              const uint32_t ba = pa[e0 / 8], bb = pb[e0 / 8];
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const float2 ma = make_float2((float)((ba >> (2 * u)) & 1u),
                                             (float)((ba >> (2 * u + 1)) & 1u));
                const float2 mb = make_float2((float)((bb >> (2 * u)) & 1u),
                                             (float)((bb >> (2 * u + 1)) & 1u));
#pragma unroll
                for (int q = 0; q < QB; ++q) {
                  aa[q] = __ffma2_rn(qreg[q][j][u], ma, aa[q]);
                  ab[q] = __ffma2_rn(qreg[q][j][u], mb, ab[q]);
                }
              }
            }
          }
#pragma unroll
          for (int q = 0; q < QB; ++q) {
            pa_acc[q] = aa[q].x + aa[q].y;
            pb_acc[q] = ab[q].x + ab[q].y;
          }
        }
        // lanes 0-15 finish row rr, lanes 16-31 row rb (its factors are unused
        // when the pair has no second row)
        const float c1 = (FMT == LAM_ROWS_INT8 && CC) ? pair_sum(pa_c1, pb_c1, lane) : 0.0f;
        const float c2 = (FMT != LAM_ROWS_SIGN && CC) ? pair_sum(pa_c2, pb_c2, lane) : 0.0f;
        float xx = 0.0f;
        if (CC) {
          if (FMT == LAM_ROWS_INT8)
            xx = fmaf(sr * sr, c2, fmaf(2.0f * sr * orr, c1, (float)D * orr * orr));
          else if (FMT == LAM_ROWS_FP16)
            xx = c2;
          else
            xx = (float)D * sr * sr;
        }
#pragma unroll
        for (int q = 0; q < QB; ++q) {
          const float acc = pair_sum(pa_acc[q], pb_acc[q], lane) * qinv[q];
          float dot;
          if (FMT == LAM_ROWS_INT8) dot = fmaf(sr, acc, orr * qs[q]);
          else if (FMT == LAM_ROWS_FP16) dot = acc;
          else dot = sr * fmaf(2.0f, acc, -qs[q]);
          float sc;
          if (a.metric == LAM_METRIC_IP) sc = dot;
          else if (a.metric == LAM_METRIC_COSINE)
            sc = (qn[q] == 0.0f || xx == 0.0f) ? 0.0f : dot / (qn[q] * sqrtf(xx));
          else sc = fmaf(-2.0f, dot, qq[q] + xx);
          const float sa = __shfl_sync(0xffffffffu, sc, 0);
          const float sb = __shfl_sync(0xffffffffu, sc, 16);
          if (q >= a.B) continue;
          if (desc ? sa > thr_s[q] : sa < thr_s[q]) {
            lists[q].insert(make_key(sa, (uint32_t)(r0 + (int64_t)t * tr + rr), desc), lane);
            const uint64_t kk = lists[q].kth(a.k);
            thr_s[q] = kk == kSentinel ? (desc ? -INFINITY : INFINITY)
                                       : rank_key32_score((uint32_t)(kk >> 32), desc);
          }
          if (has_b && (desc ? sb > thr_s[q] : sb < thr_s[q])) {
            lists[q].insert(make_key(sb, (uint32_t)(r0 + (int64_t)t * tr + rb), desc), lane);
            const uint64_t kk = lists[q].kth(a.k);
            thr_s[q] = kk == kSentinel ? (desc ? -INFINITY : INFINITY)
                                       : rank_key32_score((uint32_t)(kk >> 32), desc);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }
  }
  __syncthreads();
  uint64_t *cand = reinterpret_cast<uint64_t *>(smem);
  if (warp < kBwWarps) {
#pragma unroll
    for (int q = 0; q < QB; ++q)
      lists[q].store(cand + ((size_t)q * kBwWarps + warp) * a.k, a.k, lane);
  }
  __syncthreads();
  for (int q = 0; q < QB && q < a.B; ++q)
    rank_merge(cand + (size_t)q * kBwWarps * a.k, kBwWarps, a.k,
               a.partial + ((size_t)blockIdx.x * a.B + q) * a.k, threadIdx.x, kBwThreads);
}

// ---------------------------------------------------------------------------
// Sign-bit rows (per-vector codec), B <= 2: one lane per row.  The dot product
// with the query is q . xhat = alpha (2 S - sum(q)), S = the sum of q_d over
// the row's set bits.  S is gathered four bits at a time from per-query nibble
// tables in shared memory, T[q][p][v] = sum of q_{4p + b} over the set bits b
// of v (b = 0 .. 3, in that order), so a 768-bit row costs 192 table reads and
// adds instead of 768 masked multiply-adds.  All lanes read the same nibble
// position of their own rows at once, so a read touches at most 16 distinct
// words of one 64-byte table row: no bank conflicts.  Stages hold contiguous
// rows (bulk copies); warp w scores rows 32 w .. 32 w + 31 of each stage, and
// one ballot per query admits candidates into the warp's register top-k in
// row order.
template <int QB, int KPL, bool CC, int NCH>
__global__ void __launch_bounds__(kBwThreads, 1)
    score_bw_sign_kernel(ScoreArgs a, RowPtrs rp, int tr, int ns, int stage_bytes) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const int D = a.D;
  const int npos = D / 4;  // nibbles per row
  float *tab = reinterpret_cast<float *>(smem + (size_t)ns * stage_bytes);  // [QB][npos][16]
  float *qstat = tab + (size_t)QB * npos * 16;                               // [QB][3]
  uint64_t *full = reinterpret_cast<uint64_t *>(qstat + 4 * QB);
  uint64_t *empty = full + ns;
  volatile int *abort_flag = reinterpret_cast<volatile int *>(empty + ns);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t N = a.N;
  const int64_t r0 = (int64_t)blockIdx.x * N / gridDim.x;
  const int64_t r1 = (int64_t)(blockIdx.x + 1) * N / gridDim.x;
  const int64_t nrows = r1 - r0;
  const int ntiles = (int)((nrows + tr - 1) / tr);
  const size_t row_bytes = (size_t)D / 8;

  if (threadIdx.x == 0) {
    for (int s = 0; s < ns; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kBwWarps);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  // the nibble tables, from a copy of the queries in the first (still empty) stage
  float *qsm = reinterpret_cast<float *>(smem);
  for (int e = threadIdx.x; e < QB * D; e += blockDim.x)
    qsm[e] = e < a.B * D ? a.queries[e] : 0.0f;
  __syncthreads();
  for (int e = threadIdx.x; e < QB * npos * 16; e += blockDim.x) {
    const int q = e / (npos * 16), pv = e - q * npos * 16, pos = pv >> 4, v = pv & 15;
    const float *qr = qsm + q * D + 4 * pos;
    float t = 0.0f;
#pragma unroll
    for (int b = 0; b < 4; ++b)
      if (v & (1 << b)) t += qr[b];
    tab[e] = t;
  }
  // sum(q), ||q|| and ||q||^2 per query (the norm from the query scaled near 1)
  if (warp < QB) {
    const int q = warp;
    float sum = 0.0f, mx = 0.0f;
    for (int d = lane; d < D; d += 32) {
      const float v = qsm[q * D + d];
      sum += v;
      mx = fmaxf(mx, fabsf(v));
    }
    const float nsc = norm_scale(warp_max(mx));
    float part = 0.0f;
    for (int d = lane; d < D; d += 32) {
      const float u = qsm[q * D + d] * nsc;
      part = fmaf(u, u, part);
    }
    sum = warp_sum(sum);
    const float qn = sqrtf(warp_sum(part)) / nsc;
    if (lane == 0) {
      qstat[3 * q] = sum;
      qstat[3 * q + 1] = qn;
      qstat[3 * q + 2] = qn * qn;
    }
  }
  __syncthreads();

  WarpList<KPL> lists[QB];
#pragma unroll
  for (int q = 0; q < QB; ++q) lists[q].init();

  if (warp == kBwWarps) {
    if (lane == 0) {
      int issued = 0;
      const int nt = producers_stalled(a.gflags) ? 0 : ntiles;
      for (int t = 0; t < nt; ++t) {
        const int s = t % ns, r = t / ns;
        if (r > 0 && !mbar_wait(&empty[s], (r - 1) & 1, abort_flag, a.gflags)) break;
        const int64_t nr = min((int64_t)tr, nrows - (int64_t)t * tr);
        const uint32_t bytes = (uint32_t)(nr * row_bytes);
        mbar_arrive_expect_tx(&full[s], bytes);
        bulk_g2s(smem + (size_t)s * stage_bytes,
                 static_cast<const uint8_t *>(a.codes) + (r0 + (int64_t)t * tr) * row_bytes,
                 bytes, &full[s]);
        issued = t + 1;
      }
      for (int t = max(0, issued - ns); t < issued; ++t) drain_wait(&full[t % ns], (t / ns) & 1);
    }
  } else {
    const bool desc = a.metric != LAM_METRIC_L2;
    float qs[QB], qn[QB], qq[QB], thr_s[QB];
#pragma unroll
    for (int q = 0; q < QB; ++q) {
      qs[q] = qstat[3 * q];
      qn[q] = qstat[3 * q + 1];
      qq[q] = qstat[3 * q + 2];
      thr_s[q] = desc ? -INFINITY : INFINITY;
    }
    // 16-byte pieces per row (128 bits); NCH > 0: that count, fully unrolled
    const int nchunk = NCH > 0 ? NCH : (int)(row_bytes / 16);
    // the row scale one pass ahead (the warp's passes are 32 kBwWarps rows
    // apart, or start the next tile at the same offset)
    float p_alpha = 0.0f;
    {
      const int64_t row = r0 + warp * 32 + lane;
      if (warp * 32 < tr && row < r1) p_alpha = rp.scale[row];
    }
    for (int t = 0; t < ntiles; ++t) {
      const int st = t % ns, r = t / ns;
      if (!mbar_wait(&full[st], r & 1, abort_flag, a.gflags)) break;
      const int nr = (int)min((int64_t)tr, nrows - (int64_t)t * tr);
      const uint8_t *stage = smem + (size_t)st * stage_bytes;
      for (int rb = warp * 32; rb < nr; rb += kBwWarps * 32) {
        const int rr = rb + lane;
        const bool valid = rr < nr;
        const float alpha = valid ? p_alpha : 0.0f;
        {
          const int nb = rb + kBwWarps * 32;
          const int64_t nrow = nb < nr ? r0 + (int64_t)t * tr + nb + lane
                                       : r0 + (int64_t)(t + 1) * tr + warp * 32 + lane;
          if (nrow < r1) p_alpha = rp.scale[nrow];
        }
        const uint8_t *rowp = stage + (size_t)(valid ? rr : 0) * row_bytes;
        float acc[QB][2];
#pragma unroll
        for (int q = 0; q < QB; ++q) acc[q][0] = acc[q][1] = 0.0f;
#pragma unroll (NCH > 0 ? NCH : 1)
        for (int c = 0; c < nchunk; ++c) {
          const uint4 v = *reinterpret_cast<const uint4 *>(rowp + (size_t)c * 16);
          const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int pos0 = (c * 4 + u) * 8;  // first nibble position of this word
#pragma unroll
            for (int n = 0; n < 8; ++n) {
              const uint32_t nib = (w4[u] >> (4 * n)) & 15u;
#pragma unroll
              for (int q = 0; q < QB; ++q)
                acc[q][n & 1] += tab[((size_t)q * npos + pos0 + n) * 16 + nib];
            }
          }
        }
        const float xx = CC ? (float)D * alpha * alpha : 0.0f;
#pragma unroll
        for (int q = 0; q < QB; ++q) {
          const float S = acc[q][0] + acc[q][1];
          const float dot = alpha * fmaf(2.0f, S, -qs[q]);
          float sc;
          if (a.metric == LAM_METRIC_IP) sc = dot;
          else if (a.metric == LAM_METRIC_COSINE)
            sc = (qn[q] == 0.0f || xx == 0.0f) ? 0.0f : dot / (qn[q] * sqrtf(xx));
          else sc = fmaf(-2.0f, dot, qq[q] + xx);
          if (q >= a.B) continue;
          uint32_t m = __ballot_sync(0xffffffffu, valid && (desc ? sc > thr_s[q] : sc < thr_s[q]));
          while (m != 0) {
            const int l = __ffs(m) - 1;
            m &= m - 1;
            const float sl = __shfl_sync(0xffffffffu, sc, l);
            if (desc ? sl > thr_s[q] : sl < thr_s[q]) {
              lists[q].insert(make_key(sl, (uint32_t)(r0 + (int64_t)t * tr + rb + l), desc), lane);
              const uint64_t kk = lists[q].kth(a.k);
              thr_s[q] = kk == kSentinel ? (desc ? -INFINITY : INFINITY)
                                         : rank_key32_score((uint32_t)(kk >> 32), desc);
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }
  }
  __syncthreads();
  uint64_t *cand = reinterpret_cast<uint64_t *>(smem);
  if (warp < kBwWarps) {
#pragma unroll
    for (int q = 0; q < QB; ++q)
      lists[q].store(cand + ((size_t)q * kBwWarps + warp) * a.k, a.k, lane);
  }
  __syncthreads();
  for (int q = 0; q < QB && q < a.B; ++q)
    rank_merge(cand + (size_t)q * kBwWarps * a.k, kBwWarps, a.k,
               a.partial + ((size_t)blockIdx.x * a.B + q) * a.k, threadIdx.x, kBwThreads);
}

// ---------------------------------------------------------------------------
// Generic path: any D, width 1/2/4, k <= 1024, any batch.  Grid (ctas, B):
// a CTA scores one query against a range of rows, warp per row with plain
// global loads, per-warp top-k lists in shared memory, then a rank merge.
constexpr int kGenWarps = 8;

__device__ __forceinline__ int32_t load_code(const void *codes, int width, int64_t i) {
  if (width == 1) return reinterpret_cast<const int8_t *>(codes)[i];
  if (width == 2) return reinterpret_cast<const int16_t *>(codes)[i];
  return reinterpret_cast<const int32_t *>(codes)[i];
}

__global__ void __launch_bounds__(kGenWarps * 32) score_generic_kernel(ScoreArgs a, RowPtrs rp) {
  const int width = codes_width(a, rp);
  if (rp.qst != nullptr && (!status_ok(rp.qst) || (width != 1 && width != 2))) return;
  extern __shared__ __align__(16) uint8_t gsmem[];
  uint64_t *lists = reinterpret_cast<uint64_t *>(gsmem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int D = a.D, k = a.k;
  uint64_t *L = lists + (size_t)warp * k;
  for (int64_t b = blockIdx.y; b < a.B; b += gridDim.y) {
  const float *q = a.queries + b * D;
  for (int i = lane; i < k; i += 32) L[i] = kSentinel;
  __syncwarp();
  uint64_t thr = kSentinel;

  float part = 0.0f;
  float mx = 0.0f;
  for (int d = lane; d < D; d += 32) mx = fmaxf(mx, fabsf(q[d]));
  const float ns = norm_scale(warp_max(mx));
  for (int d = lane; d < D; d += 32) part = fmaf(q[d] * ns, q[d] * ns, part);
  const float qn = sqrtf(warp_sum(part)) / ns, qq = qn * qn;
  const bool desc = a.metric != LAM_METRIC_L2;
  // per-row codecs score the decoded rows themselves (unit step)
  const float s = a.fmt ? 1.0f : a.s, s2 = s * s;

  const int64_t r0 = (int64_t)blockIdx.x * a.N / gridDim.x;
  const int64_t r1 = (int64_t)(blockIdx.x + 1) * a.N / gridDim.x;
  for (int64_t row = r0 + warp; row < r1; row += kGenWarps) {
    float acc = 0.0f, cc = 0.0f;
    const int64_t base = row * D;
    for (int d = lane; d < D; d += 32) {
      const float c = a.fmt ? row_value(a, rp, row, d) : (float)load_code(a.codes, width, base + d);
      acc = fmaf(q[d], c, acc);
      cc = fmaf(c, c, cc);
    }
    acc = warp_sum(acc);
    cc = warp_sum(cc);
    const float sc = finish_score(a.metric, acc, cc, s, s2, qq, qn);
    const uint64_t key = make_key(sc, (uint32_t)row, desc);
    if (key < thr) smem_list_insert(L, k, key, lane, thr);
  }
  __syncthreads();
  rank_merge(lists, kGenWarps, k, a.partial + ((size_t)blockIdx.x * a.B + b) * k, threadIdx.x,
             kGenWarps * 32);
  __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// Final merge: per query, n_lists partial lists of k keys -> the k best,
// decoded to (score, id).  Bitonic sort in shared memory; when the candidates
// exceed one buffer, chunks are sorted together with the running top-k.
constexpr int kMergeThreads = 1024;
constexpr int kMergeCap = 16384;

__device__ __forceinline__ int next_pow2_dev(int x) {
  int p = 1;
  while (p < x) p <<= 1;
  return p;
}

__device__ void bitonic_sort(uint64_t *buf, int P) {
  for (int size = 2; size <= P; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < P / 2; i += blockDim.x) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool up = (lo & size) == 0;
        const uint64_t x = buf[lo], y = buf[hi];
        if ((x > y) == up) {
          buf[lo] = y;
          buf[hi] = x;
        }
      }
      __syncthreads();
    }
  }
}

__global__ void __launch_bounds__(kMergeThreads) topk_merge_kernel(ScoreArgs a, int P,
                                                                   RowPtrs rp) {
  if (rp.qst != nullptr && (!status_ok(rp.qst) || (status_width(rp.qst) != 1 &&
                                                   status_width(rp.qst) != 2))) {
    if (blockIdx.x == 0 && threadIdx.x == 0) atomicOr(a.gflags, kFlagInput);
    return;
  }
  extern __shared__ __align__(16) uint8_t msmem[];
  uint64_t *buf = reinterpret_cast<uint64_t *>(msmem);
  const int64_t b = blockIdx.x;
  const int k = a.k;
  const int64_t total = (int64_t)a.n_lists * k;
  // candidate e of query b lives at partial[(l * B + b) * k + i], e = l*k + i
  auto cand = [&](int64_t e) -> uint64_t {
    const int64_t l = e / k, i = e - l * k;
    return a.partial[((size_t)l * a.B + b) * k + i];
  };
  if (total <= P) {
    for (int i = threadIdx.x; i < P; i += blockDim.x) buf[i] = i < total ? cand(i) : kSentinel;
    __syncthreads();
    bitonic_sort(buf, P);
  } else {
    for (int i = threadIdx.x; i < k; i += blockDim.x) buf[i] = kSentinel;
    const int chunk = P - k;
    for (int64_t c0 = 0; c0 < total; c0 += chunk) {
      for (int i = threadIdx.x; i < chunk; i += blockDim.x)
        buf[k + i] = (c0 + i < total) ? cand(c0 + i) : kSentinel;
      __syncthreads();
      bitonic_sort(buf, P);
    }
  }
  const bool desc = a.metric != LAM_METRIC_L2;
  if (!desc) {
    // Squared L2 was ranked through ||q||^2 + s^2||c||^2 - 2 s q.c, which
    // cancels for near neighbours; the k survivors are rescored in the direct
    // form sum_d (q_d - s c_d)^2 and re-sorted.
    uint64_t *rescored = buf + P;
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
    const float *q = a.queries + b * a.D;
    for (int i = warp; i < k; i += nw) {
      const uint64_t key = buf[i];
      const uint32_t row = (uint32_t)(key & 0xffffffffu);
      float acc = 0.0f;
      if (row < a.N) {
        for (int d = lane; d < a.D; d += 32) {
          const float xh = a.fmt ? row_value(a, rp, row, d)
                                 : __fmul_rn(a.s, (float)load_code(a.codes, codes_width(a, rp),
                                                                   (int64_t)row * a.D + d));
          const float df = __fsub_rn(q[d], xh);
          acc = fmaf(df, df, acc);
        }
      }
      acc = warp_sum(acc);
      if (lane == 0) rescored[i] = row < a.N ? make_key(acc, row, false) : kSentinel;
    }
    __syncthreads();
    const int P2 = next_pow2_dev(k);
    for (int i = threadIdx.x; i < P2; i += blockDim.x) buf[i] = i < k ? rescored[i] : kSentinel;
    __syncthreads();
    bitonic_sort(buf, P2);
  }
  for (int i = threadIdx.x; i < k; i += blockDim.x) {
    const uint64_t key = buf[i];
    uint32_t o = (uint32_t)(key >> 32);
    if (desc) o = ~o;
    a.scores[b * k + i] = unord_f32(o);
    a.ids[b * k + i] = (int64_t)(uint32_t)(key & 0xffffffffu);
  }
}

// k-way merge of the sorted partial lists, one warp per query.  The CTA first
// copies the candidate lists of its qpc queries to shared memory; lane l then
// owns lists l, l + 32, ... and keeps their heads in registers; each of the k
// steps takes the warp-wide smallest head and advances that list.  Squared L2
// survivors are rescored in the direct form (all warps of the CTA share the
// rows of its queries) and re-sorted, as in the block-sort merge above.
constexpr int kKmWarps = 8;

// Eight consecutive codes of width w (1, 2 or 4) from index i (a multiple of
// 8; the address 8 w-byte aligned) as exact fp32 values.
__device__ __forceinline__ void load8_codes(const void *codes, int w, int64_t i, float (&c)[8]) {
  if (w == 1) {
    const uint2 v = *reinterpret_cast<const uint2 *>(static_cast<const int8_t *>(codes) + i);
#pragma unroll
    for (int t = 0; t < 8; ++t) c[t] = (float)(int8_t)((t < 4 ? v.x : v.y) >> (8 * (t & 3)));
  } else if (w == 2) {
    const uint4 v = *reinterpret_cast<const uint4 *>(static_cast<const int16_t *>(codes) + i);
    const uint32_t x[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int t = 0; t < 8; ++t) c[t] = (float)(int16_t)(x[t >> 1] >> (16 * (t & 1)));
  } else {
    const int4 *p = reinterpret_cast<const int4 *>(static_cast<const int32_t *>(codes) + i);
    const int4 v0 = p[0], v1 = p[1];
    c[0] = (float)v0.x; c[1] = (float)v0.y; c[2] = (float)v0.z; c[3] = (float)v0.w;
    c[4] = (float)v1.x; c[5] = (float)v1.y; c[6] = (float)v1.z; c[7] = (float)v1.w;
  }
}

template <int HPL>
__global__ void __launch_bounds__(kKmWarps * 32) topk_kmerge_kernel(ScoreArgs a, int qpc,
                                                                    RowPtrs rp, int mode,
                                                                    int kout) {
  if (rp.qst != nullptr && (!status_ok(rp.qst) || (status_width(rp.qst) != 1 &&
                                                   status_width(rp.qst) != 2))) {
    if (blockIdx.x == 0 && threadIdx.x == 0) atomicOr(a.gflags, kFlagInput);
    return;
  }
  // the merge of the gated full pass: nothing to do when every query passed
  if (mode == 2 && hi_all_certified(a.gflags)) return;
  extern __shared__ __align__(16) uint8_t ksmem[];
  const int L = a.n_lists, k = a.k;
  const bool cert = mode == 1;
  const int ko = cert ? kout : k;  // entries written per query
  uint64_t *cand = reinterpret_cast<uint64_t *>(ksmem);            // [qpc][L][k]
  uint64_t *outk = cand + (size_t)qpc * L * k;                       // [kKmWarps][P2]
  const int P2 = next_pow2_dev(k);
  const int64_t b0 = (int64_t)blockIdx.x * qpc;
  const int per_q = L * k;  // fits: the candidates of qpc queries fit in shared memory
  // (unrolled: eight independent loads in flight per thread)
#pragma unroll 8
  for (int e = threadIdx.x; e < qpc * per_q; e += blockDim.x) {
    const int qi = e / per_q, rem = e - qi * per_q;
    const int l = rem / k, i = rem - l * k;
    const int64_t b = b0 + qi;
    cand[e] = b < a.B ? a.partial[((size_t)l * a.B + b) * k + i] : kSentinel;
  }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool desc = a.metric != LAM_METRIC_L2;
  // qpc <= kKmWarps: warp qi owns query b0 + qi
  const int qi = warp;
  const int64_t b = b0 + qi;
  const bool mine = qi < qpc && b < a.B;
  uint64_t *O = outk + (size_t)warp * P2;
  uint64_t tkey = kSentinel;  // cert: the k-th (last) candidate's key by the hi-only score
  if (mine) {
    const uint64_t *C = cand + (size_t)qi * per_q;
    int pos[HPL];
    uint64_t head[HPL];
#pragma unroll
    for (int h = 0; h < HPL; ++h) {
      const int l = lane + 32 * h;
      pos[h] = 0;
      head[h] = l < L ? C[(size_t)l * k] : kSentinel;
    }
    for (int i = 0; i < k; ++i) {
      uint64_t m = head[0];
      int mh = 0;
#pragma unroll
      for (int h = 1; h < HPL; ++h)
        if (head[h] < m) {
          m = head[h];
          mh = h;
        }
      // warp minimum of the 64-bit heads: the high words by one reduction,
      // then the low words of the lanes that hold the smallest high word
      const uint32_t mhi = (uint32_t)(m >> 32);
      const uint32_t ghi = __reduce_min_sync(0xffffffffu, mhi);
      const uint32_t glo = __reduce_min_sync(0xffffffffu, mhi == ghi ? (uint32_t)m : 0xffffffffu);
      const uint64_t gm = ((uint64_t)ghi << 32) | glo;
      const unsigned bal = __ballot_sync(0xffffffffu, m == gm);
      if (lane == __ffs(bal) - 1) {
#pragma unroll
        for (int h = 0; h < HPL; ++h)
          if (h == mh) {
            ++pos[h];
            head[h] = pos[h] < k ? C[(size_t)(lane + 32 * h) * k + pos[h]] : kSentinel;
          }
      }
      if (lane == 0) O[i] = gm;
      tkey = gm;
    }
  }
  if (!desc || cert) {
    // Survivors rescored in the direct form (squared L2: the ranking form
    // ||q||^2 + s^2||c||^2 - 2 s q.c cancels for near neighbours), and every
    // candidate of the certifying merge exactly (it was ranked by the hi-only
    // score).  Every warp rescores candidates of every query of the CTA, kRs
    // rows at a time so that their code loads are in flight together (each
    // row's sum keeps the order of a one-row loop).
    constexpr int kRs = 4;
    __shared__ float qnq[kKmWarps][2];  // cert: ||q|| and ||q||^2 of the CTA's queries
    if (cert && mine) {
      const float *q = a.queries + b * a.D;
      float mx = 0.0f;
      for (int d = lane; d < a.D; d += 32) mx = fmaxf(mx, fabsf(q[d]));
      const float sc = norm_scale(warp_max(mx));
      float part = 0.0f;
      for (int d = lane; d < a.D; d += 32) part = fmaf(q[d] * sc, q[d] * sc, part);
      const float qn = sqrtf(warp_sum(part)) / sc;
      if (lane == 0) {
        qnq[warp][0] = qn;
        qnq[warp][1] = qn * qn;
      }
    }
    __syncthreads();
    const float s2 = a.s * a.s;
    // vector loads when Q_eps code rows and query rows are 16-byte aligned
    const bool vec = a.fmt == 0 && (a.D & 7) == 0 &&
                     ((reinterpret_cast<uintptr_t>(a.codes) |
                       reinterpret_cast<uintptr_t>(a.queries)) & 15u) == 0;
    for (int t0 = warp; t0 < qpc * k; t0 += kKmWarps * kRs) {
      uint32_t row[kRs];
      const float *q[kRs];
      uint64_t *slot[kRs];
      float acc[kRs], cc[kRs];
      int tqs[kRs];
#pragma unroll
      for (int u = 0; u < kRs; ++u) {
        const int t = t0 + u * kKmWarps;
        const int tq = t / k, i = t - tq * k;
        const int64_t tb = b0 + tq;
        const bool ok = t < qpc * k && tb < a.B;
        tqs[u] = ok ? tq : 0;
        slot[u] = ok ? outk + (size_t)tq * P2 + i : nullptr;
        row[u] = ok ? (uint32_t)(*slot[u] & 0xffffffffu) : 0xffffffffu;
        q[u] = a.queries + (ok ? tb : 0) * a.D;
        acc[u] = 0.0f;
        cc[u] = 0.0f;
      }
      if (vec) {
        // eight consecutive coordinates per lane and 256-wide slice: one 8- or
        // 16-byte code load (int8 / int16) and two float4 query loads per row
        const int w = codes_width(a, rp);
#pragma unroll 2
        for (int d0 = lane * 8; d0 < a.D; d0 += 256) {
#pragma unroll
          for (int u = 0; u < kRs; ++u) {
            if (row[u] < a.N) {
              float c[8];
              load8_codes(a.codes, w, (int64_t)row[u] * a.D + d0, c);
              const float4 qa = *reinterpret_cast<const float4 *>(q[u] + d0);
              const float4 qb = *reinterpret_cast<const float4 *>(q[u] + d0 + 4);
              const float qv[8] = {qa.x, qa.y, qa.z, qa.w, qb.x, qb.y, qb.z, qb.w};
#pragma unroll
              for (int t = 0; t < 8; ++t) {
                if (!desc) {
                  const float df = __fsub_rn(qv[t], __fmul_rn(a.s, c[t]));
                  acc[u] = fmaf(df, df, acc[u]);
                } else {
                  acc[u] = fmaf(qv[t], c[t], acc[u]);
                  cc[u] = fmaf(c[t], c[t], cc[u]);
                }
              }
            }
          }
        }
      } else if (!desc) {
#pragma unroll 4
        for (int d = lane; d < a.D; d += 32) {
#pragma unroll
          for (int u = 0; u < kRs; ++u) {
            if (row[u] < a.N) {
              const float xh =
                  a.fmt ? row_value(a, rp, row[u], d)
                        : __fmul_rn(a.s, (float)load_code(a.codes, codes_width(a, rp),
                                                          (int64_t)row[u] * a.D + d));
              const float df = __fsub_rn(q[u][d], xh);
              acc[u] = fmaf(df, df, acc[u]);
            }
          }
        }
      } else {  // cert, inner product or cosine: sum q_d c_d and sum c_d^2
#pragma unroll 4
        for (int d = lane; d < a.D; d += 32) {
#pragma unroll
          for (int u = 0; u < kRs; ++u) {
            if (row[u] < a.N) {
              const float c =
                  (float)load_code(a.codes, codes_width(a, rp), (int64_t)row[u] * a.D + d);
              acc[u] = fmaf(q[u][d], c, acc[u]);
              cc[u] = fmaf(c, c, cc[u]);
            }
          }
        }
      }
#pragma unroll
      for (int u = 0; u < kRs; ++u) {
        float tot = warp_sum(acc[u]);
        if (desc) {
          const float tcc = a.metric == LAM_METRIC_COSINE ? warp_sum(cc[u]) : 0.0f;
          tot = finish_score(a.metric, tot, tcc, a.s, s2, qnq[tqs[u]][1], qnq[tqs[u]][0]);
        }
        if (lane == 0 && slot[u] != nullptr)
          *slot[u] = row[u] < a.N ? make_key(tot, row[u], desc) : kSentinel;
      }
    }
    __syncthreads();
    if (mine) {
      for (int i = k + lane; i < P2; i += 32) O[i] = kSentinel;
      __syncwarp();
      for (int size = 2; size <= P2; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
          for (int t = lane; t < P2 / 2; t += 32) {
            const int lo = 2 * t - (t & (stride - 1));
            const int hi = lo + stride;
            const bool up = (lo & size) == 0;
            const uint64_t x = O[lo], y = O[hi];
            if ((x > y) == up) {
              O[lo] = y;
              O[hi] = x;
            }
          }
          __syncwarp();
        }
      }
      if (cert && lane == 0) {
        // Certification: a row outside the candidates scored no better than
        // the last candidate by the hi-only score T, and its exact score lies
        // within Bq of that score (the dropped lo term, |q_lo . c| <=
        // 2^-11 ||q|| ||c||, plus fp32 accumulation, D 2^-21 of ||q|| ||c||).
        // The top-kout is exact when the kout-th exact score beats T by more
        // than Bq; otherwise the query is counted and the full pass reruns.
        bool ok = tkey == kSentinel;  // fewer rows than candidates: all were rescored
        if (!ok) {
          const float T = rank_key32_score((uint32_t)(tkey >> 32), desc);
          const uint64_t kk = O[ko - 1];
          const float ek = rank_key32_score((uint32_t)(kk >> 32), desc);
          const float maxc = sqrtf(__uint_as_float(
                                 *reinterpret_cast<volatile uint32_t *>(a.gflags + kHdrMaxCC))) *
                             1.0001f;
          const float coef = 0x1p-11f + (float)a.D * 0x1p-21f;
          const float qn = qnq[warp][0];
          float bq;
          if (a.metric == LAM_METRIC_COSINE) bq = coef;
          else if (a.metric == LAM_METRIC_IP) bq = coef * a.s * qn * maxc;
          else  // also the fp32 rounding of the ranking form ||q||^2 + s^2||c||^2 - 2 s q.c
            bq = 2.0f * coef * a.s * qn * maxc + 0x1p-21f * (qn * qn + s2 * maxc * maxc);
          ok = kk != kSentinel && (desc ? ek > T + bq : ek < T - bq) &&
               a.gflags[kHdrForceFail] == 0u;
        }
        if (!ok) atomicAdd(a.gflags + kHdrHiFail, 1u);
      }
    }
  }
  __syncwarp();
  if (mine) {
    for (int i = lane; i < ko; i += 32) {
      const uint64_t key = O[i];
      uint32_t o = (uint32_t)(key >> 32);
      if (desc) o = ~o;
      a.scores[b * ko + i] = unord_f32(o);
      a.ids[b * ko + i] = (int64_t)(uint32_t)(key & 0xffffffffu);
    }
  }
}

// Per-slab merge of a multi-slab search: per query the nsplit partial lists
// of one slab (lists list0 .. list0 + n_lists - 1) become one sorted list of
// k keys, slab `slab` of `out` ([nslabs][B][k], the partial-list layout), so
// the final merge sees one list per slab.  With `seed` it also writes the
// ranking-form score of the k-th key (+-inf when the slab holds fewer than k
// rows): the first slab's k-th best bounds what the later slabs may offer.
// One warp per query, lists staged in shared memory when they fit; the merge
// stops at the first sentinel (later slabs offer few rows).
constexpr int kSmWarps = 8;

template <int HPL>
__global__ void __launch_bounds__(kSmWarps * 32)
    slab_merge_kernel(ScoreArgs a, int list0, int n_lists, int qpc, bool staged, int slab,
                      uint64_t *__restrict__ out, float *__restrict__ seed) {
  extern __shared__ __align__(16) uint8_t smsmem[];
  uint64_t *cand = reinterpret_cast<uint64_t *>(smsmem);  // [qpc][n_lists][k]
  const int k = a.k;
  const int per_q = n_lists * k;
  const int64_t b0 = (int64_t)blockIdx.x * qpc;
  if (staged) {
    for (int e = threadIdx.x; e < qpc * per_q; e += blockDim.x) {
      const int qi = e / per_q, rem = e - qi * per_q;
      const int l = rem / k, i = rem - l * k;
      const int64_t b = b0 + qi;
      cand[e] = b < a.B ? a.partial[((size_t)(list0 + l) * a.B + b) * k + i] : kSentinel;
    }
    __syncthreads();
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool desc = a.metric != LAM_METRIC_L2;
  for (int qi = warp; qi < qpc; qi += kSmWarps) {
    const int64_t b = b0 + qi;
    if (b >= a.B) break;
    // key i of list l of this query
    auto at = [&](int l, int i) -> uint64_t {
      return staged ? cand[(size_t)qi * per_q + (size_t)l * k + i]
                    : a.partial[((size_t)(list0 + l) * a.B + b) * k + i];
    };
    int pos[HPL];
    uint64_t head[HPL];
#pragma unroll
    for (int h = 0; h < HPL; ++h) {
      const int l = lane + 32 * h;
      pos[h] = 0;
      head[h] = l < n_lists ? at(l, 0) : kSentinel;
    }
    uint64_t *o = out + ((size_t)slab * a.B + b) * k;
    uint64_t gm = kSentinel;
    int i = 0;
    for (; i < k; ++i) {
      uint64_t m = head[0];
      int mh = 0;
#pragma unroll
      for (int h = 1; h < HPL; ++h)
        if (head[h] < m) {
          m = head[h];
          mh = h;
        }
      gm = m;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const uint64_t v = __shfl_xor_sync(0xffffffffu, gm, off);
        gm = v < gm ? v : gm;
      }
      if (gm == kSentinel) break;  // every list is exhausted
      if (lane == 0) o[i] = gm;
      const unsigned bal = __ballot_sync(0xffffffffu, m == gm);
      if (lane == __ffs(bal) - 1) {
#pragma unroll
        for (int h = 0; h < HPL; ++h)
          if (h == mh) {
            ++pos[h];
            head[h] = pos[h] < k ? at(lane + 32 * h, pos[h]) : kSentinel;
          }
      }
    }
    for (int j = i + lane; j < k; j += 32) o[j] = kSentinel;
    if (seed != nullptr && lane == 0) {
      float v = desc ? -INFINITY : INFINITY;
      if (i == k) {
        uint32_t ok = (uint32_t)(gm >> 32);
        if (desc) ok = ~ok;
        v = unord_f32(ok);
      }
      seed[b] = v;
    }
  }
}

constexpr size_t kKmCandBytes = 160 * 1024;

inline int next_pow2(int64_t x) {
  int p = 1;
  while (p < x) p <<= 1;
  return p;
}

}  // namespace

int bandwidth_ctas(int64_t N, int D, int width, int sms) {
  const BwShape sh = bw_shape(D, width);
  int64_t c = (N + sh.tr - 1) / sh.tr;
  if (c > sms) c = sms;
  if (c < 1) c = 1;
  return (int)c;
}

int generic_ctas(int64_t B, int64_t N, int sms) {
  int64_t per_q = (2LL * sms + B - 1) / B;
  int64_t by_rows = (N + 63) / 64;
  int64_t c = per_q < by_rows ? per_q : by_rows;
  if (c > 2LL * sms) c = 2LL * sms;
  if (c < 1) c = 1;
  return (int)c;
}

template <int W, int QB, int KPL>
static cudaError_t launch_bw_t(const ScoreArgs &a, const BwShape &sh, const QuantStatus *qst,
                               cudaStream_t st) {
  const size_t smem = (size_t)sh.ns * sh.stage_bytes + 2 * sh.ns * sizeof(uint64_t) + 16;
  auto kern = a.metric == LAM_METRIC_IP ? score_bw_kernel<W, QB, KPL, false>
                                        : score_bw_kernel<W, QB, KPL, true>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  timing_launch_begin(LAM_TIME_SCORE, st);
  kern<<<a.n_lists, kBwThreads, smem, st>>>(a, sh.tr, sh.ns, sh.stage_bytes, qst);
  timing_launch_end(LAM_TIME_SCORE, st);
  return cudaGetLastError();
}

template <int W, int QB>
static cudaError_t launch_bw_k(const ScoreArgs &a, const BwShape &sh, const QuantStatus *qst,
                               cudaStream_t st) {
  if (a.k <= 32) return launch_bw_t<W, QB, 1>(a, sh, qst, st);
  return launch_bw_t<W, QB, 4>(a, sh, qst, st);
}

template <int W>
static cudaError_t launch_bw_w(const ScoreArgs &a, const QuantStatus *qst, cudaStream_t st) {
  const BwShape sh = bw_shape(a.D, W);
  // merge scratch (QB * 8 warps * k keys) must fit in the stage buffers
  if ((size_t)2 * kBwWarps * a.k * 8 > (size_t)sh.ns * sh.stage_bytes) return cudaErrorInvalidValue;
  return a.B == 1 ? launch_bw_k<W, 1>(a, sh, qst, st) : launch_bw_k<W, 2>(a, sh, qst, st);
}

cudaError_t launch_score_bandwidth(const ScoreArgs &a, cudaStream_t st, const QuantStatus *qst) {
  if (qst != nullptr) {  // width on the device: both variants, one runs
    const cudaError_t e = launch_bw_w<1>(a, qst, st);
    return e != cudaSuccess ? e : launch_bw_w<2>(a, qst, st);
  }
  return a.width == 1 ? launch_bw_w<1>(a, nullptr, st) : launch_bw_w<2>(a, nullptr, st);
}

template <int FMT, int QB, int KPL>
static cudaError_t launch_bw_rows_t(const ScoreArgs &a, const RowPtrs &rp, const BwShape &sh,
                                   cudaStream_t st) {
  const size_t smem = (size_t)sh.ns * sh.stage_bytes + 2 * sh.ns * sizeof(uint64_t) + 16;
  auto kern = a.metric == LAM_METRIC_IP ? score_bw_rows_kernel<FMT, QB, KPL, false>
                                        : score_bw_rows_kernel<FMT, QB, KPL, true>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  timing_launch_begin(LAM_TIME_SCORE, st);
  kern<<<a.n_lists, kBwThreads, smem, st>>>(a, rp, sh.tr, sh.ns, sh.stage_bytes);
  timing_launch_end(LAM_TIME_SCORE, st);
  return cudaGetLastError();
}

template <int FMT>
static cudaError_t launch_bw_rows_f(const ScoreArgs &a, const RowPtrs &rp, const BwShape &sh,
                                   cudaStream_t st) {
  if (a.B == 1)
    return a.k <= 32 ? launch_bw_rows_t<FMT, 1, 1>(a, rp, sh, st)
                     : launch_bw_rows_t<FMT, 1, 4>(a, rp, sh, st);
  return a.k <= 32 ? launch_bw_rows_t<FMT, 2, 1>(a, rp, sh, st)
                   : launch_bw_rows_t<FMT, 2, 4>(a, rp, sh, st);
}

template <int QB, int KPL>
static cudaError_t launch_bw_sign_t(const ScoreArgs &a, const RowPtrs &rp, const BwShape &sh,
                                   cudaStream_t st) {
  const size_t smem = (size_t)sh.ns * sh.stage_bytes + (size_t)QB * (a.D / 4) * 16 * 4 +
                      16 * QB + 2 * sh.ns * sizeof(uint64_t) + 16;
  auto pick = [&](auto cc) {
    constexpr bool CC = decltype(cc)::value;
    return a.D == 768    ? score_bw_sign_kernel<QB, KPL, CC, 6>
           : a.D == 1024 ? score_bw_sign_kernel<QB, KPL, CC, 8>
                         : score_bw_sign_kernel<QB, KPL, CC, 0>;
  };
  auto kern = a.metric == LAM_METRIC_IP ? pick(std::integral_constant<bool, false>{})
                                        : pick(std::integral_constant<bool, true>{});
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  timing_launch_begin(LAM_TIME_SCORE, st);
  kern<<<a.n_lists, kBwThreads, smem, st>>>(a, rp, sh.tr, sh.ns, sh.stage_bytes);
  timing_launch_end(LAM_TIME_SCORE, st);
  return cudaGetLastError();
}

static cudaError_t launch_bw_sign(const ScoreArgs &a, const RowPtrs &rp, const BwShape &sh,
                                  cudaStream_t st) {
  if (a.B == 1)
    return a.k <= 32 ? launch_bw_sign_t<1, 1>(a, rp, sh, st) : launch_bw_sign_t<1, 4>(a, rp, sh, st);
  return a.k <= 32 ? launch_bw_sign_t<2, 1>(a, rp, sh, st) : launch_bw_sign_t<2, 4>(a, rp, sh, st);
}

int rows_row_bytes(int fmt, int D) {
  return fmt == LAM_ROWS_INT8 ? D : fmt == LAM_ROWS_FP16 ? 2 * D : D / 8;
}

int bandwidth_rows_ctas(int64_t N, int fmt, int D, int sms) {
  return bandwidth_ctas(N, rows_row_bytes(fmt, D), 1, sms);
}

cudaError_t launch_score_bandwidth_rows(const ScoreArgs &a, const RowPtrs &rp, cudaStream_t st) {
  const BwShape sh = bw_shape(rows_row_bytes(a.fmt, a.D), 1);
  if ((size_t)2 * kBwWarps * a.k * 8 > (size_t)sh.ns * sh.stage_bytes) return cudaErrorInvalidValue;
  if (a.fmt == LAM_ROWS_INT8) return launch_bw_rows_f<LAM_ROWS_INT8>(a, rp, sh, st);
  if (a.fmt == LAM_ROWS_FP16) return launch_bw_rows_f<LAM_ROWS_FP16>(a, rp, sh, st);
  return launch_bw_sign(a, rp, sh, st);
}

cudaError_t launch_score_generic(const ScoreArgs &a, cudaStream_t st, const RowPtrs &rp) {
  const size_t smem = (size_t)kGenWarps * a.k * sizeof(uint64_t);
  cudaError_t e = cudaFuncSetAttribute(score_generic_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(a.n_lists, (unsigned)(a.B < 65535 ? a.B : 65535));
  timing_launch_begin(LAM_TIME_SCORE, st);
  score_generic_kernel<<<grid, kGenWarps * 32, smem, st>>>(a, rp);
  timing_launch_end(LAM_TIME_SCORE, st);
  return cudaGetLastError();
}

template <int HPL>
static cudaError_t launch_kmerge_t(const ScoreArgs &a, cudaStream_t st, const RowPtrs &rp,
                                   int mode, int kout) {
  const size_t per_q = (size_t)a.n_lists * a.k * 8;
  int64_t qpc = (int64_t)(kKmCandBytes / per_q);
  if (qpc > kKmWarps) qpc = kKmWarps;  // one query per warp
  // at least ~2 CTAs per SM when the batch allows: the merge is latency-bound
  const int64_t spread = (a.B + 2LL * a.sms - 1) / (2LL * a.sms);
  if (qpc > spread) qpc = spread;
  if (qpc > a.B) qpc = a.B;
  if (qpc < 1) qpc = 1;
  const size_t smem = (size_t)qpc * per_q + (size_t)kKmWarps * next_pow2(a.k) * 8;
  auto kern = topk_kmerge_kernel<HPL>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  // (the gated merge of a two-pass search counts as an auxiliary launch)
  const int kind = mode == 2 ? LAM_TIME_AUX : LAM_TIME_MERGE;
  timing_launch_begin(kind, st);
  kern<<<(unsigned)((a.B + qpc - 1) / qpc), kKmWarps * 32, smem, st>>>(a, (int)qpc, rp, mode,
                                                                       kout);
  timing_launch_end(kind, st);
  return cudaGetLastError();
}

template <int HPL>
static cudaError_t launch_slab_merge_t(const ScoreArgs &a, int list0, int n_lists, int slab,
                                      uint64_t *out, float *seed, cudaStream_t st) {
  const size_t per_q = (size_t)n_lists * a.k * 8;
  const bool staged = per_q <= kKmCandBytes;
  int64_t qpc = staged ? (int64_t)(kKmCandBytes / per_q) : kSmWarps;
  if (qpc > kSmWarps) qpc = kSmWarps;
  const int64_t spread = (a.B + 2LL * a.sms - 1) / (2LL * a.sms);
  if (qpc > spread) qpc = spread;
  if (qpc < 1) qpc = 1;
  const size_t smem = staged ? (size_t)qpc * per_q : 0;
  auto kern = slab_merge_kernel<HPL>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kern<<<(unsigned)((a.B + qpc - 1) / qpc), kSmWarps * 32, smem, st>>>(a, list0, n_lists, (int)qpc,
                                                                      staged, slab, out, seed);
  return cudaGetLastError();
}

cudaError_t launch_slab_merge(const ScoreArgs &a, int list0, int n_lists, int slab, uint64_t *out,
                              float *seed, cudaStream_t st) {
  if (n_lists <= 32) return launch_slab_merge_t<1>(a, list0, n_lists, slab, out, seed, st);
  if (n_lists <= 64) return launch_slab_merge_t<2>(a, list0, n_lists, slab, out, seed, st);
  if (n_lists <= 128) return launch_slab_merge_t<4>(a, list0, n_lists, slab, out, seed, st);
  if (n_lists <= 256) return launch_slab_merge_t<8>(a, list0, n_lists, slab, out, seed, st);
  return cudaErrorInvalidValue;
}

bool kmerge_fits(int n_lists, int k) {
  return (size_t)n_lists * k * 8 <= kKmCandBytes && n_lists <= 512;
}

cudaError_t launch_topk_merge(const ScoreArgs &a, cudaStream_t st, const RowPtrs &rp, int mode,
                              int kout) {
  // warp k-way merge when one query's candidates fit the shared-memory budget
  if (kmerge_fits(a.n_lists, a.k)) {
    if (a.n_lists <= 32) return launch_kmerge_t<1>(a, st, rp, mode, kout);
    if (a.n_lists <= 64) return launch_kmerge_t<2>(a, st, rp, mode, kout);
    if (a.n_lists <= 128) return launch_kmerge_t<4>(a, st, rp, mode, kout);
    if (a.n_lists <= 256) return launch_kmerge_t<8>(a, st, rp, mode, kout);
    return launch_kmerge_t<16>(a, st, rp, mode, kout);
  }
  if (mode != 0) return cudaErrorInvalidValue;  // two-pass searches plan for the k-way merge
  const int64_t total = (int64_t)a.n_lists * a.k;
  int P = total <= kMergeCap ? next_pow2(total) : kMergeCap;
  if (P < 64) P = 64;
  const size_t smem = ((size_t)P + kMaxK) * sizeof(uint64_t);  // + rescoring scratch
  cudaError_t e = cudaFuncSetAttribute(topk_merge_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int threads = P / 2 < 32 ? 32 : (P / 2 > kMergeThreads ? kMergeThreads : P / 2);
  timing_launch_begin(LAM_TIME_MERGE, st);
  topk_merge_kernel<<<(unsigned)a.B, threads, smem, st>>>(a, P, rp);
  timing_launch_end(LAM_TIME_MERGE, st);
  return cudaGetLastError();
}

}  // namespace lam
