// score_tm.cu -- exact search on the codes for small query batches (3 to 64
// queries) on the tcgen05 tensor cores, with the codes in the MMA M dimension
// (Sec. "Brute-force scan crossover": the scan over the retained memory is a
// matrix-vector product per query; a few queries sharing one pass over the
// codes keep it bandwidth-bound, so the MMAs must stay off its critical path).
//
// Orientation.  A = 128 code rows (fp16, converted from the raw int8/int16
// codes straight into tensor memory by the converter warps: no fp16 copy of
// the codes in shared memory), B = the NQ query rows' fp16 hi terms followed
// by their lo terms (N = 2 NQ: one MMA per K step), D = 128 rows x 2 NQ fp32
// in tensor memory; the score's accumulator is D[hi column] + D[lo column].
// Exactness is that of the other tensor path: codes with |c| <= 2048 are
// exact in fp16, each query is scaled by 2^e and split as hi + lo with
// |q 2^e - hi - lo| <= 2^-22 |q 2^e|, every product is exact in fp32, only
// the accumulation order differs from the CUDA cores.
//
// CTA: a contiguous range of 128-row tiles.  Per 64-wide K slice of a tile:
// one A stage in tensor memory (32 columns of fp16 pairs), fed by a 16 KB raw
// stage (2-D TMA, 128 rows x 128 bytes, 128-byte swizzle; an int8 stage spans
// two K slices), and one query slice (hi and lo images of the query block's
// two 32-wide K chunks, NQ x 64 bytes each).  Tensor memory (512 columns):
// two accumulators at 0 and 128 (2 NQ <= 128 columns), eight A stages at
// 256 + 32 s.
//
// Warp roles (warp w reaches TMEM lanes 32 (w % 4) .. + 31):
//   warp 0       raw-code TMA producer;
//   warp 1       TMEM allocation; one lane issues the MMAs and commits;
//   warp 2       query-slice producer (bulk copies);
//   converters   kTmSets sets of 4 warps, thread = code row; set j converts
//                the raw stages j, j + kTmSets, ... (so the sets' load ->
//                convert -> tensor-memory store chains overlap): raw codes ->
//                fp16 pairs -> tcgen05.st into the A stage; each row's sum of
//                c^2 (cosine / L2) in integers, added across the sets;
//   epilogue     4 warps.  Thread = code row: tcgen05.ld of the row's hi and
//                lo columns, summed, scored and written to a shared-memory
//                score tile S[row][query] (the accumulator is then free);
//                then thread = (query, slice of rows): a scan of its column
//                of S in increasing row order into a per-thread register
//                top-k (all lanes insert in parallel, each for its own
//                query); at the end the 2 to 8 lists of each query merge.
// Every wait is bounded; a timeout records LAM_ERR_TIMEOUT and unwinds.
#include "score_common.cuh"
#include "tc_common.cuh"

#include <type_traits>

namespace lam {

namespace {

constexpr int kTmRows = 128;          // code rows per tile (MMA M)
constexpr int kTmK = 64;              // K of one A stage / query slice
constexpr int kTmRawRow = 128;        // bytes of one code row per raw stage
constexpr int kTmRawBytes = kTmRows * kTmRawRow;  // 16 KB
constexpr int kTmSets = 2;            // converter sets
constexpr int kTmConvWarps = 4 * kTmSets;
constexpr int kTmEpiWarps = 4;
constexpr int kTmThreads = 32 * (3 + kTmConvWarps + kTmEpiWarps);
constexpr int kTmEpi0 = 3 + kTmConvWarps;  // first epilogue warp
constexpr int kTmAStages = 8;         // A stages in tensor memory
constexpr int kTmRawMax = 12;
constexpr int kTmRawMin = 6;          // raw stages beside a resident query
constexpr int kTmRawRing = 8;         // raw stages beside a query ring
constexpr int kTmQMax = 24;
constexpr int kTmMaxB = 64;
constexpr int kTmMaxK = 32;
constexpr int kTmMaxDynSmem = 232448;  // 227 KB
constexpr uint32_t kTmCols = 512;
constexpr uint32_t kTmAccCols = 128;   // per accumulator buffer: hi and lo columns
constexpr uint32_t kTmACol0 = 256;     // first A-stage column

// The MMAs of one A slice from one asm block (see umma_f16_x4):
// D[tmem] (+)= A[tmem] * B[smem]^T with A: 128 lanes = M rows, each 32-bit
// column two consecutive K elements.  Per 32-wide K chunk c < nc and K step
// j: the A columns a[2c + j] times the chunk's stacked hi/lo query operand
// b[c] (32 bytes per K step).
__device__ __forceinline__ void umma_ts_slice(uint32_t d, int nc, const uint32_t (&a)[4],
                                              const uint64_t (&b)[2], uint32_t idesc,
                                              uint32_t accumulate) {
  constexpr uint64_t k1 = (16 * 2) >> 4;
  if (nc == 2) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %10, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %5, %9, p;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%2], %6, %9, 1;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%3], %7, %9, 1;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%4], %8, %9, 1;\n\t}" ::"r"(d),
        "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "l"(b[0]), "l"(b[0] + k1), "l"(b[1]),
        "l"(b[1] + k1), "r"(idesc), "r"(accumulate)
        : "memory");
  } else {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %6, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %3, %5, p;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%2], %4, %5, 1;\n\t}" ::"r"(d),
        "r"(a[0]), "r"(a[1]), "l"(b[0]), "l"(b[0] + k1), "r"(idesc), "r"(accumulate)
        : "memory");
  }
}

// 32 consecutive 32-bit columns of this warp's 32 TMEM lanes (register i ->
// column i), then wait until the stores have landed.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
      "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
      "r"(v[15]), "r"(v[16]), "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]),
      "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]),
      "r"(v[29]), "r"(v[30]), "r"(v[31])
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// Named barrier of the epilogue warps (id 1; 0 is __syncthreads).
__device__ __forceinline__ void epi_sync() {
  asm volatile("bar.sync 1, %0;" ::"r"(kTmEpiWarps * 32) : "memory");
}

}  // namespace

// Shared memory: [raw stages][query slots][score tile: 128 rows x (NQ2 + 1)
// floats, or the threads' final lists, whichever is larger][factor fq,
// ||q||^2 per query][sum of c^2, 2 x 128 rows, 64-bit][barriers, TMEM slot,
// abort flag].  NQ2: the queries' column block of the score tile (16, 32 or
// 64; 128 / NQ2 threads share a query).
struct TmLayout {
  int nr, nq, nqp;  // raw stages, query slots, queries padded to 16
  int qslot_bytes;
  int resident;     // the query slots hold every slice: loaded once, never freed
  size_t q_off, s_off, f_off, cc_off, bar_off, smem_bytes;
};

// Column block of the score tile for B queries (a power of two >= 16).
__host__ __device__ inline int tm_nq2(int64_t B) { return B > 32 ? 64 : B > 16 ? 32 : 16; }

inline TmLayout tm_layout(int64_t B, int D, int k) {
  TmLayout L;
  L.nqp = (int)((B + 15) / 16 * 16);
  L.qslot_bytes = L.nqp * 256;  // hi and lo of two 32-wide K chunks, 64 bytes per row
  const int nka = (D + kTmK - 1) / kTmK;
  const int nq2 = tm_nq2(B);
  const size_t stile = (size_t)kTmRows * (nq2 + 1) * 4, flists = (size_t)kTmRows * k * 8;
  const size_t sbuf = stile > flists ? stile : flists;
  const size_t fac = (size_t)L.nqp * 8;
  const size_t cc = 2 * kTmRows * 8;
  const size_t tailb = 112 * 8 + 1024;  // barriers, slot, flag, alignment slack
  const size_t fixed = sbuf + fac + cc + tailb;
  L.nr = 0;
  L.nq = 0;
  L.resident = 0;
  if (fixed < (size_t)kTmMaxDynSmem) {
    const size_t avail = kTmMaxDynSmem - fixed;
    const size_t all_q = (size_t)nka * L.qslot_bytes;
    if (all_q + (size_t)kTmRawMin * kTmRawBytes <= avail) {
      // every query slice stays resident (each tile reads the same ones)
      L.resident = 1;
      L.nq = nka;
      L.nr = (int)((avail - all_q) / kTmRawBytes);
    } else {
      // a ring: raw stages enough for the HBM latency, query slots with the rest
      L.nr = kTmRawRing;
      L.nq = avail > (size_t)L.nr * kTmRawBytes
                 ? (int)((avail - (size_t)L.nr * kTmRawBytes) / L.qslot_bytes) : 0;
      if (L.nq > kTmQMax) L.nq = kTmQMax;
      while (L.nq < 2 && L.nr > kTmRawMin) {  // (large k: fewer raw stages)
        --L.nr;
        L.nq = (int)((avail - (size_t)L.nr * kTmRawBytes) / L.qslot_bytes);
      }
    }
    if (L.nr > kTmRawMax) L.nr = kTmRawMax;
  }
  L.q_off = (size_t)L.nr * kTmRawBytes;
  L.s_off = L.q_off + (size_t)L.nq * L.qslot_bytes;
  L.f_off = L.s_off + (sbuf + 15) / 16 * 16;
  L.cc_off = (L.f_off + fac + 7) / 8 * 8;
  L.bar_off = L.cc_off + cc;
  L.smem_bytes = L.bar_off + tailb;
  return L;
}

struct TmGeom {
  int nr, nq, nqp, qslot_bytes, resident;
  int q_off, s_off, f_off, cc_off, bar_off;
  const QuantStatus *qst;  // status-driven calls: the codes' width is read here
};

}  // namespace lam

namespace lam {
namespace {

template <int MET>
__device__ __forceinline__ float tm_score(float acc, float fq, float qq, float rf) {
  if constexpr (MET == LAM_METRIC_IP) return fq * acc;
  else if constexpr (MET == LAM_METRIC_COSINE) return (fq * acc) * rf;
  else return fmaf(fq, acc, qq + rf);
}

template <int W, int MET, int KR>
__global__ void __launch_bounds__(kTmThreads, 1)
    score_tm_kernel(const __grid_constant__ CUtensorMap cmap, ScoreArgs a, TmGeom g) {
  // status-driven call: only the variant of the codes' width runs
  if (g.qst != nullptr && (!status_ok(g.qst) || status_width(g.qst) != (uint32_t)W)) return;
  extern __shared__ uint8_t tm_smem_raw[];
  // 1024-byte alignment for the swizzled tiles
  const uint32_t base_u32 = smem_u32(tm_smem_raw);
  uint8_t *smem = tm_smem_raw + (((base_u32 + 1023u) & ~1023u) - base_u32);
  const int nr = g.nr, nq = g.nq, NQ = g.nqp;
  uint8_t *raw_ring = smem;
  uint8_t *qring = smem + g.q_off;
  float *stile = reinterpret_cast<float *>(smem + g.s_off);  // score tile / final lists
  float *fq_s = reinterpret_cast<float *>(smem + g.f_off);
  float *qq_s = fq_s + NQ;
  unsigned long long *ccsum = reinterpret_cast<unsigned long long *>(smem + g.cc_off);
  uint64_t *rfull = reinterpret_cast<uint64_t *>(smem + g.bar_off);
  uint64_t *rempty = rfull + nr;
  uint64_t *qfull = rempty + nr;
  uint64_t *qempty = qfull + nq;
  uint64_t *afull = qempty + nq;
  uint64_t *aempty = afull + kTmAStages;
  uint64_t *accf = aempty + kTmAStages;
  uint64_t *acce = accf + 2;
  uint64_t *ccf = acce + 2;
  uint64_t *cce = ccf + 2;
  uint64_t *done = cce + 2;
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t n_tiles = (a.N + kTmRows - 1) / kTmRows;
  const int64_t tb = (int64_t)blockIdx.x * n_tiles / gridDim.x;
  const int64_t te = (int64_t)(blockIdx.x + 1) * n_tiles / gridDim.x;
  const int ntl = (int)(te - tb);
  const int nk32 = (a.D + 31) / 32;          // 32-wide K chunks of the query image
  const int nka = (a.D + kTmK - 1) / kTmK;   // A slices per tile
  constexpr int SPR = W == 1 ? 2 : 1;        // A slices per raw stage
  const int rpt = (nka + SPR - 1) / SPR;     // raw stages per tile
  constexpr bool CC = MET != LAM_METRIC_IP;
  const int k = a.k;
  const int B = (int)a.B;
  const uint32_t part = (uint32_t)NQ * 64;   // one hi or lo image of one K chunk
  const uint8_t *qA = static_cast<const uint8_t *>(a.qprep);

  if (threadIdx.x == 0) {
    for (int r = 0; r < nr; ++r) {
      mbar_init(&rfull[r], 1);
      mbar_init(&rempty[r], 4);  // the four warps of the set that converts it
    }
    for (int q = 0; q < nq; ++q) {
      mbar_init(&qfull[q], 1);
      mbar_init(&qempty[q], 1);
    }
    for (int s = 0; s < kTmAStages; ++s) {
      mbar_init(&afull[s], 4);
      mbar_init(&aempty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], kTmEpiWarps);
      mbar_init(&ccf[b], kTmConvWarps);
      mbar_init(&cce[b], kTmEpiWarps);
    }
    mbar_init(done, 1);
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  // per-query factor of the score (s 2^-e, 2^-e / ||q|| or -2 s 2^-e, see
  // tm_score) and ||q||^2
  for (int j = threadIdx.x; j < NQ; j += blockDim.x) {
    float fq = 0.0f, qq = 0.0f;
    if (j < B) {
      const float4 qi = reinterpret_cast<const float4 *>(qA + (size_t)nk32 * 16384)[j];
      fq = MET == LAM_METRIC_IP       ? a.s * qi.x
           : MET == LAM_METRIC_COSINE ? (qi.y > 0.0f ? qi.x / qi.y : 0.0f)
                                      : -2.0f * a.s * qi.x;
      qq = qi.z;
    }
    fq_s[j] = fq;
    qq_s[j] = qq;
  }
  for (int i = threadIdx.x; i < 2 * kTmRows; i += blockDim.x) ccsum[i] = 0ull;
  if (warp == 1) tmem_alloc(tmem_slot, kTmCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------ raw-code producer --
    if (lane == 0) {
      const int r_total = producers_stalled(a.gflags) ? 0 : ntl * rpt;
      int gr = 0;
      for (; gr < r_total; ++gr) {
        const int rs = gr % nr, rr = gr / nr;
        if (rr > 0 && !mbar_wait(&rempty[rs], (rr - 1) & 1, abort_flag, a.gflags)) break;
        const int lt = gr / rpt, j = gr - lt * rpt;
        mbar_arrive_expect_tx(&rfull[rs], kTmRawBytes);
        tma_load_2d(raw_ring + (size_t)rs * kTmRawBytes, &cmap, j * (kTmRawRow / W),
                    (int)((tb + lt) * kTmRows), &rfull[rs]);
      }
      for (int t = max(0, gr - nr); t < gr; ++t) drain_wait_tc(&rfull[t % nr], (t / nr) & 1);
    }
  } else if (warp == 2) {
    // ------------------------------------------------ query producer -----
    // slice i of a tile: K chunks 2i and 2i + 1 of the query image, each as
    // its hi rows then its lo rows (one stacked B operand per chunk)
    if (lane == 0) {
      const int q_total = producers_stalled(a.gflags) ? 0 : g.resident ? nka : ntl * nka;
      int it = 0;
      for (; it < q_total; ++it) {
        const int qs = it % nq, rq = it / nq;
        if (rq > 0 && !mbar_wait(&qempty[qs], (rq - 1) & 1, abort_flag, a.gflags)) break;
        const int ai = it % nka, c0 = 2 * ai;
        const int nc = nk32 - c0 < 2 ? nk32 - c0 : 2;
        uint8_t *dst = qring + (size_t)qs * g.qslot_bytes;
        mbar_arrive_expect_tx(&qfull[qs], (uint32_t)nc * 2u * part);
        for (int c = 0; c < nc; ++c)
          for (int h = 0; h < 2; ++h)
            bulk_g2s(dst + (size_t)(2 * c + h) * part, qA + (size_t)(c0 + c) * 16384 + h * 8192,
                     part, &qfull[qs]);
      }
      for (int t = max(0, it - nq); t < it; ++t) drain_wait_tc(&qfull[t % nq], (t / nq) & 1);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer ---------
    if (lane == 0) {
      const uint32_t idesc = idesc_f16(kTmRows, 2 * NQ);
      int it = 0;
      bool ok = true;
      for (int lt = 0; lt < ntl && ok; ++lt) {
        const int buf = lt & 1, u = lt >> 1;
        if (u > 0 && !mbar_wait(&acce[buf], (u - 1) & 1, abort_flag, a.gflags)) break;
        tc_fence_after();
        const uint32_t d = tmem_base + (uint32_t)buf * kTmAccCols;
        for (int ai = 0; ai < nka; ++ai, ++it) {
          const int s = it % kTmAStages, qs = it % nq;
          const uint32_t qpar = g.resident ? 0u : (uint32_t)((it / nq) & 1);
          if (!mbar_wait(&afull[s], (it / kTmAStages) & 1, abort_flag, a.gflags) ||
              ((!g.resident || lt == 0) && !mbar_wait(&qfull[qs], qpar, abort_flag, a.gflags))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t qbase = smem_u32(qring + (size_t)qs * g.qslot_bytes);
          const int nc = nk32 - 2 * ai < 2 ? nk32 - 2 * ai : 2;
          // A: 8 columns per K16 step; B: chunk c's hi and lo rows
          const uint32_t acol = tmem_base + kTmACol0 + (uint32_t)s * 32u;
          const uint32_t aa[4] = {acol, acol + 8u, acol + 16u, acol + 24u};
          const uint64_t bq[2] = {desc_sw64(qbase), desc_sw64(qbase + 2u * part)};
          umma_ts_slice(d, nc, aa, bq, idesc, ai > 0 ? 1u : 0u);
          umma_commit(&aempty[s]);
          if (!g.resident) umma_commit(&qempty[qs]);
        }
        if (ok) umma_commit(&accf[buf]);
      }
      umma_commit(done);
      drain_wait_tc(done, 0);
    }
  } else if (warp < kTmEpi0) {
    // ------------------------------------------------ converters ---------
    const int set = (warp - 3) >> 2;                    // this warp's converter set
    const int quad = warp & 3;                          // its TMEM lane quarter
    const int rloc = quad * 32 + lane;                  // its code row in the tile
    const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
    const __half2 bias = __float2half2_rn(1152.0f);
    bool ok = true;
    float amax = 0.0f;
    for (int lt = 0; lt < ntl && ok; ++lt) {
      const int buf = lt & 1, u = lt >> 1;
      unsigned long long ccp = 0ull;  // the row's sum of c^2 over this set's stages
      for (int ri = 0; ri < rpt; ++ri) {
        const int gr = lt * rpt + ri;
        if (gr % kTmSets != set) continue;
        const int rs = gr % nr;
        if (!warp_wait(&rfull[rs], (gr / nr) & 1, abort_flag, a.gflags)) {
          ok = false;
          break;
        }
        // the row's 128 bytes: 16-byte piece p at p ^ (row & 7) (128-byte swizzle)
        const uint8_t *rowp = raw_ring + (size_t)rs * kTmRawBytes + (size_t)rloc * kTmRawRow;
        uint4 rv[8];
#pragma unroll
        for (int p = 0; p < 8; ++p)
          rv[p] = *reinterpret_cast<const uint4 *>(rowp + ((p ^ (rloc & 7)) << 4));
        __syncwarp();
        if (lane == 0) mbar_arrive(&rempty[rs]);
        int c2 = 0;  // exact: at most 128 int8 or 64 int16 (|c| <= 2048) squares
#pragma unroll
        for (int h = 0; h < SPR; ++h) {
          const int ai = ri * SPR + h;
          if (ai >= nka) break;
          const int it = lt * nka + ai, s = it % kTmAStages, ra = it / kTmAStages;
          if (ra > 0 && !warp_wait(&aempty[s], (ra - 1) & 1, abort_flag, a.gflags)) {
            ok = false;
            break;
          }
          tc_fence_after();
          // 64 codes -> 32 fp16 pairs, word t = codes (2t, 2t + 1) of the slice
          uint32_t o[32];
          if constexpr (W == 1) {
#pragma unroll
            for (int pp = 0; pp < 4; ++pp) {
              const uint4 r4 = rv[4 * h + pp];
              const uint32_t w4[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
              for (int t = 0; t < 4; ++t) {
                // fp16 bits 0x64uu = 1024 + u with u = code + 128; minus 1152 = code
                const uint32_t x = w4[t] ^ 0x80808080u;
                o[8 * pp + 2 * t] =
                    h2_as_u32(__hsub2(u32_as_h2(__byte_perm(x, 0x64646464u, 0x5140)), bias));
                o[8 * pp + 2 * t + 1] =
                    h2_as_u32(__hsub2(u32_as_h2(__byte_perm(x, 0x64646464u, 0x7362)), bias));
                if (CC) c2 = __dp4a((int)w4[t], (int)w4[t], c2);
              }
            }
          } else {
#pragma unroll
            for (int p = 0; p < 8; ++p) {
              const uint32_t w4[4] = {rv[p].x, rv[p].y, rv[p].z, rv[p].w};
#pragma unroll
              for (int t = 0; t < 4; ++t) {
                // each half biased to c + 32768 below 2^23 + 2^16: exact fp32 c
                const uint32_t x = w4[t] ^ 0x80008000u;
                const float f0 = __int_as_float(__byte_perm(x, 0x4B000000u, 0x7410)) - 8421376.0f;
                const float f1 = __int_as_float(__byte_perm(x, 0x4B000000u, 0x7432)) - 8421376.0f;
                amax = fmaxf(amax, fmaxf(fabsf(f0), fabsf(f1)));
                if (CC) {
                  const int c0 = (int)(w4[t] << 16) >> 16, c1 = (int)w4[t] >> 16;
                  c2 += c0 * c0 + c1 * c1;
                }
                o[4 * p + t] = h2_as_u32(__floats2half2_rn(f0, f1));
              }
            }
          }
          tmem_st32(tmem_base + lane_off + kTmACol0 + (uint32_t)s * 32u, o);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&afull[s]);
        }
        if (!ok) break;
        ccp += (unsigned long long)(unsigned)c2;
      }
      if (!ok) break;
      if (CC) {
        // the sets' partial sums of c^2 meet in the tile's row slot
        if (u > 0 && !warp_wait(&cce[buf], (u - 1) & 1, abort_flag, a.gflags)) break;
        if (ccp != 0ull) atomicAdd(&ccsum[buf * kTmRows + rloc], ccp);
        __syncwarp();
        if (lane == 0) mbar_arrive(&ccf[buf]);
      }
    }
    if (W == 2 && amax > 2048.0f) atomicOr(a.gflags, kFlagRange);
  } else {
    // ------------------------------------------------ epilogue -----------
    const int et = threadIdx.x - 32 * kTmEpi0;  // 0 .. 127
    const int quad = warp & 3;
    const int rloc = quad * 32 + lane;           // phase 1: thread = code row
    const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
    const int nq2 = tm_nq2(B), sst = nq2 + 1;    // score tile row stride (no bank conflicts)
    const int sq = et % nq2, sh = et / nq2;      // phase 2: query, slice of nq2 rows
    constexpr bool desc = MET != LAM_METRIC_L2;
    RegTopK<KR> reg;
    reg.init(k);
    float thr = desc ? -INFINITY : INFINITY;  // score of the thread's k-th best
    for (int lt = 0; lt < ntl; ++lt) {
      const int buf = lt & 1, u = lt >> 1;
      if (!warp_wait(&accf[buf], u & 1, abort_flag, a.gflags)) break;
      if (CC && !warp_wait(&ccf[buf], u & 1, abort_flag, a.gflags)) break;
      tc_fence_after();
      const int64_t row0 = (tb + lt) * kTmRows;
      float rf = 0.0f;
      if (CC) {
        // the row's score factor: 1/||c|| (cosine) or s^2 ||c||^2 (L2)
        const float t = (float)ccsum[buf * kTmRows + rloc];
        rf = MET == LAM_METRIC_COSINE ? (t > 0.0f ? 1.0f / sqrtf(t) : 0.0f) : a.s * a.s * t;
        ccsum[buf * kTmRows + rloc] = 0ull;
      }
      // the row's scores for queries 0 .. nq2 - 1 (accumulator = hi + lo column)
      const uint32_t acc0 = tmem_base + lane_off + (uint32_t)buf * kTmAccCols;
      float *srow = stile + rloc * sst;
      for (int c = 0; c * 32 < nq2 && c * 32 < B; ++c) {
        uint32_t hv[32], lv[32];
        tmem_ld32(acc0 + (uint32_t)c * 32u, hv);
        tmem_ld32(acc0 + (uint32_t)NQ + (uint32_t)c * 32u, lv);
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int q = c * 32 + i;
          if (q < nq2 && q < B)
            srow[q] = tm_score<MET>(__uint_as_float(hv[i]) + __uint_as_float(lv[i]), fq_s[q],
                                    qq_s[q], rf);
        }
      }
      // the accumulator is free again before the scores are ranked
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&acce[buf]);
        if (CC) mbar_arrive(&cce[buf]);
      }
      epi_sync();
      if (sq < B) {
        // rows sh * nq2 .. + nq2 - 1 of the tile, in increasing order; a row
        // enters when it beats the k-th best strictly (an equal score of a
        // later row ranks after it)
        const int r0 = sh * nq2;
        const int64_t nvalid = a.N - (row0 + r0);
        const int nrow = nvalid < nq2 ? (int)(nvalid > 0 ? nvalid : 0) : nq2;
        for (int r = 0; r < nrow; ++r) {
          const float sc = stile[(r0 + r) * sst + sq];
          if (desc ? sc > thr : sc < thr) {
            reg.insert(rank_key32(sc, desc), (uint32_t)(row0 + r0 + r));
            const uint32_t tk = reg.key[KR - 1];
            thr = tk == 0xffffffffu ? (desc ? -INFINITY : INFINITY) : rank_key32_score(tk, desc);
          }
        }
      }
      epi_sync();  // (the next tile overwrites the score tile)
    }
    // each thread's list -> shared memory [query][slice][k], then per query
    // the 128 / nq2 lists merge into the CTA's partial list
    uint64_t *fl = reinterpret_cast<uint64_t *>(stile);
    const int tpq = kTmRows / nq2;
    if (sq < B) {
      uint64_t *dst = fl + ((size_t)sq * tpq + sh) * k;
#pragma unroll
      for (int i = 0; i < KR; ++i)
        if (i >= KR - k) dst[i - (KR - k)] = ((uint64_t)reg.key[i] << 32) | reg.id[i];
    }
    epi_sync();
    const int ew = warp - kTmEpi0;
    for (int q = ew; q < B; q += kTmEpiWarps)
      rank_merge(fl + (size_t)q * tpq * k, tpq, k, a.partial + ((size_t)blockIdx.x * a.B + q) * k,
                 lane, 32);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmCols);
  }
}

}  // namespace

bool tm_fits(int64_t B, int D, int k) {
  if (B < 1 || B > kTmMaxB || k < 1 || k > kTmMaxK || D < 1) return false;
  const TmLayout L = tm_layout(B, D, k);
  return L.nr >= 2 && L.nq >= 2 && L.smem_bytes <= (size_t)kTmMaxDynSmem;
}

int tm_box_rows() { return kTmRows; }

cudaError_t launch_score_tm(const ScoreArgs &a, const QuantStatus *qst, const CUtensorMap &cmap1,
                            const CUtensorMap &cmap2, cudaStream_t st) {
  if (!tm_fits(a.B, a.D, a.k)) return cudaErrorInvalidValue;
  const TmLayout L = tm_layout(a.B, a.D, a.k);
  TmGeom g;
  g.nr = L.nr;
  g.nq = L.nq;
  g.nqp = L.nqp;
  g.qslot_bytes = L.qslot_bytes;
  g.resident = L.resident;
  g.q_off = (int)L.q_off;
  g.s_off = (int)L.s_off;
  g.f_off = (int)L.f_off;
  g.cc_off = (int)L.cc_off;
  g.bar_off = (int)L.bar_off;
  g.qst = qst;
  auto run = [&](auto kern, const CUtensorMap &cmap) -> cudaError_t {
    cudaError_t r =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)L.smem_bytes);
    if (r != cudaSuccess) return r;
    timing_launch_begin(LAM_TIME_SCORE, st);
    kern<<<(unsigned)a.n_lists, kTmThreads, L.smem_bytes, st>>>(cmap, a, g);
    timing_launch_end(LAM_TIME_SCORE, st);
    return cudaGetLastError();
  };
  auto by_k = [&](auto wtag, auto mtag, const CUtensorMap &cmap) -> cudaError_t {
    constexpr int W = decltype(wtag)::value, MET = decltype(mtag)::value;
    return a.k <= 16 ? run(score_tm_kernel<W, MET, 16>, cmap) : run(score_tm_kernel<W, MET, 32>, cmap);
  };
  auto by_metric = [&](auto wtag, const CUtensorMap &cmap) -> cudaError_t {
    if (a.metric == LAM_METRIC_IP)
      return by_k(wtag, std::integral_constant<int, LAM_METRIC_IP>{}, cmap);
    if (a.metric == LAM_METRIC_COSINE)
      return by_k(wtag, std::integral_constant<int, LAM_METRIC_COSINE>{}, cmap);
    return by_k(wtag, std::integral_constant<int, LAM_METRIC_L2>{}, cmap);
  };
  if (qst != nullptr) {
    const cudaError_t r = by_metric(std::integral_constant<int, 1>{}, cmap1);
    return r != cudaSuccess ? r : by_metric(std::integral_constant<int, 2>{}, cmap2);
  }
  return a.width == 1 ? by_metric(std::integral_constant<int, 1>{}, cmap1)
                      : by_metric(std::integral_constant<int, 2>{}, cmap2);
}

}  // namespace lam
