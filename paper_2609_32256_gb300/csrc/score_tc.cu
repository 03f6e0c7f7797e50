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
// CTA: 128 queries (MMA M) x a contiguous range of 256-row tiles (MMA N).
// Two shared-memory rings:
//   MMA stages (two K = 32 chunks): the query block's hi/lo tiles, laid out by
//     the query preparation kernel exactly as the 64-byte-swizzled UMMA
//     operand, so one 32 KB bulk copy fills them; and the fp16 code tiles the
//     converters write;
//   raw stages (two to four): 256 code rows x 128 bytes (K = 128 int8 / 64
//     int16) by one 2-D TMA load with the 128-byte swizzle.
// Warp roles (352 threads; warp w runs on SM sub-partition w % 4):
//   warp 0      producer of the raw-code TMA loads;
//   warp 1      TMEM allocation; one lane issues tcgen05.mma (2 K-steps x
//               hi/lo per chunk) and commits stage/accumulator barriers;
//   warps 2-5   convert raw int8/int16 codes to fp16 in the UMMA K-major
//               64B-swizzled layout, and sum c^2 per row for cosine / L2;
//   warps 6-9   epilogue: tcgen05.ld of the 128x256 fp32 accumulator (double
//               buffered, 2 x 256 TMEM columns), scores, per-query top-k; a
//               warp whose 32 MMA rows hold no query sits out;
//   warp 10     producer of the query-block bulk copies.
// Every wait is bounded; a timeout records LAM_ERR_TIMEOUT and unwinds.
#include "score_common.cuh"
#include "tc_common.cuh"

#include <cstdio>
#include <cstdlib>
#include <cstring>

namespace lam {

namespace {

constexpr int kBM = 128;        // queries per CTA (MMA M)
constexpr int kBN = 256;        // code rows per tile (MMA N)
constexpr int kBK = 32;         // fp16 per stage along D (64-byte rows)
static_assert(kBK == 32, "tensor_k_extent (lam_internal.cuh) rounds D to 32-wide K chunks");
constexpr int kTcThreads = 352;  // 11 warps, roles below
constexpr int kConvThreads = 128;
constexpr int kABytes = kBM * kBK * 2;    // one of hi / lo: 8 KB
constexpr int kAStage = 2 * kABytes;      // hi + lo, one bulk copy: 16 KB
constexpr int kB16Bytes = kBN * kBK * 2;  // converted codes: 16 KB
constexpr int kStageBytes = kAStage + kB16Bytes;  // one MMA stage: 32 KB
constexpr int kRawRow = 128;              // bytes of one code row per raw stage
constexpr int kRawBytes = kBN * kRawRow;  // one raw stage: 32 KB
constexpr int kRawMax = 4;                // raw stages at most
constexpr int kCBuf = 16;                 // k > 32: heap candidate buffer depth at most
constexpr int kTcChunks = 2;              // K chunks per MMA stage of the stage-loop kernel
constexpr uint32_t kTmemCols = 512;       // two 256-column accumulators
constexpr int kMaxDynSmem = 232448;       // 227 KB
constexpr int kTcMaxK = 128;
// M = 128 queries, N = 256 code rows
constexpr uint32_t kIdesc = idesc_f16(kBM, kBN);
constexpr uint32_t kIdescPair = idesc_f16(2 * kBM, kBN);  // a CTA pair: M = 256

// Candidate mask of one 32-column chunk: bit j is set when column j's score
// (tile_score, the same roundings) beats thr: greater for inner product and
// cosine, smaller for L2.  rf(j) gives column j's row factor.  The metric is a
// template argument so that the 32-wide loop carries no per-element dispatch.
template <int MET, typename RF>
__device__ __forceinline__ uint32_t chunk_mask_m(const uint32_t (&v)[32], float fq, float qq,
                                                 float thr, RF rf) {
  uint32_t mask = 0;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const float acc = __uint_as_float(v[j]);
    float sc;
    if constexpr (MET == LAM_METRIC_IP) sc = fq * acc;
    else if constexpr (MET == LAM_METRIC_COSINE) sc = (fq * acc) * rf(j);
    else sc = fmaf(fq, acc, qq + rf(j));
    const bool beat = MET == LAM_METRIC_L2 ? sc < thr : sc > thr;
    mask |= (uint32_t)beat << j;
  }
  return mask;
}
template <typename RF>
__device__ __forceinline__ uint32_t chunk_mask(int metric, const uint32_t (&v)[32], float fq,
                                               float qq, float thr, RF rf) {
  if (metric == LAM_METRIC_IP) return chunk_mask_m<LAM_METRIC_IP>(v, fq, qq, thr, rf);
  if (metric == LAM_METRIC_COSINE) return chunk_mask_m<LAM_METRIC_COSINE>(v, fq, qq, thr, rf);
  return chunk_mask_m<LAM_METRIC_L2>(v, fq, qq, thr, rf);
}

// k > 32 heaps: candidates that beat the heap root are buffered per query
// (cbn slots per query in shared memory, stride kBM) and poured into the heaps
// when one query's buffer is full, so the lanes of a warp sift together
// instead of one at a time (sparse candidates otherwise leave 31 lanes idle
// for every insertion).
__device__ __forceinline__ void heap_pour(uint64_t *lists, int k, const uint64_t *hb, int m,
                                          int &cnt, float &thr_s, bool desc) {
  for (int i = 0; i < cnt; ++i) {
    const uint64_t key = hb[(size_t)i * kBM + m];
    if (key < lists[m]) heap_replace_root(lists, k, kBM, m, key);
  }
  cnt = 0;
  const uint64_t root = lists[m];
  thr_s = root == kSentinel ? (desc ? -INFINITY : INFINITY)
                            : rank_key32_score((uint32_t)(root >> 32), desc);
}

__device__ __forceinline__ float warp_sum_tc(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

__device__ __forceinline__ float warp_max_tc(float v) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
  return v;
}

// Converter thread -> (tile row, 16-byte piece) of its i-th task, chosen so
// that each quarter-warp's 16-byte accesses fall in distinct banks both when
// reading the raw rows (128 bytes, piece ^ row & 7) and when writing the fp16
// rows (64 bytes, piece ^ (row >> 1) & 3).  int16: a quarter-warp takes rows
// {j, j ^ 5} of an 8-row block (four pieces each); int8: rows {0, 2, 5, 7} or
// {1, 3, 4, 6} of the block (two pieces each).  Lanes of one row differ in
// the low bits of the thread index (for the c^2 shuffles).
template <int W>
__device__ __forceinline__ int conv_row(int ct, int i) {
  const int q = ct >> 3, e = ct & 7;
  if (W == 2) {
    const int j = q & 3;
    return 32 * i + 8 * (q >> 2) + ((e >> 2) ? (j ^ 5) : j);
  }
  const int slot = e >> 1;
  return 64 * i + 8 * (q >> 1) + ((2 * slot + (slot >> 1)) ^ (q & 1));
}
template <int W>
__device__ __forceinline__ int conv_sub(int ct) {
  return W == 2 ? ct & 3 : ct & 1;
}

template <bool B>
struct BoolTag {
  static constexpr bool value = B;
};

struct TcLayout {
  int ns, nr, chunks;  // MMA stages, raw stages, K chunks per MMA stage
  size_t raw_off, lists_off, cbuf_off, cc_off, bar_off, smem_bytes;
};

// Shared memory: [MMA stages][raw stages][k > 32: per-query heaps and their
// candidate buffers][cosine / L2: c^2 per row, 2 tiles][barriers, TMEM slot,
// abort flag].  The heaps' buffers take up to kCBuf slots per query, as many
// as leave room for two single-chunk MMA stages and one raw stage (the kernel
// reads the depth back from the offsets).  Raw stages fill what is left, up to
// kRawMax: the deeper the ring, the more code bytes are in flight while the
// converters work.  (The inner-product layout, without the c^2 buffers, fits
// a third raw stage beside two double-chunk MMA stages.)
inline TcLayout tc_layout(int width, int k, bool cc_rows = true) {
  (void)width;
  TcLayout L;
  const size_t lists = k > 32 ? (size_t)kBM * k * 8 : 0;
  const size_t cc = cc_rows ? 2 * kBN * 4 : 0;
  const size_t tailb = 64 * 8 + 1024;  // barriers, slots, alignment slack
  size_t cbuf = 0;
  if (k > 32) {
    const size_t room = kMaxDynSmem - lists - cc - tailb;
    const size_t need = 2 * (size_t)kStageBytes + kRawBytes;
    const size_t slots = room > need ? (room - need) / ((size_t)kBM * 8) : 0;
    cbuf = (slots < (size_t)kCBuf ? slots : (size_t)kCBuf) * kBM * 8;
  }
  const size_t avail = kMaxDynSmem - lists - cbuf - cc - tailb;
  // two K chunks per MMA stage (one 32 KB copy of the query blocks, 8 MMAs
  // per barrier round trip) when two such stages and two raw stages fit
  L.chunks = (size_t)2 * kTcChunks * kStageBytes + (size_t)2 * kRawBytes <= avail ? kTcChunks : 1;
  int ns = L.chunks > 1 ? 2 : 3, nr = 0;
  for (;; --ns) {
    const size_t mma = (size_t)ns * L.chunks * kStageBytes;
    nr = mma < avail ? (int)((avail - mma) / kRawBytes) : 0;
    if (nr > kRawMax) nr = kRawMax;
    if (nr >= 2 || ns == 2) break;
  }
  if (nr < 1) ns = 0;
  L.ns = ns;
  L.nr = nr;
  L.raw_off = (size_t)ns * L.chunks * kStageBytes;
  L.lists_off = L.raw_off + (size_t)nr * kRawBytes;
  L.cbuf_off = L.lists_off + lists;
  L.cc_off = L.cbuf_off + cbuf;
  L.bar_off = L.cc_off + cc;
  L.smem_bytes = L.bar_off + tailb;
  return L;
}

struct TcGeom {
  int ns, nr, chunks;  // MMA stages, raw stages, 32-wide K chunks per MMA stage
  int raw_off, lists_off, cbuf_off, cc_off, bar_off;
  int qoff;  // MMA row of the block's first query (64 for one block of <= 64)
  const QuantStatus *qst;  // status-driven calls: the codes' width is read here
  int hi;    // hi-only pass: the lo term of the query is neither copied nor multiplied
  int gate;  // full pass of a two-pass search: runs only if a query was not certified
};

template <int W, int KR>
__global__ void __launch_bounds__(kTcThreads, 1)
    score_tc_kernel(const __grid_constant__ CUtensorMap cmap, ScoreArgs a, TcGeom g) {
  // status-driven call: only the variant of the codes' width runs
  if (g.qst != nullptr && (!status_ok(g.qst) || status_width(g.qst) != (uint32_t)W)) return;
  if (g.gate && hi_all_certified(a.gflags)) return;
  extern __shared__ uint8_t tc_smem_raw[];
  // 1024-byte alignment for the swizzled tiles (address bits drive the swizzle)
  const uint32_t base_u32 = smem_u32(tc_smem_raw);
  uint8_t *smem = tc_smem_raw + (((base_u32 + 1023u) & ~1023u) - base_u32);
  const int ns = g.ns, nr = g.nr, C = g.chunks;
  const size_t stage_stride = (size_t)C * kStageBytes;  // [C query blocks][C code blocks]
  uint8_t *raw_ring = smem + g.raw_off;
  uint64_t *lists = reinterpret_cast<uint64_t *>(smem + g.lists_off);
  uint8_t *cbuf = smem + g.cbuf_off;  // k > 32: the heaps' candidate buffers
  float *ccbuf = reinterpret_cast<float *>(smem + g.cc_off);
  uint64_t *afull = reinterpret_cast<uint64_t *>(smem + g.bar_off);
  uint64_t *conv = afull + ns;
  uint64_t *empty = conv + ns;
  uint64_t *rfull = empty + ns;
  uint64_t *rempty = rfull + nr;
  uint64_t *accf = rempty + nr;
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
  constexpr int R = kRawRow / (kBK * W);  // K chunks per raw stage: 4 (int8), 2 (int16)
  const bool need_cc = a.metric != LAM_METRIC_IP;
  const uint8_t *qA = static_cast<const uint8_t *>(a.qprep);
  // Epilogue warps whose 32 MMA rows hold queries; the others sit out (the
  // query rows are g.qoff .. row_end - 1 of the block).
  const int64_t q_left = a.B - (int64_t)qb * kBM;
  const int row_end = g.qoff + (int)(q_left < kBM - g.qoff ? q_left : kBM - g.qoff);
  auto quad_used = [&](int q) { return 32 * q < row_end && 32 * q + 32 > g.qoff; };
  const uint32_t n_epi = 32u * (uint32_t)(quad_used(0) + quad_used(1) + quad_used(2) + quad_used(3));

  if (threadIdx.x == 0) {
    for (int s = 0; s < ns; ++s) {
      mbar_init(&afull[s], 1);
      mbar_init(&conv[s], kConvThreads);
      mbar_init(&empty[s], 1);
    }
    for (int r = 0; r < nr; ++r) {
      mbar_init(&rfull[r], 1);
      mbar_init(&rempty[r], kConvThreads);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], n_epi);
      mbar_init(&ccf[b], kConvThreads);
      mbar_init(&cce[b], n_epi);
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
    // ------------------------------------------------ producer -----------
    if (lane == 0) {
      // raw code stages, freed by the converters
      const int rpt = (nk + R - 1) / R;  // raw stages per tile
      const int r_total = producers_stalled(a.gflags) ? 0 : ntl * rpt;
      int gr = 0;
      for (; gr < r_total; ++gr) {
        const int rs = gr % nr, rr = gr / nr;
        if (rr > 0 && !mbar_wait(&rempty[rs], (rr - 1) & 1, abort_flag, a.gflags)) break;
        const int lt = gr / rpt, j = gr - lt * rpt;
        mbar_arrive_expect_tx(&rfull[rs], kRawBytes);
        tma_load_2d(raw_ring + (size_t)rs * kRawBytes, &cmap, j * (kRawRow / W),
                    (int)(tb + lt) * kBN, &rfull[rs]);
      }
      for (int t = max(0, gr - nr); t < gr; ++t) drain_wait_tc(&rfull[t % nr], (t / nr) & 1);
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
        for (int kc = 0; kc < nk; kc += C, ++it) {
          const int s = it % ns, r = it / ns;
          const int nc = nk - kc < C ? nk - kc : C;
          if (!mbar_wait(&afull[s], r & 1, abort_flag, a.gflags) ||
              !mbar_wait(&conv[s], r & 1, abort_flag, a.gflags)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = smem_u32(smem + (size_t)s * stage_stride);
          // the stage's MMAs from one asm block (see umma_chunks)
          uint64_t ahi[2], alo[2], bd[2];
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            ahi[c] = desc_sw64(st + c * kAStage);
            alo[c] = desc_sw64(st + c * kAStage + kABytes);
            bd[c] = desc_sw64(st + C * kAStage + c * kB16Bytes);
          }
          umma_chunks(d_tmem, nc, ahi, alo, bd, g.hi != 0, kIdesc, kc > 0 ? 1u : 0u);
          umma_commit(&empty[s]);
        }
        if (ok) umma_commit(&accf[buf]);
      }
      umma_commit(done);
      drain_wait_tc(done, 0);
    }
  } else if (warp < 6) {
    // ------------------------------------------------ converters ---------
    // (CC: the row's sum of c^2 is needed, cosine and L2)
    auto converters = [&](auto cc_tag) {
      constexpr bool CC = decltype(cc_tag)::value;
      const int ct = threadIdx.x - 64;  // 0 .. 127
      constexpr int kTasks = (W == 1 ? 512 : 1024) / kConvThreads;  // 16-byte chunks per thread
      const __half2 bias = __float2half2_rn(1152.0f);
      int it = 0, gr = 0;
      bool ok = true;
      float amax = 0.0f, ccmax = 0.0f;
      for (int lt = 0; lt < ntl && ok; ++lt) {
        const int buf = lt & 1, u = lt >> 1;
        float ccp[kTasks];
#pragma unroll
        for (int i = 0; i < kTasks; ++i) ccp[i] = 0.0f;
        for (int kc = 0; kc < nk; ++kc) {
          const int rs = gr % nr;
          if (kc % R == 0 && !mbar_wait(&rfull[rs], (gr / nr) & 1, abort_flag, a.gflags)) {
            ok = false;
            break;
          }
          const int s = it % ns, r = it / ns;
          if (kc % C == 0 && r > 0 && !mbar_wait(&empty[s], (r - 1) & 1, abort_flag, a.gflags)) {
            ok = false;
            break;
          }
          const uint8_t *__restrict__ raw = raw_ring + (size_t)rs * kRawBytes;
          uint8_t *__restrict__ b16 =
              smem + (size_t)s * stage_stride + (size_t)C * kAStage + (size_t)(kc % C) * kB16Bytes;
          const int j0 = (kc % R) * (kBK * W / 16);  // first 16-byte chunk of this K slice
          // All loads first: the stores below could alias them as far as the
          // compiler knows, which would otherwise serialise the tasks.  Raw rows
          // are 128 bytes in the 128-byte swizzle (chunk ^ row & 7).
          uint4 rv[kTasks];
#pragma unroll
          for (int i = 0; i < kTasks; ++i) {
            const int row = conv_row<W>(ct, i), sub = conv_sub<W>(ct);
            rv[i] = *reinterpret_cast<const uint4 *>(raw + row * kRawRow +
                                                     (((j0 + sub) ^ (row & 7)) << 4));
          }
          if constexpr (W == 1) {
#pragma unroll
            for (int i = 0; i < kTasks; ++i) {
              const int row = conv_row<W>(ct, i), h = conv_sub<W>(ct);
              const uint32_t w[4] = {rv[i].x, rv[i].y, rv[i].z, rv[i].w};
              uint32_t o[8];
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                const uint32_t x = w[j] ^ 0x80808080u;
                // fp16 bits 0x64uu = 1024 + u with u = code + 128; minus 1152 = code
                o[2 * j] = h2_as_u32(__hsub2(u32_as_h2(__byte_perm(x, 0x64646464u, 0x5140)), bias));
                o[2 * j + 1] =
                    h2_as_u32(__hsub2(u32_as_h2(__byte_perm(x, 0x64646464u, 0x7362)), bias));
              }
              const int sw = (row >> 1) & 3;
              uint8_t *rowp = b16 + row * 64;
              *reinterpret_cast<uint4 *>(rowp + (((2 * h) ^ sw) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
              *reinterpret_cast<uint4 *>(rowp + (((2 * h + 1) ^ sw) << 4)) =
                  make_uint4(o[4], o[5], o[6], o[7]);
              if (CC) {
                int c2 = 0;
#pragma unroll
                for (int j = 0; j < 4; ++j) c2 = __dp4a((int)w[j], (int)w[j], c2);
                ccp[i] += (float)c2;
              }
            }
          } else {
            // Each 16-bit half biased to c + 0x8080 (no carry between the
            // halves while c is small): its high byte is 0x80 exactly when c
            // lies in [-128, 127], and its low byte is then c + 128.  One vote
            // per chunk picks the path for all of the warp's tasks, so that
            // the tasks stay independent and interleave.
            uint32_t xb[kTasks][4], tor = 0;
#pragma unroll
            for (int i = 0; i < kTasks; ++i) {
              const uint32_t w[4] = {rv[i].x, rv[i].y, rv[i].z, rv[i].w};
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                xb[i][j] = (w[j] ^ 0x80008000u) + 0x00800080u;
                tor |= xb[i][j] ^ 0x80008000u;
              }
            }
            if (__all_sync(0xffffffffu, (tor & 0xff00ff00u) == 0u)) {
              // the int8 conversion on the low bytes
#pragma unroll
              for (int i = 0; i < kTasks; ++i) {
                const int row = conv_row<W>(ct, i), qt = conv_sub<W>(ct);
                uint32_t o[4];
#pragma unroll
                for (int j = 0; j < 4; ++j)
                  o[j] = h2_as_u32(__hsub2(u32_as_h2(__byte_perm(xb[i][j], 0x64646464u, 0x4240)), bias));
                *reinterpret_cast<uint4 *>(b16 + row * 64 + ((qt ^ ((row >> 1) & 3)) << 4)) =
                    make_uint4(o[0], o[1], o[2], o[3]);
                if (CC) {
                  const int p0 = (int)__byte_perm(rv[i].x, rv[i].y, 0x6420);
                  const int p1 = (int)__byte_perm(rv[i].z, rv[i].w, 0x6420);
                  ccp[i] += (float)__dp4a(p1, p1, __dp4a(p0, p0, 0));
                }
              }
            } else {
#pragma unroll
              for (int i = 0; i < kTasks; ++i) {
                const int row = conv_row<W>(ct, i), qt = conv_sub<W>(ct);
                const uint32_t w[4] = {rv[i].x, rv[i].y, rv[i].z, rv[i].w};
                uint32_t o[4];
                float c2 = 0.0f;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                  const uint32_t x = w[j] ^ 0x80008000u;
                  const float f0 = __int_as_float(__byte_perm(x, 0x4B000000u, 0x7410)) - 8421376.0f;
                  const float f1 = __int_as_float(__byte_perm(x, 0x4B000000u, 0x7432)) - 8421376.0f;
                  amax = fmaxf(amax, fmaxf(fabsf(f0), fabsf(f1)));
                  if (CC) c2 = fmaf(f0, f0, fmaf(f1, f1, c2));
                  o[j] = h2_as_u32(__floats2half2_rn(f0, f1));
                }
                *reinterpret_cast<uint4 *>(b16 + row * 64 + ((qt ^ ((row >> 1) & 3)) << 4)) =
                    make_uint4(o[0], o[1], o[2], o[3]);
                if (CC) ccp[i] += c2;
              }
            }
          }
          if (kc % C == C - 1 || kc == nk - 1) {  // the stage's chunks are all converted
            fence_proxy_async_smem();
            mbar_arrive(&conv[s]);
            ++it;
          }
          if (kc % R == R - 1 || kc == nk - 1) {
            mbar_arrive(&rempty[rs]);
            ++gr;
          }
        }
        if (!ok) break;
        if (CC) {
          float tr[kTasks];  // the rows' sums of c^2
#pragma unroll
          for (int i = 0; i < kTasks; ++i) {
            float t = ccp[i] + __shfl_xor_sync(0xffffffffu, ccp[i], 1);
            if (W == 2) t += __shfl_xor_sync(0xffffffffu, t, 2);
            tr[i] = t;
            ccmax = fmaxf(ccmax, t);
          }
          if (need_cc) {
            if (u > 0 && !mbar_wait(&cce[buf], (u - 1) & 1, abort_flag, a.gflags)) break;
#pragma unroll
            for (int i = 0; i < kTasks; ++i) {
              const float t = tr[i];
              const bool writer = conv_sub<W>(ct) == 0;
              // per-row factor of the score: 1/||c|| for cosine, s^2 ||c||^2 for L2
              const float rowf = a.metric == LAM_METRIC_COSINE
                                     ? (t > 0.0f ? 1.0f / sqrtf(t) : 0.0f)
                                     : a.s * a.s * t;
              if (writer) ccbuf[buf * kBN + conv_row<W>(ct, i)] = rowf;
            }
            mbar_arrive(&ccf[buf]);
          }
        }
      }
      if (W == 2 && amax > 2048.0f) atomicOr(a.gflags, kFlagRange);
      // hi-only pass: the largest row norm bounds what the dropped lo term
      // could add to any row's score (the certification in the merge)
      if (CC && g.hi) {
        const float m = warp_max_tc(ccmax);
        if (lane == 0) note_max_cc(a.gflags, m);
      }
    };
    if (need_cc || g.hi)
      converters(BoolTag<true>{});
    else
      converters(BoolTag<false>{});
  } else if (warp == 10) {
    // ------------------------------------------------ query producer -----
    if (lane == 0) {
      // the query blocks of the MMA stages, freed by the MMAs
      const int spt = (nk + C - 1) / C;  // MMA stages per tile
      const int a_total = producers_stalled(a.gflags) ? 0 : ntl * spt;
      int it = 0;
      for (; it < a_total; ++it) {
        const int s = it % ns, r = it / ns;
        if (r > 0 && !mbar_wait(&empty[s], (r - 1) & 1, abort_flag, a.gflags)) break;
        const int kc = (it % spt) * C;
        const int nc = nk - kc < C ? nk - kc : C;
        uint8_t *dst = smem + (size_t)s * stage_stride;
        const uint8_t *src = qA + ((size_t)qb * nk + kc) * kAStage;
        const int nh = g.hi ? 1 : 2;  // the hi image, and the lo image unless hi-only
        if (g.qoff == 0) {
          mbar_arrive_expect_tx(&afull[s], (uint32_t)(nc * nh) * kABytes);
          if (nh == 2) {
            bulk_g2s(dst, src, (uint32_t)nc * kAStage, &afull[s]);
          } else {
            for (int c = 0; c < nc; ++c)
              bulk_g2s(dst + (size_t)c * kAStage, src + (size_t)c * kAStage, kABytes, &afull[s]);
          }
        } else {
          // queries in MMA rows 64 .. 127 only: the hi and lo rows 0 .. 63
          // (64-byte rows, the first 4 KB of each 8 KB tile) feed TMEM lanes
          // that no epilogue warp reads, so they are not copied
          mbar_arrive_expect_tx(&afull[s], (uint32_t)(nc * nh) * (kABytes / 2));
          for (int c = 0; c < nc; ++c)
            for (int h = 0; h < nh; ++h) {
              const size_t off = (size_t)c * kAStage + (size_t)h * kABytes + kABytes / 2;
              bulk_g2s(dst + off, src + off, kABytes / 2, &afull[s]);
            }
        }
      }
      for (int t = max(0, it - ns); t < it; ++t) drain_wait_tc(&afull[t % ns], (t / ns) & 1);
    }
  } else if (quad_used(warp & 3)) {
    // ------------------------------------------------ epilogue -----------
    // (warp w may read TMEM lanes 32 (w % 4) .. 32 (w % 4) + 31)
    const int quad = warp & 3;
    const int m = quad * 32 + lane;  // TMEM lane = MMA row of the query block
    const int64_t qidx = (int64_t)qb * kBM + m - g.qoff;
    const bool qvalid = m >= g.qoff && qidx < a.B;
    const int k = a.k;
    const bool desc = a.metric != LAM_METRIC_L2;
    const float s = a.s;
    float pw = 0.0f, qn = 0.0f, qq = 0.0f;
    if (qvalid) {
      const float4 qi = reinterpret_cast<const float4 *>(
          qA + (size_t)(a.Bpad / kBM) * nk * kAStage)[qidx];
      pw = qi.x;
      qn = qi.y;
      qq = qi.z;
    }
    // per-query factor of the score: s 2^-e (IP), 2^-e / ||q|| (cosine),
    // -2 s 2^-e (L2); see tile_score
    const float fq = a.metric == LAM_METRIC_IP ? s * pw
                     : a.metric == LAM_METRIC_COSINE ? (qn > 0.0f ? pw / qn : 0.0f)
                                                     : -2.0f * s * pw;
    constexpr int RK = KR > 0 ? KR : 1;
    RegTopK<RK> reg;
    reg.init(k);
    float thr_s = desc ? -INFINITY : INFINITY;  // score of the k-th best so far
    float seed = desc ? -INFINITY : INFINITY;   // admission bound before the list fills
    // k > 32: the heaps' candidate buffers (depth from the layout)
    uint64_t *hb = reinterpret_cast<uint64_t *>(cbuf);
    const int hbn = KR == 0 ? (g.cc_off - g.cbuf_off) / (kBM * 8) : 0;
    int hcnt = 0;
    if (KR == 0)
      for (int i = 0; i < k; ++i) lists[(size_t)i * kBM + m] = kSentinel;
    for (int lt = 0; lt < ntl; ++lt) {
      const int buf = lt & 1, u = lt >> 1;
      if (!warp_wait(&accf[buf], u & 1, abort_flag, a.gflags)) break;
      if (need_cc && !warp_wait(&ccf[buf], u & 1, abort_flag, a.gflags)) break;
      tc_fence_after();
      const int64_t row0 = (tb + lt) * kBN;
      const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(buf * kBN);
      if (KR > 0 && lt == 0 && row0 + kBN <= a.N) {
        // First (full) tile: the k-th best of RK group bests bounds the k-th
        // best score from below (as in the batched kernel).
        constexpr int NG = KR > 0 ? KR : 1, GR = kBN / NG, P = 32 / GR;
        float gb[NG];
#pragma unroll 1
        for (int c = 0; c < kBN / 32; ++c) {
          uint32_t v[32];
          tmem_ld32(taddr + c * 32, v);
#pragma unroll
          for (int i = 0; i < NG - P; ++i) gb[i] = gb[i + P];
#pragma unroll
          for (int h = 0; h < P; ++h) {
            float best = -INFINITY;
#pragma unroll
            for (int j = h * GR; j < (h + 1) * GR; ++j) {
              const float rf = need_cc ? ccbuf[buf * kBN + c * 32 + j] : 0.0f;
              const float sc = tile_score(a.metric, __uint_as_float(v[j]), fq, qq, rf);
              best = fmaxf(best, desc ? sc : -sc);
            }
            gb[NG - P + h] = best;
          }
        }
        const float kth = kth_largest(gb, k);
        seed = desc ? nextafterf(kth, -INFINITY) : nextafterf(-kth, INFINITY);
      }
      const float thr = desc ? fmaxf(thr_s, seed) : fminf(thr_s, seed);
#pragma unroll 1
      for (int c = 0; c < kBN / 32; ++c) {
        uint32_t v[32];
        tmem_ld32(taddr + c * 32, v);
        if (KR > 0) {
          // Candidates must beat the k-th score strictly (rows arrive in
          // increasing order, so an equal score ranks later).  A compact pass
          // marks them in a 32-bit mask; the warp then inserts them into the
          // register lists, one per lane per step, each re-tested against the
          // threshold the earlier steps tightened.
          const int64_t nvalid = a.N - (row0 + c * 32);
          const float thr_c = desc ? fmaxf(thr_s, thr) : fminf(thr_s, thr);
          const float *ccc = ccbuf + buf * kBN + c * 32;
          uint32_t mask = chunk_mask(a.metric, v, fq, qq, thr_c, [&](int j) { return ccc[j]; });
          if (!qvalid || nvalid <= 0) mask = 0;
          else if (nvalid < 32) mask &= (1u << nvalid) - 1u;
          while (__any_sync(0xffffffffu, mask != 0)) {
            uint32_t kc = 0xffffffffu, ic = 0xffffffffu;
            if (mask != 0) {
              const int j = __ffs(mask) - 1;
              mask &= mask - 1;
              const float rf = need_cc ? ccc[j] : 0.0f;
              const float sc = tile_score(a.metric, __uint_as_float(select32(v, j)), fq, qq, rf);
              if (desc ? sc > thr_s : sc < thr_s) {
                kc = rank_key32(sc, desc);
                ic = (uint32_t)(row0 + c * 32 + j);
              }
            }
            reg.insert(kc, ic);
            const uint32_t tk = reg.key[RK - 1];
            thr_s = tk == 0xffffffffu ? (desc ? -INFINITY : INFINITY) : rank_key32_score(tk, desc);
          }
        } else if (KR == 0) {
          // k > 32: a max-heap per query in shared memory (root = the worst
          // key kept); a candidate replaces the root and sifts down.
          const int64_t nvalid = a.N - (row0 + c * 32);
          const float *ccc = ccbuf + buf * kBN + c * 32;
          uint32_t mask = chunk_mask(a.metric, v, fq, qq, thr_s, [&](int j) { return ccc[j]; });
          if (!qvalid || nvalid <= 0) mask = 0;
          else if (nvalid < 32) mask &= (1u << nvalid) - 1u;
          if (hbn > 0) {
            while (__any_sync(0xffffffffu, mask != 0)) {
              if (mask != 0) {
                const int j = __ffs(mask) - 1;
                mask &= mask - 1;
                const float rf = need_cc ? ccbuf[buf * kBN + c * 32 + j] : 0.0f;
                const float sc =
                    tile_score(a.metric, __uint_as_float(select32(v, j)), fq, qq, rf);
                const uint64_t key = make_key(sc, (uint32_t)(row0 + c * 32 + j), desc);
                if (key < lists[m]) hb[(size_t)(hcnt++) * kBM + m] = key;
              }
              if (__any_sync(0xffffffffu, hcnt == hbn)) heap_pour(lists, k, hb, m, hcnt, thr_s, desc);
            }
          } else {
            while (mask != 0) {
              const int j = __ffs(mask) - 1;
              mask &= mask - 1;
              const float rf = need_cc ? ccbuf[buf * kBN + c * 32 + j] : 0.0f;
              const float sc = tile_score(a.metric, __uint_as_float(select32(v, j)), fq, qq, rf);
              const uint64_t key = make_key(sc, (uint32_t)(row0 + c * 32 + j), desc);
              if (key < lists[m]) {
                heap_replace_root(lists, k, kBM, m, key);
                const uint64_t root = lists[m];
                thr_s = root == kSentinel ? (desc ? -INFINITY : INFINITY)
                                          : rank_key32_score((uint32_t)(root >> 32), desc);
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
      if (KR > 0) {
#pragma unroll
        for (int i = 0; i < RK; ++i)
          if (i >= RK - k) out[i - (RK - k)] = ((uint64_t)reg.key[i] << 32) | reg.id[i];
      } else {
        if (hcnt > 0) heap_pour(lists, k, hb, m, hcnt, thr_s, desc);
        heap_sort_ascending(lists, k, kBM, m);
        for (int i = 0; i < k; ++i) out[i] = lists[(size_t)i * kBM + m];
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// Query preparation, one warp per query: the power-of-two scale 2^e, the fp16
// split hi + lo of q 2^e written straight into the operand image the MMA
// stages load (per query block and 32-wide K slice: [hi 128 x 64 B | lo], rows
// 64 bytes apart with the 16-byte chunks of row r XOR-ed by (r >> 1) & 3, the
// 64-byte swizzle), zeros for padding rows and columns; then (2^-e, ||q||,
// ||q||^2, sum_d q_d) per query after the images.  With dup = 2 (int16 codes
// split as 256 h + l, two K chunks per 32 coordinates) every K slice of the
// query is written twice, as image chunks 2 j and 2 j + 1.
__device__ __forceinline__ void qprep_block(const float *__restrict__ q, int64_t B, int D,
                                            int64_t Bpad, uint8_t *__restrict__ qA, int64_t blk,
                                            int qoff = 0, int dup = 1) {
  const int64_t b = blk * 8 + (threadIdx.x >> 5);  // MMA row over all query blocks
  const int lane = threadIdx.x & 31;
  if (b >= Bpad) return;
  const int nk = (D + kBK - 1) / kBK * dup;
  const int64_t qb = b / kBM;
  const int r = (int)(b % kBM);
  float4 *qinfo = reinterpret_cast<float4 *>(qA + (size_t)(Bpad / kBM) * nk * kAStage);
  const int64_t qi = b - qoff;  // the query of this row (qoff > 0 only with one block)
  const bool valid = qi >= 0 && qi < B;
  const float *qr = valid ? q + qi * D : q;
  float mx = 0.0f, qs = 0.0f;
  if (valid) {
    for (int d = lane; d < D; d += 32) {
      const float v = qr[d];
      mx = fmaxf(mx, fabsf(v));
      qs += v;
    }
  }
  for (int off = 16; off > 0; off >>= 1) {
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
    qs += __shfl_xor_sync(0xffffffffu, qs, off);
  }
  int e = 0, ex = 0;
  if (mx > 0.0f) {
    frexpf(mx, &ex);  // mx = f * 2^ex, f in [0.5, 1)
    e = 15 - ex;      // mx * 2^e in [2^14, 2^15)
    e = max(-126, min(126, e));
  }
  const float sc = ldexpf(1.0f, e);
  // ||q|| from the query scaled near 1 (no under- or overflow of the squares)
  const float ns = mx > 0.0f ? ldexpf(1.0f, max(-126, min(126, -ex))) : 1.0f;
  float ss = 0.0f;
  if (valid)
    for (int d = lane; d < D; d += 32) ss = fmaf(qr[d] * ns, qr[d] * ns, ss);
  for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
  const float qn = sqrtf(ss) / ns, qq = qn * qn;
  // lane writes whole 16-byte chunks (8 fp16) of the hi and lo images
  for (int ch = lane; ch < nk * (kBK / 8); ch += 32) {
    const int kc = ch / (kBK / 8), c16 = ch % (kBK / 8);
    const int d0 = (kc / dup) * kBK + c16 * 8;  // the query coordinates of this piece
    uint32_t hw[4], lw[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int d = d0 + 2 * t;
      const float v0 = (valid && d < D) ? qr[d] * sc : 0.0f;
      const float v1 = (valid && d + 1 < D) ? qr[d + 1] * sc : 0.0f;
      const __half2 h = __floats2half2_rn(v0, v1);
      const float2 hf = __half22float2(h);
      const __half2 l = __floats2half2_rn(v0 - hf.x, v1 - hf.y);
      hw[t] = h2_as_u32(h);
      lw[t] = h2_as_u32(l);
    }
    const size_t off = ((size_t)qb * nk + kc) * kAStage + (size_t)r * 64 +
                       (size_t)((c16 ^ ((r >> 1) & 3)) << 4);
    *reinterpret_cast<uint4 *>(qA + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
    *reinterpret_cast<uint4 *>(qA + off + kABytes) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
  }
  if (lane == 0 && qi >= 0)
    qinfo[qi] = valid ? make_float4(ldexpf(1.0f, -e), qn, qq, qs)
                      : make_float4(0.f, 0.f, 0.f, 0.f);
}

__global__ void __launch_bounds__(256) qprep_kernel(const float *__restrict__ q, int64_t B, int D,
                                                    int64_t Bpad, uint8_t *__restrict__ qA,
                                                    int qoff) {
  qprep_block(q, B, D, Bpad, qA, blockIdx.x, qoff);
}


// ===========================================================================
// Batched path for two or more query blocks.  A separate pass converts the
// codes once per call into fp16 rows (and the per-row score factor), so the
// scoring kernel is a plain TMA -> tcgen05 pipeline: no conversion sits in
// its stage loop.  Rows are processed in slabs to bound the fp16 copy.
// ===========================================================================
constexpr int kTc2Threads = 192;  // warp 0 producer, warp 1 MMA, warps 2-5 epilogue
// 32-wide K chunks per pipeline stage: one bulk copy brings the query and one
// the code blocks of all of them (they lie back to back), so a stage is two
// 32 KB copies and one barrier round trip for 8 MMAs.  Measured against one
// chunk per stage: 66 instead of 72 us at 27,986 rows x 1,024 queries.
constexpr int kTc2Chunks = 2;

// codes [row_base, row_base + nrows) -> the fp16 operand image of the scoring
// kernel: for each tile of 256 rows and each 32-wide K chunk, one contiguous
// 16 KB block of 64-byte rows in the 64-byte swizzle (16-byte piece j of row r
// at piece j ^ ((r >> 1) & 3)), so that one bulk copy stages it.  Rows past
// nrows and columns past D are zero.  Also the per-row factor rowf (1/||c|| for
// cosine, s^2 ||c||^2 for L2).  One warp per row of the padded slab.
//
// Wide (int16 codes beyond +-2048, or no known bound): each code is split as
// c = 256 h + l with h = c >> 8 in [-128, 127] and l = c & 255 in [0, 255];
// 256 h and l are both exact in fp16.  K chunk j of the codes becomes image
// chunks 2 j (the 256 h values) and 2 j + 1 (the l values), and the query
// image repeats each K slice (qprep_block with dup = 2), so the scoring
// kernel runs unchanged over 2 D columns: q . c = q . (256 h) + q . l, every
// product exact in fp32 (11 x 8 significant bits at most).
template <int W>
__device__ __forceinline__ void convert_block(const void *__restrict__ codes, int64_t row_base,
                                              int64_t nrows, int64_t nrows_pad, int D,
                                              uint8_t *__restrict__ out,
                                              float *__restrict__ rowf, int metric, float s,
                                              uint32_t *gflags, int64_t blk, bool wide = false,
                                              bool track = false) {
  const int64_t r = blk * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= nrows_pad) return;
  const bool valid = r < nrows;
  const int nk = (D + kBK - 1) / kBK;
  const int rr = (int)(r % kBN);
  const int sw = (rr >> 1) & 3;
  uint8_t *dst = out + (size_t)(r / kBN) * nk * (wide ? 2 : 1) * kB16Bytes + (size_t)rr * 64;
  const uint8_t *src = static_cast<const uint8_t *>(codes) + (row_base + r) * (int64_t)D * W;
  float cc = 0.0f, amax = 0.0f;
  for (int ch = lane; ch < nk * (kBK / 8); ch += 32) {
    const int d0 = ch * 8;
    float f[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) f[t] = 0.0f;
    if (valid && d0 < D) {  // D is a multiple of 16: a chunk is all in or all out
      if (W == 1) {
        const uint2 v = *reinterpret_cast<const uint2 *>(src + d0);
#pragma unroll
        for (int t = 0; t < 8; ++t) f[t] = (float)(int8_t)((t < 4 ? v.x : v.y) >> (8 * (t & 3)));
      } else {
        const uint4 v = *reinterpret_cast<const uint4 *>(src + d0 * 2);
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int t = 0; t < 8; ++t) f[t] = (float)(int16_t)(w[t >> 1] >> (16 * (t & 1)));
      }
    }
    uint32_t o[4];
    const size_t piece = (size_t)(((ch & 3) ^ sw) << 4);
    if (W == 2 && wide) {
      uint32_t ol[4];
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        cc = fmaf(f[2 * t], f[2 * t], fmaf(f[2 * t + 1], f[2 * t + 1], cc));
        const int c0 = (int)f[2 * t], c1 = (int)f[2 * t + 1];
        o[t] = h2_as_u32(__floats2half2_rn((float)((c0 >> 8) * 256), (float)((c1 >> 8) * 256)));
        ol[t] = h2_as_u32(__floats2half2_rn((float)(c0 & 255), (float)(c1 & 255)));
      }
      uint8_t *d2 = dst + (size_t)(ch >> 2) * 2 * kB16Bytes + piece;
      *reinterpret_cast<uint4 *>(d2) = make_uint4(o[0], o[1], o[2], o[3]);
      *reinterpret_cast<uint4 *>(d2 + kB16Bytes) = make_uint4(ol[0], ol[1], ol[2], ol[3]);
      continue;
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      amax = fmaxf(amax, fmaxf(fabsf(f[2 * t]), fabsf(f[2 * t + 1])));
      cc = fmaf(f[2 * t], f[2 * t], fmaf(f[2 * t + 1], f[2 * t + 1], cc));
      o[t] = h2_as_u32(__floats2half2_rn(f[2 * t], f[2 * t + 1]));
    }
    *reinterpret_cast<uint4 *>(dst + (size_t)(ch >> 2) * kB16Bytes + piece) =
        make_uint4(o[0], o[1], o[2], o[3]);
  }
  cc = warp_sum_tc(cc);
  if (lane == 0 && valid && metric != LAM_METRIC_IP)
    rowf[r] = metric == LAM_METRIC_COSINE ? (cc > 0.0f ? 1.0f / sqrtf(cc) : 0.0f) : s * s * cc;
  // (a hi-only pass follows: the largest row norm, for the certification)
  if (track && lane == 0 && valid) note_max_cc(gflags, cc);
  if (W == 2 && !wide && amax > 2048.0f) atomicOr(gflags, kFlagRange);
}

// (qst: status-driven calls launch both widths; only the codes' width converts)
__device__ __forceinline__ bool width_gate(const QuantStatus *qst, int W) {
  return qst == nullptr || (status_ok(qst) && status_width(qst) == (uint32_t)W);
}

template <int W>
__global__ void __launch_bounds__(256) convert_codes_kernel(const void *__restrict__ codes,
                                                            int64_t row_base, int64_t nrows,
                                                            int64_t nrows_pad, int D,
                                                            uint8_t *__restrict__ out,
                                                            float *__restrict__ rowf, int metric,
                                                            float s, uint32_t *gflags,
                                                            const QuantStatus *qst,
                                                            int wide = 0, int track = 0) {
  if (!width_gate(qst, W)) return;
  convert_block<W>(codes, row_base, nrows, nrows_pad, D, out, rowf, metric, s, gflags, blockIdx.x,
                   wide != 0, track != 0);
}

// Query preparation and the first slab's conversion in one launch: blocks
// [0, q_blocks) prepare queries, the rest convert code rows (independent work).
template <int W>
__global__ void __launch_bounds__(256) prep_convert_kernel(
    const float *__restrict__ q, int64_t B, int D, int64_t Bpad, uint8_t *__restrict__ qA,
    unsigned q_blocks, const void *__restrict__ codes, int64_t nrows, int64_t nrows_pad,
    uint8_t *__restrict__ out, float *__restrict__ rowf, int metric, float s, uint32_t *gflags,
    const QuantStatus *qst, int wide = 0, int track = 0) {
  if (blockIdx.x < q_blocks)
    qprep_block(q, B, D, Bpad, qA, blockIdx.x, 0, wide ? 2 : 1);
  else if (width_gate(qst, W))
    convert_block<W>(codes, 0, nrows, nrows_pad, D, out, rowf, metric, s, gflags,
                     blockIdx.x - q_blocks, wide != 0, track != 0);
}

// Status-driven calls: one launch converts at the width the quantize status
// holds (a launch per width would schedule a whole grid of idle blocks).
__global__ void __launch_bounds__(256) convert_codes_from_kernel(
    const void *__restrict__ codes, int64_t row_base, int64_t nrows, int64_t nrows_pad, int D,
    uint8_t *__restrict__ out, float *__restrict__ rowf, int metric, float s, uint32_t *gflags,
    const QuantStatus *qst) {
  if (width_gate(qst, 1))
    convert_block<1>(codes, row_base, nrows, nrows_pad, D, out, rowf, metric, s, gflags, blockIdx.x);
  else if (width_gate(qst, 2))
    convert_block<2>(codes, row_base, nrows, nrows_pad, D, out, rowf, metric, s, gflags, blockIdx.x);
}

__global__ void __launch_bounds__(256) prep_convert_from_kernel(
    const float *__restrict__ q, int64_t B, int D, int64_t Bpad, uint8_t *__restrict__ qA,
    unsigned q_blocks, const void *__restrict__ codes, int64_t nrows, int64_t nrows_pad,
    uint8_t *__restrict__ out, float *__restrict__ rowf, int metric, float s, uint32_t *gflags,
    const QuantStatus *qst) {
  if (blockIdx.x < q_blocks)
    qprep_block(q, B, D, Bpad, qA, blockIdx.x);
  else if (width_gate(qst, 1))
    convert_block<1>(codes, 0, nrows, nrows_pad, D, out, rowf, metric, s, gflags,
                     blockIdx.x - q_blocks);
  else if (width_gate(qst, 2))
    convert_block<2>(codes, 0, nrows, nrows_pad, D, out, rowf, metric, s, gflags,
                     blockIdx.x - q_blocks);
}

// Per-row codecs: the stored codes become the fp16 operand image as they are
// (int8 codes c, fp16 values, sign bits as +-1), and the decoding moves into
// per-row factors (u, w, z) of the score
//   q . xhat = pw (q 2^e) . c * a + (sum q) * o      (a, o: scale, offset)
//   inner product / squared L2   u = a, w = o, z = ||xhat||^2
//   cosine                       u = a / ||xhat||, w = o / ||xhat||
// with ||xhat||^2 summed over xhat_d exactly as the decoder forms it.
template <int FMT>
__device__ __forceinline__ void convert_rows_block(const void *__restrict__ codes,
                                                   const float *__restrict__ rscale,
                                                   const float *__restrict__ roff,
                                                   int64_t row_base, int64_t nrows,
                                                   int64_t nrows_pad, int D,
                                                   uint8_t *__restrict__ out,
                                                   float4 *__restrict__ rowf4, int metric,
                                                   int64_t blk) {
  const int64_t r = blk * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= nrows_pad) return;
  const bool valid = r < nrows;
  const int nk = (D + kBK - 1) / kBK;
  const int rr = (int)(r % kBN);
  const int sw = (rr >> 1) & 3;
  uint8_t *dst = out + (size_t)(r / kBN) * nk * kB16Bytes + (size_t)rr * 64;
  const int64_t grow = row_base + r;
  float sa = 1.0f, so = 0.0f;
  if (valid && FMT != LAM_ROWS_FP16) sa = rscale[grow];
  if (valid && FMT == LAM_ROWS_INT8) so = roff[grow];
  float xx = 0.0f;
  for (int ch = lane; ch < nk * (kBK / 8); ch += 32) {
    const int d0 = ch * 8;
    uint32_t o[4] = {0u, 0u, 0u, 0u};
    if (valid && d0 < D) {  // D is a multiple of 16: a chunk is all in or all out
      if (FMT == LAM_ROWS_INT8) {
        const uint2 v = *reinterpret_cast<const uint2 *>(static_cast<const int8_t *>(codes) +
                                                         grow * D + d0);
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const uint32_t wv = t < 2 ? v.x : v.y;
          const float c0 = (float)(int8_t)(wv >> (16 * (t & 1)));
          const float c1 = (float)(int8_t)(wv >> (16 * (t & 1) + 8));
          const float x0 = __fadd_rn(so, __fmul_rn(sa, c0));
          const float x1 = __fadd_rn(so, __fmul_rn(sa, c1));
          xx = fmaf(x0, x0, fmaf(x1, x1, xx));
          o[t] = h2_as_u32(__floats2half2_rn(c0, c1));
        }
      } else if (FMT == LAM_ROWS_FP16) {
        const uint4 v = *reinterpret_cast<const uint4 *>(static_cast<const __half *>(codes) +
                                                         grow * D + d0);
        o[0] = v.x;
        o[1] = v.y;
        o[2] = v.z;
        o[3] = v.w;
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          __half2 h;
          memcpy(&h, &o[t], 4);
          const float2 f = __half22float2(h);
          xx = fmaf(f.x, f.x, fmaf(f.y, f.y, xx));
        }
      } else {
        const uint32_t byte = static_cast<const uint8_t *>(codes)[grow * (D / 8) + ch];
#pragma unroll
        for (int t = 0; t < 4; ++t) {  // +1 = 0x3C00, -1 = 0xBC00 in binary16
          const uint32_t lo = ((byte >> (2 * t)) & 1u) ? 0x3C00u : 0xBC00u;
          const uint32_t hi = ((byte >> (2 * t + 1)) & 1u) ? 0x3C00u : 0xBC00u;
          o[t] = lo | (hi << 16);
          xx = fmaf(sa, sa, fmaf(sa, sa, xx));
        }
      }
    }
    *reinterpret_cast<uint4 *>(dst + (size_t)(ch >> 2) * kB16Bytes + (((ch & 3) ^ sw) << 4)) =
        make_uint4(o[0], o[1], o[2], o[3]);
  }
  xx = warp_sum_tc(xx);
  if (lane == 0 && valid) {
    float u = sa, w = so;
    if (metric == LAM_METRIC_COSINE) {
      const float inv = xx > 0.0f ? 1.0f / sqrtf(xx) : 0.0f;
      u = sa * inv;
      w = so * inv;
    }
    rowf4[r] = make_float4(u, w, xx, 0.0f);
  }
}

template <int FMT>
__global__ void __launch_bounds__(256) convert_rows_kernel(
    const void *__restrict__ codes, const float *__restrict__ rscale,
    const float *__restrict__ roff, int64_t row_base, int64_t nrows, int64_t nrows_pad, int D,
    uint8_t *__restrict__ out, float4 *__restrict__ rowf4, int metric) {
  convert_rows_block<FMT>(codes, rscale, roff, row_base, nrows, nrows_pad, D, out, rowf4, metric,
                          blockIdx.x);
}

template <int FMT>
__global__ void __launch_bounds__(256) prep_convert_rows_kernel(
    const float *__restrict__ q, int64_t B, int D, int64_t Bpad, uint8_t *__restrict__ qA,
    unsigned q_blocks, const void *__restrict__ codes, const float *__restrict__ rscale,
    const float *__restrict__ roff, int64_t nrows, int64_t nrows_pad, uint8_t *__restrict__ out,
    float4 *__restrict__ rowf4, int metric) {
  if (blockIdx.x < q_blocks)
    qprep_block(q, B, D, Bpad, qA, blockIdx.x);
  else
    convert_rows_block<FMT>(codes, rscale, roff, 0, nrows, nrows_pad, D, out, rowf4, metric,
                            blockIdx.x - q_blocks);
}

struct Tc2Layout {
  int ns, chunks;
  size_t lists_off, cbuf_off, bar_off, smem_bytes;
};

inline Tc2Layout tc2_layout(int k, bool pair = false) {
  Tc2Layout L;
  // (pair: each CTA of a 2-CTA cluster stages half of each chunk's code rows)
  const size_t stage = (size_t)kAStage + (pair ? kB16Bytes / 2 : kB16Bytes);
  // (k <= 32 keeps its candidates in registers, k > 32 a heap per query in
  // shared memory; stages of kTc2Chunks chunks while two of them fit beside
  // the heaps, else single-chunk stages)
  const size_t lists = k > 32 ? (size_t)kBM * k * 8 : 0;
  const size_t tailb = 64 * 8 + 1024;
  size_t cbuf = 0;  // k > 32: the heaps' candidate buffers (as in the stage-loop kernel)
  if (k > 32) {
    const size_t room = kMaxDynSmem - lists - tailb;
    const size_t need = 2 * stage;
    const size_t slots = room > need ? (room - need) / ((size_t)kBM * 8) : 0;
    cbuf = (slots < (size_t)kCBuf ? slots : (size_t)kCBuf) * kBM * 8;
  }
  const size_t avail = kMaxDynSmem - lists - cbuf - tailb;
  L.chunks = avail / ((size_t)kTc2Chunks * stage) >= 2 ? kTc2Chunks : 1;
  int ns = (int)(avail / ((size_t)L.chunks * stage));
  if (ns > 8) ns = 8;
  L.ns = ns;
  L.lists_off = (size_t)ns * L.chunks * stage;
  L.cbuf_off = L.lists_off + lists;
  L.bar_off = L.cbuf_off + cbuf;
  L.smem_bytes = L.bar_off + tailb;
  return L;
}

struct Tc2Geom {
  int ns, chunks;  // stages, 32-wide K chunks per stage
  int lists_off, cbuf_off, bar_off;
  int64_t row_base, nrows;  // the slab
  int list_base;            // partial-list index of this slab's split 0
  const uint8_t *b16;       // fp16 operand image of the slab
  const float *seed;        // later slabs: per query, the first slab's k-th best score
  const float *rowf;        // per-row factors of the slab (Q_eps codes)
  const float4 *rowf4;      // per-row (u, w, z) of the slab (per-row codecs)
  int hi;    // hi-only pass: the lo term of the query is neither copied nor multiplied
  int gate;  // full pass of a two-pass search: runs only if a query was not certified
};

// Per-row score factors of the per-row codecs for one 32-row chunk, one row
// per lane, and their broadcast for row j (all lanes must call at()).
template <bool RC>
struct RowFac;
template <>
struct RowFac<false> {  // (the Q_eps path keeps its single factor in `rfl`)
  __device__ __forceinline__ void load(const Tc2Geom &, int64_t, bool, bool) {}
  __device__ __forceinline__ RowFac at(int, bool) const { return *this; }
};
template <>
struct RowFac<true> {
  float u, w, z;
  __device__ __forceinline__ void load(const Tc2Geom &g, int64_t i, bool ok, bool) {
    const float4 v = ok ? g.rowf4[i] : make_float4(0.f, 0.f, 0.f, 0.f);
    u = v.x;
    w = v.y;
    z = v.z;
  }
  __device__ __forceinline__ RowFac at(int j, bool l2) const {
    RowFac f;
    f.u = __shfl_sync(0xffffffffu, u, j);
    f.w = __shfl_sync(0xffffffffu, w, j);
    f.z = l2 ? __shfl_sync(0xffffffffu, z, j) : 0.0f;
    return f;
  }
};
// Per-query factors: fq multiplies the accumulator, fs the row offset term.
struct QFac {
  float fq, fs, qq;
  int metric;
};
__device__ __forceinline__ float fac_score(const RowFac<false> &, float, const QFac &) {
  return 0.0f;
}
__device__ __forceinline__ float fac_score(const RowFac<true> &f, float acc, const QFac &q) {
  const float dot = fmaf(q.fq * f.u, acc, q.fs * f.w);
  return q.metric == LAM_METRIC_L2 ? fmaf(-2.0f, dot, q.qq + f.z) : dot;
}

// PAIR: the CTAs of a 2-CTA cluster take query blocks 2j and 2j + 1 over the
// same code tiles.  Each stages its 128 queries and half of each chunk's 256
// code rows (the even CTA rows 0-127, the odd one rows 128-255); the even
// CTA's issuer waits for both halves (the odd CTA's MMA warp relays "stage s
// landed" by a remote arrive) and issues M = 256 MMAs, so each accumulator
// holds its CTA's 128 queries x all 256 rows while each SM takes in 24 KB per
// chunk instead of 32 KB.  Its commits free the stage and fill the
// accumulator in both CTAs; the accumulator is free again when the epilogue
// threads of both CTAs arrived.  Two-pass (hi / gated) launches are not pairs.
template <int KR, bool RC, bool PAIR = false>
__global__ void __launch_bounds__(kTc2Threads, 1)
    score_tc2_kernel(ScoreArgs a, Tc2Geom g) {
  if (!PAIR && g.gate && hi_all_certified(a.gflags)) return;
  extern __shared__ uint8_t tc_smem_raw[];
  const uint32_t base_u32 = smem_u32(tc_smem_raw);
  uint8_t *smem = tc_smem_raw + (((base_u32 + 1023u) & ~1023u) - base_u32);
  const int ns = g.ns, C = g.chunks;
  uint64_t *lists = reinterpret_cast<uint64_t *>(smem + g.lists_off);
  uint64_t *full = reinterpret_cast<uint64_t *>(smem + g.bar_off);
  uint64_t *empty = full + ns;
  uint64_t *accf = empty + ns;
  uint64_t *acce = accf + 2;
  uint64_t *done = acce + 2;
  uint64_t *pfull = done + 1;  // PAIR, even CTA: the odd CTA's stage s landed
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(pfull + ns);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
  constexpr int kBSlot = PAIR ? kB16Bytes / 2 : kB16Bytes;  // code bytes per chunk staged here
  const size_t stage_bytes = (size_t)kAStage + kBSlot;
  const uint32_t rank = PAIR ? cluster_rank() : 0u;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // grid: (splits of the code tiles, query blocks); pairs take (query blocks,
  // splits), the pair along the cluster's x dimension as the MMA pair needs
  const int qb = PAIR ? blockIdx.x : blockIdx.y;
  const int split = PAIR ? blockIdx.y : blockIdx.x, nsplit = PAIR ? gridDim.y : gridDim.x;
  const int64_t n_tiles = (g.nrows + kBN - 1) / kBN;
  const int64_t tb = (int64_t)split * n_tiles / nsplit;
  const int64_t te = (int64_t)(split + 1) * n_tiles / nsplit;
  const int ntl = (int)(te - tb);
  const int nk = (a.D + kBK - 1) / kBK;
  const bool need_cc = RC || a.metric != LAM_METRIC_IP;
  const uint8_t *qA = static_cast<const uint8_t *>(a.qprep);

  if (threadIdx.x == 0) {
    for (int s = 0; s < ns; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], PAIR ? 256 : 128);
    }
    mbar_init(done, 1);
    if (PAIR)
      for (int s = 0; s < ns; ++s) mbar_init(&pfull[s], 1);
    *abort_flag = 0;
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if constexpr (PAIR) {
    if (warp == 1) tmem_alloc_pair(tmem_slot, kTmemCols);
    tc_fence_before();
    cluster_sync_all();  // (both CTAs' barriers initialised before any remote arrive)
  } else {
    if (warp == 1) tmem_alloc(tmem_slot, kTmemCols);
    tc_fence_before();
    __syncthreads();
  }
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------ producer -----------
    if (lane == 0) {
      int it = 0, issued = 0;
      bool ok = !producers_stalled(a.gflags);
      for (int lt = 0; lt < ntl && ok; ++lt) {
        const int tile = (int)(tb + lt);
        for (int kc = 0; kc < nk; kc += C, ++it) {
          const int s = it % ns, r = it / ns;
          const int nc = nk - kc < C ? nk - kc : C;
          if (r > 0 && !mbar_wait(&empty[s], (r - 1) & 1, abort_flag, a.gflags)) {
            ok = false;
            break;
          }
          // stage: [query blocks of the nc chunks][code blocks of the nc chunks]
          uint8_t *st = smem + (size_t)s * C * stage_bytes;
          const uint8_t *qsrc = qA + ((size_t)qb * nk + kc) * kAStage;
          mbar_arrive_expect_tx(&full[s], (uint32_t)nc * ((g.hi ? kABytes : kAStage) + kBSlot));
          if (!g.hi) {
            bulk_g2s(st, qsrc, (uint32_t)nc * kAStage, &full[s]);
          } else {  // the hi images only
            for (int c = 0; c < nc; ++c)
              bulk_g2s(st + (size_t)c * kAStage, qsrc + (size_t)c * kAStage, kABytes, &full[s]);
          }
          if constexpr (PAIR) {  // this CTA's 128 of each chunk's 256 code rows
            for (int c = 0; c < nc; ++c)
              bulk_g2s(st + C * kAStage + c * kBSlot,
                       g.b16 + ((size_t)tile * nk + kc + c) * kB16Bytes + rank * kBSlot, kBSlot,
                       &full[s]);
          } else {
            bulk_g2s(st + C * kAStage, g.b16 + ((size_t)tile * nk + kc) * kB16Bytes,
                     (uint32_t)nc * kB16Bytes, &full[s]);
          }
          issued = it + 1;
        }
      }
      for (int t = max(0, issued - ns); t < issued; ++t) drain_wait_tc(&full[t % ns], (t / ns) & 1);
    }
  } else if (warp == 1) {
    if (PAIR && rank == 1) {
      // ---------------------------------- odd CTA of a pair: stage relay ---
      if (lane == 0) {
        int it = 0;
        bool ok = true;
        for (int lt = 0; lt < ntl && ok; ++lt)
          for (int kc = 0; kc < nk; kc += C, ++it) {
            const int s = it % ns, r = it / ns;
            if (!mbar_wait(&full[s], r & 1, abort_flag, a.gflags)) {
              ok = false;
              break;
            }
            mbar_arrive_peer(&pfull[s], 0);
          }
      }
    } else if (lane == 0) {
      // ------------------------------------------------ MMA issuer ---------
      int it = 0;
      bool ok = true;
      for (int lt = 0; lt < ntl && ok; ++lt) {
        const int buf = lt & 1, u = lt >> 1;
        if (u > 0 && !(PAIR ? mbar_wait_cl(&acce[buf], (u - 1) & 1, abort_flag, a.gflags)
                            : mbar_wait(&acce[buf], (u - 1) & 1, abort_flag, a.gflags)))
          break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(buf * kBN);
        for (int kc = 0; kc < nk; kc += C, ++it) {
          const int s = it % ns, r = it / ns;
          const int nc = nk - kc < C ? nk - kc : C;
          if (!mbar_wait(&full[s], r & 1, abort_flag, a.gflags) ||
              (PAIR && !mbar_wait_cl(&pfull[s], r & 1, abort_flag, a.gflags))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t st = smem_u32(smem + (size_t)s * C * stage_bytes);
          // the stage's MMAs from one asm block (see umma_chunks)
          uint64_t ahi[2], alo[2], bd[2];
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            ahi[c] = desc_sw64(st + c * kAStage);
            alo[c] = desc_sw64(st + c * kAStage + kABytes);
            bd[c] = desc_sw64(st + C * kAStage + c * kBSlot);
          }
          if constexpr (PAIR) {
            umma_chunks<2>(d_tmem, nc, ahi, alo, bd, g.hi != 0, kIdescPair, kc > 0 ? 1u : 0u);
            umma_commit_pair(&empty[s], 3);
          } else {
            umma_chunks(d_tmem, nc, ahi, alo, bd, g.hi != 0, kIdesc, kc > 0 ? 1u : 0u);
            umma_commit(&empty[s]);
          }
        }
        if (ok) {
          if constexpr (PAIR) umma_commit_pair(&accf[buf], 3);
          else umma_commit(&accf[buf]);
        }
      }
      if constexpr (PAIR) umma_commit_pair(done, 1);
      else umma_commit(done);
      drain_wait_tc(done, 0);
    }
  } else {
    // ------------------------------------------------ epilogue -----------
    // (warps 2-5: warp w may read TMEM lanes 32 (w % 4) .. 32 (w % 4) + 31)
    const int quad = warp & 3;
    const int m = quad * 32 + lane;
    const int64_t qidx = (int64_t)qb * kBM + m;
    const bool qvalid = qidx < a.B;
    const int k = a.k;
    const bool desc = a.metric != LAM_METRIC_L2;
    const float s = a.s;
    float pw = 0.0f, qn = 0.0f, qq = 0.0f, qs = 0.0f;
    if (qvalid) {
      const float4 qi = reinterpret_cast<const float4 *>(
          qA + (size_t)(a.Bpad / kBM) * nk * kAStage)[qidx];
      pw = qi.x;
      qn = qi.y;
      qq = qi.z;
      qs = qi.w;
    }
    const float fq = a.metric == LAM_METRIC_IP ? s * pw
                     : a.metric == LAM_METRIC_COSINE ? (qn > 0.0f ? pw / qn : 0.0f)
                                                     : -2.0f * s * pw;
    QFac qf;  // per-row codecs
    {
      const float inv = a.metric == LAM_METRIC_COSINE ? (qn > 0.0f ? 1.0f / qn : 0.0f) : 1.0f;
      qf.fq = pw * inv;
      qf.fs = qs * inv;
      qf.qq = qq;
      qf.metric = a.metric;
    }
    const bool l2 = a.metric == LAM_METRIC_L2;
    constexpr int RK = KR > 0 ? KR : 1;
    RegTopK<RK> reg;
    reg.init(k);
    float thr_s = desc ? -INFINITY : INFINITY;
    float seed = desc ? -INFINITY : INFINITY;  // admission bound before the list fills
    if (g.seed != nullptr && qvalid) {
      // rows worse than the first slab's k-th best cannot enter the final top-k
      // (equal ones are still offered)
      const float t = g.seed[qidx];
      seed = desc ? nextafterf(t, -INFINITY) : nextafterf(t, INFINITY);
    }
    // k > 32: the heaps' candidate buffers (depth from the layout)
    uint64_t *hb = reinterpret_cast<uint64_t *>(smem + g.cbuf_off);
    const int hbn = KR == 0 ? (g.bar_off - g.cbuf_off) / (kBM * 8) : 0;
    int hcnt = 0;
    if (KR == 0)
      for (int i = 0; i < k; ++i) lists[(size_t)i * kBM + m] = kSentinel;
    for (int lt = 0; lt < ntl; ++lt) {
      const int buf = lt & 1, u = lt >> 1;
      const int64_t row0 = (tb + lt) * kBN;  // slab-local
      if (!warp_wait(&accf[buf], u & 1, abort_flag, a.gflags)) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(buf * kBN);
      if (KR > 0 && lt == 0 && row0 + kBN <= g.nrows) {
        // First (full) tile: the best score of each of RK row groups gives RK
        // >= k distinct rows, so the k-th best of these group bests bounds the
        // k-th best score from below; rows worse than it are never offered
        // (equal ones are).  Saves most of the candidates of the empty list.
        constexpr int GR = kBN / (KR > 0 ? KR : 1);  // rows per group
        constexpr int NG = KR > 0 ? KR : 1, P = 32 / GR;  // groups, groups per chunk
        float gb[NG];
#pragma unroll 1
        for (int c = 0; c < kBN / 32; ++c) {
          uint32_t v[32];
          RowFac<RC> rl;
          rl.load(g, row0 + c * 32 + lane, true, need_cc);
          const float rfl = RC ? 0.0f : need_cc ? g.rowf[row0 + c * 32 + lane] : 0.0f;
          tmem_ld32(taddr + c * 32, v);
          // shift register: the P bests of this chunk enter at the top
#pragma unroll
          for (int i = 0; i < NG - P; ++i) gb[i] = gb[i + P];
#pragma unroll
          for (int h = 0; h < P; ++h) {
            float best = -INFINITY;
#pragma unroll
            for (int j = h * GR; j < (h + 1) * GR; ++j) {
              const float sc =
                  RC ? fac_score(rl.at(j, l2), __uint_as_float(v[j]), qf)
                     : tile_score(a.metric, __uint_as_float(v[j]), fq, qq,
                                  __shfl_sync(0xffffffffu, rfl, j));
              best = fmaxf(best, desc ? sc : -sc);
            }
            gb[NG - P + h] = best;
          }
        }
        const float kth = kth_largest(gb, k);  // in "larger is better" units
        seed = desc ? fmaxf(seed, nextafterf(kth, -INFINITY))
                    : fminf(seed, nextafterf(-kth, INFINITY));
      }
#pragma unroll 1
      for (int c = 0; c < kBN / 32; ++c) {
        uint32_t v[32];
        const int64_t nvalid = g.nrows - (row0 + c * 32);
        // lane j holds the factors of row j of this chunk
        RowFac<RC> rl;
        rl.load(g, row0 + c * 32 + lane, lane < nvalid, need_cc);
        const float rfl =
            RC ? 0.0f : need_cc && lane < nvalid ? g.rowf[row0 + c * 32 + lane] : 0.0f;
        tmem_ld32(taddr + c * 32, v);
        const float thr = desc ? fmaxf(thr_s, seed) : fminf(thr_s, seed);
        uint32_t mask = 0;
        if constexpr (RC) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const float sc = fac_score(rl.at(j, l2), __uint_as_float(v[j]), qf);
            mask |= (uint32_t)(desc ? sc > thr : sc < thr) << j;
          }
        } else {
          mask = chunk_mask(a.metric, v, fq, qq, thr,
                            [&](int j) { return __shfl_sync(0xffffffffu, rfl, j); });
        }
        if (!qvalid || nvalid <= 0) mask = 0;
        else if (nvalid < 32) mask &= (1u << nvalid) - 1u;
        const uint32_t grow0 = (uint32_t)(g.row_base + row0 + c * 32);  // global row id
        if (KR > 0) {
          // one candidate per lane per step straight into the register list
          // (re-tested against the threshold the earlier steps tightened)
          while (__any_sync(0xffffffffu, mask != 0)) {
            const int j = mask != 0 ? __ffs(mask) - 1 : 0;
            const RowFac<RC> rfc = RC ? rl.at(j, l2) : rl;
            const float rf = RC ? 0.0f : __shfl_sync(0xffffffffu, rfl, j);
            uint32_t kc = 0xffffffffu, ic = 0xffffffffu;
            if (mask != 0) {
              mask &= mask - 1;
              const float sc = RC ? fac_score(rfc, __uint_as_float(select32(v, j)), qf)
                                  : tile_score(a.metric, __uint_as_float(select32(v, j)), fq,
                                               qq, rf);
              if (desc ? sc > thr_s : sc < thr_s) {
                kc = rank_key32(sc, desc);
                ic = grow0 + j;
              }
            }
            reg.insert(kc, ic);
            const uint32_t tk = reg.key[RK - 1];
            thr_s = tk == 0xffffffffu ? (desc ? -INFINITY : INFINITY) : rank_key32_score(tk, desc);
          }
        } else if (hbn > 0) {
          while (__any_sync(0xffffffffu, mask != 0)) {
            const int j = mask != 0 ? __ffs(mask) - 1 : 0;
            const RowFac<RC> rfc = RC ? rl.at(j, l2) : rl;
            const float rf = RC ? 0.0f : __shfl_sync(0xffffffffu, rfl, j);
            if (mask != 0) {
              mask &= mask - 1;
              const float sc = RC ? fac_score(rfc, __uint_as_float(select32(v, j)), qf)
                                  : tile_score(a.metric, __uint_as_float(select32(v, j)), fq,
                                               qq, rf);
              const uint64_t key = make_key(sc, grow0 + j, desc);
              if (key < lists[m]) hb[(size_t)(hcnt++) * kBM + m] = key;
            }
            if (__any_sync(0xffffffffu, hcnt == hbn)) heap_pour(lists, k, hb, m, hcnt, thr_s, desc);
          }
        } else {
          while (__any_sync(0xffffffffu, mask != 0)) {
            const int j = mask != 0 ? __ffs(mask) - 1 : 0;
            const RowFac<RC> rfc = RC ? rl.at(j, l2) : rl;
            const float rf = RC ? 0.0f : __shfl_sync(0xffffffffu, rfl, j);
            if (mask == 0) continue;
            mask &= mask - 1;
            const float sc = RC ? fac_score(rfc, __uint_as_float(select32(v, j)), qf)
                                : tile_score(a.metric, __uint_as_float(select32(v, j)), fq, qq,
                                             rf);
            const uint64_t key = make_key(sc, grow0 + j, desc);
            if (key < lists[m]) {
              heap_replace_root(lists, k, kBM, m, key);
              const uint64_t root = lists[m];
              thr_s = root == kSentinel ? (desc ? -INFINITY : INFINITY)
                                        : rank_key32_score((uint32_t)(root >> 32), desc);
            }
          }
        }
      }
      tc_fence_before();
      if (PAIR && rank == 1) mbar_arrive_peer(&acce[buf], 0);  // (the even CTA's issuer)
      else mbar_arrive(&acce[buf]);
    }
    if (qvalid) {
      uint64_t *out = a.partial + ((size_t)(g.list_base + split) * a.B + qidx) * k;
      if (KR > 0) {
#pragma unroll
        for (int i = 0; i < RK; ++i)
          if (i >= RK - k) out[i - (RK - k)] = ((uint64_t)reg.key[i] << 32) | reg.id[i];
      } else {
        if (hcnt > 0) heap_pour(lists, k, hb, m, hcnt, thr_s, desc);
        heap_sort_ascending(lists, k, kBM, m);
        for (int i = 0; i < k; ++i) out[i] = lists[(size_t)i * kBM + m];
      }
    }
  }

  tc_fence_before();
  if constexpr (PAIR) {
    // (the even CTA's MMAs, which read this CTA's stages, have drained)
    cluster_sync_all();
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc_pair(tmem_base, kTmemCols);
    }
    cluster_sync_all();
  } else {
    __syncthreads();
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc(tmem_base, kTmemCols);
    }
  }
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

// Four or more query blocks: the codes are converted once per call (each
// code tile would otherwise be converted once per query block); one to three
// blocks convert in the stage loop.  Measured: B = 256 over 8.4M int8 rows
// takes 8.3 ms in the stage loop against 9.4 ms with the conversion pass (3.1
// of them); B = 1,024 over 27,986 rows 88 us against 72 + 12.
constexpr int64_t kPreBlocks = 4;

// Opt-in (LAM_SCORE_TM=1): the small-batch kernel with the codes in the MMA M
// dimension.  Measured against the stage-loop kernel over 361,802 int16 rows:
// 145 / 155 / 170 / 172 / 230 us at B = 3 / 8 / 16 / 32 / 64 against 153 /
// 157 / 159 / 162 / 162 us, and slower on int8 codes; both are bound by the
// raw-code supply of 128-byte row segments and their hand-offs, not by the
// MMAs.
bool tm_enabled() {
  const char *e = getenv("LAM_SCORE_TM");
  return e != nullptr && strcmp(e, "1") == 0;
}

// Opt-in (LAM_SCORE_PAIR=1): CTA pairs for the batched kernel (an even number
// of query blocks, one pass).  Measured: 77.7 against 68.0 us at 27,986 rows x
// 1,024 queries, 2.82 against 2.37 ms at 361,802 x 4,096, results bit-identical.
// A pair MMA (M = 256, N = 256) runs at the single-CTA rate per SM (128.7 cycles,
// twice the work) and each SM stages 24 instead of 32 KB per chunk, but these
// shapes are bound by the stage hand-offs and the epilogue, which the pair
// couples across two SMs (spinning instead of sleeping waits changed nothing).
bool pair_enabled() {
  const char *e = getenv("LAM_SCORE_PAIR");
  return e != nullptr && strcmp(e, "1") == 0;
}

// One launch of the batched kernel over grid (splits, query blocks); pairs as
// 2-CTA clusters of query blocks 2j, 2j + 1 (an even count), launched over
// (query blocks, splits): the driver takes an MMA pair only along the
// cluster's x dimension (a cluster of 1 x 2 is refused at launch).
cudaError_t launch_tc2(void (*kern)(ScoreArgs, Tc2Geom), dim3 grid, size_t smem,
                       cudaStream_t st, bool pair, const ScoreArgs &x, const Tc2Geom &g) {
  if (!pair) {
    kern<<<grid, kTc2Threads, smem, st>>>(x, g);
    return cudaGetLastError();
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid.y, grid.x);  // (query blocks, splits): the pair along x
  cfg.blockDim = dim3(kTc2Threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 2;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, x, g);
  if (e != cudaSuccess && getenv("LAM_DEBUG") != nullptr) {
    int nc = -1, cs = -1;
    const cudaError_t e1 = cudaOccupancyMaxActiveClusters(&nc, kern, &cfg);
    cfg.numAttrs = 0;
    const cudaError_t e2 = cudaOccupancyMaxPotentialClusterSize(&cs, kern, &cfg);
    cudaFuncAttributes fa;
    cudaFuncGetAttributes(&fa, kern);
    fprintf(stderr,
            "pair launch: grid (%u, %u) smem %zu: %s; max active clusters %d (%s), potential "
            "cluster size %d (%s); regs %d, static smem %zu, max dyn smem %d, cluster dims "
            "required %d, non-portable %d\n",
            grid.x, grid.y, smem, cudaGetErrorString(e), nc, cudaGetErrorString(e1), cs,
            cudaGetErrorString(e2), fa.numRegs, fa.sharedSizeBytes,
            fa.maxDynamicSharedSizeBytes, fa.requiredClusterWidth,
            fa.nonPortableClusterSizeAllowed);
  }
  return e;
}

bool tensor_fits(int width, int k, int64_t B) {
  if (k > kTcMaxK || (width != 1 && width != 2)) return false;
  if ((B + kBM - 1) / kBM >= kPreBlocks) return tc2_layout(k).ns >= 2;
  return tc_layout(width, k).ns >= 2;
}

bool tensor_fits_pre(int k) { return k <= kTcMaxK && tc2_layout(k).ns >= 2; }

int tensor_splits(int64_t B, int64_t N, int sms) {
  const int64_t nqb = (B + kBM - 1) / kBM;
  const int64_t n_tiles = (N + kBN - 1) / kBN;
  // splits x query blocks a multiple of the SM count: whole waves of CTAs
  int64_t ns = sms / gcd_i(sms, (int)(nqb % (1 << 30)));
  if (ns > n_tiles) ns = n_tiles;
  if (ns < 1) ns = 1;
  return (int)ns;
}

TensorPlan tensor_plan(int64_t B, int64_t N, int D, int k, int sms, bool force_pre) {
  TensorPlan p;
  const int64_t Bpad = (B + kBM - 1) / kBM * kBM;
  const int64_t nk = (D + kBK - 1) / kBK;
  p.pre = force_pre || Bpad / kBM >= kPreBlocks;
  p.qinfo_off = (size_t)(Bpad / kBM) * nk * kAStage;
  size_t off = p.qinfo_off + (size_t)Bpad * 16;
  off = (off + 255) / 256 * 256;
  if (!p.pre) {
    p.slab_rows = N;
    p.nslabs = 1;
    p.nsplit = tensor_splits(B, N, sms);
    p.fp16_off = p.rowf_off = p.seed_off = p.slabl_off = off;
    p.bytes = off;
  } else {
    int64_t cap = ((int64_t)1 << 30) / (nk * kBK * 2) / kBN * kBN;  // ~1 GiB of fp16 rows
    if (cap < kBN) cap = kBN;
    p.slab_rows = N < cap ? N : cap;
    p.nslabs = (int)((N + p.slab_rows - 1) / p.slab_rows);
    p.nsplit = tensor_splits(B, p.slab_rows, sms);
    p.fp16_off = off;
    p.rowf_off = p.fp16_off + (size_t)((p.slab_rows + kBN - 1) / kBN) * nk * kB16Bytes;
    p.seed_off = p.rowf_off + (size_t)p.slab_rows * 16;
    p.slabl_off = (p.seed_off + (size_t)Bpad * 4 + 255) / 256 * 256;
    p.bytes = p.slabl_off + (p.nslabs > 1 ? (size_t)p.nslabs * B * k * 8 : 0);
  }
  p.n_lists = p.nslabs * p.nsplit;
  return p;
}

cudaError_t launch_score_tensor(const ScoreArgs &a, cudaStream_t st, const RowPtrs &rp,
                                ScoreArgs *merge, int *merge_mode) {
  if (merge != nullptr) *merge = a;
  if (merge_mode != nullptr) *merge_mode = 0;
  const bool rc = a.fmt != 0;
  // status-driven call (codes' width on the device): both widths launch, one works
  const QuantStatus *qst = rc ? nullptr : rp.qst;
  if (a.k > kTcMaxK || (!rc && !qst && a.width != 1 && a.width != 2)) return cudaErrorInvalidValue;
  // int16 codes split as 256 h + l: the operand images span 2 D columns
  const bool wide = !rc && !qst && tensor_wide(a.width, a.code_bound);
  const int Dk = tensor_k_extent(a.D, wide);
  const TensorPlan P = tensor_plan(a.B, a.N, Dk, a.k, a.sms, rc || wide);
  if (P.n_lists != a.n_lists) return cudaErrorInvalidValue;
  // Two passes (Q_eps codes): the hi-only pass keeps kp candidates per list,
  // the certifying merge rescores them exactly and writes the top-k, and the
  // full (hi + lo) pass with its merge runs only for an uncertified query.
  const bool hi = !rc && !qst && tensor_hi(a.B, a.N, a.D, a.k, a.width, a.code_bound, a.sms);
  ScoreArgs ah = a;
  if (hi) ah.k = hi_list(a.k);
  uint8_t *qA = static_cast<uint8_t *>(a.qprep);
  const unsigned q_blocks = (unsigned)((a.Bpad + 7) / 8);
  cudaError_t e = cudaSuccess;

  if (!P.pre) {
    timing_launch_begin(LAM_TIME_AUX, st);
    // one block of at most 64 queries: they take MMA rows 64 .. 127, read by
    // the epilogue warps that share the SM sub-partitions of the converters
    // only (the producer and MMA warps sit on the other two)
    // Opt-in: up to 64 queries with k <= 32 on the kernel with the codes in
    // the MMA M dimension (queries from MMA row 0 of the image).
    const bool tm = !hi && !rc && tm_fits(a.B, a.D, a.k) && tm_enabled();
    const int qoff = !tm && a.Bpad == kBM && a.B <= kBM / 2 ? kBM / 2 : 0;
    qprep_kernel<<<q_blocks, 256, 0, st>>>(a.queries, a.B, a.D, a.Bpad, qA, qoff);
    timing_launch_end(LAM_TIME_AUX, st);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    CUtensorMap cmap1, cmap2;  // the codes as int8 and as int16 rows
    const uint32_t box_rows = tm ? (uint32_t)tm_box_rows() : (uint32_t)kBN;
    if ((qst || a.width == 1) &&
        !make_map_2d(&cmap1, CU_TENSOR_MAP_DATA_TYPE_UINT8, a.codes, (uint64_t)a.D, (uint64_t)a.N,
                     (uint64_t)a.D, (uint32_t)kRawRow, box_rows, CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
    if ((qst || a.width == 2) &&
        !make_map_2d(&cmap2, CU_TENSOR_MAP_DATA_TYPE_UINT16, a.codes, (uint64_t)a.D,
                     (uint64_t)a.N, (uint64_t)a.D * 2, (uint32_t)(kRawRow / 2), box_rows,
                     CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
    if (tm) return launch_score_tm(a, qst, cmap1, cmap2, st);
    const dim3 grid((unsigned)a.n_lists, (unsigned)(a.Bpad / kBM));
    // one pass of the stage-loop kernel over the lists of x.k keys
    auto pass = [&](const ScoreArgs &x, int hi_pass, int gate, int kind) -> cudaError_t {
      const TcLayout L = tc_layout(x.width, x.k, x.metric != LAM_METRIC_IP);
      if (L.ns < 2) return cudaErrorInvalidValue;
      TcGeom g;
      g.qst = qst;
      g.qoff = qoff;
      g.ns = L.ns;
      g.nr = L.nr;
      g.chunks = L.chunks;
      g.raw_off = (int)L.raw_off;
      g.lists_off = (int)L.lists_off;
      g.cbuf_off = (int)L.cbuf_off;
      g.cc_off = (int)L.cc_off;
      g.bar_off = (int)L.bar_off;
      g.hi = hi_pass;
      g.gate = gate;
      auto run = [&](auto kern, const CUtensorMap &cmap) -> cudaError_t {
        cudaError_t r = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)L.smem_bytes);
        if (r != cudaSuccess) return r;
        timing_launch_begin(kind, st);
        kern<<<grid, kTcThreads, L.smem_bytes, st>>>(cmap, x, g);
        timing_launch_end(kind, st);
        return cudaGetLastError();
      };
      auto run1 = [&]() -> cudaError_t {
        if (x.k <= 16) return run(score_tc_kernel<1, 16>, cmap1);
        if (x.k <= 32) return run(score_tc_kernel<1, 32>, cmap1);
        return run(score_tc_kernel<1, 0>, cmap1);
      };
      auto run2 = [&]() -> cudaError_t {
        if (x.k <= 16) return run(score_tc_kernel<2, 16>, cmap2);
        if (x.k <= 32) return run(score_tc_kernel<2, 32>, cmap2);
        return run(score_tc_kernel<2, 0>, cmap2);
      };
      if (qst) {
        const cudaError_t r = run1();
        return r != cudaSuccess ? r : run2();
      }
      return x.width == 1 ? run1() : run2();
    };
    if (!hi) return pass(a, 0, 0, LAM_TIME_SCORE);
    e = pass(ah, 1, 0, LAM_TIME_SCORE);
    if (e != cudaSuccess) return e;
    e = launch_topk_merge(ah, st, RowPtrs(), 1, a.k);
    if (e != cudaSuccess) return e;
    e = pass(a, 0, 1, LAM_TIME_AUX);  // (a no-op unless a query was not certified)
    if (merge_mode != nullptr) *merge_mode = 2;
    return e;
  }
  // two or more query blocks: convert each slab once, then the pure MMA kernel
  const bool pair = !hi && (a.Bpad / kBM) % 2 == 0 && pair_enabled();
  const Tc2Layout L = tc2_layout(a.k, pair);
  if (L.ns < 2) return cudaErrorInvalidValue;
  const Tc2Layout LH = tc2_layout(ah.k);  // the hi-only pass's lists
  if (LH.ns < 2) return cudaErrorInvalidValue;
  uint8_t *f16 = static_cast<uint8_t *>(a.qprep) + P.fp16_off;
  float *rowf = reinterpret_cast<float *>(static_cast<uint8_t *>(a.qprep) + P.rowf_off);
  Tc2Geom g;
  g.ns = L.ns;
  g.chunks = L.chunks;
  g.lists_off = (int)L.lists_off;
  g.cbuf_off = (int)L.cbuf_off;
  g.bar_off = (int)L.bar_off;
  g.b16 = f16;
  g.rowf = rowf;
  g.rowf4 = reinterpret_cast<const float4 *>(rowf);
  g.seed = nullptr;
  float *seed = reinterpret_cast<float *>(static_cast<uint8_t *>(a.qprep) + P.seed_off);
  uint64_t *slabl = reinterpret_cast<uint64_t *>(static_cast<uint8_t *>(a.qprep) + P.slabl_off);
  // several slabs: each slab's lists are merged into one, and the first slab's
  // k-th best bounds what the later slabs may offer
  const bool per_slab = P.nslabs > 1 && P.nsplit <= 256;
  auto kern_for = [&](int kk, bool pr) {
    if (pr)
      return rc ? (kk <= 16   ? score_tc2_kernel<16, true, true>
                   : kk <= 32 ? score_tc2_kernel<32, true, true>
                              : score_tc2_kernel<0, true, true>)
                : (kk <= 16   ? score_tc2_kernel<16, false, true>
                   : kk <= 32 ? score_tc2_kernel<32, false, true>
                              : score_tc2_kernel<0, false, true>);
    return rc ? (kk <= 16   ? score_tc2_kernel<16, true>
                 : kk <= 32 ? score_tc2_kernel<32, true>
                            : score_tc2_kernel<0, true>)
              : (kk <= 16   ? score_tc2_kernel<16, false>
                 : kk <= 32 ? score_tc2_kernel<32, false>
                            : score_tc2_kernel<0, false>);
  };
  // (the two passes may share one instantiation with different layouts: the
  // shared-memory limit is set right before each launch)
  auto kern = kern_for(a.k, pair);
  auto kern_h = kern_for(ah.k, false);
  const dim3 grid((unsigned)P.nsplit, (unsigned)(a.Bpad / kBM));
  for (int j = 0; j < P.nslabs; ++j) {
    const int64_t row_base = (int64_t)j * P.slab_rows;
    const int64_t nrows = a.N - row_base < P.slab_rows ? a.N - row_base : P.slab_rows;
    const int64_t nrows_pad = (nrows + kBN - 1) / kBN * kBN;
    const unsigned cg = (unsigned)((nrows_pad + 7) / 8);
    timing_launch_begin(LAM_TIME_AUX, st);
    float4 *rowf4 = reinterpret_cast<float4 *>(rowf);
    if (rc) {
      auto conv = [&](auto first, auto rest) {
        if (j == 0)
          first<<<q_blocks + cg, 256, 0, st>>>(a.queries, a.B, a.D, a.Bpad, qA, q_blocks, a.codes,
                                               rp.scale, rp.offset, nrows, nrows_pad, f16,
                                               rowf4, a.metric);
        else
          rest<<<cg, 256, 0, st>>>(a.codes, rp.scale, rp.offset, row_base, nrows,
                                   nrows_pad, a.D, f16, rowf4, a.metric);
      };
      if (a.fmt == LAM_ROWS_INT8)
        conv(prep_convert_rows_kernel<LAM_ROWS_INT8>, convert_rows_kernel<LAM_ROWS_INT8>);
      else if (a.fmt == LAM_ROWS_FP16)
        conv(prep_convert_rows_kernel<LAM_ROWS_FP16>, convert_rows_kernel<LAM_ROWS_FP16>);
      else
        conv(prep_convert_rows_kernel<LAM_ROWS_SIGN>, convert_rows_kernel<LAM_ROWS_SIGN>);
    } else if (qst) {  // status-driven: the width is read on the device
      if (j == 0)
        prep_convert_from_kernel<<<q_blocks + cg, 256, 0, st>>>(
            a.queries, a.B, a.D, a.Bpad, qA, q_blocks, a.codes, nrows, nrows_pad, f16, rowf,
            a.metric, a.s, a.gflags, qst);
      else
        convert_codes_from_kernel<<<cg, 256, 0, st>>>(a.codes, row_base, nrows, nrows_pad, a.D,
                                                      f16, rowf, a.metric, a.s, a.gflags, qst);
    } else if (j == 0) {  // the first slab's conversion shares a launch with the query prep
      if (a.width == 1)
        prep_convert_kernel<1><<<q_blocks + cg, 256, 0, st>>>(
            a.queries, a.B, a.D, a.Bpad, qA, q_blocks, a.codes, nrows, nrows_pad, f16, rowf,
            a.metric, a.s, a.gflags, nullptr, 0, hi ? 1 : 0);
      else
        prep_convert_kernel<2><<<q_blocks + cg, 256, 0, st>>>(
            a.queries, a.B, a.D, a.Bpad, qA, q_blocks, a.codes, nrows, nrows_pad, f16, rowf,
            a.metric, a.s, a.gflags, nullptr, wide ? 1 : 0, hi ? 1 : 0);
    } else if (a.width == 1) {
      convert_codes_kernel<1><<<cg, 256, 0, st>>>(a.codes, row_base, nrows, nrows_pad, a.D, f16,
                                                  rowf, a.metric, a.s, a.gflags, nullptr);
    } else {
      convert_codes_kernel<2><<<cg, 256, 0, st>>>(a.codes, row_base, nrows, nrows_pad, a.D, f16,
                                                  rowf, a.metric, a.s, a.gflags, nullptr,
                                                  wide ? 1 : 0);
    }
    timing_launch_end(LAM_TIME_AUX, st);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    g.row_base = row_base;
    g.nrows = nrows;
    g.list_base = j * P.nsplit;
    g.hi = 0;
    g.gate = 0;
    if (hi) {  // (one slab): the hi-only pass, its certifying merge, the gated full pass
      ScoreArgs akh = ah;  // the kernel sees the K extent of the operand images
      akh.D = Dk;
      Tc2Geom gh = g;
      gh.ns = LH.ns;
      gh.chunks = LH.chunks;
      gh.lists_off = (int)LH.lists_off;
      gh.cbuf_off = (int)LH.cbuf_off;
      gh.bar_off = (int)LH.bar_off;
      gh.hi = 1;
      e = cudaFuncSetAttribute(kern_h, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)LH.smem_bytes);
      if (e != cudaSuccess) return e;
      timing_launch_begin(LAM_TIME_SCORE, st);
      kern_h<<<grid, kTc2Threads, LH.smem_bytes, st>>>(akh, gh);
      timing_launch_end(LAM_TIME_SCORE, st);
      e = cudaGetLastError();
      if (e != cudaSuccess) return e;
      e = launch_topk_merge(ah, st, RowPtrs(), 1, a.k);
      if (e != cudaSuccess) return e;
      g.gate = 1;
    }
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)L.smem_bytes);
    if (e != cudaSuccess) return e;
    timing_launch_begin(hi ? LAM_TIME_AUX : LAM_TIME_SCORE, st);
    ScoreArgs ak = a;  // the kernel sees the K extent of the operand images
    ak.D = Dk;
    e = launch_tc2(kern, grid, L.smem_bytes, st, pair, ak, g);
    timing_launch_end(hi ? LAM_TIME_AUX : LAM_TIME_SCORE, st);
    if (e == cudaSuccess) e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (per_slab) {
      timing_launch_begin(LAM_TIME_MERGE, st);
      e = launch_slab_merge(a, j * P.nsplit, P.nsplit, j, slabl, j == 0 ? seed : nullptr, st);
      timing_launch_end(LAM_TIME_MERGE, st);
      if (e != cudaSuccess) return e;
      if (j == 0) g.seed = seed;
    }
  }
  if (per_slab && merge != nullptr) {
    merge->partial = slabl;
    merge->n_lists = P.nslabs;
  }
  if (hi && merge_mode != nullptr) *merge_mode = 2;
  return cudaSuccess;
}

bool tensor_hi(int64_t B, int64_t N, int D, int k, int width, int code_bound, int sms) {
  const char *env = getenv("LAM_SCORE_HI");
  if (env == nullptr || strcmp(env, "1") != 0) return false;  // opt-in
  const int kp = hi_list(k);
  if (kp == 0 || (width != 1 && width != 2)) return false;
  const bool wide = tensor_wide(width, code_bound);
  const TensorPlan P = tensor_plan(B, N, tensor_k_extent(D, wide), k, sms, wide);
  if (P.nslabs != 1 || !kmerge_fits(P.n_lists, kp)) return false;
  return P.pre ? tc2_layout(kp).ns >= 2 : tc_layout(width, kp).ns >= 2;
}


}  // namespace lam
