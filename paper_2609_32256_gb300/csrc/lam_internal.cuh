// lam_internal.cuh -- shared device helpers and launcher declarations of the
// sm_103a library.  Nothing here is visible through the C ABI.
#pragma once

#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/lam.h"

namespace lam {

// ---------------------------------------------------------------- constants --
constexpr uint32_t kFlagNonfinite = 1u;   // quantize: NaN/Inf seen
constexpr uint32_t kFlagRange = 2u;       // codes beyond a width / code bound
constexpr uint32_t kFlagWorkspace = 4u;   // codes buffer too small (AUTO)
constexpr uint32_t kFlagTimeout = 8u;     // a bounded wait gave up
constexpr uint32_t kFlagInput = 16u;      // the codes' quantize status reports an error
                                          // or a width the call does not take

constexpr int kMaxK = 1024;
constexpr int kHeaderBytes = 256;         // status block at the head of a workspace

// Wait budget of every device-side spin: ~1 s of SM clock.
constexpr long long kWaitCycles = 2000000000LL;

// 32-bit words of a search's status header (zeroed by every call): the flags
// above, and two test hooks the host sets only when asked to (the tests of
// the timeout path): a wait budget in SM cycles (0: kWaitCycles) and a stall
// word that makes the copy producers issue nothing.
constexpr int kHdrFlags = 0;
constexpr int kHdrWaitCycles = 2;
constexpr int kHdrStall = 3;
// Two-pass tensor search (hi-only candidates, then exact rescoring): the
// count of queries whose candidates could not be certified, the largest
// sum_d c_d^2 of any row (fp32 bits), and a test hook that fails every query.
constexpr int kHdrHiFail = 4;
constexpr int kHdrMaxCC = 5;
constexpr int kHdrForceFail = 6;

// Status block of lam_quantize (32 bytes, zeroed before each call).
struct QuantStatus {
  uint32_t neg_min;   // max over inputs of ~ord(x)   (0: no finite input seen)
  uint32_t max;       // max over inputs of ord(x)
  uint32_t flags;
  uint32_t width;     // width the AUTO kernel resolved
  uint32_t bar;       // blocks of the AUTO kernel that have finished
  uint32_t s_neg_min; // (unused)
  uint32_t s_max;     // width the AUTO kernel speculated from its sample
  uint32_t passes;    // 1: codes written at the resolved width; 2: a second pass is needed
};

// ----------------------------------------------------- ordered float keys --
// ord() maps fp32 to uint32 so that unsigned order equals numeric order
// (-0 is first folded into +0).
__device__ __forceinline__ uint32_t ord_f32(float f) {
  f = f + 0.0f;
  uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float unord_f32(uint32_t o) {
  uint32_t b = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
  return __uint_as_float(b);
}
// 64-bit selection key: smaller is better.  High word: the score in rank
// order (complemented for descending metrics); low word: the row id, so
// equal scores rank the lower id first.
__device__ __forceinline__ uint64_t make_key(float score, uint32_t row, bool desc) {
  uint32_t o = ord_f32(score);
  if (desc) o = ~o;
  return ((uint64_t)o << 32) | (uint64_t)row;
}
constexpr uint64_t kSentinel = ~0ull;

// ------------------------------------------------------------ PTX helpers --
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}
__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// As mbar_try_wait, but the thread may sleep (up to about a millisecond)
// until the phase completes instead of spinning on the issue slots.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(1000000u)
      : "memory");
  return ok != 0;
}
// The wait budget of a search: its header's test word, else kWaitCycles.
__device__ __forceinline__ long long wait_budget(const uint32_t *gflags) {
  const uint32_t v = gflags ? *reinterpret_cast<const volatile uint32_t *>(gflags + kHdrWaitCycles)
                            : 0u;
  return v ? (long long)v : kWaitCycles;
}
// Raises the header's largest row sum of squares to cc (cc >= 0: its fp32
// bits order as unsigned integers); reads first, so most rows add no atomic.
__device__ __forceinline__ void note_max_cc(uint32_t *gflags, float cc) {
  uint32_t *p = gflags + kHdrMaxCC;
  const uint32_t b = __float_as_uint(cc);
  if (b > *reinterpret_cast<volatile uint32_t *>(p)) atomicMax(p, b);
}
// Whether every query of a two-pass tensor search was certified (the
// fallback pass then has nothing to do).
__device__ __forceinline__ bool hi_all_certified(const uint32_t *gflags) {
  return *reinterpret_cast<const volatile uint32_t *>(gflags + kHdrHiFail) == 0u;
}
// Whether the copy producers of a search must issue nothing (test hook).
__device__ __forceinline__ bool producers_stalled(const uint32_t *gflags) {
  return gflags && *reinterpret_cast<const volatile uint32_t *>(gflags + kHdrStall) != 0u;
}
// Bounded wait for phase `parity` of `bar`.  Gives up after the search's wait
// budget (read only once the wait has slept; ~1 s unless a test set it) or as
// soon as *abort is set; on giving up sets *abort and the timeout flag.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity,
                                          volatile int *abort, uint32_t *gflags) {
  if (mbar_try_wait(bar, parity)) return true;
  long long t0 = clock64();
  long long budget = -1;
  while (true) {
    if (mbar_try_wait_sleep(bar, parity)) return true;
    if (*abort) return false;
    if (budget < 0) budget = wait_budget(gflags);
    if (clock64() - t0 > budget) {
      *abort = 1;
      if (gflags) atomicOr(gflags, kFlagTimeout);
      return false;
    }
  }
}

// 1-D bulk copy global -> shared, completing on an mbarrier (16-byte
// aligned addresses, size a multiple of 16).
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes,
                                         uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// 2-D tiled TMA load (coordinates: x = innermost element index, y = row).
__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, int32_t x,
                                            int32_t y, uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

// The Q_eps quotient x / s rounded to nearest, equal bit for bit to one IEEE
// division, from y = RN(1/s) and two FMA steps (cheaper than the division):
// q0 = x y is within two ulps of x / s; q1 = q0 + (x - s q0) y is faithful;
// and by Markstein's theorem (a faithful quotient, a reciprocal with relative
// error below 2^-24, the residual and the update each rounded once to
// nearest) q2 = q1 + (x - s q1) y is the correctly rounded quotient, as long
// as nothing over- or underflows.  Hence the guards: s in [2^-40, 2^40]
// (otherwise every value takes the division) and |q0| < 2^100 (otherwise,
// and for non-finite x, this value does); below |x| = 2^-80 the residual may
// be subnormal, but the quotient is then under 2^-40 and rounds to code 0
// either way.  (Checked against IEEE single division for every finite x and
// 18 divisors, among them 2^-40, 2^40 and all-ones significands.)
struct QDiv {
  float s, y;
  bool fast;
  __device__ __forceinline__ static QDiv of(float s_) {
    QDiv d;
    d.s = s_;
    d.y = __frcp_rn(s_);
    d.fast = s_ >= 0x1p-40f && s_ <= 0x1p40f;
    return d;
  }
  __device__ __forceinline__ float quot(float x) const {
    float q = __fmul_rn(x, y);
    if (fast && fabsf(q) < 0x1p100f) {
      q = __fmaf_rn(__fmaf_rn(-s, q, x), y, q);
      q = __fmaf_rn(__fmaf_rn(-s, q, x), y, q);
    } else {
      q = __fdiv_rn(x, s);
    }
    return q;
  }
  // Q_eps(x): the quotient rounded half to even
  __device__ __forceinline__ int32_t code(float x) const { return __float2int_rn(quot(x)); }
};

// ------------------------------------------------------------- launchers --
// (defined in quantize.cu / score_bw.cu / score_tc.cu; all launch on `st`)
cudaError_t launch_quant_range(const float *x, int64_t n, QuantStatus *status, int sms,
                               cudaStream_t st);
cudaError_t launch_quantize(const float *x, int64_t n, float s, int width_req, void *codes,
                            size_t codes_bytes, QuantStatus *status, int sms,
                            cudaStream_t st);
// Q_eps fused with the band digests (width_req 1/2/4 forced, 0 AUTO).
cudaError_t launch_quantize_bands(const float *x, int64_t N, int D, int r, float s,
                                  int width_req, void *codes, size_t codes_bytes,
                                  uint64_t *digests, QuantStatus *st, int sms,
                                  cudaStream_t stream);
// Batch admission (admit.cu).
size_t admit_workspace_bytes(int64_t N, int nb, int64_t max_pairs);
cudaError_t launch_admit_batch(const float *e, int64_t N, int D, const uint64_t *dig, int nb,
                               double delta, int32_t *rep, double *dist, void *ws,
                               int64_t max_pairs, int sms, cudaStream_t st, int64_t *n_pairs,
                               double *delta_hat, int64_t *n_retained, bool *overflow);
// Error-bounded byte codec (lamz.cu).
size_t lamz_head_bytes(int64_t n);
size_t lamz_bound_bytes(int64_t n);
size_t lamz_workspace_bytes(int64_t n);
cudaError_t launch_lamz_compress(const float *x, int64_t n, float rel, uint8_t *out, size_t cap,
                                 void *ws, int sms, cudaStream_t stream, size_t *bytes,
                                 bool *fits, bool *nonfinite, bool *timed_out);
cudaError_t launch_lamz_decompress(const uint8_t *in, size_t in_bytes, float *out, int64_t n,
                                   void *ws, int sms, cudaStream_t stream, bool *bad);
cudaError_t launch_code_sqnorms(const void *codes, int width, int64_t N, int D, float *out,
                                int sms, cudaStream_t st);
cudaError_t launch_dequantize(const void *codes, int width, int64_t n, float s, float *out,
                              int sms, cudaStream_t st);
// AUTO width: one launch; if the status ends with passes == 2 the caller
// quantizes again with launch_quantize at the resolved width.
cudaError_t launch_quantize_auto(const float *x, int64_t n, float s, void *codes,
                                 size_t codes_bytes, QuantStatus *status, int sms,
                                 cudaStream_t st);
// Asynchronous quantization: settles the status on the device after the AUTO
// or forced kernel (range error for a forced width, AUTO's second pass).
cudaError_t launch_quantize_settle(const float *x, int64_t n, float s, int width_req, void *codes,
                                   size_t codes_bytes, QuantStatus *status, int sms,
                                   cudaStream_t st);
cudaError_t launch_dequantize_from(const void *codes, const QuantStatus *status, int64_t n,
                                   float s, float *out, int sms, cudaStream_t st);

struct ScoreArgs {
  const float *queries;
  int64_t B;
  const void *codes;
  int width;
  int64_t N;
  int D;
  float s;         // 2 eps
  int code_bound;  // tensor path limit check
  int k;
  int metric;
  float *scores;
  int64_t *ids;
  uint32_t *gflags;     // workspace status flags
  uint64_t *partial;    // [n_lists][B][k] keys
  int n_lists;
  void *qprep;          // tensor path: fp16 [2*Bpad][D] then float4 [Bpad]
  int64_t Bpad;
  int sms;
  // Per-row codecs (lam_score_topk_rows): LAM_ROWS_*, 0 for Q_eps codes.
  // (It sits in the struct's tail padding: a larger kernel parameter block
  // costs the tensor-core kernel registers and time.)
  int fmt = 0;
};

// Per-row factors of a per-row codec, passed beside ScoreArgs; for the
// status-driven calls (lam_score_topk_from) the quantize status that holds
// the codes' width (a.width is then ignored).
struct RowPtrs {
  const float *scale = nullptr;
  const float *offset = nullptr;
  const QuantStatus *qst = nullptr;
};

// A quantize status that finished without error.  The consumers run after
// the quantize kernels in stream order and nothing writes the block while
// they read it, so every thread may take it through the read-only cache (one
// address read by every thread of a grid: a coherent load per thread would
// queue on that one L2 line).
__device__ __forceinline__ bool status_ok(const QuantStatus *st) {
  const uint32_t f = __ldg(&st->flags);
  return !(f & (kFlagNonfinite | kFlagRange | kFlagWorkspace | kFlagTimeout));
}
__device__ __forceinline__ uint32_t status_width(const QuantStatus *st) {
  return __ldg(&st->width);
}
// Width of the codes: from the status when there is one.
__device__ __forceinline__ int codes_width(const ScoreArgs &a, const RowPtrs &rp) {
  return rp.qst != nullptr ? (int)status_width(rp.qst) : a.width;
}

// Decoded value xhat_d of row `row` of a per-row codec, evaluated exactly as
// lam_decode_rows writes it.
__device__ __forceinline__ float row_value(const ScoreArgs &a, const RowPtrs &rp, int64_t row,
                                           int d) {
  if (a.fmt == LAM_ROWS_INT8)
    return __fadd_rn(rp.offset[row],
                     __fmul_rn(rp.scale[row],
                               (float)static_cast<const int8_t *>(a.codes)[row * a.D + d]));
  if (a.fmt == LAM_ROWS_FP16)
    return __half2float(static_cast<const __half *>(a.codes)[row * a.D + d]);
  const uint8_t byte = static_cast<const uint8_t *>(a.codes)[row * (a.D / 8) + d / 8];
  return ((byte >> (d & 7)) & 1u) ? rp.scale[row] : -rp.scale[row];
}

cudaError_t launch_encode_rows(const float *x, int64_t N, int D, int fmt, void *codes,
                               float *scale, float *offset, int sms, cudaStream_t st);
cudaError_t launch_decode_rows(const void *codes, int fmt, int64_t N, int D, const float *scale,
                               const float *offset, float *out, int sms, cudaStream_t st);

// `qst` (status-driven calls): the codes' width is read on the device.
cudaError_t launch_score_bandwidth(const ScoreArgs &a, cudaStream_t st,
                                   const QuantStatus *qst = nullptr);
// Per-vector codecs, B <= 2: row bytes (D, 2D or D/8) a multiple of 16, D <= 1024, k <= 128.
cudaError_t launch_score_bandwidth_rows(const ScoreArgs &a, const RowPtrs &rp, cudaStream_t st);
int bandwidth_rows_ctas(int64_t N, int fmt, int D, int sms);
cudaError_t launch_score_generic(const ScoreArgs &a, cudaStream_t st,
                                 const RowPtrs &rp = RowPtrs());
// `merge` (optional) receives the arguments of the final merge: a search of
// several slabs leaves one merged list per slab in its workspace.
// `merge_mode` (optional) receives the mode of that merge (launch_topk_merge):
// 2 after a two-pass search, whose final merge belongs to the gated full pass.
cudaError_t launch_score_tensor(const ScoreArgs &a, cudaStream_t st,
                                const RowPtrs &rp = RowPtrs(), ScoreArgs *merge = nullptr,
                                int *merge_mode = nullptr);
// mode 0: the merge of a search; 1: the certifying merge of a two-pass
// tensor search (a.k = candidate lists; every candidate rescored exactly,
// the best kout written, uncertified queries counted in the header); 2: the
// merge of the gated full pass (does nothing when every query was certified).
cudaError_t launch_topk_merge(const ScoreArgs &a, cudaStream_t st, const RowPtrs &rp = RowPtrs(),
                              int mode = 0, int kout = 0);
// Multi-slab searches: the partial lists [list0, list0 + n_lists) of one slab
// merged into slab `slab` of `out` ([nslabs][B][k] keys); with `seed`, also
// per query the ranking-form score of the slab's k-th best key.
cudaError_t launch_slab_merge(const ScoreArgs &a, int list0, int n_lists, int slab, uint64_t *out,
                              float *seed, cudaStream_t st);

// Planning shared by the workspace-size query and the launch.
enum Path { kPathBandwidth = 0, kPathTensor = 1, kPathGeneric = 2 };
int bandwidth_ctas(int64_t N, int D, int width, int sms);
int tensor_splits(int64_t B, int64_t N, int sms);
bool tensor_fits(int width, int k, int64_t B);  // shared memory holds >= 2 stages
bool tensor_fits_pre(int k);         // the same for the converting-pass kernel alone
// Tensor-path workspace (after the partial lists): [query images][query info]
// and, for two or more query blocks, [fp16 code slab][per-row factors].
struct TensorPlan {
  bool pre;            // codes converted to fp16 by a separate pass
  int64_t slab_rows;   // rows per slab (pre), else N
  int nslabs, nsplit, n_lists;
  // rowf: 16 bytes per slab row; seed: 4 bytes per query; slab lists: the
  // merged list of each slab, nslabs x B x k keys (several slabs only)
  size_t qinfo_off, fp16_off, rowf_off, seed_off, slabl_off, bytes;
};
// (force_pre: the per-row codecs always take the converting pass)
TensorPlan tensor_plan(int64_t B, int64_t N, int D, int k, int sms, bool force_pre = false);
// int16 codes the fp16 operands cannot hold exactly (a bound above 2048, or
// no bound given): the tensor path splits each code as 256 h + l, two exact
// fp16 values, and converts with the separate pass over 2 D image columns.
inline bool tensor_wide(int width, int code_bound) {
  return width == 2 && !(code_bound > 0 && code_bound <= 2048);
}
// Candidate list length of the hi-only tensor pass for a final top-k: k plus
// a margin (6 for k < 12, else 16), rounded up to the 16- and 32-entry
// register lists; 0 when that exceeds the largest tensor-path list (128).
inline int hi_list(int k) {
  int kp = k + (k < 12 ? 6 : 16);
  if (kp <= 16) kp = 16;
  else if (kp <= 32) kp = 32;
  return kp <= 128 ? kp : 0;
}
// Whether a tensor-path search of this shape runs as two passes: the hi-only
// pass (fp16 hi term of the query only, half the MMAs) keeping hi_list(k)
// candidates, exact rescoring and certification in the merge, and the full
// (hi + lo) pass gated on a certification failure.  Opt-in: LAM_SCORE_HI=1
// (measured, it does not beat the single full pass on this part: the
// kernels are bound by shared-memory ingress and the epilogue as much as by
// the MMAs, and the extra candidates, the rescoring merge and the gated
// launches cost what the halved MMAs save).
bool tensor_hi(int64_t B, int64_t N, int D, int k, int width, int code_bound, int sms);
// Small query batches on the tensor cores with the codes in the MMA M
// dimension (score_tm.cu): whether the kernel takes B queries and top-k, and
// its launch over a.n_lists CTAs of 256-row tiles.  The query images are the
// tensor path's (one block, queries from MMA row 0); cmap1 / cmap2 map the
// codes as int8 / int16 rows (boxes of 128 bytes x tm_box_rows() rows,
// 128-byte swizzle).
bool tm_fits(int64_t B, int D, int k);
int tm_box_rows();
cudaError_t launch_score_tm(const ScoreArgs &a, const QuantStatus *qst, const CUtensorMap &cmap1,
                            const CUtensorMap &cmap2, cudaStream_t st);
// The warp k-way merge takes n_lists sorted lists of k keys per query.
bool kmerge_fits(int n_lists, int k);

// K extent of the tensor path's operand images: D, or for the split two
// image chunks per 32-wide K chunk of the codes (D rounded up to 32, doubled).
inline int tensor_k_extent(int D, bool wide) { return wide ? 2 * ((D + 31) / 32 * 32) : D; }

// Synchronous read-back of a small device status block into host memory:
// queued on `st`, then waits for `st`.
cudaError_t read_back(void *dst, const void *src, size_t n, cudaStream_t st);

// Launch bracketing for lam_timing_* (no-ops unless timing is on for `kind`).
void timing_launch_begin(int kind, cudaStream_t st);
void timing_launch_end(int kind, cudaStream_t st);
int generic_ctas(int64_t B, int64_t N, int sms);

}  // namespace lam
