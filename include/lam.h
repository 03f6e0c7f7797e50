/*
 * lam.h -- C ABI of the GB300 (sm_103a) library for LAM's quantized memory.
 *
 * The method (paper: "LAM: Lossy Agent Memory"):
 *   - Q_eps(x) = round(x / 2 eps), coordinatewise with one global eps
 *     (Sec. 3.2 "Three layers", layer L1; Algorithm 1 applies it to every
 *     arriving embedding).
 *   - Dequantisation xhat = 2 eps * Q_eps(x): a cell of the quantizer has
 *     half-width eps (Sec. 3.1; App. "Rank invariance, in full").
 *   - Exact search over the stored vectors is one matrix-vector product per
 *     query followed by a top-k (Sec. "Brute-force scan crossover"); here it
 *     runs directly on the integer codes, with dequantisation folded into the
 *     score.
 *
 * Conventions shared by every call:
 *   - Every array argument is a DEVICE pointer on the current CUDA device,
 *     allocated and owned by the caller.  The library allocates no memory.
 *     Only the scalar outputs of the synchronous calls are host pointers.
 *   - Arrays are dense and row-major.  Codes are two's-complement integers of
 *     1, 2 or 4 bytes ("width").
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).  Work is
 *     queued on it; lam_quantize and lam_score_topk_status also wait for it.
 *   - Arguments are checked on the host before anything is queued; a bad
 *     argument returns LAM_ERR_INVALID and queues nothing.
 *   - Rounding: the quotient x / 2eps is one IEEE fp32 division by
 *     s = fl32(2 * eps) and is rounded half-to-even; dequantisation is one
 *     fp32 multiply s * code.  No fast-math arithmetic is used.
 */
#ifndef LAM_H
#define LAM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A cudaStream_t. */
typedef struct CUstream_st *lam_stream_t;

typedef enum lam_status {
  LAM_OK = 0,
  LAM_ERR_INVALID = 1,     /* bad argument; nothing was queued             */
  LAM_ERR_RANGE = 2,       /* codes do not fit the requested/needed width  */
  LAM_ERR_NONFINITE = 3,   /* NaN or Inf in the input of lam_quantize      */
  LAM_ERR_WORKSPACE = 4,   /* an output or workspace buffer is too small   */
  LAM_ERR_CUDA = 5,        /* a CUDA runtime call or launch failed         */
  LAM_ERR_TIMEOUT = 6,     /* a bounded device-side wait gave up           */
  LAM_ERR_UNSUPPORTED = 7  /* a forced kernel path cannot take this shape  */
} lam_status;

/* Code widths, in bytes.  LAM_WIDTH_AUTO asks lam_quantize for the narrowest. */
enum { LAM_WIDTH_AUTO = 0, LAM_I8 = 1, LAM_I16 = 2, LAM_I32 = 4 };

/* Scores: inner product and cosine rank descending, squared L2 ascending. */
enum { LAM_METRIC_IP = 0, LAM_METRIC_COSINE = 1, LAM_METRIC_L2 = 2 };

/* Library version, major*10000 + minor*100 + patch. */
int32_t lam_version(void);

/* Static text for a status code. */
const char *lam_status_string(int32_t status);

/* Bytes of device workspace lam_quantize needs (a 32-byte status block). */
size_t lam_quantize_workspace_size(void);

/*
 * lam_quantize -- Q_eps over n fp32 values (Sec. 3.2, layer L1).
 *
 *   code_i = round_half_even(fl32(x_i / s)),  s = fl32(2 * eps)
 *
 * x          [n] fp32, device, 4-byte aligned (16-byte alignment of x and
 *            codes selects the 128-bit vector path).
 * n          number of values, 0 <= n < 2^62.
 * eps        finite, > 0, and 2*eps a normal fp32 number.
 * width_req  LAM_I8, LAM_I16, LAM_I32, or LAM_WIDTH_AUTO for the narrowest
 *            width whose range holds [min code, max code] (int8 when n == 0).
 * codes      [n] codes of the resolved width, device, aligned to the width
 *            (AUTO: 4-byte aligned); may be NULL to ask only for the range and
 *            width.  Contents are undefined unless LAM_OK.
 * codes_bytes  size of `codes`; must be >= n * width (AUTO: of the width that
 *            is resolved -- n * 4 always suffices).
 * workspace  >= lam_quantize_workspace_size() bytes of device memory,
 *            16-byte aligned; it may be reused between calls on one stream.
 * width_out, scale_out, code_min_out, code_max_out   host outputs (any may be
 *            NULL): the width used, s = 2*eps, and the smallest and largest
 *            code.  They are written for LAM_OK and LAM_ERR_RANGE.
 *
 * With LAM_WIDTH_AUTO one launch speculates the width from a fixed sample
 * of x (four values at each of 64 evenly spaced positions), quantizes at
 * it while measuring the exact range, and a second launch quantizes again
 * only if the exact range needs a wider type.
 *
 * Synchronous on `stream`: the status block is read back, because the width
 * and the range are outputs.  Errors: LAM_ERR_NONFINITE (NaN/Inf in x),
 * LAM_ERR_RANGE (a forced width, or int32, cannot hold the codes),
 * LAM_ERR_WORKSPACE (codes_bytes or the workspace is too small), LAM_ERR_CUDA.
 * (LAM_ERR_TIMEOUT is not returned by this call.)
 */
lam_status lam_quantize(const float *x, int64_t n, float eps, int32_t width_req,
                        void *codes, size_t codes_bytes, void *workspace,
                        size_t workspace_bytes, int32_t *width_out,
                        float *scale_out, int32_t *code_min_out,
                        int32_t *code_max_out, lam_stream_t stream);

/*
 * lam_quantize_bands -- Q_eps fused with the band digests of the quantized
 * rows (Sec. 3.2, layer L1: quantize, divide each vector into bands of r
 * coordinates and hash each band; records sharing a band digest are
 * candidates.  Algorithm 1: B <- BandHash(Q_eps(e))).  One pass over x.
 *
 * x        [N, D] fp32 rows, device, 4-byte aligned; D a multiple of r and
 *          D / r <= 65536.
 * r        band width in coordinates (the paper sweeps 2, 4, 8, 16, 32).
 * codes    as for lam_quantize (may be NULL: digests only).
 * digests  [N, D / r] uint64, device, 8-byte aligned: digests[i * (D/r) + b]
 *          is the 64-bit FNV-1a (offset basis 14695981039346656037, prime
 *          1099511628211, one xor and one multiply per byte) of band b of
 *          row i: the band index as 2 little-endian bytes, then the band's r
 *          codes as their `width` little-endian two's-complement bytes.  The
 *          paper names no hash; this reading is exact and portable.
 * The width, workspace, outputs, synchrony and errors are those of
 * lam_quantize (with AUTO, the digests use the resolved width); on an error
 * the digests are undefined.  LAM_ERR_INVALID also for r outside 1..D, D not
 * a multiple of r, or a misaligned digests pointer.
 */
lam_status lam_quantize_bands(const float *x, int64_t N, int32_t D, float eps,
                              int32_t width_req, int32_t r, void *codes,
                              size_t codes_bytes, uint64_t *digests,
                              void *workspace, size_t workspace_bytes,
                              int32_t *width_out, float *scale_out,
                              int32_t *code_min_out, int32_t *code_max_out,
                              lam_stream_t stream);

/*
 * lam_admit_batch -- the batch form of the admission rule (Algorithm 2;
 * Sec. 3.3): records 0..N-1 in order; the candidates of record i are the
 * retained records that share a band digest with it in the same band (the
 * digests of lam_quantize_bands); its representative is the lowest-indexed
 * candidate within l2 distance delta of it (delta = sqrt(2 - 2t) for merge
 * threshold t, Eq. 2), else record i is retained.  Distances are taken in
 * full precision: per coordinate the difference of the two fp32 values in
 * double, squared, summed in coordinate order without fused multiply-adds,
 * then one sqrt; a pair is within delta when that distance is <= delta.
 *
 * e         [N, D] fp32 embeddings, device, 4-byte aligned.
 * digests   [N, nb] uint64 band digests, device, 8-byte aligned.
 * rep       [N] int32 out: representative of each record (itself if retained).
 * dist      [N] double out: distance to the representative (0 if retained).
 * workspace >= lam_admit_batch_workspace_size(N, nb, max_pairs) bytes of
 *           device memory, 256-byte aligned; max_pairs bounds the number of
 *           (row, lower row) candidate pairs before de-duplication.
 * delta_hat_out (host, may be NULL): the measured bound, the largest merge
 *           distance (0 when nothing merges); n_retained_out: |R|;
 *           n_pairs_out: candidate pairs found.
 * Synchronous on `stream`.  Errors: LAM_ERR_INVALID (bad sizes, NULL or
 * misaligned pointers, delta negative or not finite, N > 2^31 - 1, N * nb >=
 * 2^32), LAM_ERR_WORKSPACE (workspace too small, or more candidate pairs than
 * max_pairs: *n_pairs_out then holds the count needed), LAM_ERR_CUDA.
 */
size_t lam_admit_batch_workspace_size(int64_t N, int32_t nb, int64_t max_pairs);
lam_status lam_admit_batch(const float *e, int64_t N, int32_t D,
                           const uint64_t *digests, int32_t nb, double delta,
                           int32_t *rep, double *dist, void *workspace,
                           size_t workspace_bytes, int64_t max_pairs,
                           double *delta_hat_out, int64_t *n_retained_out,
                           int64_t *n_pairs_out, lam_stream_t stream);

/*
 * Error-bounded byte codec for retained embeddings (Sec. 3.2, layer L2:
 * "error-bounded byte compression" under a relative codec error bound; the
 * paper deploys 1% of max|x|).  The paper uses a third-party codec; this is a
 * self-contained format of the same family:
 *   eb = fl32(rel * max|x|), s = fl32(2 eb) (s = 1 when every x is 0); the
 *   codes are Q_eps at eps = eb (the quantizer's division and rounding);
 *   blocks of 32 codes; inside a block the deltas d_0 = q_0, d_j = q_j -
 *   q_{j-1} (a tail block repeats its last code); L = bit length of the
 *   block's largest |d| (0..31).
 * Stream (little-endian): "LAMZ", n (int64), s (fp32), one byte L per block,
 * zero padding to a multiple of 4, then for each block with L > 0 a 32-bit
 * sign word (bit j: d_j < 0) and L 32-bit bit planes (bit j of plane p: bit p
 * of |d_j|).  Decoding returns fl32(s * q): |x - x_hat| <= eb (+ fp32
 * rounding of the quotient and the product), exactly the error of Q_eps.
 *
 * lam_lamz_bound(n): the largest stream for n values.
 * lam_lamz_workspace_size(n): device scratch for either direction.
 * lam_lamz_compress: x [n] fp32 device (4-byte aligned), rel in [1e-6, 1],
 *   out (device, 4-byte aligned) of out_capacity bytes, *out_bytes (host) the
 *   stream size.  Synchronous (one pass over x after its max|x|; blocks of
 *   32 values are placed by a decoupled look-back across the device, a
 *   bounded wait).  Errors: LAM_ERR_INVALID, LAM_ERR_NONFINITE,
 *   LAM_ERR_WORKSPACE (workspace too small, or the stream exceeds
 *   out_capacity: *out_bytes then holds the size needed and the bytes of out
 *   past the header are unspecified), LAM_ERR_TIMEOUT (the look-back gave
 *   up; out unspecified), LAM_ERR_CUDA.
 * lam_lamz_decompress: the stream (device, in_bytes) into out [n] fp32
 *   (device).  LAM_ERR_INVALID for a stream that is not LAMZ, has another n,
 *   a bit length above 31, or is truncated (checked on the device before any
 *   payload word is read; out is then not written).  Synchronous: one wait,
 *   after the decode.
 */
size_t lam_lamz_bound(int64_t n);
size_t lam_lamz_workspace_size(int64_t n);
lam_status lam_lamz_compress(const float *x, int64_t n, float rel, void *out,
                             size_t out_capacity, size_t *out_bytes, void *workspace,
                             size_t workspace_bytes, lam_stream_t stream);
lam_status lam_lamz_decompress(const void *in, size_t in_bytes, float *out, int64_t n,
                               void *workspace, size_t workspace_bytes,
                               lam_stream_t stream);

/*
 * Device-resident form of the same steps, for pipelines that must not wait
 * for the host: lam_quantize_async queues Q_eps exactly as lam_quantize
 * computes it (same codes, same AUTO width) but reads nothing back.  The
 * outcome stays in the workspace's 32-byte status block: the width, the code
 * range, the errors.  lam_dequantize_from and lam_score_topk_from take the
 * codes' width from that block on the device, so quantize -> dequantize ->
 * search can be queued back to back on streams (or captured in a CUDA graph)
 * with no host round trip; lam_quantize_result reads the block when the host
 * needs it.
 *
 * lam_quantize_async: arguments as for lam_quantize without the host
 *   outputs.  AUTO writes the codes at the narrowest width; when the width
 *   it speculated from a sample was too narrow, a second pass on the device
 *   rewrites them (the codes buffer must hold n times that width).  A forced
 *   width too narrow for the codes is recorded as a range error.  Keep the
 *   workspace (and codes) alive and unchanged until their consumers ran.
 *   Asynchronous.  Errors now: LAM_ERR_INVALID, LAM_ERR_WORKSPACE (workspace
 *   below 32 bytes, or codes_bytes < n * forced width), LAM_ERR_CUDA.
 * lam_quantize_result: waits for `stream` and decodes the status block of
 *   the workspace as lam_quantize reports it (same eps and width_req as the
 *   call; outputs and errors as for lam_quantize).
 * lam_dequantize_from: xhat = fl32(2 eps * code) at the width in the status
 *   block `quant_workspace` (codes and out 4-byte aligned).  Nothing is
 *   written when the status holds an error.  Asynchronous.
 * lam_score_topk_from: lam_score_topk with the width and validity taken from
 *   `quant_workspace` (widths 1 and 2; eps the quantizer's).  The path is
 *   chosen without the width, from shapes that both widths take; the tensor
 *   cores take int16 codes up to +-2048 only, larger ones give LAM_ERR_RANGE
 *   from lam_score_topk_status.  A status with an error, or width 4, gives
 *   LAM_ERR_UNSUPPORTED there (the scores are then undefined).  Workspace
 *   size and path queries as for lam_score_topk.  Asynchronous.
 */
lam_status lam_quantize_async(const float *x, int64_t n, float eps, int32_t width_req,
                              void *codes, size_t codes_bytes, void *workspace,
                              size_t workspace_bytes, lam_stream_t stream);
lam_status lam_quantize_result(const void *workspace, float eps, int32_t width_req,
                               lam_stream_t stream, int32_t *width_out, float *scale_out,
                               int32_t *code_min_out, int32_t *code_max_out);
lam_status lam_dequantize_from(const void *codes, const void *quant_workspace, int64_t n,
                               float eps, float *out, lam_stream_t stream);
size_t lam_score_topk_from_workspace_size(int64_t B, int64_t N, int32_t D, int32_t k);
int32_t lam_score_topk_from_path(int64_t B, int64_t N, int32_t D, int32_t k);
lam_status lam_score_topk_from(const float *queries, int64_t B, const void *codes,
                               const void *quant_workspace, int64_t N, int32_t D, float eps,
                               int32_t k, int32_t metric, float *scores, int64_t *ids,
                               void *workspace, size_t workspace_bytes, lam_stream_t stream);

/*
 * lam_dequantize -- xhat_i = fl32(scale * code_i), the inverse map of Q_eps
 * up to the cell half-width eps (|x - xhat| <= eps, Sec. 3.1).
 *
 * codes  [n] of `width` bytes (1, 2 or 4), device, aligned to the width.
 * out    [n] fp32, device, 4-byte aligned.
 * scale  the step s returned by lam_quantize (s = 2 eps).
 * Asynchronous on `stream`.  Errors: LAM_ERR_INVALID, LAM_ERR_CUDA.
 */
lam_status lam_dequantize(const void *codes, int32_t width, int64_t n,
                          float scale, float *out, lam_stream_t stream);

/*
 * Bytes of device workspace lam_score_topk needs for this shape on the
 * current device (arguments as for lam_score_topk).  0 for invalid shapes.
 */
size_t lam_score_topk_workspace_size(int64_t B, int64_t N, int32_t D,
                                     int32_t k, int32_t width,
                                     int32_t code_bound);

/*
 * lam_score_topk -- exact search on the codes (Sec. "Brute-force scan
 * crossover"): every query against every stored row, dequantisation folded
 * into the score, then the k best per query.
 *
 *   inner product  s * sum_d q_d c_d                     (descending)
 *   cosine         sum_d q_d c_d / (||q|| ||c||)          (descending; 0 if a
 *                  norm is 0 -- the norm of the dequantised row, s cancels)
 *   squared L2     ||q||^2 - 2 s q.c + s^2 ||c||^2        (ascending)
 *
 * with s = fl32(2 * eps).  Ties between equal fp32 scores go to the lower row
 * id (the paper's lowest-index rule, Algorithm 1).
 *
 * queries    [B, D] fp32, device, 4-byte aligned.  B >= 1.
 * codes      [N, D] codes of `width` bytes, device, aligned to the width (a
 *            16-byte aligned base enables the bulk-copy and TMA paths).
 *            1 <= k <= N < 2^31.
 * code_bound the largest |code| if known (e.g. max(-code_min, code_max) from
 *            lam_quantize), else 0; with int16 codes a bound <= 2048 enables
 *            the tensor-core path.  A bound smaller than the real codes gives
 *            LAM_ERR_RANGE from lam_score_topk_status.
 * k          1 <= k <= min(N, 1024).
 * scores     [B, k] fp32, device, best first.  ids [B, k] int64, device
 *            (naturally aligned).
 * workspace  >= lam_score_topk_workspace_size(...) bytes, device, 256-byte
 *            aligned.  Calls that share a workspace must not overlap.
 *
 * Asynchronous on `stream`.  Device-side faults of the data (a code beyond
 * code_bound) and bounded-wait timeouts are recorded in the workspace; read
 * them with lam_score_topk_status.  The environment variable LAM_SCORE_PATH
 * (auto|bandwidth|tensor|generic) forces one kernel path for testing; a
 * forced path that cannot take the shape returns LAM_ERR_UNSUPPORTED.
 */
lam_status lam_score_topk(const float *queries, int64_t B, const void *codes,
                          int32_t width, int64_t N, int32_t D, float eps,
                          int32_t code_bound, int32_t k, int32_t metric,
                          float *scores, int64_t *ids, void *workspace,
                          size_t workspace_bytes, lam_stream_t stream);

/*
 * Per-vector byte codecs of the composite-reduction experiment (Sec.
 * "Composite reduction", Table "composite": fp16, per-vector int8 and
 * sign-binary next to the error-bounded codec).  The paper names them with
 * their ratios only (3.96x and 30.72x over fp32 at D = 768); the library's
 * definitions, per row x of D values:
 *
 *   LAM_ROWS_INT8  lo = min x, hi = max x, scale = fl32((hi - lo) / 255),
 *                  c_d = rint_half_even(fl32(fl32(x_d - lo) / scale)) - 128
 *                  (-128 where scale = 0), offset = fl32(lo + 128 scale);
 *                  xhat_d = fl32(offset + fl32(scale c_d)).  Codes int8
 *                  [N, D], scale and offset fp32 [N]: D + 8 bytes a row.
 *   LAM_ROWS_FP16  c_d = fp16(x_d), round to nearest even; xhat_d = c_d.
 *                  Codes [N, D] binary16; scale and offset unused.
 *   LAM_ROWS_SIGN  bit d of row byte d/8 at position d % 8 is (x_d >= 0);
 *                  scale = alpha = fl32(sum_d |x_d| / D) with the sum in fp64
 *                  (the least-squares scale for the signs); xhat_d = alpha or
 *                  -alpha.  Codes uint8 [N, D/8] (D a multiple of 8), scale
 *                  fp32 [N]: D/8 + 4 bytes a row.
 *
 * The alpha of a row may differ by one fp32 ulp from a sum in another order
 * (the fp64 sum's own error is far below half an fp32 ulp); everything else
 * is exact.
 */
enum { LAM_ROWS_INT8 = 1, LAM_ROWS_FP16 = 2, LAM_ROWS_SIGN = 3 };

/*
 * lam_encode_rows -- x [N, D] fp32 (device, 4-byte aligned) into the codes
 * and per-row factors of `fmt` (layouts above; device buffers owned by the
 * caller, codes aligned to their element, scale/offset 4-byte aligned, NULL
 * where the codec has none).  Non-finite inputs give unspecified codes.
 * Asynchronous on `stream`.  Errors: LAM_ERR_INVALID, LAM_ERR_CUDA.
 *
 * lam_decode_rows -- the codes back to xhat [N, D] fp32 (device).
 * Asynchronous.  Errors: LAM_ERR_INVALID, LAM_ERR_CUDA.
 */
lam_status lam_encode_rows(const float *x, int64_t N, int32_t D, int32_t fmt, void *codes,
                           float *scale, float *offset, lam_stream_t stream);
lam_status lam_decode_rows(const void *codes, int32_t fmt, int64_t N, int32_t D,
                           const float *scale, const float *offset, float *out,
                           lam_stream_t stream);

/*
 * lam_score_topk_rows -- exact search over rows stored in a per-row codec:
 * the scores of lam_score_topk on the decoded rows xhat (inner product,
 * cosine with the norm of xhat, squared L2; same ordering and tie rule), with
 * the decoding folded into the score.  For int8 rows
 *   q . xhat = scale_i (q . c_i) + offset_i sum_d q_d,
 * so the codes enter the tensor-core product as they are stored.
 *
 * codes, scale, offset as written by lam_encode_rows for `fmt` (a 16-byte
 * aligned code base enables the bulk-copy and tensor-core paths: B <= 2 takes
 * the bandwidth kernel when D <= 1024, k <= 128 and a row is a multiple of 16
 * bytes, larger batches the tensor cores).  Other arguments, the workspace
 * rule, LAM_SCORE_PATH and the status read (lam_score_topk_status) as for
 * lam_score_topk.  Asynchronous.
 * Errors: LAM_ERR_INVALID, LAM_ERR_WORKSPACE, LAM_ERR_UNSUPPORTED,
 * LAM_ERR_CUDA.
 */
size_t lam_score_topk_rows_workspace_size(int64_t B, int64_t N, int32_t D, int32_t k,
                                          int32_t fmt);
int32_t lam_score_topk_rows_path(int64_t B, int64_t N, int32_t D, int32_t k, int32_t fmt);
lam_status lam_score_topk_rows(const float *queries, int64_t B, const void *codes, int32_t fmt,
                               const float *scale, const float *offset, int64_t N, int32_t D,
                               int32_t k, int32_t metric, float *scores, int64_t *ids,
                               void *workspace, size_t workspace_bytes, lam_stream_t stream);

/*
 * Waits for `stream`, then reads the device status the last lam_score_topk
 * on this workspace recorded: LAM_OK, LAM_ERR_RANGE, LAM_ERR_TIMEOUT, or
 * LAM_ERR_UNSUPPORTED when a lam_score_topk_from found an error or width 4 in
 * its quantize status (written to *status_out).  Returns LAM_ERR_CUDA if the
 * read fails.
 */
lam_status lam_score_topk_status(const void *workspace, lam_stream_t stream,
                                 int32_t *status_out);

/*
 * The kernel path lam_score_topk takes for a shape: 0 bandwidth (CUDA cores,
 * small batches), 1 tensor (tcgen05), 2 generic; -1 if the shape is invalid.
 */
int32_t lam_score_topk_path(int64_t B, int64_t N, int32_t D, int32_t k,
                            int32_t width, int32_t code_bound);

/*
 * lam_code_sqnorms -- sqnorm_out[i] = fl32(sum_d c_{i,d}^2) for each code row:
 * the exact integer sum, rounded once to fp32.  It is the per-row side array
 * an exact scan on codes can keep for cosine and squared L2 (Eq. 1 splits the
 * L2 distance into the two norms and the inner product); lam_score_topk
 * computes the same sums internally where it already reads the codes, so it
 * does not take this array.
 *
 * codes       [N, D] row-major device codes of `width` bytes (1 or 2),
 *             aligned to the width.
 * sqnorm_out  [N] device fp32, 4-byte aligned.
 * Asynchronous on `stream`.  Errors: LAM_ERR_INVALID (N < 0, D < 1, NULL or
 * misaligned pointers, width not 1 or 2), LAM_ERR_CUDA.
 */
lam_status lam_code_sqnorms(const void *codes, int32_t width, int64_t N, int32_t D,
                            float *sqnorm_out, lam_stream_t stream);

/*
 * Kernel timing (measurement support, not part of the method).
 *
 * lam_timing_begin(mask, capacity) makes the library bracket each launch of
 * the kernels selected by `mask` with a pair of CUDA events recorded on the
 * launching stream, for at most `capacity` launches in total, and count every
 * launch of its kernels by kind.  Kinds:
 *   LAM_TIME_QUANTIZE    the Q_eps kernel of lam_quantize
 *   LAM_TIME_DEQUANTIZE  the kernel of lam_dequantize
 *   LAM_TIME_SCORE       the fused score + top-k kernel of lam_score_topk
 *                        (one launch per row slab)
 *   LAM_TIME_AUX         every other kernel (query preparation, operand
 *                        conversion, range pass, admission)
 *   LAM_TIME_MERGE       the merge of partial top-k lists of lam_score_topk
 * The events are created here (no allocation happens later on the timed
 * path).  Intended for one host thread driving one device; a later begin
 * replaces the earlier state.  Errors: LAM_ERR_INVALID for mask outside
 * 1..31 or capacity outside 0..1048576; LAM_ERR_CUDA if event creation fails.
 *
 * lam_timing_read(kind, total_ms, timed, launches) waits for the recorded
 * events of one kind (a single bit of the mask) and returns the summed device
 * time of its bracketed launches, how many were bracketed, and how many were
 * launched since begin.  Any output pointer may be NULL.
 *
 * lam_timing_end() stops timing and destroys the events.
 */
#define LAM_TIME_QUANTIZE 1
#define LAM_TIME_DEQUANTIZE 2
#define LAM_TIME_SCORE 4
#define LAM_TIME_AUX 8
#define LAM_TIME_MERGE 16

lam_status lam_timing_begin(int32_t mask, int64_t capacity);
lam_status lam_timing_read(int32_t kind, double *total_ms, int64_t *timed,
                           int64_t *launches);
lam_status lam_timing_end(void);

/*
 * lam_score_topk_noalloc -- lam_score_topk for callers that cannot allocate
 * device memory.  (The paper has no counterpart: this is a packaging of the
 * same search.)
 *
 * Who needs it: a caller whose host framework owns all device memory through
 * its own pool and forbids allocations it did not make, or a latency-critical
 * caller that cannot afford cudaMalloc's implicit synchronisation, has no way
 * to provide the workspace lam_score_topk asks for.  This call takes the same
 * inputs and outputs (all caller-owned device buffers) but keeps its scratch
 * in a fixed 16 MiB array inside the library, which every GPU that loads the
 * library holds until the process exits.  It calls no cudaMalloc, cudaFree or
 * other allocating routine.
 *
 * Limits and behaviour:
 *   - Arguments, the path forced by LAM_SCORE_PATH and the shape are checked
 *     exactly as lam_score_topk checks them, with the same statuses
 *     (LAM_ERR_INVALID, LAM_ERR_UNSUPPORTED, LAM_ERR_CUDA).  Shapes whose
 *     search needs more than 16 MiB (16777216 bytes) of scratch return
 *     LAM_ERR_WORKSPACE; in every such case nothing is queued.
 *   - The scratch belongs to the current device: `stream` must be a stream of
 *     the current device (or NULL).
 *   - The array's device address is looked up (cudaGetSymbolAddress, with the
 *     device current) on the first call in each CUDA context on a device, and
 *     again after that context changed (e.g. cudaDeviceReset); make the first
 *     call on a device before any stream capture begins.
 *   - All calls share the one array, which keeps the last call's contents;
 *     the status word is cleared at the start of every call.  Calls that
 *     overlap on the GPU (other streams, other host threads) race on it and
 *     must be serialised by the caller.
 *   - Synchronous on `stream`: it waits for the search and returns the device
 *     status as its own return value: LAM_ERR_RANGE, LAM_ERR_TIMEOUT or
 *     LAM_ERR_UNSUPPORTED as lam_score_topk_status would report them.
 */
lam_status lam_score_topk_noalloc(const float *queries, int64_t B,
                                  const void *codes, int32_t width, int64_t N,
                                  int32_t D, float eps, int32_t code_bound,
                                  int32_t k, int32_t metric, float *scores,
                                  int64_t *ids, lam_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* LAM_H */
