// lam_api.cu -- the C ABI (include/lam.h): argument checks, planning of the
// scoring path and its workspace, and the launches.  The library allocates no
// device memory; its only state is a per-device cache of the SM count.
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <mutex>
#include <vector>

#include "lam_internal.cuh"

namespace {

using namespace lam;

int device_sms() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (dev >= 0 && dev < 64 && cache[dev] > 0) return cache[dev];
  int v = 0;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  if (dev >= 0 && dev < 64) cache[dev] = v;
  return v;
}

bool valid_width(int32_t w) { return w == 1 || w == 2 || w == 4; }

// eps finite, > 0, and s = 2 eps a normal fp32 number.
bool valid_eps(float eps) {
  if (!(eps > 0.0f) || !isfinite(eps)) return false;
  const float s = 2.0f * eps;
  return isfinite(s) && isnormal(s);
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Host replica of the device width resolution (same fp32 ops, half-to-even).
float host_qround(float x, float s) {
  const float q = x / s;
  return nearbyintf(q);
}

float unord_host(uint32_t o) {
  uint32_t b = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
  float f;
  memcpy(&f, &b, 4);
  return f;
}

int width_of(float rmin, float rmax) {
  if (rmin >= -128.0f && rmax <= 127.0f) return 1;
  if (rmin >= -32768.0f && rmax <= 32767.0f) return 2;
  if (rmin >= -2147483648.0f && rmax < 2147483648.0f) return 4;
  return 0;
}

struct Plan {
  int path = -1;
  int n_lists = 0;
  int64_t Bpad = 0;
  size_t partial_off = 0, qprep_off = 0, total = 0;
};

int forced_path() {
  const char *e = getenv("LAM_SCORE_PATH");
  if (e == nullptr || *e == 0 || strcmp(e, "auto") == 0) return -1;
  if (strcmp(e, "bandwidth") == 0) return kPathBandwidth;
  if (strcmp(e, "tensor") == 0) return kPathTensor;
  if (strcmp(e, "generic") == 0) return kPathGeneric;
  return -2;
}

bool shape_ok(int64_t B, int64_t N, int32_t D, int32_t k, int32_t width, int32_t code_bound) {
  return B >= 1 && B <= (1LL << 31) && N >= 1 && N < 2147483647LL && D >= 1 &&
         D <= (1 << 20) && k >= 1 && k <= kMaxK && k <= N && valid_width(width) &&
         code_bound >= 0 && (int64_t)N * D < (1LL << 46);
}

bool bandwidth_ok(int64_t B, int32_t D, int32_t k, int32_t width) {
  return B <= 2 && (width == 1 || width == 2) && D % 8 == 0 && (D * width) % 16 == 0 &&
         D <= 1024 && k <= 128;
}

// int8 codes and int16 codes within +-2048 are exact fp16 operands; other
// int16 codes take the split (256 h + l) through the converting pass.
bool tensor_ok(int64_t B, int64_t N, int32_t D, int32_t k, int32_t width, int32_t code_bound) {
  (void)N;
  if (width != 1 && width != 2) return false;
  const bool fits = tensor_wide(width, code_bound) ? tensor_fits_pre(k) : tensor_fits(width, k, B);
  return D % 16 == 0 && fits && B <= (1LL << 23);
}

TensorPlan tensor_plan_for(int64_t B, int64_t N, int32_t D, int32_t k, int32_t width,
                           int32_t code_bound, int sms) {
  return tensor_wide(width, code_bound) ? tensor_plan(B, N, tensor_k_extent(D, true), k, sms, true)
                                        : tensor_plan(B, N, D, k, sms);
}

// Test hooks, read from the environment at every search (unset in normal
// use): LAM_TEST_WAIT_CYCLES=<n> gives the search's device waits a budget of
// n SM cycles instead of ~1 s and LAM_TEST_STALL=1 makes its copy producers
// issue nothing, so that every consumer's wait runs out (the timeout path);
// LAM_TEST_HI_FAIL=1 makes the certifying merge of a two-pass tensor search
// reject every query, so that the gated full pass runs.
}  // namespace

namespace lam {
__global__ void set_test_words_kernel(uint32_t *hdr, uint32_t wait_cycles, uint32_t stall,
                                      uint32_t force_fail) {
  hdr[kHdrWaitCycles] = wait_cycles;
  hdr[kHdrStall] = stall;
  hdr[kHdrForceFail] = force_fail;
}
}  // namespace lam

namespace {

// LAM_DEBUG=1: the CUDA error behind a LAM_ERR_CUDA, on stderr.
void debug_report(const char *where, cudaError_t e) {
  const char *d = getenv("LAM_DEBUG");
  if (d != nullptr && strcmp(d, "1") == 0)
    fprintf(stderr, "%s: %s (%d)\n", where, cudaGetErrorString(e), (int)e);
}

cudaError_t apply_test_hooks(void *ws, cudaStream_t st) {
  const char *w = getenv("LAM_TEST_WAIT_CYCLES");
  const char *z = getenv("LAM_TEST_STALL");
  const char *f = getenv("LAM_TEST_HI_FAIL");
  const uint32_t wait_cycles = (w && *w) ? (uint32_t)strtoul(w, nullptr, 10) : 0u;
  const uint32_t stall = (z && strcmp(z, "1") == 0) ? 1u : 0u;
  const uint32_t force_fail = (f && strcmp(f, "1") == 0) ? 1u : 0u;
  if (wait_cycles == 0 && stall == 0 && force_fail == 0) return cudaSuccess;
  set_test_words_kernel<<<1, 1, 0, st>>>(static_cast<uint32_t *>(ws), wait_cycles, stall,
                                         force_fail);
  return cudaGetLastError();
}

// Chooses the path (or honours LAM_SCORE_PATH) and lays out the workspace:
// [status 256 B][partial lists n_lists x B x k keys][tensor: query prep].
bool make_plan(int64_t B, int64_t N, int32_t D, int32_t k, int32_t width, int32_t code_bound,
               int sms, Plan *p) {
  if (!shape_ok(B, N, D, k, width, code_bound) || sms <= 0) return false;
  const bool bw = bandwidth_ok(B, D, k, width);
  const bool tc = tensor_ok(B, N, D, k, width, code_bound);
  const int f = forced_path();
  if (f == -2) return false;
  int path;
  if (f >= 0) {
    if ((f == kPathBandwidth && !bw) || (f == kPathTensor && !tc)) {
      p->path = -2;
      return false;
    }
    path = f;
  } else if (bw) {
    path = kPathBandwidth;
  } else if (tc) {
    path = kPathTensor;
  } else {
    path = kPathGeneric;
  }
  p->path = path;
  if (path == kPathBandwidth) p->n_lists = bandwidth_ctas(N, D, width, sms);
  else if (path == kPathTensor)
    p->n_lists = tensor_plan_for(B, N, D, k, width, code_bound, sms).n_lists;
  else p->n_lists = generic_ctas(B, N, sms);
  p->Bpad = (B + 127) / 128 * 128;
  p->partial_off = kHeaderBytes;
  // (a two-pass tensor search keeps hi_list(k) candidates per list)
  const int kl = path == kPathTensor && tensor_hi(B, N, D, k, width, code_bound, sms)
                     ? hi_list(k) : k;
  const size_t partial = (size_t)p->n_lists * (size_t)B * (size_t)kl * 8;
  p->qprep_off = align_up(p->partial_off + partial, 256);
  p->total = p->qprep_off;
  if (path == kPathTensor)
    p->total += align_up(tensor_plan_for(B, N, D, k, width, code_bound, sms).bytes, 256);
  return true;
}

// Status-driven search (codes' width on the device, 1 or 2): the path cannot
// depend on the width, so each test holds for both.
bool make_from_plan(int64_t B, int64_t N, int32_t D, int32_t k, int sms, Plan *p) {
  if (!shape_ok(B, N, D, k, 2, 0) || sms <= 0) return false;
  const bool bw = bandwidth_ok(B, D, k, 1) && bandwidth_ok(B, D, k, 2);
  const bool tc = D % 16 == 0 && tensor_fits(1, k, B) && tensor_fits(2, k, B) &&
                  B <= (1LL << 23);
  const int f = forced_path();
  if (f == -2) return false;
  int path = bw ? kPathBandwidth : tc ? kPathTensor : kPathGeneric;
  if (f >= 0) {
    if ((f == kPathBandwidth && !bw) || (f == kPathTensor && !tc)) {
      p->path = -2;
      return false;
    }
    path = f;
  }
  p->path = path;
  p->n_lists = path == kPathBandwidth ? bandwidth_ctas(N, D, 2, sms)
               : path == kPathTensor  ? tensor_plan(B, N, D, k, sms).n_lists
                                      : generic_ctas(B, N, sms);
  p->Bpad = (B + 127) / 128 * 128;
  p->partial_off = kHeaderBytes;
  const size_t partial = (size_t)p->n_lists * (size_t)B * (size_t)k * 8;
  p->qprep_off = align_up(p->partial_off + partial, 256);
  p->total = p->qprep_off;
  if (path == kPathTensor) p->total += align_up(tensor_plan(B, N, D, k, sms).bytes, 256);
  return true;
}

// Per-row codecs: shape checks and the plan (tensor path with the converting
// pass, else the generic path; no bandwidth kernel).
bool rows_shape_ok(int64_t B, int64_t N, int32_t D, int32_t k, int32_t fmt) {
  if (fmt != LAM_ROWS_INT8 && fmt != LAM_ROWS_FP16 && fmt != LAM_ROWS_SIGN) return false;
  if (fmt == LAM_ROWS_SIGN && D % 8 != 0) return false;
  return shape_ok(B, N, D, k, 1, 0);
}

bool make_rows_plan(int64_t B, int64_t N, int32_t D, int32_t k, int32_t fmt, int sms, Plan *p) {
  if (!rows_shape_ok(B, N, D, k, fmt) || sms <= 0) return false;
  const bool tc = D % 16 == 0 && tensor_fits_pre(k) && B <= (1LL << 23);
  const int row_bytes = fmt == LAM_ROWS_INT8 ? D : fmt == LAM_ROWS_FP16 ? 2 * D : D / 8;
  const bool bw = B <= 2 && k <= 128 && D <= 1024 && D % 8 == 0 && row_bytes % 16 == 0;
  const int f = forced_path();
  if (f == -2) return false;
  int path = bw ? kPathBandwidth : tc ? kPathTensor : kPathGeneric;
  if (f >= 0) {
    if ((f == kPathBandwidth && !bw) || (f == kPathTensor && !tc)) {
      p->path = -2;
      return false;
    }
    path = f;
  }
  p->path = path;
  p->n_lists = path == kPathTensor      ? tensor_plan(B, N, D, k, sms, true).n_lists
               : path == kPathBandwidth ? bandwidth_rows_ctas(N, fmt, D, sms)
                                        : generic_ctas(B, N, sms);
  p->Bpad = (B + 127) / 128 * 128;
  p->partial_off = kHeaderBytes;
  const size_t partial = (size_t)p->n_lists * (size_t)B * (size_t)k * 8;
  p->qprep_off = align_up(p->partial_off + partial, 256);
  p->total = p->qprep_off;
  if (path == kPathTensor) p->total += align_up(tensor_plan(B, N, D, k, sms, true).bytes, 256);
  return true;
}

}  // namespace

namespace lam {

cudaError_t read_back(void *dst, const void *src, size_t n, cudaStream_t st) {
  cudaError_t e = cudaMemcpyAsync(dst, src, n, cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  return e;
}

namespace {

// Event pairs around selected kernel launches (lam_timing_*).
struct Timing {
  std::mutex mu;
  int mask = 0;
  std::vector<cudaEvent_t> ev;  // 2 per bracketed launch
  std::vector<int> kind;        // kind of each bracketed launch
  int64_t cap = 0, used = 0;
  int64_t launches[5] = {0, 0, 0, 0, 0};
  bool open = false;  // a begin without its end
};
Timing g_timing;

int kind_index(int kind) {
  return kind == LAM_TIME_QUANTIZE ? 0 : kind == LAM_TIME_DEQUANTIZE ? 1
         : kind == LAM_TIME_SCORE  ? 2 : kind == LAM_TIME_MERGE ? 4 : 3;
}

void timing_release() {
  for (cudaEvent_t e : g_timing.ev) cudaEventDestroy(e);
  g_timing.ev.clear();
  g_timing.kind.clear();
  g_timing.cap = g_timing.used = 0;
  g_timing.mask = 0;
  g_timing.open = false;
  for (int64_t &c : g_timing.launches) c = 0;
}

}  // namespace

void timing_launch_begin(int kind, cudaStream_t st) {
  std::lock_guard<std::mutex> lk(g_timing.mu);
  if (g_timing.mask == 0) return;
  ++g_timing.launches[kind_index(kind)];
  if (!(g_timing.mask & kind) || g_timing.used >= g_timing.cap) return;
  cudaEventRecord(g_timing.ev[2 * g_timing.used], st);
  g_timing.open = true;
}

void timing_launch_end(int kind, cudaStream_t st) {
  std::lock_guard<std::mutex> lk(g_timing.mu);
  if (!g_timing.open || !(g_timing.mask & kind)) return;
  cudaEventRecord(g_timing.ev[2 * g_timing.used + 1], st);
  g_timing.kind.push_back(kind);
  ++g_timing.used;
  g_timing.open = false;
}

}  // namespace lam

namespace lam {
namespace {
// Host outputs and status of a finished Q_eps pass from its status block.
lam_status decode_quant_status(const QuantStatus &h, int32_t width_req, float s,
                               int32_t *width_out, float *scale_out, int32_t *code_min_out,
                               int32_t *code_max_out) {
  if (h.flags & kFlagTimeout) return LAM_ERR_TIMEOUT;
  if (h.flags & kFlagNonfinite) return LAM_ERR_NONFINITE;
  float rmin = 0.0f, rmax = 0.0f;
  if (h.neg_min != 0) {
    rmin = host_qround(unord_host(~h.neg_min), s);
    rmax = host_qround(unord_host(h.max), s);
  }
  const int need = width_of(rmin, rmax);
  const int w = width_req == LAM_WIDTH_AUTO ? need : width_req;
  if (scale_out) *scale_out = s;
  if (width_out) *width_out = w;
  if (need != 0) {
    if (code_min_out) *code_min_out = (int32_t)rmin;
    if (code_max_out) *code_max_out = (int32_t)rmax;
  } else {
    if (code_min_out) *code_min_out = rmin < -2147483648.0f ? INT32_MIN : (int32_t)rmin;
    if (code_max_out) *code_max_out = rmax >= 2147483648.0f ? INT32_MAX : (int32_t)rmax;
  }
  if (need == 0 || (h.flags & kFlagRange)) return LAM_ERR_RANGE;
  if (width_req != LAM_WIDTH_AUTO && need > width_req) return LAM_ERR_RANGE;
  if (width_req == LAM_WIDTH_AUTO && (int)h.width != need) return LAM_ERR_CUDA;  // must agree
  if (h.flags & kFlagWorkspace) return LAM_ERR_WORKSPACE;
  return LAM_OK;
}

}  // namespace
}  // namespace lam

extern "C" {

int32_t lam_version(void) { return 100; }

const char *lam_status_string(int32_t status) {
  switch (status) {
    case LAM_OK: return "ok";
    case LAM_ERR_INVALID: return "invalid argument";
    case LAM_ERR_RANGE: return "codes out of range for the width";
    case LAM_ERR_NONFINITE: return "non-finite input";
    case LAM_ERR_WORKSPACE: return "buffer or workspace too small";
    case LAM_ERR_CUDA: return "CUDA error";
    case LAM_ERR_TIMEOUT: return "device wait timed out";
    case LAM_ERR_UNSUPPORTED: return "forced kernel path cannot take this shape";
    default: return "unknown status";
  }
}

size_t lam_quantize_workspace_size(void) { return sizeof(QuantStatus); }

lam_status lam_quantize(const float *x, int64_t n, float eps, int32_t width_req, void *codes,
                        size_t codes_bytes, void *workspace, size_t workspace_bytes,
                        int32_t *width_out, float *scale_out, int32_t *code_min_out,
                        int32_t *code_max_out, lam_stream_t stream) {
  if (n < 0 || n >= (1LL << 62) || !valid_eps(eps)) return LAM_ERR_INVALID;
  if (width_req != LAM_WIDTH_AUTO && !valid_width(width_req)) return LAM_ERR_INVALID;
  if (n > 0 && x == nullptr) return LAM_ERR_INVALID;
  // natural alignment: fp32 input; codes aligned to their width (AUTO: 4 bytes)
  if ((reinterpret_cast<uintptr_t>(x) & 3u) != 0) return LAM_ERR_INVALID;
  const uintptr_t calign = width_req == LAM_WIDTH_AUTO ? 4u : (uintptr_t)width_req;
  if (codes != nullptr && (reinterpret_cast<uintptr_t>(codes) & (calign - 1)) != 0)
    return LAM_ERR_INVALID;
  const float s = 2.0f * eps;
  if (n == 0) {
    if (width_out) *width_out = width_req == LAM_WIDTH_AUTO ? 1 : width_req;
    if (scale_out) *scale_out = s;
    if (code_min_out) *code_min_out = 0;
    if (code_max_out) *code_max_out = 0;
    return LAM_OK;
  }
  if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) & 15u) != 0)
    return LAM_ERR_INVALID;
  if (workspace_bytes < sizeof(QuantStatus)) return LAM_ERR_WORKSPACE;
  if (codes != nullptr && width_req != LAM_WIDTH_AUTO &&
      (unsigned long long)n * (unsigned long long)width_req > codes_bytes)
    return LAM_ERR_WORKSPACE;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  QuantStatus *dst = static_cast<QuantStatus *>(workspace);
  if (cudaMemsetAsync(dst, 0, sizeof(QuantStatus), st) != cudaSuccess) return LAM_ERR_CUDA;
  cudaError_t e = cudaSuccess;
  const int tkind = (width_req == LAM_WIDTH_AUTO || codes != nullptr) ? LAM_TIME_QUANTIZE
                                                                       : LAM_TIME_AUX;
  timing_launch_begin(tkind, st);
  if (width_req == LAM_WIDTH_AUTO) {
    e = launch_quantize_auto(x, n, s, codes, codes_bytes, dst, sms, st);
  } else if (codes != nullptr) {
    e = launch_quantize(x, n, s, width_req, codes, codes_bytes, dst, sms, st);
  } else {
    e = launch_quant_range(x, n, dst, sms, st);
  }
  timing_launch_end(tkind, st);
  if (e != cudaSuccess) return LAM_ERR_CUDA;
  QuantStatus h;
  if (read_back(&h, dst, sizeof(h), st) != cudaSuccess) return LAM_ERR_CUDA;
  if (width_req == LAM_WIDTH_AUTO && codes != nullptr && h.passes == 2 &&
      !(h.flags & (kFlagTimeout | kFlagNonfinite | kFlagRange | kFlagWorkspace)) &&
      (h.width == 1 || h.width == 2 || h.width == 4)) {
    // the width speculated from the sample was too narrow: quantize again
    timing_launch_begin(LAM_TIME_QUANTIZE, st);
    e = launch_quantize(x, n, s, (int)h.width, codes, codes_bytes, dst, sms, st);
    timing_launch_end(LAM_TIME_QUANTIZE, st);
    if (e != cudaSuccess) return LAM_ERR_CUDA;
    const uint32_t width_resolved = h.width;
    if (read_back(&h, dst, sizeof(h), st) != cudaSuccess) return LAM_ERR_CUDA;
    h.width = width_resolved;
  }
  return lam::decode_quant_status(h, width_req, s, width_out, scale_out, code_min_out,
                                  code_max_out);
}

lam_status lam_quantize_bands(const float *x, int64_t N, int32_t D, float eps, int32_t width_req,
                              int32_t r, void *codes, size_t codes_bytes, uint64_t *digests,
                              void *workspace, size_t workspace_bytes, int32_t *width_out,
                              float *scale_out, int32_t *code_min_out, int32_t *code_max_out,
                              lam_stream_t stream) {
  if (N < 0 || D < 1 || r < 1 || r > D || D % r != 0 || D / r > 65536 || !valid_eps(eps))
    return LAM_ERR_INVALID;
  if (N > (1LL << 62) / D) return LAM_ERR_INVALID;
  if (width_req != LAM_WIDTH_AUTO && !valid_width(width_req)) return LAM_ERR_INVALID;
  const int64_t n = N * (int64_t)D;
  if (n > 0 && (x == nullptr || digests == nullptr)) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(x) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(digests) & 7u) != 0)
    return LAM_ERR_INVALID;
  const uintptr_t calign = width_req == LAM_WIDTH_AUTO ? 4u : (uintptr_t)width_req;
  if (codes != nullptr && (reinterpret_cast<uintptr_t>(codes) & (calign - 1)) != 0)
    return LAM_ERR_INVALID;
  const float s = 2.0f * eps;
  if (n == 0) {
    if (width_out) *width_out = width_req == LAM_WIDTH_AUTO ? 1 : width_req;
    if (scale_out) *scale_out = s;
    if (code_min_out) *code_min_out = 0;
    if (code_max_out) *code_max_out = 0;
    return LAM_OK;
  }
  if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) & 15u) != 0)
    return LAM_ERR_INVALID;
  if (workspace_bytes < sizeof(QuantStatus)) return LAM_ERR_WORKSPACE;
  if (codes != nullptr && width_req != LAM_WIDTH_AUTO &&
      (unsigned long long)n * (unsigned long long)width_req > codes_bytes)
    return LAM_ERR_WORKSPACE;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  QuantStatus *dst = static_cast<QuantStatus *>(workspace);
  if (cudaMemsetAsync(dst, 0, sizeof(QuantStatus), st) != cudaSuccess) return LAM_ERR_CUDA;
  timing_launch_begin(LAM_TIME_QUANTIZE, st);
  cudaError_t e = launch_quantize_bands(x, N, D, r, s, width_req, codes, codes_bytes, digests,
                                        dst, sms, st);
  timing_launch_end(LAM_TIME_QUANTIZE, st);
  if (e != cudaSuccess) return LAM_ERR_CUDA;
  QuantStatus h;
  if (read_back(&h, dst, sizeof(h), st) != cudaSuccess) return LAM_ERR_CUDA;
  if (width_req == LAM_WIDTH_AUTO && h.passes == 2 &&
      !(h.flags & (kFlagTimeout | kFlagNonfinite | kFlagRange | kFlagWorkspace)) &&
      (h.width == 1 || h.width == 2 || h.width == 4)) {
    // the width speculated from the sample was too narrow: hash again at the exact one
    timing_launch_begin(LAM_TIME_QUANTIZE, st);
    e = launch_quantize_bands(x, N, D, r, s, (int)h.width, codes, codes_bytes, digests, dst, sms,
                              st);
    timing_launch_end(LAM_TIME_QUANTIZE, st);
    if (e != cudaSuccess) return LAM_ERR_CUDA;
    const uint32_t width_resolved = h.width;
    if (read_back(&h, dst, sizeof(h), st) != cudaSuccess) return LAM_ERR_CUDA;
    h.width = width_resolved;
  }
  return lam::decode_quant_status(h, width_req, s, width_out, scale_out, code_min_out,
                                  code_max_out);
}

size_t lam_admit_batch_workspace_size(int64_t N, int32_t nb, int64_t max_pairs) {
  if (N < 0 || N > INT32_MAX || nb < 1 || max_pairs < 0 || max_pairs > INT32_MAX ||
      (N * (int64_t)nb) > (int64_t)UINT32_MAX)
    return 0;
  return admit_workspace_bytes(N, nb, max_pairs);
}

lam_status lam_admit_batch(const float *e, int64_t N, int32_t D, const uint64_t *digests,
                           int32_t nb, double delta, int32_t *rep, double *dist,
                           void *workspace, size_t workspace_bytes, int64_t max_pairs,
                           double *delta_hat_out, int64_t *n_retained_out,
                           int64_t *n_pairs_out, lam_stream_t stream) {
  if (N < 0 || N > INT32_MAX || D < 1 || nb < 1 || max_pairs < 0 || max_pairs > INT32_MAX ||
      !(delta >= 0.0) || !isfinite(delta) || (N * (int64_t)nb) > (int64_t)UINT32_MAX)
    return LAM_ERR_INVALID;
  if (n_pairs_out) *n_pairs_out = 0;
  if (N == 0) {
    if (delta_hat_out) *delta_hat_out = 0.0;
    if (n_retained_out) *n_retained_out = 0;
    return LAM_OK;
  }
  if (e == nullptr || digests == nullptr || rep == nullptr || dist == nullptr ||
      workspace == nullptr)
    return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(e) & 3u) || (reinterpret_cast<uintptr_t>(digests) & 7u) ||
      (reinterpret_cast<uintptr_t>(rep) & 3u) || (reinterpret_cast<uintptr_t>(dist) & 7u) ||
      (reinterpret_cast<uintptr_t>(workspace) & 255u))
    return LAM_ERR_INVALID;
  if (workspace_bytes < admit_workspace_bytes(N, nb, max_pairs)) return LAM_ERR_WORKSPACE;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int64_t np = 0, kept = 0;
  double dh = 0.0;
  bool overflow = false;
  timing_launch_begin(LAM_TIME_AUX, st);
  const cudaError_t err = launch_admit_batch(e, N, D, digests, nb, delta, rep, dist, workspace,
                                             max_pairs, sms, st, &np, &dh, &kept, &overflow);
  timing_launch_end(LAM_TIME_AUX, st);
  if (err != cudaSuccess) return LAM_ERR_CUDA;
  if (n_pairs_out) *n_pairs_out = np;
  if (overflow) return LAM_ERR_WORKSPACE;
  if (delta_hat_out) *delta_hat_out = dh;
  if (n_retained_out) *n_retained_out = kept;
  return LAM_OK;
}

size_t lam_lamz_bound(int64_t n) { return n < 0 ? 0 : lamz_bound_bytes(n); }

size_t lam_lamz_workspace_size(int64_t n) { return n < 0 ? 0 : lamz_workspace_bytes(n); }

lam_status lam_lamz_compress(const float *x, int64_t n, float rel, void *out, size_t out_capacity,
                             size_t *out_bytes, void *workspace, size_t workspace_bytes,
                             lam_stream_t stream) {
  if (n < 0 || n > (1LL << 40) || !(rel >= 1e-6f) || !(rel <= 1.0f)) return LAM_ERR_INVALID;
  if (n > 0 && (x == nullptr || out == nullptr || workspace == nullptr)) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(x) & 3u) || (reinterpret_cast<uintptr_t>(out) & 3u) ||
      (reinterpret_cast<uintptr_t>(workspace) & 255u))
    return LAM_ERR_INVALID;
  if (workspace_bytes < lamz_workspace_bytes(n)) return LAM_ERR_WORKSPACE;
  if (out_capacity < lamz_head_bytes(n)) {
    if (out_bytes) *out_bytes = lamz_head_bytes(n);
    return LAM_ERR_WORKSPACE;
  }
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  size_t bytes = 0;
  bool fits = false, nonfinite = false, timed_out = false;
  timing_launch_begin(LAM_TIME_AUX, st);
  const cudaError_t e = launch_lamz_compress(x, n, rel, static_cast<uint8_t *>(out), out_capacity,
                                             workspace, sms, st, &bytes, &fits, &nonfinite,
                                             &timed_out);
  timing_launch_end(LAM_TIME_AUX, st);
  if (e != cudaSuccess) return LAM_ERR_CUDA;
  if (out_bytes) *out_bytes = bytes;
  if (nonfinite) return LAM_ERR_NONFINITE;
  if (timed_out) return LAM_ERR_TIMEOUT;
  return fits ? LAM_OK : LAM_ERR_WORKSPACE;
}

lam_status lam_lamz_decompress(const void *in, size_t in_bytes, float *out, int64_t n,
                               void *workspace, size_t workspace_bytes, lam_stream_t stream) {
  if (n < 0 || n > (1LL << 40)) return LAM_ERR_INVALID;
  if (n > 0 && (in == nullptr || out == nullptr || workspace == nullptr)) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(in) & 3u) || (reinterpret_cast<uintptr_t>(out) & 3u) ||
      (reinterpret_cast<uintptr_t>(workspace) & 255u))
    return LAM_ERR_INVALID;
  if (workspace_bytes < lamz_workspace_bytes(n)) return LAM_ERR_WORKSPACE;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  bool bad = true;
  timing_launch_begin(LAM_TIME_AUX, st);
  const cudaError_t e = launch_lamz_decompress(static_cast<const uint8_t *>(in), in_bytes, out, n,
                                               workspace, sms, st, &bad);
  timing_launch_end(LAM_TIME_AUX, st);
  if (e != cudaSuccess) return LAM_ERR_CUDA;
  return bad ? LAM_ERR_INVALID : LAM_OK;
}

lam_status lam_dequantize(const void *codes, int32_t width, int64_t n, float scale, float *out,
                          lam_stream_t stream) {
  if (n < 0 || !valid_width(width) || !isfinite(scale)) return LAM_ERR_INVALID;
  if (n == 0) return LAM_OK;
  if (codes == nullptr || out == nullptr) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(codes) & (uintptr_t)(width - 1)) != 0 ||
      (reinterpret_cast<uintptr_t>(out) & 3u) != 0)
    return LAM_ERR_INVALID;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  timing_launch_begin(LAM_TIME_DEQUANTIZE, st);
  const cudaError_t e = launch_dequantize(codes, width, n, scale, out, sms, st);
  timing_launch_end(LAM_TIME_DEQUANTIZE, st);
  return e == cudaSuccess ? LAM_OK : LAM_ERR_CUDA;
}

lam_status lam_code_sqnorms(const void *codes, int32_t width, int64_t N, int32_t D,
                            float *sqnorm_out, lam_stream_t stream) {
  if (N < 0 || D < 1 || (width != 1 && width != 2)) return LAM_ERR_INVALID;
  if (N == 0) return LAM_OK;
  if (codes == nullptr || sqnorm_out == nullptr) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(codes) & (uintptr_t)(width - 1)) != 0 ||
      (reinterpret_cast<uintptr_t>(sqnorm_out) & 3u) != 0)
    return LAM_ERR_INVALID;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  timing_launch_begin(LAM_TIME_AUX, st);
  const cudaError_t e = launch_code_sqnorms(codes, width, N, D, sqnorm_out, sms, st);
  timing_launch_end(LAM_TIME_AUX, st);
  return e == cudaSuccess ? LAM_OK : LAM_ERR_CUDA;
}

size_t lam_score_topk_workspace_size(int64_t B, int64_t N, int32_t D, int32_t k, int32_t width,
                                     int32_t code_bound) {
  Plan p;
  const int sms = device_sms();
  if (!make_plan(B, N, D, k, width, code_bound, sms, &p)) return 0;
  // misaligned codes fall back to the generic path at call time
  const size_t generic = align_up(kHeaderBytes + (size_t)generic_ctas(B, N, sms) * B * k * 8, 256);
  return p.total > generic ? p.total : generic;
}

int32_t lam_score_topk_path(int64_t B, int64_t N, int32_t D, int32_t k, int32_t width,
                            int32_t code_bound) {
  Plan p;
  if (!make_plan(B, N, D, k, width, code_bound, device_sms(), &p)) return -1;
  return p.path;
}

lam_status lam_score_topk(const float *queries, int64_t B, const void *codes, int32_t width,
                          int64_t N, int32_t D, float eps, int32_t code_bound, int32_t k,
                          int32_t metric, float *scores, int64_t *ids, void *workspace,
                          size_t workspace_bytes, lam_stream_t stream) {
  if (queries == nullptr || codes == nullptr || scores == nullptr || ids == nullptr ||
      workspace == nullptr)
    return LAM_ERR_INVALID;
  if (metric != LAM_METRIC_IP && metric != LAM_METRIC_COSINE && metric != LAM_METRIC_L2)
    return LAM_ERR_INVALID;
  if (!valid_eps(eps)) return LAM_ERR_INVALID;
  if (!shape_ok(B, N, D, k, width, code_bound)) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(codes) & (uintptr_t)(width - 1)) != 0 ||
      (reinterpret_cast<uintptr_t>(queries) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(scores) & 3u) != 0 || (reinterpret_cast<uintptr_t>(ids) & 7u) != 0)
    return LAM_ERR_INVALID;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  Plan p;
  if (!make_plan(B, N, D, k, width, code_bound, sms, &p))
    return p.path == -2 ? LAM_ERR_UNSUPPORTED : LAM_ERR_INVALID;
  // TMA and bulk copies need a 16-byte aligned code base
  const bool aligned = (reinterpret_cast<uintptr_t>(codes) & 15u) == 0;
  if (!aligned && p.path != kPathGeneric) {
    if (forced_path() >= 0) return LAM_ERR_UNSUPPORTED;
    p.path = kPathGeneric;
    p.n_lists = generic_ctas(B, N, sms);
    p.qprep_off = align_up(p.partial_off + (size_t)p.n_lists * B * k * 8, 256);
    p.total = p.qprep_off;
  }
  if (workspace_bytes < p.total) return LAM_ERR_WORKSPACE;

  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  if (cudaMemsetAsync(ws, 0, kHeaderBytes, st) != cudaSuccess) return LAM_ERR_CUDA;
  if (apply_test_hooks(ws, st) != cudaSuccess) return LAM_ERR_CUDA;
  ScoreArgs a;
  a.queries = queries;
  a.B = B;
  a.codes = codes;
  a.width = width;
  a.N = N;
  a.D = D;
  a.s = 2.0f * eps;
  a.code_bound = code_bound;
  a.k = k;
  a.metric = metric;
  a.scores = scores;
  a.ids = ids;
  a.gflags = reinterpret_cast<uint32_t *>(ws);
  a.partial = reinterpret_cast<uint64_t *>(ws + p.partial_off);
  a.n_lists = p.n_lists;
  a.qprep = ws + p.qprep_off;
  a.Bpad = p.Bpad;
  a.sms = sms;
  cudaError_t e;
  ScoreArgs m = a;  // the final merge's lists
  int merge_mode = 0;
  if (p.path == kPathBandwidth) e = launch_score_bandwidth(a, st);
  else if (p.path == kPathTensor) e = launch_score_tensor(a, st, RowPtrs(), &m, &merge_mode);
  else e = launch_score_generic(a, st);
  if (e == cudaSuccess) e = launch_topk_merge(m, st, RowPtrs(), merge_mode);
  if (e != cudaSuccess) {
    debug_report("lam_score_topk", e);
    return LAM_ERR_CUDA;
  }
  return LAM_OK;
}

lam_status lam_encode_rows(const float *x, int64_t N, int32_t D, int32_t fmt, void *codes,
                           float *scale, float *offset, lam_stream_t stream) {
  if (N < 0 || D < 1 || D > (1 << 20)) return LAM_ERR_INVALID;
  if (fmt != LAM_ROWS_INT8 && fmt != LAM_ROWS_FP16 && fmt != LAM_ROWS_SIGN) return LAM_ERR_INVALID;
  if (fmt == LAM_ROWS_SIGN && D % 8 != 0) return LAM_ERR_INVALID;
  if (N >= (1LL << 40) / D) return LAM_ERR_INVALID;
  if (N == 0) return LAM_OK;
  if (x == nullptr || codes == nullptr) return LAM_ERR_INVALID;
  if (fmt != LAM_ROWS_FP16 && scale == nullptr) return LAM_ERR_INVALID;
  if (fmt == LAM_ROWS_INT8 && offset == nullptr) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(x) & 3u) != 0 ||
      (fmt == LAM_ROWS_FP16 && (reinterpret_cast<uintptr_t>(codes) & 1u) != 0) ||
      (reinterpret_cast<uintptr_t>(scale) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(offset) & 3u) != 0)
    return LAM_ERR_INVALID;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  timing_launch_begin(LAM_TIME_QUANTIZE, st);
  const cudaError_t e = launch_encode_rows(x, N, D, fmt, codes, scale, offset, sms, st);
  timing_launch_end(LAM_TIME_QUANTIZE, st);
  return e == cudaSuccess ? LAM_OK : LAM_ERR_CUDA;
}

lam_status lam_decode_rows(const void *codes, int32_t fmt, int64_t N, int32_t D,
                           const float *scale, const float *offset, float *out,
                           lam_stream_t stream) {
  if (N < 0 || D < 1 || D > (1 << 20)) return LAM_ERR_INVALID;
  if (fmt != LAM_ROWS_INT8 && fmt != LAM_ROWS_FP16 && fmt != LAM_ROWS_SIGN) return LAM_ERR_INVALID;
  if (fmt == LAM_ROWS_SIGN && D % 8 != 0) return LAM_ERR_INVALID;
  if (N >= (1LL << 40) / D) return LAM_ERR_INVALID;
  if (N == 0) return LAM_OK;
  if (codes == nullptr || out == nullptr) return LAM_ERR_INVALID;
  if (fmt != LAM_ROWS_FP16 && scale == nullptr) return LAM_ERR_INVALID;
  if (fmt == LAM_ROWS_INT8 && offset == nullptr) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(out) & 3u) != 0 ||
      (fmt == LAM_ROWS_FP16 && (reinterpret_cast<uintptr_t>(codes) & 1u) != 0) ||
      (reinterpret_cast<uintptr_t>(scale) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(offset) & 3u) != 0)
    return LAM_ERR_INVALID;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  timing_launch_begin(LAM_TIME_DEQUANTIZE, st);
  const cudaError_t e = launch_decode_rows(codes, fmt, N, D, scale, offset, out, sms, st);
  timing_launch_end(LAM_TIME_DEQUANTIZE, st);
  return e == cudaSuccess ? LAM_OK : LAM_ERR_CUDA;
}

size_t lam_score_topk_rows_workspace_size(int64_t B, int64_t N, int32_t D, int32_t k,
                                          int32_t fmt) {
  Plan p;
  const int sms = device_sms();
  if (!make_rows_plan(B, N, D, k, fmt, sms, &p)) return 0;
  const size_t generic = align_up(kHeaderBytes + (size_t)generic_ctas(B, N, sms) * B * k * 8, 256);
  return p.total > generic ? p.total : generic;
}

int32_t lam_score_topk_rows_path(int64_t B, int64_t N, int32_t D, int32_t k, int32_t fmt) {
  Plan p;
  if (!make_rows_plan(B, N, D, k, fmt, device_sms(), &p)) return -1;
  return p.path;
}

lam_status lam_score_topk_rows(const float *queries, int64_t B, const void *codes, int32_t fmt,
                               const float *scale, const float *offset, int64_t N, int32_t D,
                               int32_t k, int32_t metric, float *scores, int64_t *ids,
                               void *workspace, size_t workspace_bytes, lam_stream_t stream) {
  if (queries == nullptr || codes == nullptr || scores == nullptr || ids == nullptr ||
      workspace == nullptr)
    return LAM_ERR_INVALID;
  if (metric != LAM_METRIC_IP && metric != LAM_METRIC_COSINE && metric != LAM_METRIC_L2)
    return LAM_ERR_INVALID;
  if (!rows_shape_ok(B, N, D, k, fmt)) return LAM_ERR_INVALID;
  if (fmt != LAM_ROWS_FP16 && scale == nullptr) return LAM_ERR_INVALID;
  if (fmt == LAM_ROWS_INT8 && offset == nullptr) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return LAM_ERR_INVALID;
  if ((fmt == LAM_ROWS_FP16 && (reinterpret_cast<uintptr_t>(codes) & 1u) != 0) ||
      (reinterpret_cast<uintptr_t>(scale) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(offset) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(queries) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(scores) & 3u) != 0 || (reinterpret_cast<uintptr_t>(ids) & 7u) != 0)
    return LAM_ERR_INVALID;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  Plan p;
  if (!make_rows_plan(B, N, D, k, fmt, sms, &p))
    return p.path == -2 ? LAM_ERR_UNSUPPORTED : LAM_ERR_INVALID;
  // the converting pass reads 8- or 16-byte code vectors: a 16-byte aligned base
  const bool aligned = (reinterpret_cast<uintptr_t>(codes) & 15u) == 0;
  if (!aligned && p.path != kPathGeneric) {
    if (forced_path() >= 0) return LAM_ERR_UNSUPPORTED;
    p.path = kPathGeneric;
    p.n_lists = generic_ctas(B, N, sms);
    p.qprep_off = align_up(p.partial_off + (size_t)p.n_lists * B * k * 8, 256);
    p.total = p.qprep_off;
  }
  if (workspace_bytes < p.total) return LAM_ERR_WORKSPACE;

  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  if (cudaMemsetAsync(ws, 0, kHeaderBytes, st) != cudaSuccess) return LAM_ERR_CUDA;
  if (apply_test_hooks(ws, st) != cudaSuccess) return LAM_ERR_CUDA;
  ScoreArgs a{};
  a.queries = queries;
  a.B = B;
  a.codes = codes;
  a.width = 1;
  a.N = N;
  a.D = D;
  a.s = 1.0f;
  a.code_bound = 0;
  a.k = k;
  a.metric = metric;
  a.scores = scores;
  a.ids = ids;
  a.gflags = reinterpret_cast<uint32_t *>(ws);
  a.partial = reinterpret_cast<uint64_t *>(ws + p.partial_off);
  a.n_lists = p.n_lists;
  a.qprep = ws + p.qprep_off;
  a.Bpad = p.Bpad;
  a.sms = sms;
  a.fmt = fmt;
  RowPtrs rp;
  rp.scale = scale;
  rp.offset = offset;
  ScoreArgs m = a;  // the final merge's lists
  const cudaError_t e = p.path == kPathTensor      ? launch_score_tensor(a, st, rp, &m)
                        : p.path == kPathBandwidth ? launch_score_bandwidth_rows(a, rp, st)
                                                   : launch_score_generic(a, st, rp);
  if (e != cudaSuccess) return LAM_ERR_CUDA;
  if (launch_topk_merge(m, st, rp) != cudaSuccess) return LAM_ERR_CUDA;
  return LAM_OK;
}

lam_status lam_quantize_async(const float *x, int64_t n, float eps, int32_t width_req, void *codes,
                              size_t codes_bytes, void *workspace, size_t workspace_bytes,
                              lam_stream_t stream) {
  if (n < 0 || n >= (1LL << 62) || !valid_eps(eps)) return LAM_ERR_INVALID;
  if (width_req != LAM_WIDTH_AUTO && !valid_width(width_req)) return LAM_ERR_INVALID;
  if (n > 0 && x == nullptr) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(x) & 3u) != 0) return LAM_ERR_INVALID;
  const uintptr_t calign = width_req == LAM_WIDTH_AUTO ? 4u : (uintptr_t)width_req;
  if (codes != nullptr && (reinterpret_cast<uintptr_t>(codes) & (calign - 1)) != 0)
    return LAM_ERR_INVALID;
  if (workspace == nullptr || (reinterpret_cast<uintptr_t>(workspace) & 15u) != 0)
    return LAM_ERR_INVALID;
  if (workspace_bytes < sizeof(QuantStatus)) return LAM_ERR_WORKSPACE;
  if (codes != nullptr && width_req != LAM_WIDTH_AUTO &&
      (unsigned long long)n * (unsigned long long)width_req > codes_bytes)
    return LAM_ERR_WORKSPACE;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  const float s = 2.0f * eps;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  QuantStatus *dst = static_cast<QuantStatus *>(workspace);
  if (cudaMemsetAsync(dst, 0, sizeof(QuantStatus), st) != cudaSuccess) return LAM_ERR_CUDA;
  cudaError_t e = cudaSuccess;
  if (n > 0) {
    timing_launch_begin(LAM_TIME_QUANTIZE, st);
    if (width_req == LAM_WIDTH_AUTO) e = launch_quantize_auto(x, n, s, codes, codes_bytes, dst, sms, st);
    else if (codes != nullptr) e = launch_quantize(x, n, s, width_req, codes, codes_bytes, dst, sms, st);
    else e = launch_quant_range(x, n, dst, sms, st);
    timing_launch_end(LAM_TIME_QUANTIZE, st);
    if (e != cudaSuccess) return LAM_ERR_CUDA;
  }
  // settle on the device: the forced width and its range check, or AUTO's
  // second pass (n == 0: the width alone)
  timing_launch_begin(LAM_TIME_AUX, st);
  e = launch_quantize_settle(x, n, s, width_req, codes, codes_bytes, dst, sms, st);
  timing_launch_end(LAM_TIME_AUX, st);
  return e == cudaSuccess ? LAM_OK : LAM_ERR_CUDA;
}

lam_status lam_quantize_result(const void *workspace, float eps, int32_t width_req,
                               lam_stream_t stream, int32_t *width_out, float *scale_out,
                               int32_t *code_min_out, int32_t *code_max_out) {
  if (workspace == nullptr || !valid_eps(eps)) return LAM_ERR_INVALID;
  if (width_req != LAM_WIDTH_AUTO && !valid_width(width_req)) return LAM_ERR_INVALID;
  QuantStatus h;
  if (read_back(&h, workspace, sizeof(h), reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
    return LAM_ERR_CUDA;
  return lam::decode_quant_status(h, width_req, 2.0f * eps, width_out, scale_out, code_min_out,
                                  code_max_out);
}

lam_status lam_dequantize_from(const void *codes, const void *quant_workspace, int64_t n,
                               float eps, float *out, lam_stream_t stream) {
  if (n < 0 || !valid_eps(eps)) return LAM_ERR_INVALID;
  if (n == 0) return LAM_OK;
  if (codes == nullptr || out == nullptr || quant_workspace == nullptr) return LAM_ERR_INVALID;
  // any width may come back: 4-byte alignment covers them all
  if ((reinterpret_cast<uintptr_t>(codes) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(out) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(quant_workspace) & 15u) != 0)
    return LAM_ERR_INVALID;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  timing_launch_begin(LAM_TIME_DEQUANTIZE, st);
  const cudaError_t e = launch_dequantize_from(
      codes, static_cast<const QuantStatus *>(quant_workspace), n, 2.0f * eps, out, sms, st);
  timing_launch_end(LAM_TIME_DEQUANTIZE, st);
  return e == cudaSuccess ? LAM_OK : LAM_ERR_CUDA;
}

size_t lam_score_topk_from_workspace_size(int64_t B, int64_t N, int32_t D, int32_t k) {
  Plan p;
  const int sms = device_sms();
  if (!make_from_plan(B, N, D, k, sms, &p)) return 0;
  const size_t generic = align_up(kHeaderBytes + (size_t)generic_ctas(B, N, sms) * B * k * 8, 256);
  return p.total > generic ? p.total : generic;
}

int32_t lam_score_topk_from_path(int64_t B, int64_t N, int32_t D, int32_t k) {
  Plan p;
  if (!make_from_plan(B, N, D, k, device_sms(), &p)) return -1;
  return p.path;
}

lam_status lam_score_topk_from(const float *queries, int64_t B, const void *codes,
                               const void *quant_workspace, int64_t N, int32_t D, float eps,
                               int32_t k, int32_t metric, float *scores, int64_t *ids,
                               void *workspace, size_t workspace_bytes, lam_stream_t stream) {
  if (queries == nullptr || codes == nullptr || quant_workspace == nullptr || scores == nullptr ||
      ids == nullptr || workspace == nullptr)
    return LAM_ERR_INVALID;
  if (metric != LAM_METRIC_IP && metric != LAM_METRIC_COSINE && metric != LAM_METRIC_L2)
    return LAM_ERR_INVALID;
  if (!valid_eps(eps) || !shape_ok(B, N, D, k, 2, 0)) return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0 ||
      (reinterpret_cast<uintptr_t>(quant_workspace) & 15u) != 0)
    return LAM_ERR_INVALID;
  if ((reinterpret_cast<uintptr_t>(codes) & 1u) != 0 ||
      (reinterpret_cast<uintptr_t>(queries) & 3u) != 0 ||
      (reinterpret_cast<uintptr_t>(scores) & 3u) != 0 || (reinterpret_cast<uintptr_t>(ids) & 7u) != 0)
    return LAM_ERR_INVALID;
  const int sms = device_sms();
  if (sms <= 0) return LAM_ERR_CUDA;
  Plan p;
  if (!make_from_plan(B, N, D, k, sms, &p))
    return p.path == -2 ? LAM_ERR_UNSUPPORTED : LAM_ERR_INVALID;
  const bool aligned = (reinterpret_cast<uintptr_t>(codes) & 15u) == 0;
  if (!aligned && p.path != kPathGeneric) {
    if (forced_path() >= 0) return LAM_ERR_UNSUPPORTED;
    p.path = kPathGeneric;
    p.n_lists = generic_ctas(B, N, sms);
    p.qprep_off = align_up(p.partial_off + (size_t)p.n_lists * B * k * 8, 256);
    p.total = p.qprep_off;
  }
  if (workspace_bytes < p.total) return LAM_ERR_WORKSPACE;

  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  if (cudaMemsetAsync(ws, 0, kHeaderBytes, st) != cudaSuccess) return LAM_ERR_CUDA;
  if (apply_test_hooks(ws, st) != cudaSuccess) return LAM_ERR_CUDA;
  ScoreArgs a;
  a.queries = queries;
  a.B = B;
  a.codes = codes;
  a.width = 1;  // unused: the kernels take the width from the status
  a.N = N;
  a.D = D;
  a.s = 2.0f * eps;
  a.code_bound = 0;
  a.k = k;
  a.metric = metric;
  a.scores = scores;
  a.ids = ids;
  a.gflags = reinterpret_cast<uint32_t *>(ws);
  a.partial = reinterpret_cast<uint64_t *>(ws + p.partial_off);
  a.n_lists = p.n_lists;
  a.qprep = ws + p.qprep_off;
  a.Bpad = p.Bpad;
  a.sms = sms;
  RowPtrs rp;
  rp.qst = static_cast<const QuantStatus *>(quant_workspace);
  ScoreArgs m = a;  // the final merge's lists
  cudaError_t e;
  if (p.path == kPathBandwidth) e = launch_score_bandwidth(a, st, rp.qst);
  else if (p.path == kPathTensor) e = launch_score_tensor(a, st, rp, &m);
  else e = launch_score_generic(a, st, rp);
  if (e != cudaSuccess) return LAM_ERR_CUDA;
  if (launch_topk_merge(m, st, rp) != cudaSuccess) return LAM_ERR_CUDA;
  return LAM_OK;
}

lam_status lam_score_topk_status(const void *workspace, lam_stream_t stream, int32_t *status_out) {
  if (workspace == nullptr || status_out == nullptr) return LAM_ERR_INVALID;
  uint32_t flags = 0;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (read_back(&flags, workspace, 4, st) != cudaSuccess) return LAM_ERR_CUDA;
  if (flags & kFlagTimeout) *status_out = LAM_ERR_TIMEOUT;
  else if (flags & kFlagInput) *status_out = LAM_ERR_UNSUPPORTED;
  else if (flags & kFlagRange) *status_out = LAM_ERR_RANGE;
  else *status_out = LAM_OK;
  return LAM_OK;
}


lam_status lam_timing_begin(int32_t mask, int64_t capacity) {
  if (mask < 1 || mask > 31 || capacity < 0 || capacity > (1 << 20)) return LAM_ERR_INVALID;
  std::lock_guard<std::mutex> lk(lam::g_timing.mu);
  lam::timing_release();
  lam::g_timing.ev.reserve((size_t)capacity * 2);
  for (int64_t i = 0; i < capacity * 2; ++i) {
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) {
      lam::timing_release();
      return LAM_ERR_CUDA;
    }
    lam::g_timing.ev.push_back(e);
  }
  lam::g_timing.kind.reserve((size_t)capacity);
  lam::g_timing.cap = capacity;
  lam::g_timing.mask = mask;
  return LAM_OK;
}

lam_status lam_timing_read(int32_t kind, double *total_ms, int64_t *timed, int64_t *launches) {
  if (kind != LAM_TIME_QUANTIZE && kind != LAM_TIME_DEQUANTIZE && kind != LAM_TIME_SCORE &&
      kind != LAM_TIME_AUX && kind != LAM_TIME_MERGE)
    return LAM_ERR_INVALID;
  std::lock_guard<std::mutex> lk(lam::g_timing.mu);
  double tot = 0.0;
  int64_t cnt = 0;
  for (int64_t i = 0; i < lam::g_timing.used; ++i) {
    if (lam::g_timing.kind[(size_t)i] != kind) continue;
    if (cudaEventSynchronize(lam::g_timing.ev[2 * i + 1]) != cudaSuccess) return LAM_ERR_CUDA;
    float ms = 0.0f;
    if (cudaEventElapsedTime(&ms, lam::g_timing.ev[2 * i], lam::g_timing.ev[2 * i + 1]) !=
        cudaSuccess)
      return LAM_ERR_CUDA;
    tot += ms;
    ++cnt;
  }
  if (total_ms) *total_ms = tot;
  if (timed) *timed = cnt;
  if (launches) *launches = lam::g_timing.launches[lam::kind_index(kind)];
  return LAM_OK;
}

lam_status lam_timing_end(void) {
  std::lock_guard<std::mutex> lk(lam::g_timing.mu);
  lam::timing_release();
  return LAM_OK;
}

}  // extern "C"
