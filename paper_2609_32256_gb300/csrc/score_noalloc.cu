// score_noalloc.cu -- lam_score_topk_noalloc: exact search on the codes for
// callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc: a host framework that owns every byte
// of device memory through its own pool and forbids allocations it did not
// make, or a latency-critical path where cudaMalloc's implicit device-wide
// synchronisation is not acceptable.  Such a caller still owns the queries,
// codes, scores and ids; the search's scratch (status word, per-CTA top-k
// lists, split queries) lives in the fixed device array below instead of a
// caller-provided workspace.
#include <mutex>

#include "lam_internal.cuh"

namespace {

constexpr size_t kNoallocScratchBytes = (size_t)16 << 20;  // 16 MiB per GPU

// Scratch of lam_score_topk_noalloc.  Every GPU that loads the library holds
// it until the process exits.  In host code this name is only a stand-in for
// the device symbol; its device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

constexpr int kMaxDevices = 64;
void *g_scratch_addr[kMaxDevices] = {};
std::mutex g_setup_mutex;

// Device address of the scratch on the current device (set up once per device).
void *scratch_address(int dev) {
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (g_scratch_addr[dev] == nullptr) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
    g_scratch_addr[dev] = p;
  }
  return g_scratch_addr[dev];
}

}  // namespace

extern "C" lam_status lam_score_topk_noalloc(const float *queries, int64_t B, const void *codes,
                                             int32_t width, int64_t N, int32_t D, float eps,
                                             int32_t code_bound, int32_t k, int32_t metric,
                                             float *scores, int64_t *ids, lam_stream_t stream) {
  const size_t need = lam_score_topk_workspace_size(B, N, D, k, width, code_bound);
  if (need == 0) return LAM_ERR_INVALID;
  if (need > kNoallocScratchBytes) return LAM_ERR_WORKSPACE;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return LAM_ERR_CUDA;
  void *scratch = scratch_address(dev);
  if (scratch == nullptr) return LAM_ERR_CUDA;
  // lam_score_topk clears the status word at the head of the scratch; the
  // kernels overwrite every other byte they read.
  lam_status st = lam_score_topk(queries, B, codes, width, N, D, eps, code_bound, k, metric,
                                 scores, ids, scratch, kNoallocScratchBytes, stream);
  if (st != LAM_OK) return st;
  int32_t dev_status = LAM_OK;
  st = lam_score_topk_status(scratch, stream, &dev_status);
  if (st != LAM_OK) return st;
  return static_cast<lam_status>(dev_status);
}
