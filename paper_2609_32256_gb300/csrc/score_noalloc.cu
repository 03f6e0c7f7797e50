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
#include <cuda.h>  // CUcontext / CUresult types only; the driver calls come from the runtime

#include <mutex>

#include "lam_internal.cuh"

namespace {

constexpr size_t kNoallocScratchBytes = (size_t)16 << 20;  // 16 MiB per GPU

// Scratch of lam_score_topk_noalloc.  Every GPU that loads the library holds
// it until the process exits.  In host code this name is only a stand-in for
// the device symbol; its device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

constexpr int kMaxDevices = 64;

// The scratch address found for a device, and the CUDA context it belongs to.
struct ScratchSlot {
  unsigned long long ctx = 0;
  void *addr = nullptr;
};
ScratchSlot g_slot[kMaxDevices];
std::mutex g_setup_mutex;

typedef CUresult (*CtxGetCurrentFn)(CUcontext *);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long *);

// Unique id of the calling thread's current CUDA context (0 when there is
// none yet or it cannot be read).  The driver entry points come through the
// runtime, so the library does not link the driver library itself.
unsigned long long current_context_id() {
  static std::once_flag once;
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void *f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(f);
    f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(f);
  });
  if (get_current == nullptr || get_id == nullptr) return 0;
  CUcontext c = nullptr;
  if (get_current(&c) != CUDA_SUCCESS || c == nullptr) return 0;
  unsigned long long id = 0;
  if (get_id(c, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Device address of the scratch on the current device.  It is looked up with
// cudaGetSymbolAddress the first time a context on the device uses it, and
// again whenever that context has changed (e.g. after cudaDeviceReset), so a
// stale address is never reused; if the context cannot be identified the
// lookup runs on every call.
void *scratch_address(int dev) {
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  unsigned long long ctx = current_context_id();
  if (ctx != 0 && g_slot[dev].addr != nullptr && g_slot[dev].ctx == ctx) return g_slot[dev].addr;
  void *p = nullptr;
  if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
  if (ctx == 0) ctx = current_context_id();  // the lookup may have made the context current
  g_slot[dev].ctx = ctx;
  g_slot[dev].addr = p;
  return p;
}

}  // namespace

extern "C" lam_status lam_score_topk_noalloc(const float *queries, int64_t B, const void *codes,
                                             int32_t width, int64_t N, int32_t D, float eps,
                                             int32_t code_bound, int32_t k, int32_t metric,
                                             float *scores, int64_t *ids, lam_stream_t stream) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return LAM_ERR_CUDA;
  void *scratch = scratch_address(dev);
  if (scratch == nullptr) return LAM_ERR_CUDA;
  // lam_score_topk checks every argument in its own order and returns the
  // same statuses (LAM_ERR_WORKSPACE when the shape needs more than the
  // array) before it queues anything.  It clears the status word at the head
  // of the scratch; the kernels overwrite every other byte they read.
  lam_status st = lam_score_topk(queries, B, codes, width, N, D, eps, code_bound, k, metric,
                                 scores, ids, scratch, kNoallocScratchBytes, stream);
  if (st != LAM_OK) return st;
  int32_t dev_status = LAM_OK;
  st = lam_score_topk_status(scratch, stream, &dev_status);
  if (st != LAM_OK) return st;
  return static_cast<lam_status>(dev_status);
}
