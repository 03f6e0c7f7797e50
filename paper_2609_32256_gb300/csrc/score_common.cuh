// score_common.cuh -- pieces shared by the scoring kernels: the score
// formulas on integer codes, warp-level top-k lists, and the rank merge.
#pragma once

#include "lam_internal.cuh"

namespace lam {

// Score of one query against one code row, from
//   acc = sum_d q_d c_d  and  cc = sum_d c_d^2  (both fp32),
// with s = 2 eps, s2 = fl32(s*s), qq = ||q||^2, qn = ||q||.
//   inner product: s * acc                     (= q . xhat)
//   cosine:        acc / (||q|| sqrt(cc))       (s cancels; 0 for a zero norm)
//   squared L2:    ||q||^2 + s^2 cc - 2 s acc   (two fused multiply-adds)
__device__ __forceinline__ float finish_score(int metric, float acc, float cc, float s,
                                              float s2, float qq, float qn) {
  if (metric == LAM_METRIC_IP) return s * acc;
  if (metric == LAM_METRIC_COSINE)
    return (qn == 0.0f || cc == 0.0f) ? 0.0f : acc / (qn * sqrtf(cc));
  return fmaf(-2.0f * s, acc, fmaf(s2, cc, qq));
}

// ---- register top-k list of one warp: slot i = r*32 + lane, ascending keys --
template <int KPL>
struct WarpList {
  uint64_t v[KPL];
  __device__ __forceinline__ void init() {
#pragma unroll
    for (int r = 0; r < KPL; ++r) v[r] = kSentinel;
  }
  // Current k-th smallest key (slot k-1), the admission threshold.
  __device__ __forceinline__ uint64_t kth(int k) const {
    const int r = (k - 1) >> 5, l = (k - 1) & 31;
    uint64_t x = v[0];
#pragma unroll
    for (int j = 1; j < KPL; ++j)
      if (j == r) x = v[j];
    return __shfl_sync(0xffffffffu, x, l);
  }
  // Warp-uniform insertion of `key` (the caller checked key < kth).
  __device__ __forceinline__ void insert(uint64_t key, int lane) {
    int p = 0;
#pragma unroll
    for (int r = 0; r < KPL; ++r) p += __popc(__ballot_sync(0xffffffffu, v[r] < key));
#pragma unroll
    for (int r = KPL - 1; r >= 0; --r) {
      uint64_t up = __shfl_up_sync(0xffffffffu, v[r], 1);
      uint64_t carry = (r > 0) ? __shfl_sync(0xffffffffu, v[r > 0 ? r - 1 : 0], 31) : key;
      if (lane == 0) up = carry;
      const int i = r * 32 + lane;
      v[r] = (i < p) ? v[r] : (i == p ? key : up);
    }
  }
  // Writes slots [0, k) to dst.
  __device__ __forceinline__ void store(uint64_t *dst, int k, int lane) const {
#pragma unroll
    for (int r = 0; r < KPL; ++r) {
      const int i = r * 32 + lane;
      if (i < k) dst[i] = v[r];
    }
  }
};

// ---- per-thread top-k in registers: KR slots of (32-bit rank key, row) ----
// Keys ascend (smaller is better).  The first KR - k slots hold a dummy key 0
// that nothing can displace, so slot KR-1 is always the k-th best.  Rows must
// be offered in increasing order: a new key is placed after equal keys, so
// equal scores keep the lower row first.  Insertion compares the new key with
// every slot of the unmodified list (no serial dependence) and shifts.
template <int KR>
struct RegTopK {
  uint32_t key[KR];
  uint32_t id[KR];
  __device__ __forceinline__ void init(int k) {
#pragma unroll
    for (int i = 0; i < KR; ++i) {
      key[i] = (i < KR - k) ? 0u : 0xffffffffu;
      id[i] = 0xffffffffu;
    }
  }
  // kc == 0xffffffff inserts nothing.
  __device__ __forceinline__ void insert(uint32_t kc, uint32_t ic) {
    bool lt[KR];
#pragma unroll
    for (int i = 0; i < KR; ++i) lt[i] = kc < key[i];
#pragma unroll
    for (int i = KR - 1; i > 0; --i) {
      key[i] = lt[i - 1] ? key[i - 1] : (lt[i] ? kc : key[i]);
      id[i] = lt[i - 1] ? id[i - 1] : (lt[i] ? ic : id[i]);
    }
    key[0] = lt[0] ? kc : key[0];
    id[0] = lt[0] ? ic : id[0];
  }
};

// 32-bit rank key of a score (smaller is better) and its inverse.
__device__ __forceinline__ uint32_t rank_key32(float score, bool desc) {
  const uint32_t o = ord_f32(score);
  return desc ? ~o : o;
}
__device__ __forceinline__ float rank_key32_score(uint32_t key, bool desc) {
  return unord_f32(desc ? ~key : key);
}

// k-th largest of G register values (1 <= k <= G): the smallest value that
// fewer than k values exceed.  O(G^2) compares, no stores into v.
template <int G>
__device__ __forceinline__ float kth_largest(const float (&v)[G], int k) {
  float r = INFINITY;
#pragma unroll
  for (int i = 0; i < G; ++i) {
    int above = 0;
#pragma unroll
    for (int j = 0; j < G; ++j) above += v[j] > v[i] ? 1 : 0;
    if (above < k) r = fminf(r, v[i]);
  }
  return r;
}

// ---- per-thread max-heap of k keys in shared memory -------------------------
// Entry i of this thread's heap is H[i * stride + slot]; the root (i = 0) is
// the largest key, i.e. the worst of the k kept.
__device__ __forceinline__ void heap_sift_down(uint64_t *H, int n, int stride, int slot, int i,
                                               uint64_t key) {
  while (true) {
    const int l = 2 * i + 1;
    if (l >= n) break;
    int c = l;
    uint64_t cv = H[(size_t)l * stride + slot];
    if (l + 1 < n) {
      const uint64_t cr = H[(size_t)(l + 1) * stride + slot];
      if (cr > cv) {
        cv = cr;
        c = l + 1;
      }
    }
    if (cv <= key) break;
    H[(size_t)i * stride + slot] = cv;
    i = c;
  }
  H[(size_t)i * stride + slot] = key;
}
// Replaces the root (the worst key) by a better key.
__device__ __forceinline__ void heap_replace_root(uint64_t *H, int n, int stride, int slot,
                                                  uint64_t key) {
  heap_sift_down(H, n, stride, slot, 0, key);
}
// In-place heap sort: afterwards H[0..n) ascends.
__device__ __forceinline__ void heap_sort_ascending(uint64_t *H, int n, int stride, int slot) {
  for (int end = n - 1; end > 0; --end) {
    const uint64_t top = H[slot];
    const uint64_t last = H[(size_t)end * stride + slot];
    H[(size_t)end * stride + slot] = top;
    heap_sift_down(H, end, stride, slot, 0, last);
  }
}

// ---- shared-memory top-k list of one warp (any k <= kMaxK) ----
// L[0, k) ascending; *thr mirrors L[k-1].
__device__ __forceinline__ void smem_list_insert(uint64_t *L, int k, uint64_t key, int lane,
                                                 uint64_t &thr) {
  int p = 0;
  for (int c = 0; c < k; c += 32) {
    const int i = c + lane;
    p += __popc(__ballot_sync(0xffffffffu, i < k && L[i] < key));
  }
  for (int c = ((k - 1) >> 5) << 5; c >= 0; c -= 32) {
    const int i = c + lane;
    uint64_t prev = (i >= 1 && i - 1 < k) ? L[i - 1] : 0;
    __syncwarp();
    if (i < k && i > p) L[i] = prev;
    __syncwarp();
  }
  if (lane == 0) L[p] = key;
  __syncwarp();
  thr = L[k - 1];
}

// ---- merge of nl ascending lists of length k (in shared memory) ----
// Every element finds its rank in the union by binary search in the other
// lists (ties between equal keys broken by list index); ranks < k are written
// to out[rank].  Keys are unique except the sentinel, so out gets exactly k.
__device__ __forceinline__ void rank_merge(const uint64_t *cand, int nl, int k, uint64_t *out,
                                           int tid, int nthreads) {
  for (int e = tid; e < nl * k; e += nthreads) {
    const int l = e / k, i = e - l * k;
    const uint64_t key = cand[e];
    int rank = i;
    for (int l2 = 0; l2 < nl && rank < k; ++l2) {
      if (l2 == l) continue;
      const uint64_t *L2 = cand + (size_t)l2 * k;
      int lo = 0, hi = k;
      if (l2 < l) {
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (L2[mid] <= key) lo = mid + 1; else hi = mid;
        }
      } else {
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (L2[mid] < key) lo = mid + 1; else hi = mid;
        }
      }
      rank += lo;
    }
    if (rank < k) out[rank] = key;
  }
}

}  // namespace lam
