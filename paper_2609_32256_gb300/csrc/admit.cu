// admit.cu -- batch form of the admission rule (Algorithm 2; Sec. 3.3 "The
// eps error-bounded test"): records in order; the candidates of record i are
// the retained records sharing a band digest with it in the same band; its
// representative is the lowest-indexed candidate within l2 distance delta
// (Eq. 2: delta = sqrt(2 - 2t)), else it is retained.  The measured bound
// delta_hat is the largest merge distance.
//
// The sequential rule is resolved in parallel:
//   1. every (row, band) entry gets a 32-bit bucket key from its digest and a
//      stable radix sort groups equal keys;
//   2. inside each run of equal keys, pairs of rows whose (band, digest) agree
//      exactly are the candidate pairs (counted, then written in order);
//   3. the pairs are sorted by (row, lower row) and made unique;
//   4. each pair's distance is taken in full precision (squared differences of
//      the coordinates in double, summed in coordinate order without fused
//      multiply-adds, one sqrt) and pairs within delta are kept, in order;
//   5. greedy first-occurrence over that graph: a row whose lower neighbours
//      are all decided is merged into the first retained one, or retained if
//      none is; rounds repeat until every row is decided (the lowest undecided
//      row is always decidable, so every round makes progress).
#include "lam_internal.cuh"
#include "scan.cuh"

namespace lam {

namespace {

constexpr int kRadixBits = 4, kRadix = 1 << kRadixBits;

// ---------------------------------------------------------------- sort ------
// Stable LSD radix sort of (uint32 key, uint32 value) pairs, 4 bits a pass.
__global__ void __launch_bounds__(kSortThreads) radix_hist_kernel(const uint32_t *keys, int64_t n,
                                                                  int shift, uint32_t *hist,
                                                                  int64_t nblk) {
  __shared__ uint32_t cnt[kRadix];
  if (threadIdx.x < kRadix) cnt[threadIdx.x] = 0;
  __syncthreads();
  const int64_t base = (int64_t)blockIdx.x * kTile + (int64_t)threadIdx.x * kSortItems;
#pragma unroll
  for (int k = 0; k < kSortItems; ++k)
    if (base + k < n) atomicAdd(&cnt[(keys[base + k] >> shift) & (kRadix - 1)], 1u);
  __syncthreads();
  if (threadIdx.x < kRadix) hist[(int64_t)threadIdx.x * nblk + blockIdx.x] = cnt[threadIdx.x];
}

__global__ void __launch_bounds__(kSortThreads) radix_scatter_kernel(
    const uint32_t *keys, const uint32_t *vals, int64_t n, int shift, const uint32_t *offs,
    int64_t nblk, uint32_t *okeys, uint32_t *ovals) {
  __shared__ uint32_t cnt[kRadix * kSortThreads];  // [digit][thread]
  const int t = threadIdx.x;
  for (int d = 0; d < kRadix; ++d) cnt[d * kSortThreads + t] = 0;
  const int64_t base = (int64_t)blockIdx.x * kTile + (int64_t)t * kSortItems;
#pragma unroll
  for (int k = 0; k < kSortItems; ++k)
    if (base + k < n) ++cnt[((keys[base + k] >> shift) & (kRadix - 1)) * kSortThreads + t];
  __syncthreads();
  // exclusive scan of the flat [digit][thread] counts: thread j owns 16 of them
  uint32_t v[kSortItems], s = 0;
#pragma unroll
  for (int k = 0; k < kSortItems; ++k) {
    v[k] = cnt[t * kSortItems + k];
    s += v[k];
  }
  uint32_t tot;
  uint32_t run = block_exclusive_scan_256(s, &tot);
#pragma unroll
  for (int k = 0; k < kSortItems; ++k) {
    cnt[t * kSortItems + k] = run;
    run += v[k];
  }
  __syncthreads();
  // write each entry: global base of its digit for this block, plus its rank
  // among the block's entries of that digit (stable: threads in order, items
  // in order within a thread)
  uint32_t seen[kRadix];
#pragma unroll
  for (int d = 0; d < kRadix; ++d) seen[d] = 0;
#pragma unroll
  for (int k = 0; k < kSortItems; ++k) {
    if (base + k >= n) break;
    const uint32_t key = keys[base + k];
    const int d = (key >> shift) & (kRadix - 1);
    uint32_t sd = 0;
#pragma unroll
    for (int e = 0; e < kRadix; ++e)
      if (e == d) sd = seen[e]++;
    const uint32_t local = cnt[d * kSortThreads + t] - cnt[d * kSortThreads] + sd;
    const uint32_t pos = offs[(int64_t)d * nblk + blockIdx.x] + local;
    okeys[pos] = key;
    ovals[pos] = vals[base + k];
  }
}

// --------------------------------------------------------- candidates -------
__global__ void make_keys_kernel(const uint64_t *dig, int64_t m, int nb, uint32_t *keys,
                                 uint32_t *vals) {
  for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < m;
       j += (int64_t)gridDim.x * blockDim.x) {
    const uint64_t h = dig[j];
    const uint32_t b = (uint32_t)(j % nb);
    keys[j] = (uint32_t)(h ^ (h >> 32)) ^ (b * 0x9E3779B9u);
    vals[j] = (uint32_t)j;  // entry index = row * nb + band
  }
}

// Number of later entries of the same key run that match entry p exactly
// (same band and digest) and belong to another row; with `out`, writes those
// pairs (row of p = the lower row, since the sort is stable and entries are in
// row order) from out[offs[p]].
__global__ void pairs_kernel(const uint32_t *keys, const uint32_t *vals, const uint64_t *dig,
                             int64_t m, int nb, uint32_t *counts, const uint32_t *offs,
                             uint32_t *out_lo, uint32_t *out_hi) {
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < m;
       p += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t key = keys[p], ep = vals[p];
    const uint64_t dp = dig[ep];
    const uint32_t bp = ep % (uint32_t)nb, rp = ep / (uint32_t)nb;
    uint32_t c = 0;
    for (int64_t q = p + 1; q < m && keys[q] == key; ++q) {
      const uint32_t eq = vals[q];
      if (dig[eq] != dp || eq % (uint32_t)nb != bp) continue;
      const uint32_t rq = eq / (uint32_t)nb;
      if (rq == rp) continue;
      if (out_lo != nullptr) {
        out_lo[offs[p] + c] = rp;
        out_hi[offs[p] + c] = rq;
      }
      ++c;
    }
    if (counts != nullptr) counts[p] = c;
  }
}

// flag[p] = 1 where (hi, lo) differs from the previous pair (pairs sorted by
// hi then lo)
__global__ void unique_flags_kernel(const uint32_t *hi, const uint32_t *lo, int64_t n,
                                    uint32_t *flag) {
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < n;
       p += (int64_t)gridDim.x * blockDim.x)
    flag[p] = (p == 0 || hi[p] != hi[p - 1] || lo[p] != lo[p - 1]) ? 1u : 0u;
}

// Distance of each pair in full precision; keep[p] = 1 within delta.  The
// partial sums of squares never decrease (each rounded addition of a
// non-negative term is at least the running sum), so a pair is rejected as
// soon as its partial sum passes delta^2 (1 + 2^-40), which puts even the
// rounded square root above delta; the distances of the kept pairs are
// summed in full, in coordinate order.  (Most band candidates are far apart
// and leave after the first 64 coordinates.)
__global__ void verify_kernel(const float *__restrict__ e, int D, const uint32_t *hi,
                              const uint32_t *lo, const uint32_t *uflag, int64_t n, double delta,
                              double *dist, uint32_t *keep) {
  const double over = __dmul_rn(__dmul_rn(delta, delta), 1.0 + 0x1p-40);
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < n;
       p += (int64_t)gridDim.x * blockDim.x) {
    uint32_t k = 0;
    double dd = 0.0;
    if (uflag[p]) {
      const float *a = e + (int64_t)hi[p] * D, *b = e + (int64_t)lo[p] * D;
      double acc = 0.0;
      bool far = false;
      for (int d0 = 0; d0 < D && !far; d0 += 64) {
        const int d1 = d0 + 64 < D ? d0 + 64 : D;
        for (int d = d0; d < d1; ++d) {
          const double t = __dsub_rn((double)__ldg(a + d), (double)__ldg(b + d));
          acc = __dadd_rn(acc, __dmul_rn(t, t));
        }
        far = acc > over;
      }
      dd = far ? INFINITY : sqrt(acc);
      k = dd <= delta ? 1u : 0u;
    }
    dist[p] = dd;
    keep[p] = k;
  }
}

// Order-preserving compaction of the kept edges (offs = exclusive scan of keep).
__global__ void compact_kernel(const uint32_t *hi, const uint32_t *lo, const double *dist,
                               const uint32_t *keep, const uint32_t *offs, int64_t n,
                               uint32_t *ehi, uint32_t *elo, double *edist, uint32_t *row_cnt) {
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < n;
       p += (int64_t)gridDim.x * blockDim.x)
    if (keep[p]) {
      const uint32_t o = offs[p];
      ehi[o] = hi[p];
      elo[o] = lo[p];
      edist[o] = dist[p];
      atomicAdd(&row_cnt[hi[p]], 1u);
    }
}

// Greedy first-occurrence over the verified graph in one block: rounds until
// every row is decided.  state: 0 undecided, 1 retained, 2 merged.
__global__ void __launch_bounds__(1024) resolve_kernel(int64_t N, const uint32_t *row_start,
                                                        const uint32_t *elo, const double *edist,
                                                        uint8_t *state, int32_t *rep,
                                                        double *dist_out, double *stat) {
  __shared__ int changed, undecided;
  __shared__ double dh[32];
  __shared__ unsigned long long kept[32];
  for (int64_t i = threadIdx.x; i < N; i += blockDim.x) state[i] = 0;
  __syncthreads();
  for (int64_t round = 0; round <= N; ++round) {
    if (threadIdx.x == 0) changed = undecided = 0;
    __syncthreads();
    int ch = 0, un = 0;
    for (int64_t i = threadIdx.x; i < N; i += blockDim.x) {
      if (state[i] != 0) continue;
      int verdict = 1;  // retained unless a lower neighbour says otherwise
      uint32_t y_rep = 0;
      double d_rep = 0.0;
      for (uint32_t q = row_start[i]; q < row_start[i + 1]; ++q) {
        const uint8_t sy = ((volatile uint8_t *)state)[elo[q]];
        if (sy == 2) continue;
        if (sy == 0) {
          verdict = 0;  // a lower neighbour is still open
          break;
        }
        verdict = 2;
        y_rep = elo[q];
        d_rep = edist[q];
        break;
      }
      if (verdict == 0) {
        ++un;
        continue;
      }
      rep[i] = verdict == 1 ? (int32_t)i : (int32_t)y_rep;
      dist_out[i] = verdict == 1 ? 0.0 : d_rep;
      __threadfence_block();
      ((volatile uint8_t *)state)[i] = (uint8_t)verdict;
      ++ch;
    }
    if (ch) atomicAdd(&changed, ch);
    if (un) atomicAdd(&undecided, un);
    __syncthreads();
    const bool done = undecided == 0;
    __syncthreads();
    if (done) break;
  }
  // measured bound and retained count
  double m = 0.0;
  unsigned long long kc = 0;
  for (int64_t i = threadIdx.x; i < N; i += blockDim.x) {
    if (state[i] == 2) m = fmax(m, dist_out[i]);
    if (state[i] == 1) ++kc;
  }
  for (int off = 16; off > 0; off >>= 1) {
    m = fmax(m, __shfl_xor_sync(0xffffffffu, m, off));
    kc += __shfl_xor_sync(0xffffffffu, kc, off);
  }
  if ((threadIdx.x & 31) == 0) {
    dh[threadIdx.x >> 5] = m;
    kept[threadIdx.x >> 5] = kc;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double mm = 0.0;
    unsigned long long kk = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
      mm = fmax(mm, dh[w]);
      kk += kept[w];
    }
    stat[0] = mm;
    stat[1] = (double)kk;
  }
}

inline size_t al(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace

// Workspace layout (all offsets 256-byte aligned).
struct AdmitLayout {
  size_t stat, keysA, valsA, keysB, valsB, hist, sums, cnt, plo, phi, qlo, qhi, flag, offs, dist,
      keep, elo, ehi, edist, rowc, state, total;
};

static AdmitLayout admit_layout(int64_t N, int nb, int64_t max_pairs) {
  AdmitLayout L;
  const int64_t m = N * nb;
  const int64_t big = m > max_pairs ? m : max_pairs;
  const int64_t nblk = cdiv(big, kTile) + 1;
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t r = o;
    o += al(bytes);
    return r;
  };
  L.stat = take(64);
  L.keysA = take(4 * m);
  L.valsA = take(4 * m);
  L.keysB = take(4 * m);
  L.valsB = take(4 * m);
  L.hist = take(4 * (size_t)kRadix * nblk);
  L.sums = take(4 * (size_t)nblk + 4);
  L.cnt = take(4 * (size_t)(m + 1));
  L.plo = take(4 * (size_t)max_pairs);
  L.phi = take(4 * (size_t)max_pairs);
  L.qlo = take(4 * (size_t)max_pairs);
  L.qhi = take(4 * (size_t)max_pairs);
  L.flag = take(4 * (size_t)max_pairs + 4);
  L.offs = take(4 * (size_t)max_pairs + 4);
  L.dist = take(8 * (size_t)max_pairs);
  L.keep = take(4 * (size_t)max_pairs + 4);
  L.elo = take(4 * (size_t)max_pairs);
  L.ehi = take(4 * (size_t)max_pairs);
  L.edist = take(8 * (size_t)max_pairs);
  L.rowc = take(4 * (size_t)(N + 1));
  L.state = take((size_t)N);
  L.total = o;
  return L;
}

size_t admit_workspace_bytes(int64_t N, int nb, int64_t max_pairs) {
  return admit_layout(N, nb, max_pairs).total;
}

namespace {

// Sorts (keys, vals) of n entries by key (stable); the result ends in the
// first pair of buffers (8 passes: an even count).
cudaError_t radix_sort(uint32_t *keys, uint32_t *vals, uint32_t *tk, uint32_t *tv, int64_t n,
                       uint32_t *hist, uint32_t *sums, cudaStream_t st) {
  const int64_t nblk = cdiv(n, kTile);
  if (nblk == 0) return cudaSuccess;
  uint32_t *ik = keys, *iv = vals, *ok = tk, *ov = tv;
  for (int shift = 0; shift < 32; shift += kRadixBits) {
    radix_hist_kernel<<<(unsigned)nblk, kSortThreads, 0, st>>>(ik, n, shift, hist, nblk);
    cudaError_t e = scan_u32(hist, (int64_t)kRadix * nblk, sums, nullptr, st);
    if (e != cudaSuccess) return e;
    radix_scatter_kernel<<<(unsigned)nblk, kSortThreads, 0, st>>>(ik, iv, n, shift, hist, nblk,
                                                                  ok, ov);
    uint32_t *t1 = ik, *t2 = iv;
    ik = ok;
    iv = ov;
    ok = t1;
    ov = t2;
  }
  return cudaGetLastError();
}

unsigned grid1d(int64_t n, int sms) {
  int64_t g = cdiv(n, 256);
  if (g > (int64_t)sms * 8) g = (int64_t)sms * 8;
  return (unsigned)(g < 1 ? 1 : g);
}

}  // namespace

// Runs the batch admission; returns the candidate-pair count in *n_pairs
// (device status block) so that an oversize run can be reported.
cudaError_t launch_admit_batch(const float *e, int64_t N, int D, const uint64_t *dig, int nb,
                               double delta, int32_t *rep, double *dist, void *ws,
                               int64_t max_pairs, int sms, cudaStream_t st, int64_t *n_pairs,
                               double *delta_hat, int64_t *n_retained, bool *overflow) {
  const AdmitLayout L = admit_layout(N, nb, max_pairs);
  uint8_t *w = static_cast<uint8_t *>(ws);
  auto U = [&](size_t off) { return reinterpret_cast<uint32_t *>(w + off); };
  auto Dp = [&](size_t off) { return reinterpret_cast<double *>(w + off); };
  const int64_t m = N * nb;
  uint32_t *stat32 = U(L.stat);
  double *stat64 = Dp(L.stat + 16);
  cudaError_t err = cudaMemsetAsync(w + L.stat, 0, 64, st);
  if (err != cudaSuccess) return err;
  // 1. bucket keys, stable sort
  make_keys_kernel<<<grid1d(m, sms), 256, 0, st>>>(dig, m, nb, U(L.keysA), U(L.valsA));
  err = radix_sort(U(L.keysA), U(L.valsA), U(L.keysB), U(L.valsB), m, U(L.hist), U(L.sums), st);
  if (err != cudaSuccess) return err;
  // 2. candidate pairs: count, scan, check the total against max_pairs
  pairs_kernel<<<grid1d(m, sms), 256, 0, st>>>(U(L.keysA), U(L.valsA), dig, m, nb, U(L.cnt),
                                              nullptr, nullptr, nullptr);
  err = scan_u32(U(L.cnt), m, U(L.sums), stat32 + 0, st);
  if (err != cudaSuccess) return err;
  uint32_t np = 0;
  err = read_back(&np, stat32, 4, st);
  if (err != cudaSuccess) return err;
  *n_pairs = np;
  if ((int64_t)np > max_pairs) {
    *overflow = true;
    return cudaSuccess;
  }
  *overflow = false;
  pairs_kernel<<<grid1d(m, sms), 256, 0, st>>>(U(L.keysA), U(L.valsA), dig, m, nb, nullptr,
                                              U(L.cnt), U(L.plo), U(L.phi));
  // 3. sort pairs by (higher row, lower row): by lower row, then stably by higher
  err = radix_sort(U(L.plo), U(L.phi), U(L.qlo), U(L.qhi), np, U(L.hist), U(L.sums), st);
  if (err != cudaSuccess) return err;
  // now keys = lower rows, vals = higher rows; re-sort by the higher row
  err = radix_sort(U(L.phi), U(L.plo), U(L.qhi), U(L.qlo), np, U(L.hist), U(L.sums), st);
  if (err != cudaSuccess) return err;
  // keys (phi) = higher row i, vals (plo) = lower row y, ordered by (i, y)
  unique_flags_kernel<<<grid1d(np, sms), 256, 0, st>>>(U(L.phi), U(L.plo), np, U(L.flag));
  // 4. verify, keep pairs within delta in order, count per row
  verify_kernel<<<grid1d(np, sms), 256, 0, st>>>(e, D, U(L.phi), U(L.plo), U(L.flag), np, delta,
                                                 Dp(L.dist), U(L.keep));
  err = cudaMemcpyAsync(U(L.offs), U(L.keep), 4 * (size_t)np, cudaMemcpyDeviceToDevice, st);
  if (err != cudaSuccess) return err;
  err = scan_u32(U(L.offs), np, U(L.sums), stat32 + 1, st);
  if (err != cudaSuccess) return err;
  err = cudaMemsetAsync(U(L.rowc), 0, 4 * (size_t)(N + 1), st);
  if (err != cudaSuccess) return err;
  compact_kernel<<<grid1d(np, sms), 256, 0, st>>>(U(L.phi), U(L.plo), Dp(L.dist), U(L.keep),
                                                  U(L.offs), np, U(L.ehi), U(L.elo), Dp(L.edist),
                                                  U(L.rowc));
  err = scan_u32(U(L.rowc), N + 1, U(L.sums), stat32 + 2, st);
  if (err != cudaSuccess) return err;
  // 5. greedy first-occurrence
  resolve_kernel<<<1, 1024, 0, st>>>(N, U(L.rowc), U(L.elo), Dp(L.edist), w + L.state, rep, dist,
                                     stat64);
  double h[2];
  err = read_back(h, stat64, 16, st);
  if (err != cudaSuccess) return err;
  *delta_hat = h[0];
  *n_retained = (int64_t)h[1];
  return cudaGetLastError();
}

}  // namespace lam
