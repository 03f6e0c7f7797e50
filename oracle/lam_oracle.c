/*
 * lam_oracle.c -- plain, slow CPU oracle for LAM's quantized-memory hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library links, loads or
 * calls this file.  Only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg may use it.  It shares no code, header or constant
 * generator with the CUDA path.
 *
 * What it computes (paper: "LAM: Lossy Agent Memory"):
 *   - Q_eps(x) = round(x / 2 eps), coordinatewise, one global eps
 *     (Sec. 3.2 "Three layers", layer L1; Algorithm 1 applies it to each
 *     arriving embedding).
 *   - Dequantisation xhat = 2 eps * Q_eps(x).  The paper never writes it out;
 *     it is the reading under which a quantization cell has half-width eps
 *     (Sec. 3.1, the coordinatewise tolerance ||a-b||_inf <= 2 eps between
 *     two members of one cell; App. "Rank invariance, in full").
 *   - Exact search: every query scored against every retained (here:
 *     dequantised) embedding, i.e. a matrix-vector product per query
 *     (Sec. "Brute-force scan crossover"), followed by a top-k.  Metrics:
 *     inner product, cosine, squared L2 (Eq. 1 relates L2 and cosine).
 *
 * Readings where the paper is silent:
 *   - "round" is IEEE round-half-to-even, evaluated as nearbyintf() under
 *     FE_TONEAREST on the fp32 quotient.
 *   - x / 2 eps is one fp32 IEEE division by s = fl32(2 * eps), eps given in
 *     fp32 (doubling is exact).
 *   - Dequantisation is one fp32 multiply s * (float)c.
 *   - Cosine uses the norm of the dequantised vector; a zero norm gives 0.
 *   - L2 score is the squared distance, ranked ascending; inner product and
 *     cosine rank descending.  Equal scores rank the lower id first (the
 *     paper's lowest-index rule, Algorithm 1).
 *   - Scores are accumulated in double and rounded once to fp32.
 *   - The per-vector byte codecs of the composite experiment (fp16,
 *     per-vector int8, sign-binary; Sec. "Composite reduction", Table
 *     "composite") are defined only by name and ratio; the definitions taken
 *     are given above lam_oracle_encode_int8_rows.
 *
 * Build flags matter: -O2 -ffp-contract=off -fno-fast-math, so that no
 * multiply-add is contracted into an FMA on either x86-64 or aarch64.
 */
#include <fenv.h>
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_IP 0
#define ORACLE_COSINE 1
#define ORACLE_L2 2

/* Step of the quantizer: s = 2 eps in fp32 (Sec. 3.2, L1). */
float lam_oracle_step(float eps) { return 2.0f * eps; }

/*
 * Q_eps over n fp32 values (Sec. 3.2, L1: Q_eps(x) = round(x / 2 eps)).
 *   r_i = nearbyintf(fl32(x_i / s)); codes_i = (int32) r_i when r_i fits int32.
 * Outputs: codes (may be NULL), the smallest and largest rounded quotient over
 * the finite inputs (as doubles, exact), and the count of non-finite inputs.
 * With n == 0, rmin = rmax = 0.
 */
void lam_oracle_quantize(const float *x, int64_t n, float eps, int32_t *codes,
                         double *rmin_out, double *rmax_out,
                         int64_t *n_nonfinite_out) {
  int old_mode = fegetround();
  fesetround(FE_TONEAREST);
  float s = lam_oracle_step(eps);
  double rmin = 0.0, rmax = 0.0;
  int seen = 0;
  int64_t nonfinite = 0;
  for (int64_t i = 0; i < n; ++i) {
    float xi = x[i];
    if (!isfinite(xi)) {
      nonfinite++;
      if (codes) codes[i] = 0;
      continue;
    }
    float q = xi / s;
    float r = nearbyintf(q);
    if (!seen) {
      rmin = rmax = (double)r;
      seen = 1;
    } else {
      if ((double)r < rmin) rmin = (double)r;
      if ((double)r > rmax) rmax = (double)r;
    }
    if (codes) {
      if ((double)r >= -2147483648.0 && (double)r <= 2147483647.0)
        codes[i] = (int32_t)r;
      else
        codes[i] = 0;
    }
  }
  fesetround(old_mode);
  *rmin_out = rmin;
  *rmax_out = rmax;
  *n_nonfinite_out = nonfinite;
}

/*
 * Narrowest two's-complement width (bytes: 1, 2 or 4) whose range holds
 * [rmin, rmax]; 0 when even int32 cannot hold it.
 */
int32_t lam_oracle_width(double rmin, double rmax) {
  if (rmin >= -128.0 && rmax <= 127.0) return 1;
  if (rmin >= -32768.0 && rmax <= 32767.0) return 2;
  if (rmin >= -2147483648.0 && rmax <= 2147483647.0) return 4;
  return 0;
}

/* Dequantisation xhat_i = fl32(s * (float) c_i) with s = fl32(2 eps). */
void lam_oracle_dequantize(const int32_t *codes, int64_t n, float scale,
                           float *out) {
  for (int64_t i = 0; i < n; ++i) out[i] = scale * (float)codes[i];
}

/* Squared norm of each code row, sum_d c_{i,d}^2: the exact integer sum
 * (in int64; |c| <= 32767 for the 1- and 2-byte widths, so it cannot
 * overflow for D < 2^33) rounded once to fp32.  This is the side array an
 * exact scan can keep to score cosine and squared L2 on codes (Eq. 1 expands
 * the L2 distance into the two norms and the inner product). */
void lam_oracle_code_sqnorms(const int32_t *codes, int64_t N, int32_t D,
                             float *out) {
  for (int64_t i = 0; i < N; ++i) {
    int64_t acc = 0;
    for (int32_t d = 0; d < D; ++d) {
      const int64_t c = codes[i * (int64_t)D + d];
      acc += c * c;
    }
    out[i] = (float)acc; /* one round-to-nearest conversion */
  }
}

/*
 * Band digests of quantized rows (Sec. 3.2, L1: "divide the vector into
 * bands, and hash each band; records sharing a band digest are candidates";
 * Algorithm 1, BandHash(Q_eps(e))).  The paper names no hash function; the
 * reading taken here is 64-bit FNV-1a (Fowler, Noll, Vo: offset basis
 * 14695981039346656037, prime 1099511628211, one xor then one multiply per
 * byte) over
 *   - the band's index within its row, as 2 little-endian bytes (so that
 *     equal code patterns in different bands do not share a digest), then
 *   - the band's r codes in coordinate order, each as its `width`
 *     little-endian two's-complement bytes (the bytes the code array holds).
 * Rows have D coordinates, D a multiple of r; digest[i * (D / r) + b] is band
 * b of row i.
 */
uint64_t lam_oracle_fnv1a64(const uint8_t *bytes, int64_t n, uint64_t h) {
  for (int64_t i = 0; i < n; ++i) {
    h ^= (uint64_t)bytes[i];
    h *= 1099511628211ULL;
  }
  return h;
}

void lam_oracle_band_digests(const int32_t *codes, int64_t N, int32_t D, int32_t r,
                             int32_t width, uint64_t *digest) {
  const int32_t nb = D / r;
  for (int64_t i = 0; i < N; ++i) {
    for (int32_t b = 0; b < nb; ++b) {
      uint8_t idx[2] = {(uint8_t)(b & 0xff), (uint8_t)((b >> 8) & 0xff)};
      uint64_t h = lam_oracle_fnv1a64(idx, 2, 14695981039346656037ULL);
      for (int32_t d = b * r; d < (b + 1) * r; ++d) {
        const uint32_t c = (uint32_t)codes[i * (int64_t)D + d];
        uint8_t le[4] = {(uint8_t)c, (uint8_t)(c >> 8), (uint8_t)(c >> 16), (uint8_t)(c >> 24)};
        h = lam_oracle_fnv1a64(le, width, h);
      }
      digest[i * nb + b] = h;
    }
  }
}

/*
 * Batch form of the admission rule (Algorithm 2; Sec. 3.3 "The eps
 * error-bounded test"): records 0..N-1 in order; record i's candidates are the
 * retained records that share a band digest with it in the same band
 * (BandHash(Q_eps(e_y)) and BandHash(Q_eps(e_i)) intersect; the band index
 * holds retained records only); its representative is the lowest-indexed
 * candidate within l2 distance delta (Eq. 2: delta = sqrt(2 - 2t) for merge
 * threshold t), else it is retained and becomes its own representative.
 * Distances are taken in full precision: the squared difference of each
 * coordinate in double, summed in coordinate order, then one sqrt.
 * Outputs: rep[i] (representative index, i itself when retained), dist[i]
 * (distance to it, 0 when retained) and the measured bound delta_hat = the
 * largest distance of a merge (0 when nothing merges).  Returns the number of
 * retained records.
 */
static double l2_full(const float *a, const float *b, int32_t D) {
  double acc = 0.0;
  for (int32_t d = 0; d < D; ++d) {
    const double t = (double)a[d] - (double)b[d];
    acc += t * t;
  }
  return sqrt(acc);
}

int64_t lam_oracle_admit_batch(const float *e, int64_t N, int32_t D, const uint64_t *digests,
                               int32_t nb, double delta, int32_t *rep, double *dist,
                               double *delta_hat) {
  /* per band: open-addressing table digest -> most recent retained id with it,
   * and for every (band, retained id) the previous retained id with the same
   * digest in that band (a linked list, newest first) */
  int64_t cap = 16;
  while (cap < 2 * N + 2) cap <<= 1;
  int64_t *tab_key_id = (int64_t *)malloc(sizeof(int64_t) * (size_t)cap * (size_t)nb);
  int32_t *prev = (int32_t *)malloc(sizeof(int32_t) * (size_t)N * (size_t)nb);
  int64_t *seen = (int64_t *)malloc(sizeof(int64_t) * (size_t)(N > 0 ? N : 1));
  for (int64_t i = 0; i < cap * nb; ++i) tab_key_id[i] = -1;
  for (int64_t i = 0; i < N; ++i) seen[i] = -1;
  int64_t retained = 0;
  double dh = 0.0;
  for (int64_t i = 0; i < N; ++i) {
    int64_t best = -1;
    double best_d = 0.0;
    for (int32_t b = 0; b < nb; ++b) {
      const uint64_t key = digests[i * nb + b];
      int64_t *tab = tab_key_id + (size_t)b * (size_t)cap;
      int64_t slot = (int64_t)(key & (uint64_t)(cap - 1));
      while (tab[slot] >= 0 && digests[tab[slot] * nb + b] != key) slot = (slot + 1) & (cap - 1);
      for (int64_t y = tab[slot]; y >= 0; y = prev[y * nb + b]) {
        if (seen[y] == i) continue; /* already a candidate through another band */
        seen[y] = i;
        if (best >= 0 && y > best) continue; /* cannot lower the representative */
        const double dd = l2_full(e + i * (int64_t)D, e + y * (int64_t)D, D);
        if (dd <= delta && (best < 0 || y < best)) {
          best = y;
          best_d = dd;
        }
      }
    }
    if (best >= 0) {
      rep[i] = (int32_t)best;
      dist[i] = best_d;
      if (best_d > dh) dh = best_d;
    } else {
      rep[i] = (int32_t)i;
      dist[i] = 0.0;
      ++retained;
      for (int32_t b = 0; b < nb; ++b) {
        const uint64_t key = digests[i * nb + b];
        int64_t *tab = tab_key_id + (size_t)b * (size_t)cap;
        int64_t slot = (int64_t)(key & (uint64_t)(cap - 1));
        while (tab[slot] >= 0 && digests[tab[slot] * nb + b] != key) slot = (slot + 1) & (cap - 1);
        prev[i * nb + b] = tab[slot] >= 0 ? (int32_t)tab[slot] : -1;
        tab[slot] = i;
      }
    }
  }
  free(tab_key_id);
  free(prev);
  free(seen);
  *delta_hat = dh;
  return retained;
}

/*
 * Error-bounded byte codec for retained embeddings (Sec. 3.2, layer L2:
 * "error-bounded byte compression" under a relative codec error bound; the
 * deployed bound is 1% of max|x|).  The paper uses a third-party codec; this
 * is a self-contained format of the same family, defined here:
 *   eb = fl32(rel * max|x_i|), s = fl32(2 eb) (s = 1 when every x_i is 0);
 *   q_i = Q(x_i) = rint_half_even(fl32(x_i / s)), exactly as the quantizer;
 *   blocks of 32 values; inside a block the deltas d_0 = q_0, d_j = q_j - q_{j-1}
 *   (a tail block is padded by repeating its last code, i.e. zero deltas);
 *   per block L = bit length of max_j |d_j| (0..31);
 *   layout: "LAMZ", n (int64 LE), s (fp32 LE), one byte L per block, zero
 *   padding to a multiple of 4 bytes, then for every block with L > 0 in
 *   order: a 32-bit sign word (bit j set when d_j < 0) and L 32-bit bit planes
 *   (bit j of plane p is bit p of |d_j|), all little-endian.
 * Decoding sums the deltas back into q and returns fl32(s * q): the error is
 * that of Q_eps at eps = eb.
 */
static int32_t bitlen_u32(uint32_t v) {
  int32_t b = 0;
  while (v) {
    ++b;
    v >>= 1;
  }
  return b;
}

static void put_u32(uint8_t *p, uint32_t v) {
  p[0] = (uint8_t)v;
  p[1] = (uint8_t)(v >> 8);
  p[2] = (uint8_t)(v >> 16);
  p[3] = (uint8_t)(v >> 24);
}

static uint32_t get_u32(const uint8_t *p) {
  return (uint32_t)p[0] | ((uint32_t)p[1] << 8) | ((uint32_t)p[2] << 16) | ((uint32_t)p[3] << 24);
}

/* Returns the compressed size; writes only when it fits in cap (out may be
 * NULL to ask for the size).  Returns -1 for a non-finite input. */
int64_t lam_oracle_lamz_compress(const float *x, int64_t n, float rel, uint8_t *out, int64_t cap) {
  int old_mode = fegetround();
  fesetround(FE_TONEAREST);
  float mx = 0.0f;
  for (int64_t i = 0; i < n; ++i) {
    if (!isfinite(x[i])) {
      fesetround(old_mode);
      return -1;
    }
    const float a = fabsf(x[i]);
    if (a > mx) mx = a;
  }
  const float eb = rel * mx;
  const float s = mx > 0.0f ? 2.0f * eb : 1.0f;
  const int64_t nb = (n + 31) / 32;
  const int64_t head = 16 + ((nb + 3) / 4) * 4;
  int64_t size = head;
  int32_t q[32], d[32];
  for (int pass = 0; pass < 2; ++pass) {
    int64_t pos = head;
    if (pass == 1) {
      if (out == NULL || size > cap) break;
      memset(out, 0, (size_t)head);
      out[0] = 'L';
      out[1] = 'A';
      out[2] = 'M';
      out[3] = 'Z';
      for (int k = 0; k < 8; ++k) out[4 + k] = (uint8_t)((uint64_t)n >> (8 * k));
      uint32_t sb;
      memcpy(&sb, &s, 4);
      put_u32(out + 12, sb);
    }
    for (int64_t b = 0; b < nb; ++b) {
      uint32_t mag_max = 0;
      for (int j = 0; j < 32; ++j) {
        const int64_t i = b * 32 + j;
        q[j] = i < n ? (int32_t)nearbyintf(x[i] / s) : q[j - 1];
        d[j] = j == 0 ? q[0] : q[j] - q[j - 1];
        const uint32_t m = (uint32_t)(d[j] < 0 ? -(int64_t)d[j] : d[j]);
        if (m > mag_max) mag_max = m;
      }
      const int32_t L = bitlen_u32(mag_max);
      if (pass == 0) {
        if (L > 0) size += 4 + 4 * (int64_t)L;
        continue;
      }
      out[16 + b] = (uint8_t)L;
      if (L == 0) continue;
      uint32_t sign = 0;
      for (int j = 0; j < 32; ++j)
        if (d[j] < 0) sign |= 1u << j;
      put_u32(out + pos, sign);
      pos += 4;
      for (int p = 0; p < L; ++p) {
        uint32_t plane = 0;
        for (int j = 0; j < 32; ++j) {
          const uint32_t m = (uint32_t)(d[j] < 0 ? -(int64_t)d[j] : d[j]);
          if ((m >> p) & 1u) plane |= 1u << j;
        }
        put_u32(out + pos, plane);
        pos += 4;
      }
    }
  }
  fesetround(old_mode);
  return size;
}

/* Decodes n values; returns 0, or -1 for a malformed or truncated stream. */
int32_t lam_oracle_lamz_decompress(const uint8_t *in, int64_t size, float *out, int64_t n) {
  if (size < 16 || in[0] != 'L' || in[1] != 'A' || in[2] != 'M' || in[3] != 'Z') return -1;
  uint64_t nn = 0;
  for (int k = 0; k < 8; ++k) nn |= (uint64_t)in[4 + k] << (8 * k);
  if ((int64_t)nn != n) return -1;
  const uint32_t sb = get_u32(in + 12);
  float s;
  memcpy(&s, &sb, 4);
  const int64_t nb = (n + 31) / 32;
  const int64_t head = 16 + ((nb + 3) / 4) * 4;
  if (size < head) return -1;
  int64_t pos = head;
  for (int64_t b = 0; b < nb; ++b) {
    const int32_t L = in[16 + b];
    if (L > 31 || pos + (L > 0 ? 4 + 4 * (int64_t)L : 0) > size) return -1;
    uint32_t sign = 0, planes[32];
    if (L > 0) {
      sign = get_u32(in + pos);
      pos += 4;
      for (int p = 0; p < L; ++p, pos += 4) planes[p] = get_u32(in + pos);
    }
    int32_t qv = 0;
    for (int j = 0; j < 32; ++j) {
      uint32_t m = 0;
      for (int p = 0; p < L; ++p) m |= ((planes[p] >> j) & 1u) << p;
      const int32_t dj = ((sign >> j) & 1u) ? -(int32_t)m : (int32_t)m;
      qv += dj;
      const int64_t i = b * 32 + j;
      if (i < n) out[i] = s * (float)qv;
    }
  }
  return 0;
}

/*
 * Alternative byte codecs of the composite experiment (App. "Composite
 * reduction": fp16, per-vector int8, sign-binary).  The paper names them and
 * their compression ratios only; the definitions taken here:
 *   fp16:            xhat = fp16(x) (round to nearest even).
 *   per-vector int8: lo = min_d x, hi = max_d x, scale = fl32((hi - lo) / 255),
 *                    c = rint_half_even(fl32(fl32(x - lo) / scale)) - 128 in
 *                    [-128, 127] (c = -128 when scale = 0), offset =
 *                    fl32(lo + 128 scale), xhat = fl32(offset + fl32(scale c));
 *                    two fp32 per row, i.e. 776 bytes for D = 768, the
 *                    paper's 3.96x.
 *   sign-binary:     bit b_d = (x_d >= 0), alpha = fl32(sum_d |x_d| / D)
 *                    summed in double, xhat = b ? alpha : -alpha; D/8 bytes
 *                    plus one fp32, the paper's 30.72x at D = 768.
 * Encoders write the codes and the per-row factors; lam_oracle_decode_rows
 * writes xhat.
 */
void lam_oracle_encode_int8_rows(const float *x, int64_t N, int32_t D, int8_t *codes,
                                 float *scale, float *offset) {
  int old_mode = fegetround();
  fesetround(FE_TONEAREST);
  for (int64_t i = 0; i < N; ++i) {
    const float *r = x + i * (int64_t)D;
    float lo = r[0], hi = r[0];
    for (int32_t d = 1; d < D; ++d) {
      if (r[d] < lo) lo = r[d];
      if (r[d] > hi) hi = r[d];
    }
    const float sc = (hi - lo) / 255.0f;
    for (int32_t d = 0; d < D; ++d) {
      int32_t c = -128;
      if (sc > 0.0f) {
        const float t = (r[d] - lo) / sc;
        c = (int32_t)nearbyintf(t) - 128;
        if (c < -128) c = -128;
        if (c > 127) c = 127;
      }
      codes[i * (int64_t)D + d] = (int8_t)c;
    }
    scale[i] = sc;
    offset[i] = lo + 128.0f * sc;
  }
  fesetround(old_mode);
}

void lam_oracle_encode_sign_rows(const float *x, int64_t N, int32_t D, uint8_t *bits,
                                 float *alpha) {
  for (int64_t i = 0; i < N; ++i) {
    const float *r = x + i * (int64_t)D;
    double a = 0.0;
    for (int32_t d = 0; d < D; ++d) a += fabs((double)r[d]);
    alpha[i] = (float)(a / (double)D);
    for (int32_t d = 0; d < D; d += 8) {
      uint8_t byte = 0;
      for (int t = 0; t < 8 && d + t < D; ++t)
        if (r[d + t] >= 0.0f) byte |= (uint8_t)(1u << t);
      bits[i * (int64_t)(D / 8) + d / 8] = byte;
    }
  }
}

/* fmt 1: int8 codes + scale + offset; fmt 2: fp16 bit patterns (uint16);
 * fmt 3: sign bits + alpha (in scale).  Writes xhat [N, D]. */
void lam_oracle_decode_rows(const void *codes, int32_t fmt, int64_t N, int32_t D,
                            const float *scale, const float *offset, float *out);

/* Scores [B, N] of queries against decoded rows xhat [N, D] (double, one
 * rounding; cosine 0 for a zero norm; squared L2 in the direct form). */
void lam_oracle_scores_rows(const float *queries, int64_t B, const float *rows, int64_t N,
                            int32_t D, int32_t metric, float *out) {
  for (int64_t b = 0; b < B; ++b) {
    const float *q = queries + b * (int64_t)D;
    for (int64_t i = 0; i < N; ++i) {
      const float *x = rows + i * (int64_t)D;
      double dot = 0.0, qq = 0.0, xx = 0.0, l2 = 0.0;
      if (metric == ORACLE_L2) {
        for (int32_t d = 0; d < D; ++d) {
          const double df = (double)q[d] - (double)x[d];
          l2 += df * df;
        }
      } else {
        for (int32_t d = 0; d < D; ++d) dot += (double)q[d] * (double)x[d];
      }
      if (metric == ORACLE_COSINE)
        for (int32_t d = 0; d < D; ++d) {
          qq += (double)q[d] * (double)q[d];
          xx += (double)x[d] * (double)x[d];
        }
      float v;
      if (metric == ORACLE_IP) v = (float)dot;
      else if (metric == ORACLE_COSINE) v = (qq == 0.0 || xx == 0.0) ? 0.0f : (float)(dot / (sqrt(qq) * sqrt(xx)));
      else v = (float)l2;
      out[b * N + i] = v;
    }
  }
}

/* Score of one query against one dequantised row, in double, rounded to fp32. */
static float score_one(const float *q, const int32_t *c, int32_t D, float s,
                       int metric) {
  if (metric == ORACLE_IP) {
    double acc = 0.0;
    for (int32_t d = 0; d < D; ++d) {
      float xh = s * (float)c[d];
      acc += (double)q[d] * (double)xh;
    }
    return (float)acc;
  }
  if (metric == ORACLE_COSINE) {
    double dot = 0.0, qq = 0.0, xx = 0.0;
    for (int32_t d = 0; d < D; ++d) {
      float xh = s * (float)c[d];
      dot += (double)q[d] * (double)xh;
      qq += (double)q[d] * (double)q[d];
      xx += (double)xh * (double)xh;
    }
    if (qq == 0.0 || xx == 0.0) return 0.0f;
    return (float)(dot / (sqrt(qq) * sqrt(xx)));
  }
  /* squared L2, direct form */
  double acc = 0.0;
  for (int32_t d = 0; d < D; ++d) {
    float xh = s * (float)c[d];
    double diff = (double)q[d] - (double)xh;
    acc += diff * diff;
  }
  return (float)acc;
}

/* Scores of B queries [B, D] against N code rows [N, D]: out [B, N]. */
void lam_oracle_scores(const float *queries, int64_t B, const int32_t *codes,
                       int64_t N, int32_t D, float eps, int32_t metric,
                       float *out) {
  float s = lam_oracle_step(eps);
  for (int64_t b = 0; b < B; ++b)
    for (int64_t i = 0; i < N; ++i)
      out[b * N + i] =
          score_one(queries + b * (int64_t)D, codes + i * (int64_t)D, D, s,
                    metric);
}

/* ---- top-k: full sort of (score, id), best first, ties by lower id ---- */

typedef struct {
  float score;
  int64_t id;
} scored_t;

static int cmp_desc(const void *a, const void *b) {
  const scored_t *x = (const scored_t *)a, *y = (const scored_t *)b;
  if (x->score > y->score) return -1;
  if (x->score < y->score) return 1;
  return (x->id < y->id) ? -1 : (x->id > y->id);
}

static int cmp_asc(const void *a, const void *b) {
  const scored_t *x = (const scored_t *)a, *y = (const scored_t *)b;
  if (x->score < y->score) return -1;
  if (x->score > y->score) return 1;
  return (x->id < y->id) ? -1 : (x->id > y->id);
}

/* Top-k of one row of N scores. */
static void topk_row(const float *scores, int64_t N, int32_t k, int32_t metric,
                     scored_t *tmp, float *out_scores, int64_t *out_ids) {
  for (int64_t i = 0; i < N; ++i) {
    tmp[i].score = scores[i];
    tmp[i].id = i;
  }
  qsort(tmp, (size_t)N, sizeof(scored_t),
        metric == ORACLE_L2 ? cmp_asc : cmp_desc);
  for (int32_t j = 0; j < k; ++j) {
    out_scores[j] = tmp[j].score;
    out_ids[j] = tmp[j].id;
  }
}

/* Top-k of B rows of N given scores: out [B, k]. Returns 0 on success. */
int lam_oracle_topk(const float *scores, int64_t B, int64_t N, int32_t k,
                    int32_t metric, float *out_scores, int64_t *out_ids) {
  if (k < 1 || k > N) return 1;
  scored_t *tmp = (scored_t *)malloc(sizeof(scored_t) * (size_t)N);
  if (!tmp) return 2;
  for (int64_t b = 0; b < B; ++b)
    topk_row(scores + b * N, N, k, metric, tmp, out_scores + b * (int64_t)k,
             out_ids + b * (int64_t)k);
  free(tmp);
  return 0;
}

/* ---- exhaustive search driver: score + top-k, threads split the work ---- */

typedef struct {
  const float *queries;
  const int32_t *codes;
  int64_t N;
  int32_t D;
  float s;
  int32_t metric;
  int32_t k;
  int64_t B;
  float *out_scores;
  int64_t *out_ids;
  /* scratch for the query being processed collectively */
  float *row_scores;
  int nthreads;
  int tid;
  int64_t b_single; /* query index for the row-split phase */
  int phase;        /* 0: whole queries per thread; 1: rows of b_single */
  int status;
} search_job_t;

static void *search_worker(void *arg) {
  search_job_t *j = (search_job_t *)arg;
  if (j->phase == 1) {
    /* rows [lo, hi) of one query */
    int64_t lo = j->N * j->tid / j->nthreads;
    int64_t hi = j->N * (j->tid + 1) / j->nthreads;
    const float *q = j->queries + j->b_single * (int64_t)j->D;
    for (int64_t i = lo; i < hi; ++i)
      j->row_scores[i] = score_one(q, j->codes + i * (int64_t)j->D, j->D, j->s,
                                   j->metric);
    return NULL;
  }
  float *scores = (float *)malloc(sizeof(float) * (size_t)j->N);
  scored_t *tmp = (scored_t *)malloc(sizeof(scored_t) * (size_t)j->N);
  if (!scores || !tmp) {
    j->status = 2;
    free(scores);
    free(tmp);
    return NULL;
  }
  for (int64_t b = j->tid; b < j->B; b += j->nthreads) {
    const float *q = j->queries + b * (int64_t)j->D;
    for (int64_t i = 0; i < j->N; ++i)
      scores[i] = score_one(q, j->codes + i * (int64_t)j->D, j->D, j->s,
                            j->metric);
    topk_row(scores, j->N, j->k, j->metric, tmp,
             j->out_scores + b * (int64_t)j->k, j->out_ids + b * (int64_t)j->k);
  }
  free(scores);
  free(tmp);
  return NULL;
}

/*
 * Exact search: for each of B queries, score all N dequantised rows and keep
 * the k best (Sec. "Brute-force scan crossover": a matrix-vector product per
 * query).  nthreads worker threads: whole queries per thread when B >= the
 * thread count, otherwise the rows of each query are split across threads.
 * Returns 0 on success.
 */
int lam_oracle_search(const float *queries, int64_t B, const int32_t *codes,
                      int64_t N, int32_t D, float eps, int32_t metric,
                      int32_t k, float *out_scores, int64_t *out_ids,
                      int32_t nthreads) {
  if (k < 1 || k > N || D < 1 || B < 0) return 1;
  if (nthreads < 1) nthreads = 1;
  float s = lam_oracle_step(eps);
  pthread_t *th = (pthread_t *)malloc(sizeof(pthread_t) * (size_t)nthreads);
  search_job_t *jobs =
      (search_job_t *)calloc((size_t)nthreads, sizeof(search_job_t));
  if (!th || !jobs) {
    free(th);
    free(jobs);
    return 2;
  }
  int status = 0;
  for (int t = 0; t < nthreads; ++t) {
    jobs[t].queries = queries;
    jobs[t].codes = codes;
    jobs[t].N = N;
    jobs[t].D = D;
    jobs[t].s = s;
    jobs[t].metric = metric;
    jobs[t].k = k;
    jobs[t].B = B;
    jobs[t].out_scores = out_scores;
    jobs[t].out_ids = out_ids;
    jobs[t].nthreads = nthreads;
    jobs[t].tid = t;
  }
  if (B >= nthreads) {
    for (int t = 0; t < nthreads; ++t) {
      jobs[t].phase = 0;
      pthread_create(&th[t], NULL, search_worker, &jobs[t]);
    }
    for (int t = 0; t < nthreads; ++t) {
      pthread_join(th[t], NULL);
      if (jobs[t].status) status = jobs[t].status;
    }
  } else {
    float *row_scores = (float *)malloc(sizeof(float) * (size_t)N);
    scored_t *tmp = (scored_t *)malloc(sizeof(scored_t) * (size_t)N);
    if (!row_scores || !tmp) {
      free(row_scores);
      free(tmp);
      free(th);
      free(jobs);
      return 2;
    }
    for (int64_t b = 0; b < B; ++b) {
      for (int t = 0; t < nthreads; ++t) {
        jobs[t].phase = 1;
        jobs[t].b_single = b;
        jobs[t].row_scores = row_scores;
        pthread_create(&th[t], NULL, search_worker, &jobs[t]);
      }
      for (int t = 0; t < nthreads; ++t) pthread_join(th[t], NULL);
      topk_row(row_scores, N, k, metric, tmp, out_scores + b * (int64_t)k,
               out_ids + b * (int64_t)k);
    }
    free(row_scores);
    free(tmp);
  }
  free(th);
  free(jobs);
  return status;
}

/* IEEE binary16 bit pattern to float (exact). */
static float half_to_float(uint16_t h) {
  const uint32_t sign = (uint32_t)(h >> 15) << 31;
  const int32_t e = (h >> 10) & 0x1f;
  const uint32_t m = h & 0x3ffu;
  float v;
  if (e == 0) {
    v = ldexpf((float)m, -24); /* subnormal (or zero) */
  } else if (e == 31) {
    v = m ? NAN : INFINITY;
  } else {
    v = ldexpf((float)(m | 0x400u), e - 25);
  }
  return sign ? -v : v;
}

void lam_oracle_decode_rows(const void *codes, int32_t fmt, int64_t N, int32_t D,
                            const float *scale, const float *offset, float *out) {
  for (int64_t i = 0; i < N; ++i) {
    for (int32_t d = 0; d < D; ++d) {
      float v = 0.0f;
      if (fmt == 1) {
        const int8_t c = ((const int8_t *)codes)[i * (int64_t)D + d];
        v = offset[i] + scale[i] * (float)c;
      } else if (fmt == 2) {
        v = half_to_float(((const uint16_t *)codes)[i * (int64_t)D + d]);
      } else {
        const uint8_t byte = ((const uint8_t *)codes)[i * (int64_t)(D / 8) + d / 8];
        v = ((byte >> (d % 8)) & 1u) ? scale[i] : -scale[i];
      }
      out[i * (int64_t)D + d] = v;
    }
  }
}
