/* Host check of the quotient scheme the quantize kernels use (QDiv): for a
 * divisor s and y = RN(1/s), q0 = RN(x y), then twice q <- RN(q + RN(x - s q) y)
 * with fused multiply-adds, must equal the IEEE single division RN(x / s)
 * (Markstein's theorem), with the division itself outside s in [2^-40, 2^40]
 * and for |q0| >= 2^100.  Below |x| = 2^-80 only the rounded code is compared.
 * Built with -DNO_REFINE the quotient is the plain reciprocal product x y
 * (which is not enough: the check must then find mismatches).
 * Usage: fma_quotient_check <samples per divisor>; prints the number of
 * values checked, quotient mismatches and code mismatches. */
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

static float f_of(uint32_t u) {
  float f;
  memcpy(&f, &u, 4);
  return f;
}
static uint32_t u_of(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  return u;
}
static uint64_t next64(uint64_t *st) { /* splitmix64 */
  uint64_t z = (*st += 0x9E3779B97F4A7C15ULL);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}
static volatile float sink;

int main(int argc, char **argv) {
  const long per = argc > 1 ? atol(argv[1]) : 1L << 20;
  const float ss[] = {0.02f, 0.002f, 0.0002f, 0.2f, 3.0f, 0x1.fffffep+0f, 0x1p-40f, 0x1p40f, 0.0123457f};
  long bad_q = 0, bad_c = 0, checked = 0;
  uint64_t st = 12345;
  for (unsigned k = 0; k < sizeof(ss) / sizeof(ss[0]); ++k) {
    const volatile float sv = ss[k];
    const float s = sv;
    const float y = 1.0f / s;
    const int fast = s >= 0x1p-40f && s <= 0x1p40f;
    for (long i = 0; i < per; ++i) {
      uint32_t u = (uint32_t)next64(&st);
      /* half the samples next to a quotient midpoint (k + 1/2) s */
      if (i & 1) {
        const double m = ((double)(int32_t)(u >> 8) * 0.25 + 0.5) * (double)s;
        u = u_of((float)m) + (uint32_t)((int32_t)(u & 7) - 3);
      }
      const float x = f_of(u);
      if (!isfinite(x)) continue;
      const float ref = x / s;
      float q = x * y;
      if (fast && fabsf(q) < 0x1p100f) {
#ifndef NO_REFINE
        q = fmaf(fmaf(-s, q, x), y, q);
        q = fmaf(fmaf(-s, q, x), y, q);
#endif
      } else {
        q = x / s;
      }
      sink = q;
      ++checked;
      if (u_of(q) != u_of(ref)) {
        if (fabsf(x) >= 0x1p-80f) ++bad_q;
        if (rintf(q) != rintf(ref)) ++bad_c;
      }
    }
  }
  printf("%ld %ld %ld\n", checked, bad_q, bad_c);
  return 0;
}
