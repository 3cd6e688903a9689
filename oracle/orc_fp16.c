/*
 * ORACLE -- test infrastructure only.  Nothing on the product path may link,
 * load or call this code; only tests/, __graft_entry__.smoke() and bench.py's
 * CPU-baseline leg do.
 *
 * IEEE-754 binary16 codec written from the format definition (paper Sec. 3,
 * "Precision Standard": one sign bit, an exponent field with a bias, and a
 * fraction field; the standard's arithmetic ops).  binary16 has a 5-bit
 * exponent with bias 15 and a 10-bit fraction:
 *   e = 0      : subnormal, value = f * 2^-24 (f = 0 is a signed zero)
 *   e = 1..30  : normal,    value = (1024 + f) * 2^(e - 25)
 *   e = 31     : f = 0 infinity, f != 0 NaN
 * Rounding is roundTiesToEven, the IEEE default (the paper names IEEE 754
 * and no other mode).
 *
 * A single IEEE op on two binary16 operands computed in binary64 and then
 * rounded once to binary16 gives the correctly rounded binary16 result:
 * sums, differences and products of binary16 values are exact in binary64,
 * and for division / square root binary64 has 53 >= 2*11 + 2 bits, so the
 * double rounding is innocuous.  orc_h_* use this.
 */
#include <math.h>
#include <stdint.h>

#include "oracle.h"

double orc_f16_to_f64(uint16_t h) {
  const int s = h >> 15;
  const int e = (h >> 10) & 0x1F;
  const int f = h & 0x3FF;
  double v;
  if (e == 0)
    v = ldexp((double)f, -24);
  else if (e == 31)
    v = f ? NAN : INFINITY;
  else
    v = ldexp((double)(1024 + f), e - 25);
  return s ? -v : v;
}

uint16_t orc_f64_to_f16(double x) {
  if (isnan(x)) return 0x7E00;
  const uint16_t sign = signbit(x) ? 0x8000 : 0;
  const double a = fabs(x);
  /* 65504 is the largest finite value; half its quantum above it (65520)
     is the tie, which rounds to the even significand 2048 * 32 = overflow. */
  if (a >= 65520.0) return sign | 0x7C00;
  int E;
  frexp(a, &E); /* a = m * 2^E, m in [0.5, 1): floor(log2 a) = E - 1 */
  int e = (a == 0.0) ? -14 : E - 1;
  if (e < -14) e = -14; /* subnormal range shares the quantum 2^-24 */
  const double q = ldexp(1.0, e - 10);
  const double r = nearbyint(a / q); /* a / q is exact; ties to even */
  const double v = r * q;
  if (v == 0.0) return sign;
  if (v < ldexp(1.0, -14)) return sign | (uint16_t)r; /* subnormal */
  frexp(v, &E);
  e = E - 1;
  const int mant = (int)ldexp(v, 10 - e) - 1024;
  return sign | (uint16_t)((e + 15) << 10) | (uint16_t)mant;
}

static double g_lut[65536];
static int g_lut_ready = 0;

const double* orc_f16_lut(void) {
  if (!g_lut_ready) {
    for (int i = 0; i < 65536; ++i) g_lut[i] = orc_f16_to_f64((uint16_t)i);
    g_lut_ready = 1;
  }
  return g_lut;
}

void orc_f16_decode(const uint16_t* h, double* out, int64_t n) {
  const double* lut = orc_f16_lut();
  for (int64_t i = 0; i < n; ++i) out[i] = lut[h[i]];
}

void orc_f16_encode(const double* x, uint16_t* out, int64_t n) {
  for (int64_t i = 0; i < n; ++i) out[i] = orc_f64_to_f16(x[i]);
}

uint16_t orc_h_add(uint16_t a, uint16_t b) { return orc_f64_to_f16(orc_f16_to_f64(a) + orc_f16_to_f64(b)); }
uint16_t orc_h_sub(uint16_t a, uint16_t b) { return orc_f64_to_f16(orc_f16_to_f64(a) - orc_f16_to_f64(b)); }
uint16_t orc_h_mul(uint16_t a, uint16_t b) { return orc_f64_to_f16(orc_f16_to_f64(a) * orc_f16_to_f64(b)); }
