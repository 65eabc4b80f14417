/*
 * Oracle weight draws in plain C (test infrastructure only; nothing on the
 * product path links this file).
 *
 * The same definition as oracle/weights.py, written in C so that the weights
 * of the full-size 8B- and 7B-shaped random-init models (about 7e9 draws) can
 * be generated in seconds on the host:
 *
 *   SplitMix64 (Steele, Lea & Flood, OOPSLA 2014): output n (n = 0, 1, ...) of
 *   the stream with state s is mix(s + (n + 1) * GAMMA), with the published
 *   mix function (xor-shift 30 / 27 / 31 and two odd multipliers).
 *
 *   Basic Box-Muller (Box & Muller 1958): element pair (2j, 2j + 1) takes
 *   u0 = out[2j], u1 = out[2j + 1]; a = ((u0 >> 11) + 1) 2^-53 in (0, 1],
 *   b = (u1 >> 11) 2^-53; r = sqrt(-2 ln a); z[2j] = r cos(2 pi b),
 *   z[2j + 1] = r sin(2 pi b).  Arithmetic in double precision.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

static const uint64_t GAMMA = 0x9E3779B97F4A7C15ull;

static uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

/* Round a double to the nearest bfloat16 value (ties to even), kept as a
 * double: the significand is cut to 8 bits directly, as oracle/weights.py's
 * round_bf16 does (valid in the bfloat16 normal range and for 0). */
static double round_bf16(double x) {
  uint64_t b;
  memcpy(&b, &x, 8);
  const uint64_t lsb = (b >> 45) & 1u;
  b = (b + ((1ull << 44) - 1) + lsb) & ~((1ull << 45) - 1);
  memcpy(&x, &b, 8);
  return x;
}

static double store(double x, int mode) {
  if (mode == 1) return (double)(float)x; /* float32, round to nearest even */
  if (mode == 2) return round_bf16(x);
  return x;
}

/* out[i] = store(scale * z[n0 + i]) for i < count: standard-normal draws of the
 * tensor stream with state `state`, element n0 onwards (n0 may be odd), rounded
 * to the storage type `mode` (0: none, 1: float32, 2: bfloat16). */
void oracle_normal_range(uint64_t state, int64_t n0, int64_t count, double scale, int mode, double* out) {
  const double tau = 6.283185307179586476925286766559;
  int64_t n = n0;
  const int64_t end = n0 + count;
  while (n < end) {
    const int64_t j = n / 2;
    const uint64_t u0 = mix64(state + (uint64_t)(2 * j + 1) * GAMMA);
    const uint64_t u1 = mix64(state + (uint64_t)(2 * j + 2) * GAMMA);
    const double a = (double)((u0 >> 11) + 1) * 0x1p-53;
    const double b = (double)(u1 >> 11) * 0x1p-53;
    const double r = sqrt(-2.0 * log(a));
    const double t = tau * b;
    if (n == 2 * j) out[n - n0] = store(scale * (r * cos(t)), mode);
    if (2 * j + 1 < end && 2 * j + 1 >= n0) out[2 * j + 1 - n0] = store(scale * (r * sin(t)), mode);
    n = 2 * j + 2;
  }
}

/* out[i] = the storage rounding `mode` of in[i] (the rounding the draws use). */
void oracle_round(const double* in, int64_t n, int mode, double* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = store(in[i], mode);
}
