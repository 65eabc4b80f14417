// Integer pieces of the logits -> frequency rule shared by the quantiser and
// the coders (the rule itself is written out at the top of quantize.cu):
// codes q = rint_even(min(fl32(fl32(m - l) C), 8191)), weights
// w(q) = T[q & 255] >> (q >> 8), and floor(w R / W) without a division.
#pragma once

#include "common.cuh"
#include "exp_table.inc"

namespace dlmz {

__device__ __forceinline__ uint32_t quant_w(const uint32_t* T, int q) { return T[q & 255] >> (q >> 8); }

// w(q) = T[q & 255] >> (q >> 8) is 0 for q > 7936 (T[j] < 2^31 for j >= 1; w(7936) = T[0] >> 31 = 1):
// those codes add nothing to W, A or D and need no bin
constexpr int QW0 = 31 * 256 + 1;
constexpr uint32_t QMAGIC = 0x4B400000u;  // bit pattern of 1.5 * 2^23

// QMAGIC + min(q, QW0) for d = fl32(m - l) >= 0, q = rint_even(min(fl32(d C), 8191)): clamping at
// QW0 before the rounding is the same as after it (QW0 is an integer), and every code >= QW0
// weighs nothing (NaN or +inf d land there too)
__device__ __forceinline__ uint32_t code_bits(float d) {
  const float t = fminf(__fmul_rn(d, __uint_as_float(DLMZ_QSCALE_BITS)), (float)QW0);
  return __float_as_uint(__fadd_rn(t, 12582912.0f));
}

// min(q, QW0) for d = m - l from a maximum m read back from memory: an unsigned clamp keeps the
// index in the table even if d were negative
__device__ __forceinline__ uint32_t code_index(float d) { return min(code_bits(d) - QMAGIC, (uint32_t)QW0); }

// floor(w R / W) from K = floor(R 2^64 / W) (R < W): the estimate (w K) >> 64 is the floor or
// one less, and (e + 1) W <= w R (both sides < 2^64) decides which
__device__ __forceinline__ uint32_t floor_wr_over_w(uint32_t w, uint32_t R, uint64_t Wsum, uint64_t K) {
  const uint64_t lo = (uint64_t)w * (uint32_t)K;          // w * K_lo
  const uint64_t hi = (uint64_t)w * (uint32_t)(K >> 32);  // w * K_hi
  const uint32_t est = (uint32_t)((hi + (lo >> 32)) >> 32);
  const uint64_t x = (uint64_t)w * R;
  return est + (((uint64_t)(est + 1) * Wsum) <= x ? 1u : 0u);
}

// K = floor(R 2^64 / W) for 0 < R < W < 2^53: a float64 estimate K0 (|K0 - K| <= 17: R / W is
// rounded once, and K < 2^57), then the exact remainder R 2^64 - K0 W (a signed 128-bit value
// whose high word is 0 or -1 here) corrects it in one float64 step and at most two unit steps.
__device__ __forceinline__ uint64_t recip_scaled(uint32_t R, uint64_t W) {
  const double e = ldexp((double)R / (double)W, 64);
  uint64_t K = e >= 18446744073709551615.0 ? ~0ull : (uint64_t)e;
  auto rem = [&](uint64_t k) -> int64_t {  // R 2^64 - k W; |value| < 2^62 when |k - K| <= 20
    const uint64_t plo = k * W;
    return (int64_t)(0ull - plo);  // the high word R - hi(k W) - borrow is its sign extension
  };
  K += (uint64_t)(int64_t)floor((double)rem(K) / (double)W);
  for (int it = 0; it < 4; ++it) {
    const int64_t rr = rem(K);
    if (rr < 0) --K;
    else if ((uint64_t)rr >= W) ++K;
    else break;
  }
  return K;
}

}  // namespace dlmz
