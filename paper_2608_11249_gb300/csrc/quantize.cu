// Logits -> integer frequency tables, CDFs and scores.
//
// The statistical coder (Sec. 2.1; Sec. 4 "Implementation Details") needs
// integer tables that encoder and decoder rebuild bit-identically from the
// same logits.  Per row l[0..V):
//   m = max l, top = lowest v with l_v = m
//   q_v = rint_even(min(fl32(fl32(m - l_v) * C), 8191)),  C = fl32(256 log2 e)
//   w_v = T[q_v & 255] >> (q_v >> 8),   T[j] = round(2^31 2^(-j/256))
//   W = sum w_v, A = sum w_v q_v (exact 64-bit integer sums: order-free)
//   R = 2^P - V, f_v = 1 + floor(w_v R / W), f_top += R - sum floor(w_v R / W)
//   H_q = log2q16(W) - 31*2^16 + floor(2^8 A / W)      (entropy, Sec. 3.3, 2^-16 bit)
// Only __fsub_rn / __fmul_rn / __float2int_rn touch floating point, so the
// result is independent of thread layout and reduction order.
#include <type_traits>

#include "kernels.cuh"
#include "exp_table.inc"
#include "intq.cuh"

namespace dlmz {

__constant__ uint32_t c_exp_table[256] = DLMZ_EXP_TABLE_INIT;

__device__ __forceinline__ int quant_q(float m, float l) {
  const float t = __fmul_rn(__fsub_rn(m, l), __uint_as_float(DLMZ_QSCALE_BITS));
  return __float2int_rn(fminf(t, 8191.0f));
}


// Digit-by-digit binary logarithm: ~floor(2^16 log2 W) for W >= 2^31.
__device__ __forceinline__ uint32_t log2q16(uint64_t W) {
  const int n = 63 - __clzll((long long)W);
  uint64_t y = W >> (n - 31);
  uint32_t frac = 0;
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    y = (y * y) >> 31;
    frac <<= 1;
    if (y >= (1ull << 32)) {
      frac |= 1;
      y >>= 1;
    }
  }
  return ((uint32_t)n << 16) + frac;
}

__device__ __forceinline__ int32_t entropy_q(uint64_t W, uint64_t A) {
  const uint64_t qt = A / W, rm = A % W;
  return (int32_t)((int64_t)log2q16(W) - (31ll << 16) + (int64_t)((qt << 8) + ((rm << 8) / W)));
}

__device__ __forceinline__ void argmax_merge(float& m, int& i, float m2, int i2) {
  if (m2 > m || (m2 == m && i2 < i)) {
    m = m2;
    i = i2;
  }
}

// ---- warp per row, V <= 32 * NPL, values in registers ------------------------------
template <int NPL>
__global__ void __launch_bounds__(256) quantize_warp_kernel(const float* __restrict__ logits, int rows, int V, int P,
                                                            uint32_t* __restrict__ cdf, uint64_t* __restrict__ Wout,
                                                            uint64_t* __restrict__ Aout, int32_t* __restrict__ Hq,
                                                            int32_t* __restrict__ topout, float* __restrict__ mxout,
                                                            int* err) {
  __shared__ uint32_t T[256];
  for (int i = threadIdx.x; i < 256; i += blockDim.x) T[i] = c_exp_table[i];
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  if (r >= rows) return;
  const float* lr = logits + (size_t)r * V;
  float x[NPL];
  float m = -INFINITY;
  int mi = 0x7fffffff;
  bool finite = true;
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    const int v = lane + 32 * i;
    x[i] = v < V ? lr[v] : -INFINITY;
    if (v < V) {
      finite &= isfinite(x[i]);
      argmax_merge(m, mi, x[i], v);
    }
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const int i2 = __shfl_xor_sync(0xffffffffu, mi, o);
    argmax_merge(m, mi, m2, i2);
  }
  const bool bad = !__all_sync(0xffffffffu, finite);
  if (bad) {  // the call reports EBADINPUT; m = +inf sends every code to 8191, W is pinned below
    if (lane == 0) atomicOr(err, ERR_NONFINITE);
    m = INFINITY;
  }
  uint32_t w[NPL];
  uint64_t Ws = 0, As = 0;
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    const int v = lane + 32 * i;
    if (v < V) {
      const int q = isfinite(x[i]) ? quant_q(m, x[i]) : 8191;
      w[i] = quant_w(T, q);
      Ws += w[i];
      As += (uint64_t)w[i] * (uint64_t)q;
    } else {
      w[i] = 0;
    }
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    Ws += __shfl_xor_sync(0xffffffffu, Ws, o);
    As += __shfl_xor_sync(0xffffffffu, As, o);
  }
  if (bad) {  // every w is 0: any W >= 2^31 keeps the tables defined
    Ws = 1ull << 31;
    As = 0;
  }
  if (lane == 0) {
    Wout[r] = Ws;
    if (Aout) Aout[r] = As;
    Hq[r] = entropy_q(Ws, As);
    if (topout) topout[r] = mi;
    if (mxout) mxout[r] = m;
  }
  if (!cdf) return;
  const uint64_t R = (1ull << P) - (uint64_t)V;
  uint64_t fl[NPL];
  uint64_t fsum = 0;
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    fl[i] = (uint64_t)w[i] * R / Ws;
    fsum += fl[i];
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) fsum += __shfl_xor_sync(0xffffffffu, fsum, o);
  const uint32_t D = (uint32_t)(R - fsum);
  uint32_t* cr = cdf + (size_t)r * (V + 1);
  uint32_t carry = 0;
#pragma unroll
  for (int i = 0; i < NPL; ++i) {
    const int v = lane + 32 * i;
    uint32_t f = v < V ? 1u + (uint32_t)fl[i] + (v == mi ? D : 0u) : 0u;
    uint32_t inc = f;  // inclusive scan across the warp
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t t = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += t;
    }
    if (v < V) cr[v + 1] = carry + inc;
    carry += __shfl_sync(0xffffffffu, inc, 31);
  }
  if (lane == 0) cr[0] = 0;
}

// ---- CTA per row, any V: passes over the row through L1/L2 ---------------------------
template <typename U>
__device__ __forceinline__ U block_sum(U v, U* red) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31, nw = blockDim.x >> 5;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  U t = 0;
  for (int i = 0; i < nw; ++i) t += red[i];
  return t;
}

constexpr int QT = 512;  // threads per row in the CTA kernel

__global__ void __launch_bounds__(QT) quantize_cta_kernel(const float* __restrict__ logits, int rows, int V, int P,
                                                         uint32_t* __restrict__ cdf, uint64_t* __restrict__ Wout,
                                                         uint64_t* __restrict__ Aout, int32_t* __restrict__ Hq,
                                                         int32_t* __restrict__ topout, float* __restrict__ mxout,
                                                         int* err) {
  __shared__ uint32_t T[256];
  __shared__ float redf[QT / 32];
  __shared__ int redi[QT / 32];
  __shared__ uint64_t redu[QT / 32];
  __shared__ uint64_t seg[QT];
  for (int i = threadIdx.x; i < 256; i += blockDim.x) T[i] = c_exp_table[i];
  const int r = blockIdx.x;
  const float* lr = logits + (size_t)r * V;
  // pass 1: max / lowest argmax / finiteness
  float m = -INFINITY;
  int mi = 0x7fffffff;
  int bad = 0;
  for (int v = threadIdx.x; v < V; v += QT) {
    const float x = lr[v];
    bad |= !isfinite(x);
    argmax_merge(m, mi, x, v);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    argmax_merge(m, mi, __shfl_xor_sync(0xffffffffu, m, o), __shfl_xor_sync(0xffffffffu, mi, o));
    bad |= __shfl_xor_sync(0xffffffffu, bad, o);
  }
  if ((threadIdx.x & 31) == 0) {
    redf[threadIdx.x >> 5] = m;
    redi[threadIdx.x >> 5] = mi | (bad ? 0x80000000 : 0);
  }
  __syncthreads();
  m = -INFINITY;
  mi = 0x7fffffff;
  bad = 0;
  for (int i = 0; i < QT / 32; ++i) {
    bad |= redi[i] < 0;
    argmax_merge(m, mi, redf[i], redi[i] & 0x7fffffff);
  }
  if (bad) {  // as in the warp kernel: every code 8191, W pinned to 2^31
    if (threadIdx.x == 0) atomicOr(err, ERR_NONFINITE);
    m = INFINITY;
  }
  // pass 2: W, A
  uint64_t Ws = 0, As = 0;
  for (int v = threadIdx.x; v < V; v += QT) {
    const float x = lr[v];
    const int q = isfinite(x) ? quant_q(m, x) : 8191;
    const uint32_t w = quant_w(T, q);
    Ws += w;
    As += (uint64_t)w * (uint64_t)q;
  }
  Ws = block_sum(Ws, redu);
  As = block_sum(As, redu);
  if (bad) {
    Ws = 1ull << 31;
    As = 0;
  }
  if (threadIdx.x == 0) {
    Wout[r] = Ws;
    if (Aout) Aout[r] = As;
    Hq[r] = entropy_q(Ws, As);
    if (topout) topout[r] = mi;
    if (mxout) mxout[r] = m;
  }
  if (!cdf) return;
  // pass 3: per-thread contiguous segment sums of f (without the remainder)
  const uint64_t R = (1ull << P) - (uint64_t)V;
  const int segl = (V + QT - 1) / QT;
  const int v0 = threadIdx.x * segl, v1 = min(V, v0 + segl);
  uint64_t s = 0;
  for (int v = v0; v < v1; ++v) {
    const float x = lr[v];
    const int q = isfinite(x) ? quant_q(m, x) : 8191;
    s += 1 + (uint64_t)quant_w(T, q) * R / Ws;
  }
  seg[threadIdx.x] = s;
  __syncthreads();
  // exclusive scan of the segment sums (QT entries, one warp)
  if (threadIdx.x < 32) {
    uint64_t run = 0;
    for (int base = 0; base < QT; base += 32) {
      uint64_t val = seg[base + threadIdx.x], inc = val;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint64_t t = __shfl_up_sync(0xffffffffu, inc, o);
        if (threadIdx.x >= o) inc += t;
      }
      seg[base + threadIdx.x] = run + inc - val;
      run += __shfl_sync(0xffffffffu, inc, 31);
    }
    if (threadIdx.x == 0) redu[0] = run;
  }
  __syncthreads();
  const uint32_t D = (uint32_t)((1ull << P) - redu[0]);
  // pass 4: write the CDF (remainder D added from top + 1 on)
  uint32_t* cr = cdf + (size_t)r * (V + 1);
  uint64_t c = seg[threadIdx.x] + (v0 > mi ? D : 0);
  for (int v = v0; v < v1; ++v) {
    const float x = lr[v];
    const int q = isfinite(x) ? quant_q(m, x) : 8191;
    c += 1 + (uint64_t)quant_w(T, q) * R / Ws + (v == mi ? D : 0);
    cr[v + 1] = (uint32_t)c;
  }
  if (threadIdx.x == 0) cr[0] = 0;
}

// ---- large vocabularies (V % 4 == 0): persistent, CPS CTAs of NT threads per SM ----------
// A CTA walks rows r = blockIdx.x, blockIdx.x + gridDim.x, ...; with CPS rows
// per SM in flight the row stays in L2 after the first pass (from HBM), and
// the CTAs of an SM drift apart, so one row's compute-heavy CDF pass overlaps
// another's HBM-bound first pass.  Every per-element quantity is a function
// of the integer code q in [0, 8191] alone, so the second pass only builds a
// histogram of q: W = sum hist[q] w(q), A = sum hist[q] w(q) q and the
// remainder D = R - sum hist[q] floor(w(q) R / W) come from the 8192 bins, and
// the CDF pass looks floor(w(q) R / W) up in the same shared table, rewritten
// in place.  Every CDF partial sum is at most 2^P <= 2^24, so the scan runs
// in 32-bit integers.
// floor(w R / W) without a division: K = floor(R 2^64 / W) per row (R < W); see intq.cuh.
constexpr int NQ = 8192;       // codes q = 0 .. 8191
constexpr int QNT = 256;       // threads per CTA
constexpr int QCPS = 4;        // CTAs per SM (4 x 33 KB shared memory, 64 registers per thread)

template <int NT, int CPS>
__global__ void __launch_bounds__(NT, CPS)
    quantize_persist_kernel(const float* __restrict__ logits, int rows, int V, int P, uint32_t* __restrict__ cdf,
                            uint64_t* __restrict__ Wout, uint64_t* __restrict__ Aout, int32_t* __restrict__ Hq,
                            int32_t* __restrict__ topout, float* __restrict__ mxout, int* err,
                            const float* __restrict__ pmax, const float* __restrict__ pmin, int npart) {
  constexpr int NW = NT / 32;
  static_assert(NT % 32 == 0 && NW <= 32 && NQ % NT == 0, "block shape");
  __shared__ uint32_t T[256];
  __shared__ uint32_t tab[NQ];  // histogram of q, then floor(w(q) R / W)
  __shared__ float redf[NW];
  __shared__ int redi[NW];
  __shared__ uint64_t redu[NW], redu2[NW];
  __shared__ uint32_t wtot[2][4][NW];
  __shared__ uint64_t s_K, s_W;
  __shared__ float s_m;
  __shared__ int s_top, s_bad;
  for (int i = threadIdx.x; i < 256; i += NT) T[i] = c_exp_table[i];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n4 = V >> 2;
  const uint32_t R = (1u << P) - (uint32_t)V;
  for (int r = blockIdx.x; r < rows; r += gridDim.x) {
    const float4* l4 = reinterpret_cast<const float4*>(logits + (size_t)r * V);
    // pass 1 (HBM): max; x - x is NaN exactly for non-finite x.  When the LM head's epilogue left
    // the row's maxima and minima per 128 columns (pmax: NaN-propagating), they replace the pass.
    float m = -INFINITY, nf = 0.f;
    if (pmax) {
      for (int i = threadIdx.x; i < npart; i += NT) {
        const float a = pmax[(size_t)r * npart + i], b = pmin[(size_t)r * npart + i];
        m = fmaxf(m, a);
        nf += (a - a) + (b - b);  // NaN for a NaN or infinite maximum or an infinite minimum
      }
    } else {
      constexpr int U = 4;  // independent 16-byte loads in flight per thread
      int i0 = threadIdx.x;
      for (; i0 + (U - 1) * NT < n4; i0 += U * NT) {
        float4 xv[U];
#pragma unroll
        for (int u = 0; u < U; ++u) xv[u] = l4[i0 + u * NT];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          const float4 x = xv[u];
          m = fmaxf(fmaxf(m, x.x), fmaxf(fmaxf(x.y, x.z), x.w));
          nf += (x.x - x.x) + (x.y - x.y) + (x.z - x.z) + (x.w - x.w);
        }
      }
      for (; i0 < n4; i0 += NT) {
        const float4 x = l4[i0];
        m = fmaxf(fmaxf(m, x.x), fmaxf(fmaxf(x.y, x.z), x.w));
        nf += (x.x - x.x) + (x.y - x.y) + (x.z - x.z) + (x.w - x.w);
      }
    }
    int bad = !(nf == 0.f);
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
      bad |= __shfl_xor_sync(0xffffffffu, bad, o);
    }
    __syncthreads();  // previous row done with the shared state
    for (int b = threadIdx.x; b < NQ; b += NT) tab[b] = 0;
    if (lane == 0) {
      redf[warp] = m;
      redi[warp] = bad;
    }
    __syncthreads();
    if (warp == 0) {
      float m2 = lane < NW ? redf[lane] : -INFINITY;
      int b2 = lane < NW ? redi[lane] : 0;
#pragma unroll
      for (int o = 16; o; o >>= 1) {
        m2 = fmaxf(m2, __shfl_xor_sync(0xffffffffu, m2, o));
        b2 |= __shfl_xor_sync(0xffffffffu, b2, o);
      }
      if (lane == 0) {
        if (b2) {
          // the call fails; m = +inf sends every code to 8191 (in range) and W is pinned below
          atomicOr(err, ERR_NONFINITE);
          m2 = INFINITY;
        }
        s_m = m2;
        s_bad = b2;
      }
    }
    __syncthreads();
    m = s_m;
    // pass 2 (L2): histogram of the codes q < QW0 (the others weigh nothing), lowest index of the maximum
    int topc = 0x7fffffff;
    for (int i0 = threadIdx.x; i0 < n4; i0 += 4 * NT) {
      float4 xv[4];
#pragma unroll
      for (int k = 0; k < 4; ++k)
        if (i0 + k * NT < n4) xv[k] = l4[i0 + k * NT];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int i = i0 + k * NT;
        if (i < n4) {
          const float4 x = xv[k];
          if (x.x == m || x.y == m || x.z == m || x.w == m)
            topc = min(topc, 4 * i + (x.x == m ? 0 : x.y == m ? 1 : x.z == m ? 2 : 3));
          const int q0 = quant_q(m, x.x), q1 = quant_q(m, x.y), q2 = quant_q(m, x.z), q3 = quant_q(m, x.w);
          if (q0 < QW0) atomicAdd(&tab[q0], 1u);
          if (q1 < QW0) atomicAdd(&tab[q1], 1u);
          if (q2 < QW0) atomicAdd(&tab[q2], 1u);
          if (q3 < QW0) atomicAdd(&tab[q3], 1u);
        }
      }
    }
    topc = __reduce_min_sync(0xffffffffu, topc);
    if (lane == 0) redi[warp] = topc;
    __syncthreads();
    // per-row sums over the bins (each thread owns bins threadIdx.x + k NT here and below)
    uint64_t Ws = 0, As = 0;
    for (int b = threadIdx.x; b < NQ; b += NT) {
      const uint64_t hw = (uint64_t)tab[b] * quant_w(T, b);
      Ws += hw;
      As += hw * (uint32_t)b;
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      Ws += __shfl_xor_sync(0xffffffffu, Ws, o);
      As += __shfl_xor_sync(0xffffffffu, As, o);
    }
    if (lane == 0) {
      redu[warp] = Ws;
      redu2[warp] = As;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      uint64_t tw = 0, ta = 0;
      int tp = 0x7fffffff;
      for (int i = 0; i < NW; ++i) {
        tw += redu[i];
        ta += redu2[i];
        tp = min(tp, redi[i]);
      }
      if (tp == 0x7fffffff) tp = 0;  // only for rows flagged non-finite
      if (s_bad) {                   // all codes 8191 (w = 0): any W >= 2^31 keeps the tables defined
        tw = 1ull << 31;
        ta = 0;
      }
      s_top = tp;
      s_K = (uint64_t)(((unsigned __int128)R << 64) / tw);
      s_W = tw;
      Wout[r] = tw;
      if (Aout) Aout[r] = ta;
      Hq[r] = entropy_q(tw, ta);
      if (topout) topout[r] = tp;
      if (mxout) mxout[r] = m;
    }
    __syncthreads();
    if (!cdf) continue;
    const uint64_t Wr = s_W, K = s_K;
    const int top = s_top;
    // floor(w(q) R / W) per code, over its own bin's count, and the histogram-weighted sum
    uint32_t fsum = 0;  // <= R
    for (int b = threadIdx.x; b < NQ; b += NT) {
      const uint32_t f = floor_wr_over_w(quant_w(T, b), R, Wr, K);
      fsum += tab[b] * f;
      tab[b] = f;
    }
    fsum = __reduce_add_sync(0xffffffffu, fsum);
    if (lane == 0) redi[warp] = (int)fsum;
    __syncthreads();  // the floor table complete
    const uint32_t D = R - __reduce_add_sync(0xffffffffu, lane < NW ? (uint32_t)redi[lane] : 0u);
    // CDF[v+1] = (v+1) + sum_{u<=v} (floor(w_u R / W) + (u == top ? D : 0)), scanned in
    // tiles of 4 NT float4s: sub-tile k holds float4s base + k NT + thread, so the
    // loads coalesce and the four warp scans run side by side; one barrier per tile
    uint32_t* cr = cdf + (size_t)r * (V + 1);
    if (threadIdx.x == 0) cr[0] = 0;
    // CDF entry 1 + 4 i + e starts a 16-byte quad when e == sh
    const int sh = (int)((0u - (uint32_t)(reinterpret_cast<uintptr_t>(cr + 1) >> 2)) & 3u);
    uint32_t carry = 0;
    int wb = 0;
    for (int base = 0; base < n4; base += 4 * NT) {
      uint32_t f[4][4], ts[4], inc[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int i = base + k * NT + threadIdx.x;
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (i < n4) x = __ldcs(l4 + i);
        const bool ok = i < n4;
        f[k][0] = ok ? tab[quant_q(m, x.x)] : 0u;
        f[k][1] = ok ? tab[quant_q(m, x.y)] : 0u;
        f[k][2] = ok ? tab[quant_q(m, x.z)] : 0u;
        f[k][3] = ok ? tab[quant_q(m, x.w)] : 0u;
        const uint32_t dt = (uint32_t)(top - 4 * i);  // the remainder joins the element at top and every prefix after it
        if (dt < 4u) {
          f[k][0] += dt == 0 ? D : 0u;
          f[k][1] += dt == 1 ? D : 0u;
          f[k][2] += dt == 2 ? D : 0u;
          f[k][3] += dt == 3 ? D : 0u;
        }
        ts[k] = f[k][0] + f[k][1] + f[k][2] + f[k][3];
        inc[k] = ts[k];
      }
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const uint32_t t = __shfl_up_sync(0xffffffffu, inc[k], o);
          if (lane >= o) inc[k] += t;
        }
      }
      if (lane == 31) {
#pragma unroll
        for (int k = 0; k < 4; ++k) wtot[wb][k][warp] = inc[k];
      }
      __syncthreads();
      uint32_t run = carry;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t tv = lane < NW ? wtot[wb][k][lane] : 0u;
        const uint32_t pre = __reduce_add_sync(0xffffffffu, lane < warp ? tv : 0u);
        const int i = base + k * NT + threadIdx.x;
        const int v = 4 * i;
        uint32_t o[4];  // o[e] = CDF[v + e + 1]
        uint32_t c = (uint32_t)v + run + pre + (inc[k] - ts[k]);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          c += 1u + f[k][e];
          o[e] = c;
        }
        run += __reduce_add_sync(0xffffffffu, tv);
        const uint32_t n0 = __shfl_down_sync(0xffffffffu, o[0], 1);
        const uint32_t n1 = __shfl_down_sync(0xffffffffu, o[1], 1);
        const uint32_t n2 = __shfl_down_sync(0xffffffffu, o[2], 1);
        if (i < n4) {
          uint32_t* dst = cr + 1 + v;
          if (sh == 0) {
            __stcs(reinterpret_cast<uint4*>(dst), make_uint4(o[0], o[1], o[2], o[3]));
          } else {
            // lanes 0..30 write the quad that starts at their element sh and ends in the
            // next lane's float4; a warp's first elements and its last lane's tail go singly
            if (lane == 0) {
#pragma unroll
              for (int e = 0; e < 3; ++e)
                if (e < sh) __stcs(dst + e, o[e]);
            }
            if (lane < 31 && i + 1 < n4) {
              const uint4 qv = sh == 1 ? make_uint4(o[1], o[2], o[3], n0)
                             : sh == 2 ? make_uint4(o[2], o[3], n0, n1)
                                       : make_uint4(o[3], n0, n1, n2);
              __stcs(reinterpret_cast<uint4*>(dst + sh), qv);
            } else {
#pragma unroll
              for (int e = 1; e < 4; ++e)
                if (e >= sh) __stcs(dst + e, o[e]);
            }
          }
        }
      }
      carry = run;
      wb ^= 1;
    }
  }
}

// ---- large vocabularies: a cluster of two CTAs per row -------------------------------------
// Each CTA of the pair takes one contiguous half of the row (in float4s).  With two 512-thread
// CTAs per SM, 152 rows are in flight (77 MB at V = 126464, 92 MB at 152064), so the histogram
// and CDF passes re-read the row from L2 rather than HBM.  Everything one half needs from the
// other is a value or a sum over histogram bins, so the pair exchanges scalars only, through
// distributed shared memory (thread 0 stores into both CTAs' slot and arrives on the peer's
// mbarrier; the slots and barriers alternate between two sets):
//   1. the halves' maxima (NaN-propagating) and minima -> m and the non-finite flag;
//   2. W and A over each half's bins and the lowest index of m in each half;
//   3. each half's sum of floor(w R / W) -> D and the CDF offset of the second half.
// A half's CDF pass looks up only codes that occur in it, i.e. its own non-empty bins, so each
// CTA fills the table value 1 + floor(w(q) R / W) for those bins alone.
constexpr int QP_NT = 512;  // threads per CTA (two CTAs per SM)
constexpr int QU = 8;       // float4 loads in flight per thread in the first pass
constexpr int QH = 8;       // and in the second

struct QPairSlot {  // one exchange, indexed by the sender's rank
  uint64_t W[2], A[2];
  float mx[2], mn[2];
  uint32_t fs[2];
  int top[2];
};

__device__ __forceinline__ float fmax_nan(float a, float b) {
  float d;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(d) : "f"(a), "f"(b));
  return d;
}
__device__ __forceinline__ float fmax3_nan(float a, float b, float c) {
  float d;
  asm("max.NaN.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
__device__ __forceinline__ float fmin3(float a, float b, float c) {
  float d;
  asm("min.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
// table entry q of the code bits QMAGIC + q in [QMAGIC, QMAGIC + QW0] (pair_code's range): the byte
// address base + 4 bits with base = table - 4 QMAGIC (32-bit wrap-around)
__device__ __forceinline__ uint32_t lds_code(uint32_t base, uint32_t bits) {
  uint32_t v;
  asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(base + 4u * bits));
  return v;
}
__device__ __forceinline__ void red_code(uint32_t base, uint32_t bits) {
  asm volatile("red.shared.add.u32 [%0], 1;" ::"r"(base + 4u * bits) : "memory");
}
// inclusive warp scan step: s += value of lane - d (lanes below d unchanged)
template <int d>
__device__ __forceinline__ void scan_step(uint32_t& s) {
  asm volatile(
      "{\n\t.reg .b32 t;\n\t.reg .pred p;\n\tshfl.sync.up.b32 t|p, %0, %1, 0, -1;\n\t@p add.u32 %0, %0, t;\n\t}"
      : "+r"(s)
      : "n"(d));
}

// code_bits of d = fl32(m - l) (in [QMAGIC, QMAGIC + QW0]: d >= 0 or NaN, as m is the row's maximum
// computed here).  With PART the maximum comes from another kernel, so d is also clamped below at
// 0 there: d < 0 (l above that maximum) never happens for consistent inputs, and the clamp keeps the
// table index in range whatever they are (NaN stays NaN and lands on QW0).
template <bool PART>
__device__ __forceinline__ uint32_t pair_code(float d) {
  if (!PART) return code_bits(d);
  const float t = fminf(fmax_nan(__fmul_rn(d, __uint_as_float(DLMZ_QSCALE_BITS)), 0.f), (float)QW0);
  return __float_as_uint(__fadd_rn(t, 12582912.0f));
}

template <bool PART>
__global__ void __launch_bounds__(QP_NT, 2)
    quantize_pair_kernel(const float* __restrict__ logits, int rows, int V, int P, uint32_t* __restrict__ cdf,
                         uint64_t* __restrict__ Wout, uint64_t* __restrict__ Aout, int32_t* __restrict__ Hq,
                         int32_t* __restrict__ topout, float* __restrict__ mxout, int* err,
                         const float* __restrict__ pmax, const float* __restrict__ pmin, int npart) {
  constexpr int NT = QP_NT, NW = NT / 32, BPT = NQ / NT;
  __shared__ __align__(16) uint32_t tab[NQ];  // histogram of the codes, then 1 + floor(w R / W)
  __shared__ uint32_t T[256];
  __shared__ QPairSlot xs[2];
  __shared__ __align__(8) uint64_t xbar[2];
  __shared__ float rf[2][NW];
  __shared__ uint64_t ru[2][NW];
  __shared__ int ri[NW];
  __shared__ uint32_t wsum[2][2][NW];
  __shared__ float s_m;
  __shared__ int s_bad, s_top, s_ok;
  __shared__ uint64_t s_W, s_K;
  __shared__ uint32_t s_D, s_carry;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (cluster_nctarank() != 2) {  // launched without its cluster shape: no cluster operation runs
    if (tid == 0) atomicOr(err, ERR_LAUNCH);
    return;
  }
  const uint32_t rank = cluster_ctarank(), peer = rank ^ 1u;
  for (int i = tid; i < 256; i += NT) T[i] = c_exp_table[i];
  if (tid == 0) {
    mbar_init(smem_u32(&xbar[0]), 1);
    mbar_init(smem_u32(&xbar[1]), 1);
    s_ok = 1;
    fence_mbarrier_init_cluster();
  }
  cluster_sync_all();  // the peer's barriers are initialised before any arrival on them

  const int n4 = V >> 2, half = (n4 + 1) >> 1;
  const int c0 = rank ? half : 0, n = rank ? n4 - half : half;  // this CTA's float4s [c0, c0 + n)
  const uint32_t R = (1u << P) - (uint32_t)V;
  const uint32_t tabq = smem_u32(tab) - 4u * QMAGIC;
  const uint32_t Tt = T[tid & 255];  // bins tid + k NT share T[b & 255] (NT is a multiple of 256)
  uint32_t xk = 0;                   // exchanges so far

  // thread 0: the slot of exchange xk is written (own copy and the peer's); signal the peer and wait
  // for its values.  Returns false (error word set) if the peer's arrival does not come.
  auto exchange_wait = [&]() -> bool {
    const uint32_t b = xk & 1u;
    mbar_arrive_remote(mapa_shared(smem_u32(&xbar[b]), peer));
    const bool ok = mbar_wait_cluster_bounded(smem_u32(&xbar[b]), (xk >> 1) & 1u, err);
    ++xk;
    return ok;
  };
  auto put_u64 = [&](uint64_t* p, uint64_t v) {
    *p = v;
    st_cluster_u64(mapa_shared(smem_u32(p), peer), v);
  };
  auto put_u32 = [&](uint32_t* p, uint32_t v) {
    *p = v;
    st_cluster_u32(mapa_shared(smem_u32(p), peer), v);
  };

  for (int r = blockIdx.x >> 1; r < rows; r += gridDim.x >> 1) {
    const float4* lc = reinterpret_cast<const float4*>(logits + (size_t)r * V) + c0;
    // ---- m and the non-finite flag
    float mx = -INFINITY, mn = INFINITY;
    if (PART) {  // per-128-column maxima (NaN-propagating) and minima from the LM head: the whole row
      for (int i = tid; i < npart; i += NT) {
        mx = fmax_nan(mx, pmax[(size_t)r * npart + i]);
        mn = fminf(mn, pmin[(size_t)r * npart + i]);
      }
    } else {  // pass 1 (HBM) over this half, QU float4 loads in flight per thread
      // the last round re-reads the half's last float4 past the end (a repeat leaves the maximum
      // and the minimum as they are), so every load is unconditional
      auto mxmn = [&](const float4 x) {
        mx = fmax3_nan(mx, x.x, x.y);
        mx = fmax3_nan(mx, x.z, x.w);
        mn = fmin3(mn, x.x, x.y);
        mn = fmin3(mn, x.z, x.w);
      };
      int i = tid;
      for (; i + (QU - 1) * NT < n; i += QU * NT) {
        float4 x[QU];
#pragma unroll
        for (int u = 0; u < QU; ++u) x[u] = lc[i + u * NT];
#pragma unroll
        for (int u = 0; u < QU; ++u) mxmn(x[u]);
      }
      if (i < n) {
        float4 x[QU];
#pragma unroll
        for (int u = 0; u < QU; ++u) x[u] = lc[min(i + u * NT, n - 1)];
#pragma unroll
        for (int u = 0; u < QU; ++u) mxmn(x[u]);
      }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      mx = fmax_nan(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    }
    if (lane == 0) {
      rf[0][warp] = mx;
      rf[1][warp] = mn;
    }
    __syncthreads();  // also: the previous row's CDF pass is done with tab
    for (int b = tid; b < NQ / 4; b += NT) reinterpret_cast<uint4*>(tab)[b] = make_uint4(0u, 0u, 0u, 0u);
    if (tid == 0) {
      float a = -INFINITY, z = INFINITY;
      for (int w = 0; w < NW; ++w) {
        a = fmax_nan(a, rf[0][w]);
        z = fminf(z, rf[1][w]);
      }
      bool ok = true;
      if (!PART) {
        QPairSlot& x = xs[xk & 1u];
        put_u32(reinterpret_cast<uint32_t*>(&x.mx[rank]), __float_as_uint(a));
        put_u32(reinterpret_cast<uint32_t*>(&x.mn[rank]), __float_as_uint(z));
        ok = exchange_wait();
        a = fmax_nan(x.mx[0], x.mx[1]);
        z = fminf(x.mn[0], x.mn[1]);
      }
      const int bad = !(isfinite(a) && z > -INFINITY);
      if (bad && rank == 0) atomicOr(err, ERR_NONFINITE);
      s_m = bad ? INFINITY : a;  // m = +inf sends every code to QW0 (no weight); W is pinned below
      s_bad = bad;
      s_ok = ok;
    }
    __syncthreads();
    if (!s_ok) break;
    const float m = s_m;
    // ---- pass 2 (L2): histogram of the codes (codes >= QW0 share bin QW0, which weighs nothing) and
    // the lowest index of m in this half (m - l == 0 exactly when l == m)
    int topc = 0x7fffffff;
    {
      auto hist4 = [&](const float4 x, int i) {
        const float d0 = __fsub_rn(m, x.x), d1 = __fsub_rn(m, x.y), d2 = __fsub_rn(m, x.z), d3 = __fsub_rn(m, x.w);
        red_code(tabq, pair_code<PART>(d0));
        red_code(tabq, pair_code<PART>(d1));
        red_code(tabq, pair_code<PART>(d2));
        red_code(tabq, pair_code<PART>(d3));
        if (fminf(fmin3(d0, d1, d2), d3) == 0.f)
          topc = min(topc, 4 * (c0 + i) + (d0 == 0.f ? 0 : d1 == 0.f ? 1 : d2 == 0.f ? 2 : 3));
      };
      int i = tid;
      for (; i + (QH - 1) * NT < n; i += QH * NT) {
        float4 x[QH];
#pragma unroll
        for (int u = 0; u < QH; ++u) x[u] = lc[i + u * NT];
#pragma unroll
        for (int u = 0; u < QH; ++u) hist4(x[u], i + u * NT);
      }
      if (i < n) {  // the last round: loads clamped into the half, only the elements inside it counted
        float4 x[QH];
#pragma unroll
        for (int u = 0; u < QH; ++u) x[u] = lc[min(i + u * NT, n - 1)];
#pragma unroll
        for (int u = 0; u < QH; ++u)
          if (i + u * NT < n) hist4(x[u], i + u * NT);
      }
    }
    topc = __reduce_min_sync(0xffffffffu, topc);
    if (lane == 0) ri[warp] = topc;
    __syncthreads();  // histogram complete
    // ---- W and A over this half's bins
    uint64_t Ws = 0, As = 0;
#pragma unroll 4
    for (int k = 0; k < BPT; ++k) {
      const int b = tid + k * NT;
      if (b < QW0) {
        const uint64_t hw = (uint64_t)tab[b] * (Tt >> (b >> 8));
        Ws += hw;
        As += hw * (uint32_t)b;
      }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      Ws += __shfl_xor_sync(0xffffffffu, Ws, o);
      As += __shfl_xor_sync(0xffffffffu, As, o);
    }
    if (lane == 0) {
      ru[0][warp] = Ws;
      ru[1][warp] = As;
    }
    __syncthreads();
    if (tid == 0) {
      uint64_t tw = 0, ta = 0;
      int tp = 0x7fffffff;
      for (int w = 0; w < NW; ++w) {
        tw += ru[0][w];
        ta += ru[1][w];
        tp = min(tp, ri[w]);
      }
      QPairSlot& x = xs[xk & 1u];
      put_u64(&x.W[rank], tw);
      put_u64(&x.A[rank], ta);
      put_u32(reinterpret_cast<uint32_t*>(&x.top[rank]), (uint32_t)tp);
      const bool ok = exchange_wait();
      tw = x.W[0] + x.W[1];
      ta = x.A[0] + x.A[1];
      tp = x.top[0] != 0x7fffffff ? x.top[0] : x.top[1];
      if (tp == 0x7fffffff) tp = 0;  // only for rows flagged non-finite
      if (s_bad) {                   // all codes QW0 (w = 0): any W >= 2^31 keeps the tables defined
        tw = 1ull << 31;
        ta = 0;
      }
      s_top = tp;
      s_W = tw;
      s_K = recip_scaled(R, tw);
      s_ok = ok;
      if (rank == 0) {
        Wout[r] = tw;
        if (Aout) Aout[r] = ta;
        Hq[r] = entropy_q(tw, ta);
        if (topout) topout[r] = tp;
        if (mxout) mxout[r] = m;
      }
    }
    __syncthreads();
    if (!s_ok) break;
    if (!cdf) continue;
    // ---- 1 + floor(w(q) R / W) for this half's non-empty bins, and the half's sum of the floors
    {
      const uint64_t Wr = s_W, K = s_K;
      uint32_t fs = 0;  // <= R
#pragma unroll 4
      for (int k = 0; k < BPT; ++k) {
        const int b = tid + k * NT;
        if (b < QW0) {
          const uint32_t h = tab[b];
          if (h) {
            const uint32_t f = floor_wr_over_w(Tt >> (b >> 8), R, Wr, K);
            fs += h * f;
            tab[b] = 1u + f;
          }
        }
      }
      fs = __reduce_add_sync(0xffffffffu, fs);
      if (lane == 0) ri[warp] = (int)fs;
      __syncthreads();
      if (tid == 0) {
        tab[QW0] = 1u;  // codes >= QW0: f = 0
        uint32_t t = 0;
        for (int w = 0; w < NW; ++w) t += (uint32_t)ri[w];
        QPairSlot& x = xs[xk & 1u];
        put_u32(&x.fs[rank], t);
        const bool ok = exchange_wait();
        const uint32_t D = R - x.fs[0] - x.fs[1];
        s_D = D;
        // the first half's entries sum to its element count + its floors (+ D if m's first index is there)
        s_carry = rank ? (uint32_t)(4 * half) + x.fs[0] + ((uint32_t)s_top < (uint32_t)(4 * half) ? D : 0u) : 0u;
        s_ok = ok;
      }
      __syncthreads();
      if (!s_ok) break;
    }
    // ---- pass 3 (L2): CDF[v + 1] = sum_{u <= v} (1 + floor(w_u R / W) + (u == top ? D : 0)), in tiles
    // of 2 NT float4s (layout below): running sums within each float4, warp scans of the float4
    // totals, then the CTA's offsets (one barrier per two tiles).  The row's entry 1 starts at word
    // offset e0 mod 4 from a 16-byte boundary; the pass is compiled once per e0.
    const uint32_t D = s_D;
    const int top = s_top;
    uint32_t carry = s_carry;
    uint32_t* cr = cdf + (size_t)r * (V + 1);
    if (rank == 0 && tid == 0) cr[0] = 0;
    const int e0 = (int)((0u - (uint32_t)(reinterpret_cast<uintptr_t>(cr + 1) >> 2)) & 3u);
    // A tile is 2 NT float4s; warp w takes float4s [64 w, 64 w + 64) of it as two sub-blocks of 32,
    // lane l float4s 64 w + l and 64 w + 32 + l, so loads and stores are 512 contiguous bytes per
    // instruction.  tile_local: the lane's 8 table values (plus D at m's first index, zero past this
    // half) as running sums within each float4, the warp's scans of the float4 totals, and the
    // exclusive offsets ex0 / ex1 of the lane's two float4s inside the warp's 256 elements; returns
    // the warp's total.  FULL: the tile lies inside the half (known at compile time).
    auto tile_local = [&](auto FULLc, int t0, const float4 x0, const float4 x1, uint32_t(&o)[8], uint32_t& ex0,
                          uint32_t& ex1) -> uint32_t {
      constexpr bool FULL = decltype(FULLc)::value;
      const int j0 = t0 + 64 * warp + lane, j1 = j0 + 32;
      o[0] = lds_code(tabq, pair_code<PART>(__fsub_rn(m, x0.x)));
      o[1] = lds_code(tabq, pair_code<PART>(__fsub_rn(m, x0.y)));
      o[2] = lds_code(tabq, pair_code<PART>(__fsub_rn(m, x0.z)));
      o[3] = lds_code(tabq, pair_code<PART>(__fsub_rn(m, x0.w)));
      o[4] = lds_code(tabq, pair_code<PART>(__fsub_rn(m, x1.x)));
      o[5] = lds_code(tabq, pair_code<PART>(__fsub_rn(m, x1.y)));
      o[6] = lds_code(tabq, pair_code<PART>(__fsub_rn(m, x1.z)));
      o[7] = lds_code(tabq, pair_code<PART>(__fsub_rn(m, x1.w)));
      const uint32_t dt0 = (uint32_t)(top - 4 * (c0 + j0)), dt1 = (uint32_t)(top - 4 * (c0 + j1));
      if (dt0 < 4u) {
#pragma unroll
        for (int e = 0; e < 4; ++e) o[e] += dt0 == (uint32_t)e ? D : 0u;
      }
      if (dt1 < 4u) {
#pragma unroll
        for (int e = 0; e < 4; ++e) o[4 + e] += dt1 == (uint32_t)e ? D : 0u;
      }
      if (!FULL) {  // past the end of this half (the other half's elements or the row's end): nothing
        const bool v0 = j0 < n, v1 = j1 < n;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          o[e] = v0 ? o[e] : 0u;
          o[e + 4] = v1 ? o[e + 4] : 0u;
        }
      }
#pragma unroll
      for (int e = 1; e < 4; ++e) {
        o[e] += o[e - 1];
        o[4 + e] += o[3 + e];
      }
      uint32_t s0 = o[3], s1 = o[7];
      scan_step<1>(s0);
      scan_step<1>(s1);
      scan_step<2>(s0);
      scan_step<2>(s1);
      scan_step<4>(s0);
      scan_step<4>(s1);
      scan_step<8>(s0);
      scan_step<8>(s1);
      scan_step<16>(s0);
      scan_step<16>(s1);
      const uint32_t t0tot = __shfl_sync(0xffffffffu, s0, 31), t1tot = __shfl_sync(0xffffffffu, s1, 31);
      ex0 = s0 - o[3];
      ex1 = t0tot + s1 - o[7];
      return t0tot + t1tot;
    };
    // the tile's CDF entries o[] + offsets, written out.  E0 (compile time): the first entry of a
    // float4 that starts a 16-byte quad.  Full tiles: each lane stores the quads that start at its
    // float4s' entry E0, completed by the next lane's first E0 entries (lane 31 of the first
    // sub-block by lane 0 of the second); a warp's first E0 entries and the tail of its last quad,
    // which the next warp completes, go singly.  Partial tiles: single stores.
    auto tile_store = [&](auto FULLc, auto E0c, int t0, uint32_t(&o)[8], uint32_t b0, uint32_t b1) {
      constexpr bool FULL = decltype(FULLc)::value;
      constexpr int E0 = decltype(E0c)::value;
      const int j0 = t0 + 64 * warp + lane, j1 = j0 + 32;
      uint32_t* d0 = cr + 1 + 4 * (c0 + j0);
      uint32_t* d1 = d0 + 128;
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        o[e] += b0;
        o[4 + e] += b1;
      }
      if (!FULL) {
        const bool v0 = j0 < n, v1 = j1 < n;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          if (v0) __stcs(d0 + e, o[e]);
          if (v1) __stcs(d1 + e, o[4 + e]);
        }
        return;
      }
      if (E0 == 0) {
        __stcs(reinterpret_cast<uint4*>(d0), make_uint4(o[0], o[1], o[2], o[3]));
        __stcs(reinterpret_cast<uint4*>(d1), make_uint4(o[4], o[5], o[6], o[7]));
        return;
      }
      const int nl = (lane + 1) & 31;
      uint32_t y[3], z[3];
#pragma unroll
      for (int e = 0; e < 3; ++e) {
        if (e < E0) {
          y[e] = __shfl_sync(0xffffffffu, o[e], nl);
          z[e] = __shfl_sync(0xffffffffu, o[4 + e], nl);
          if (lane == 31) y[e] = z[e];  // the first sub-block's last float4 continues into the second's first
        }
      }
      if (E0 == 1) {
        __stcs(reinterpret_cast<uint4*>(d0 + 1), make_uint4(o[1], o[2], o[3], y[0]));
      } else if (E0 == 2) {
        __stcs(reinterpret_cast<uint4*>(d0 + 2), make_uint4(o[2], o[3], y[0], y[1]));
      } else {
        __stcs(reinterpret_cast<uint4*>(d0 + 3), make_uint4(o[3], y[0], y[1], y[2]));
      }
      if (lane < 31) {
        if (E0 == 1) {
          __stcs(reinterpret_cast<uint4*>(d1 + 1), make_uint4(o[5], o[6], o[7], z[0]));
        } else if (E0 == 2) {
          __stcs(reinterpret_cast<uint4*>(d1 + 2), make_uint4(o[6], o[7], z[0], z[1]));
        } else {
          __stcs(reinterpret_cast<uint4*>(d1 + 3), make_uint4(o[7], z[0], z[1], z[2]));
        }
      } else {  // the warp block's last quad runs into the next warp's block: this lane's part only
#pragma unroll
        for (int e = E0; e < 4; ++e) __stcs(d1 + e, o[4 + e]);
      }
      if (lane == 0) {  // the warp block's first E0 entries precede its first aligned quad
#pragma unroll
        for (int e = 0; e < E0; ++e) __stcs(d0 + e, o[e]);
      }
    };
    // past the end of this half: m itself (d = 0, an in-range code; the values are dropped)
    auto ld4 = [&](int i) {
      float4 x = make_float4(m, m, m, m);
      if (i < n) x = __ldcs(lc + i);
      return x;
    };
    // two tiles per barrier: their loads and local scans run side by side; the pairs inside the
    // half first, then the last (partial) pair
    auto pass3 = [&](auto E0c) {
      const std::integral_constant<bool, true> full_c;
      const std::integral_constant<bool, false> part_c;
      int wb = 0;
      auto combine = [&](uint32_t sa, uint32_t sb, uint32_t& ba, uint32_t& bb) {
        if (lane == 0) {
          wsum[wb][0][warp] = sa;
          wsum[wb][1][warp] = sb;
        }
        __syncthreads();
        const uint32_t tva = lane < NW ? wsum[wb][0][lane] : 0u, tvb = lane < NW ? wsum[wb][1][lane] : 0u;
        wb ^= 1;
        ba = carry + __reduce_add_sync(0xffffffffu, lane < warp ? tva : 0u);
        carry += __reduce_add_sync(0xffffffffu, tva);
        bb = carry + __reduce_add_sync(0xffffffffu, lane < warp ? tvb : 0u);
        carry += __reduce_add_sync(0xffffffffu, tvb);
      };
      int t0 = 0;
      for (; t0 + 4 * NT <= n; t0 += 4 * NT) {
        const int t1 = t0 + 2 * NT;
        const int jw = 64 * warp + lane;
        const float4 xa0 = __ldcs(lc + t0 + jw), xb0 = __ldcs(lc + t0 + jw + 32);
        const float4 xa1 = __ldcs(lc + t1 + jw), xb1 = __ldcs(lc + t1 + jw + 32);
        uint32_t oa[8], ob[8], ea0, ea1, eb0, eb1, ba, bb;
        const uint32_t sa = tile_local(full_c, t0, xa0, xb0, oa, ea0, ea1);
        const uint32_t sb = tile_local(full_c, t1, xa1, xb1, ob, eb0, eb1);
        combine(sa, sb, ba, bb);
        tile_store(full_c, E0c, t0, oa, ba + ea0, ba + ea1);
        tile_store(full_c, E0c, t1, ob, bb + eb0, bb + eb1);
      }
      if (t0 < n) {  // tile t0 may still be full; t1 is partial or past the end
        const int t1 = t0 + 2 * NT;
        const int jw = 64 * warp + lane;
        const float4 xa0 = ld4(t0 + jw), xb0 = ld4(t0 + jw + 32);
        const float4 xa1 = ld4(t1 + jw), xb1 = ld4(t1 + jw + 32);
        uint32_t oa[8], ob[8], ea0, ea1, eb0, eb1, ba, bb;
        const uint32_t sa = tile_local(part_c, t0, xa0, xb0, oa, ea0, ea1);
        const uint32_t sb = tile_local(part_c, t1, xa1, xb1, ob, eb0, eb1);
        combine(sa, sb, ba, bb);
        if (t1 <= n)
          tile_store(full_c, E0c, t0, oa, ba + ea0, ba + ea1);
        else
          tile_store(part_c, E0c, t0, oa, ba + ea0, ba + ea1);
        if (t1 < n) tile_store(part_c, E0c, t1, ob, bb + eb0, bb + eb1);
      }
    };
    switch (e0) {
      case 0: pass3(std::integral_constant<int, 0>()); break;
      case 1: pass3(std::integral_constant<int, 1>()); break;
      case 2: pass3(std::integral_constant<int, 2>()); break;
      default: pass3(std::integral_constant<int, 3>()); break;
    }
  }
  cluster_sync_all();  // neither CTA leaves while the peer may still write to its shared memory
}

// clusters of quantize_pair_kernel that fit on the device at once (0: the launch shape is unavailable)
static cudaLaunchConfig_t pair_config(int grid, cudaStream_t s, cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(QP_NT);
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

static int pair_clusters() {
  static int n[kMaxDevices] = {};
  const int dev = device_ordinal();
  if (dev < 0) return 0;
  if (!n[dev]) {
    cudaLaunchAttribute attr[1];
    const cudaLaunchConfig_t cfg = pair_config(2 * 2 * num_sms(), 0, attr);
    int c = 0;
    if (cudaOccupancyMaxActiveClusters(&c, quantize_pair_kernel<false>, &cfg) != cudaSuccess || c < 1) {
      cudaGetLastError();
      c = -1;
    }
    n[dev] = c;
  }
  return n[dev] > 0 ? n[dev] : 0;
}

int quantize_rows(const float* logits, int rows, int V, int P, uint32_t* cdf, uint64_t* W, uint64_t* A, int32_t* Hq,
                  int32_t* top, float* mx, cudaStream_t s, const float* pmax, const float* pmin) {
  if (rows == 0) return DLMZ_OK;
  int* err = device_error_word();
  const int grid = (rows + 7) / 8;
  ProfScope prof(PROF_QUANT, s, 0, (double)rows * V * 4 + (cdf ? (double)rows * (V + 1) * 4 : 0.0));
  if (V <= 32) quantize_warp_kernel<1><<<grid, 256, 0, s>>>(logits, rows, V, P, cdf, W, A, Hq, top, mx, err);
  else if (V <= 64) quantize_warp_kernel<2><<<grid, 256, 0, s>>>(logits, rows, V, P, cdf, W, A, Hq, top, mx, err);
  else if (V <= 128) quantize_warp_kernel<4><<<grid, 256, 0, s>>>(logits, rows, V, P, cdf, W, A, Hq, top, mx, err);
  else if (V <= 256) quantize_warp_kernel<8><<<grid, 256, 0, s>>>(logits, rows, V, P, cdf, W, A, Hq, top, mx, err);
  else if (V <= 512) quantize_warp_kernel<16><<<grid, 256, 0, s>>>(logits, rows, V, P, cdf, W, A, Hq, top, mx, err);
  else if (V % 4 == 0 && (reinterpret_cast<uintptr_t>(logits) & 15) == 0 &&
           (reinterpret_cast<uintptr_t>(cdf) & 15) == 0 && pair_clusters() > 0) {
    cudaLaunchAttribute attr[1];
    const cudaLaunchConfig_t cfg = pair_config(2 * (rows < pair_clusters() ? rows : pair_clusters()), s, attr);
    const bool part = pmax && pmin && V % 128 == 0;
    if (part)
      cudaLaunchKernelEx(&cfg, quantize_pair_kernel<true>, logits, rows, V, P, cdf, W, A, Hq, top, mx, err, pmax, pmin,
                         V / 128);
    else
      cudaLaunchKernelEx(&cfg, quantize_pair_kernel<false>, logits, rows, V, P, cdf, W, A, Hq, top, mx, err,
                         (const float*)nullptr, (const float*)nullptr, 0);
  } else if (V % 4 == 0 && (reinterpret_cast<uintptr_t>(logits) & 15) == 0) {
    const int g = rows < QCPS * num_sms() ? rows : QCPS * num_sms();
    const bool part = pmax && pmin && V % 128 == 0;
    quantize_persist_kernel<QNT, QCPS><<<g, QNT, 0, s>>>(logits, rows, V, P, cdf, W, A, Hq, top, mx, err,
                                                         part ? pmax : nullptr, part ? pmin : nullptr, V / 128);
  } else {
    quantize_cta_kernel<<<rows, QT, 0, s>>>(logits, rows, V, P, cdf, W, A, Hq, top, mx, err);
  }
  return launch_status();
}

}  // namespace dlmz
