// CUDA-core kernels of the masked-DLM forward (Definition 3): embedding,
// RMSNorm, RoPE, SwiGLU, a tiled float32-accumulating GEMM for float32
// models and for shapes the tensor-core GEMM does not take, and a
// one-query-per-thread bidirectional attention for the same cases.
#include <math.h>

#include "kernels.cuh"

namespace dlmz {

// ---- embedding: x[t] = E[state[t]] (float32 residual stream) ---------------------
template <typename T>
__global__ void embed_kernel(const int32_t* __restrict__ state, int n, const T* __restrict__ E, int d,
                             float* __restrict__ x) {
  const int t = blockIdx.x;
  if (t >= n) return;
  const T* row = E + (size_t)state[t] * d;
  float* out = x + (size_t)t * d;
  for (int i = threadIdx.x; i < d; i += blockDim.x) out[i] = to_f(row[i]);
}

template <typename T>
int embed(const int32_t* state, int n, const T* E, int d, float* x, cudaStream_t s) {
  if (n == 0) return DLMZ_OK;
  ProfScope prof(PROF_LAYER, s, 0, (double)n * d * (sizeof(T) + 4));
  embed_kernel<T><<<n, 128, 0, s>>>(state, n, E, d, x);
  return launch_status();
}
__global__ void embed_norm_kernel(const int32_t* __restrict__ state, int n, const bf16* __restrict__ E, int d,
                                  float* __restrict__ x, bf16* __restrict__ y, float* __restrict__ ssq, int n_part) {
  const int t = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (t >= n) return;
  const bf16* row = E + (size_t)state[t] * d;
  float ss = 0.f;
  for (int i = lane; i < d; i += 32) {
    const bf16 e = row[i];
    const float v = __bfloat162float(e);
    x[(size_t)t * d + i] = v;
    y[(size_t)t * d + i] = e;
    ss += v * v;
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  for (int i = lane; i < n_part; i += 32) ssq[(size_t)t * n_part + i] = i == 0 ? ss : 0.f;
}

int embed_norm(const int32_t* state, int n, const bf16* E, int d, float* x, bf16* y, float* ssq, int n_part,
               cudaStream_t s) {
  if (n == 0) return DLMZ_OK;
  ProfScope prof(PROF_LAYER, s, 0, (double)n * d * 8);
  embed_norm_kernel<<<(n + 7) / 8, 256, 0, s>>>(state, n, E, d, x, y, ssq, n_part);
  return launch_status();
}

template int embed<float>(const int32_t*, int, const float*, int, float*, cudaStream_t);
template int embed<bf16>(const int32_t*, int, const bf16*, int, float*, cudaStream_t);

// ---- RMSNorm (one warp per row), optional row gather ------------------------------
template <typename OutT>
__global__ void rmsnorm_kernel(const float* __restrict__ x, int rows, int d, const float* __restrict__ g,
                               float eps, OutT* __restrict__ h, int L, int row0, int rpc,
                               const int32_t* __restrict__ idx) {
  const int r = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  const size_t src = idx ? (size_t)idx[r] : rpc > 0 ? (size_t)(r / rpc) * L + row0 + (r % rpc) : (size_t)r;
  const float* xr = x + src * d;
  float ss = 0.f;
  for (int i = lane; i < d; i += 32) ss += xr[i] * xr[i];
#pragma unroll
  for (int o = 16; o; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  const float inv = 1.0f / sqrtf(ss / (float)d + eps);
  OutT* hr = h + (size_t)r * d;
  for (int i = lane; i < d; i += 32) hr[i] = from_f<OutT>(xr[i] * inv * g[i]);
}

template <typename OutT>
int rmsnorm(const float* x, int rows, int d, const float* g, float eps, OutT* h, int L, int row0, int rpc,
            cudaStream_t s) {
  if (rows == 0) return DLMZ_OK;
  ProfScope prof(PROF_LAYER, s, 0, (double)rows * d * (4 + sizeof(OutT)));
  rmsnorm_kernel<OutT><<<(rows + 7) / 8, 256, 0, s>>>(x, rows, d, g, eps, h, L, row0, rpc, nullptr);
  return launch_status();
}
template int rmsnorm<float>(const float*, int, int, const float*, float, float*, int, int, int, cudaStream_t);
template int rmsnorm<bf16>(const float*, int, int, const float*, float, bf16*, int, int, int, cudaStream_t);

template <typename OutT>
int rmsnorm_gather(const float* x, const int32_t* idx, int rows, int d, const float* g, float eps, OutT* h,
                   cudaStream_t s) {
  if (rows == 0) return DLMZ_OK;
  ProfScope prof(PROF_LAYER, s, 0, (double)rows * d * (4 + sizeof(OutT)));
  rmsnorm_kernel<OutT><<<(rows + 7) / 8, 256, 0, s>>>(x, rows, d, g, eps, h, 0, 0, 0, idx);
  return launch_status();
}
template int rmsnorm_gather<float>(const float*, const int32_t*, int, int, const float*, float, float*, cudaStream_t);
template int rmsnorm_gather<bf16>(const float*, const int32_t*, int, int, const float*, float, bf16*, cudaStream_t);

// ---- RoPE in place on the Q and K heads of the fused qkv buffer -----------------
template <typename T>
__global__ void rope_kernel(T* __restrict__ qkv, int n, int ld, int nh, int hd, int L,
                            const float2* __restrict__ cs) {
  const int t = blockIdx.x;
  if (t >= n) return;
  const int pos = t % L;
  const int half = hd / 2;
  T* row = qkv + (size_t)t * ld;
  for (int j = threadIdx.x; j < nh * half; j += blockDim.x) {
    const int h = j / half, i = j % half;
    float a = to_f(row[h * hd + i]), b = to_f(row[h * hd + i + half]);
    float2 c = cs[(size_t)pos * half + i];
    row[h * hd + i] = from_f<T>(a * c.x - b * c.y);
    row[h * hd + i + half] = from_f<T>(b * c.x + a * c.y);
  }
}

template <typename T>
int rope_inplace(T* qkv, int n, int ld, int nh, int hd, int L, const float2* cs, cudaStream_t s) {
  if (n == 0) return DLMZ_OK;
  ProfScope prof(PROF_LAYER, s, 0, 2.0 * n * nh * hd * sizeof(T));
  rope_kernel<T><<<n, 128, 0, s>>>(qkv, n, ld, nh, hd, L, cs);
  return launch_status();
}
template int rope_inplace<float>(float*, int, int, int, int, int, const float2*, cudaStream_t);
template int rope_inplace<bf16>(bf16*, int, int, int, int, int, const float2*, cudaStream_t);

// ---- SwiGLU: out[t, f] = silu(g_f) * u_f from the interleaved gate/up buffer --------
template <typename T>
__global__ void swiglu_kernel(const float* __restrict__ gu, int n, int F, int gb, T* __restrict__ out) {
  const int t = blockIdx.x;
  if (t >= n) return;
  const float* r = gu + (size_t)t * 2 * F;
  for (int f = threadIdx.x; f < F; f += blockDim.x) {
    const int blk = f / gb, off = f % gb;
    const float g = r[blk * 2 * gb + off], u = r[blk * 2 * gb + gb + off];
    out[(size_t)t * F + f] = from_f<T>(g / (1.0f + expf(-g)) * u);
  }
}

template <typename T>
int swiglu(const float* gu, int n, int F, int gb, T* out, cudaStream_t s) {
  if (n == 0) return DLMZ_OK;
  ProfScope prof(PROF_LAYER, s, 0, (double)n * F * (8 + sizeof(T)));
  swiglu_kernel<T><<<n, 256, 0, s>>>(gu, n, F, gb, out);
  return launch_status();
}
template int swiglu<float>(const float*, int, int, int, float*, cudaStream_t);
template int swiglu<bf16>(const float*, int, int, int, bf16*, cudaStream_t);

// ---- tiled GEMM on CUDA cores: C[m, n] = sum_k A[m, k] B[n, k] --------------------
// 64x64 tile per 256-thread CTA, 4x4 outputs per thread, K slices of 16.
template <typename T>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const T* __restrict__ A, int lda, const T* __restrict__ B,
                                                        int ldb, int M, int N, int K, int epi, GemmEpilogue ep) {
  __shared__ float As[16][64 + 4];
  __shared__ float Bs[16][64 + 4];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += 16) {
    for (int i = threadIdx.x; i < 64 * 16; i += 256) {
      const int r = i / 16, c = i % 16;
      const int gm = m0 + r, gn = n0 + r, gk = k0 + c;
      As[c][r] = (gm < M && gk < K) ? to_f(A[(size_t)gm * lda + gk]) : 0.f;
      Bs[c][r] = (gn < N && gk < K) ? to_f(B[(size_t)gn * ldb + gk]) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = As[k][ty * 4 + i];
        b[i] = Bs[k][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= N) continue;
      const size_t o = (size_t)m * ep.ldo + n;
      if (epi == EPI_F32)
        reinterpret_cast<float*>(ep.out)[o] = acc[i][j];
      else if (epi == EPI_RESID_F32)
        reinterpret_cast<float*>(ep.out)[o] += acc[i][j];
      else
        reinterpret_cast<bf16*>(ep.out)[o] = __float2bfloat16_rn(acc[i][j]);
    }
  }
}

template <typename T>
int gemm_simt(const T* A, int lda, const T* B, int ldb, int M, int N, int K, int epi, const GemmEpilogue& ep,
              cudaStream_t s) {
  if (epi != EPI_F32 && epi != EPI_RESID_F32 && epi != EPI_BF16) return DLMZ_EINVAL;
  if (M == 0 || N == 0) return DLMZ_OK;
  dim3 grid((N + 63) / 64, (M + 63) / 64);
  ProfScope prof(PROF_GEMM_SIMT, s, 2.0 * M * N * K, (double)sizeof(T) * ((double)M * K + (double)N * K) + 4.0 * M * N);
  gemm_simt_kernel<T><<<grid, 256, 0, s>>>(A, lda, B, ldb, M, N, K, epi, ep);
  return launch_status();
}
template int gemm_simt<float>(const float*, int, const float*, int, int, int, int, int, const GemmEpilogue&,
                              cudaStream_t);
template int gemm_simt<bf16>(const bf16*, int, const bf16*, int, int, int, int, int, const GemmEpilogue&,
                             cudaStream_t);

// ---- bidirectional attention, one query per thread ---------------------------------
// CTA = (64 queries, head, window); keys/values of the window staged through
// shared memory 64 at a time; online softmax in float32.  No mask: every
// query attends to every position of its window.
template <typename T, int HD>
__global__ void __launch_bounds__(64) attention_simt_kernel(const T* __restrict__ qkv, int ld, int L, int nh,
                                                            int nkv, int d, T* __restrict__ out) {
  __shared__ float Ks[64][HD + 1];
  __shared__ float Vs[64][HD + 1];
  const int chunk = blockIdx.z, h = blockIdx.y;
  const int qi = blockIdx.x * 64 + threadIdx.x;
  const int g = h / (nh / nkv);
  const int dkv = nkv * HD;
  const size_t base = (size_t)chunk * L;
  const float scale = 1.0f / sqrtf((float)HD);
  float q[HD], o[HD];
  const bool live = qi < L;
#pragma unroll
  for (int i = 0; i < HD; ++i) {
    q[i] = live ? to_f(qkv[(base + qi) * ld + h * HD + i]) * scale : 0.f;
    o[i] = 0.f;
  }
  float mrun = -INFINITY, l = 0.f;
  for (int k0 = 0; k0 < L; k0 += 64) {
    __syncthreads();
    for (int i = threadIdx.x; i < 64 * HD; i += 64) {
      const int r = i / HD, c = i % HD;
      const bool ok = k0 + r < L;
      const size_t row = (base + k0 + r) * ld;
      Ks[r][c] = ok ? to_f(qkv[row + d + g * HD + c]) : 0.f;
      Vs[r][c] = ok ? to_f(qkv[row + d + dkv + g * HD + c]) : 0.f;
    }
    __syncthreads();
    const int kn = min(64, L - k0);
    for (int j = 0; j < kn; ++j) {
      float sc = 0.f;
#pragma unroll
      for (int i = 0; i < HD; ++i) sc = fmaf(q[i], Ks[j][i], sc);
      const float mnew = fmaxf(mrun, sc);
      const float corr = expf(mrun - mnew);
      const float p = expf(sc - mnew);
      l = l * corr + p;
#pragma unroll
      for (int i = 0; i < HD; ++i) o[i] = fmaf(o[i], corr, p * Vs[j][i]);
      mrun = mnew;
    }
  }
  if (!live) return;
  const float inv = 1.0f / l;
#pragma unroll
  for (int i = 0; i < HD; ++i) out[(base + qi) * d + h * HD + i] = from_f<T>(o[i] * inv);
}

template <typename T>
int attention_simt(const T* qkv, int ld, int n_chunks, int L, int nh, int nkv, int hd, int d, T* out,
                   cudaStream_t s) {
  if (n_chunks == 0 || L == 0) return DLMZ_OK;
  dim3 grid((L + 63) / 64, nh, n_chunks);
  ProfScope prof(PROF_ATTN, s, 4.0 * n_chunks * nh * (double)L * L * hd,
                 (double)sizeof(T) * n_chunks * L * (ld + d));
  switch (hd) {
    case 8: attention_simt_kernel<T, 8><<<grid, 64, 0, s>>>(qkv, ld, L, nh, nkv, d, out); break;
    case 16: attention_simt_kernel<T, 16><<<grid, 64, 0, s>>>(qkv, ld, L, nh, nkv, d, out); break;
    case 32: attention_simt_kernel<T, 32><<<grid, 64, 0, s>>>(qkv, ld, L, nh, nkv, d, out); break;
    case 64: attention_simt_kernel<T, 64><<<grid, 64, 0, s>>>(qkv, ld, L, nh, nkv, d, out); break;
    default: return DLMZ_EINVAL;
  }
  return launch_status();
}
template int attention_simt<float>(const float*, int, int, int, int, int, int, int, float*, cudaStream_t);
template int attention_simt<bf16>(const bf16*, int, int, int, int, int, int, int, bf16*, cudaStream_t);

}  // namespace dlmz
