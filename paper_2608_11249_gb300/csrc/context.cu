// Attention-based initial context (Sec. 3.4, policy 4).
//
// Two forwards over each window -- one with the even positions masked, one
// with the odd ones masked, the others showing their true symbols -- export
// every layer's attention averaged over heads (A_l).  Attention Rollout
// (Abnar & Zuidema 2020) with Ã_l = A_l / 2 + I / 2 and R = Ã_N ... Ã_1 scores
// position j by sum over masked i of R[i, j], taken from the pass in which j
// is visible: the row vector of masked indicators is propagated backwards,
// v <- v Ã_l for l = N .. 1.  The caller keeps the c highest scores.
#include "kernels.cuh"
#include "model.cuh"

namespace dlmz {

constexpr int MAP_THREADS = 256;
constexpr int MAP_KC = 64;  // keys per staged chunk

// Rows per CTA for window length L: the score and accumulator rows fit in shared memory.
static int map_rows(int L) {
  int r = 16384 / (L > 0 ? L : 1);  // 2 x rows x L floats <= 128 KB
  if (r > 32) r = 32;
  return r < 1 ? 1 : r;
}

// Head-averaged attention probabilities of rows [r0, r0 + R) of window w:
// maps[w][i][j] = (1 / n_heads) sum_h softmax_j(q_h,i . k_g(h),j / sqrt(hd)).
template <typename T>
__global__ void __launch_bounds__(MAP_THREADS) attn_maps_kernel(const T* __restrict__ qkv, int ld, int L, int nh,
                                                               int nkv, int hd, int d, int R, float* __restrict__ maps) {
  extern __shared__ float msm[];
  float* S = msm;                     // [R][L] scores, then probabilities of one head
  float* acc = S + (size_t)R * L;     // [R][L] head average
  float* Ks = acc + (size_t)R * L;    // [MAP_KC][hd + 1]
  float* Qs = Ks + MAP_KC * (hd + 1); // [R][hd]
  const int w = blockIdx.y, r0 = blockIdx.x * R;
  const int nr = min(R, L - r0);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, nwarp = MAP_THREADS / 32;
  const float scale = rsqrtf((float)hd);
  const T* base = qkv + (size_t)w * L * ld;
  for (int i = tid; i < R * L; i += MAP_THREADS) acc[i] = 0.f;
  for (int h = 0; h < nh; ++h) {
    const int g = h / (nh / nkv);
    __syncthreads();
    for (int i = tid; i < nr * hd; i += MAP_THREADS)
      Qs[i] = to_f(base[(size_t)(r0 + i / hd) * ld + h * hd + i % hd]);
    for (int k0 = 0; k0 < L; k0 += MAP_KC) {
      const int nk = min(MAP_KC, L - k0);
      __syncthreads();
      for (int i = tid; i < nk * hd; i += MAP_THREADS)
        Ks[(i / hd) * (hd + 1) + i % hd] = to_f(base[(size_t)(k0 + i / hd) * ld + d + g * hd + i % hd]);
      __syncthreads();
      for (int p = tid; p < nr * nk; p += MAP_THREADS) {  // (row, key) pairs
        const int r = p / nk, j = p % nk;
        const float* q = Qs + r * hd;
        const float* k = Ks + j * (hd + 1);
        float s = 0.f;
        for (int e = 0; e < hd; ++e) s = fmaf(q[e], k[e], s);
        S[(size_t)r * L + k0 + j] = s * scale;
      }
    }
    __syncthreads();
    for (int r = warp; r < nr; r += nwarp) {  // softmax of each row, one warp per row
      float* row = S + (size_t)r * L;
      float m = -INFINITY;
      for (int j = lane; j < L; j += 32) m = fmaxf(m, row[j]);
#pragma unroll
      for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
      float sum = 0.f;
      for (int j = lane; j < L; j += 32) {
        const float e = expf(row[j] - m);
        row[j] = e;
        sum += e;
      }
#pragma unroll
      for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      const float inv = 1.0f / (sum * (float)nh);
      for (int j = lane; j < L; j += 32) acc[(size_t)r * L + j] += row[j] * inv;
    }
  }
  __syncthreads();
  float* out = maps + ((size_t)w * L + r0) * L;
  for (int i = tid; i < nr * L; i += MAP_THREADS) out[i] = acc[i];
}

template <typename T>
int attention_maps(const T* qkv, int ld, int n_chunks, int L, int nh, int nkv, int hd, int d, float* maps,
                   cudaStream_t s) {
  if (n_chunks == 0) return DLMZ_OK;
  const int R = map_rows(L);
  const size_t smem = ((size_t)2 * R * L + MAP_KC * (hd + 1) + (size_t)R * hd) * 4;
  if (smem > 200 * 1024) return DLMZ_EINVAL;
  DLMZ_CUDA_TRY(cudaFuncSetAttribute(attn_maps_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  dim3 grid((L + R - 1) / R, n_chunks);
  attn_maps_kernel<T><<<grid, MAP_THREADS, smem, s>>>(qkv, ld, L, nh, nkv, hd, d, R, maps);
  return launch_status();
}
template int attention_maps<float>(const float*, int, int, int, int, int, int, int, float*, cudaStream_t);
template int attention_maps<bf16>(const bf16*, int, int, int, int, int, int, int, float*, cudaStream_t);

// state of pass `parity`: positions j with j % 2 == parity masked, the others their symbol
__global__ void parity_state_kernel(const int32_t* symbols, int64_t n, int L, int parity, int mask_id, int32_t* state) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    state[i] = (int)(i % L) % 2 == parity ? mask_id : symbols[i];
}

// v <- v (A_l / 2 + I / 2) for l = N-1 .. 0, v starting at the masked indicator; the
// visible positions' entries are this pass's scores.  One CTA per window.
__global__ void __launch_bounds__(256) rollout_kernel(const float* maps, int n_layers, int nc, int L, int parity,
                                                      float* scores) {
  extern __shared__ float v[];  // [2][L]
  const int w = blockIdx.x;
  float* cur = v;
  float* nxt = v + L;
  for (int j = threadIdx.x; j < L; j += blockDim.x) cur[j] = j % 2 == parity ? 1.f : 0.f;
  for (int l = n_layers - 1; l >= 0; --l) {
    __syncthreads();
    const float* A = maps + ((size_t)l * nc + w) * L * L;
    for (int j = threadIdx.x; j < L; j += blockDim.x) {
      float s = 0.f;
      for (int i = 0; i < L; ++i) s = fmaf(cur[i], A[(size_t)i * L + j], s);
      nxt[j] = 0.5f * s + 0.5f * cur[j];
    }
    float* t = cur;
    cur = nxt;
    nxt = t;
  }
  __syncthreads();
  for (int j = threadIdx.x; j < L; j += blockDim.x)
    if (j % 2 != parity) scores[(size_t)w * L + j] = cur[j];
}

int context_attention_scores(dlmz_model* m, const int32_t* symbols, int nc, int L, float* scores, DevBuf& maps,
                             DevBuf& state, cudaStream_t s) {
  if (nc <= 0 || L <= 0) return nc == 0 ? DLMZ_OK : DLMZ_EINVAL;
  const int N = (int)m->cfg.n_layers;
  const size_t need = (size_t)N * nc * L * L * 4;
  DLMZ_TRY(maps.ensure(need));
  DLMZ_TRY(state.ensure((size_t)nc * L * 4));
  if ((size_t)2 * L * 4 > 200 * 1024) return DLMZ_EINVAL;
  DLMZ_CUDA_TRY(cudaFuncSetAttribute(rollout_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024));
  for (int parity = 0; parity < 2; ++parity) {
    const int64_t n = (int64_t)nc * L;
    parity_state_kernel<<<(unsigned)((n + 255) / 256 < 65535 ? (n + 255) / 256 : 65535), 256, 0, s>>>(
        symbols, n, L, parity, (int)m->cfg.vocab, state.as<int32_t>());
    DLMZ_TRY(launch_status());
    DLMZ_TRY(model_attention_maps(m, state.as<int32_t>(), nc, L, maps.as<float>(), s));
    rollout_kernel<<<nc, 256, (size_t)2 * L * 4, s>>>(maps.as<float>(), N, nc, L, parity, scores);
    DLMZ_TRY(launch_status());
  }
  return DLMZ_OK;
}

}  // namespace dlmz
