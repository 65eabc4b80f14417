// Masked-DLM model: random initialisation and the forward pass (Definition 3).
//
// Weights ~ N(0, 0.02) regenerated from (seed, tensor id, element index) by
// SplitMix64 (Steele, Lea & Flood 2014) and the basic Box-Muller transform,
// evaluated in double precision and rounded to the model's storage type.
// Tensor ids: 0 embedding [(V+1) x d], 1 LM head [V x d], and per layer l
// 2+8l+{0 Wq, 1 Wk, 2 Wv, 3 Wo, 4 Wgate, 5 Wup, 6 Wdown}, each [out x in]
// row-major in its logical shape.  Physical layouts: Wq|Wk|Wv stacked into
// one [d+2 dkv x d] matrix; Wgate/Wup interleaved in blocks of gu_block rows
// so a 256-column GEMM tile holds the gate and up rows of the same features.
// On the tensor-core path the rows of Wq and Wk are also reordered inside each
// head so that RoPE's rotation pairs (i, i + hd/2) become adjacent columns
// (2i, 2i+1) of the QKV output; q.k over a head is unchanged by a permutation
// of its dimensions applied to both q and k, and V keeps its order.
#include <math.h>
#include <string.h>

#include <vector>

#include "model.cuh"

namespace dlmz {

constexpr uint64_t GAMMA = 0x9E3779B97F4A7C15ull;

__host__ __device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Round a double to bfloat16 (ties to even), for values in the normal range.
__device__ __forceinline__ __nv_bfloat16 d2bf16(double x) {
  uint64_t b = (uint64_t)__double_as_longlong(x);
  b += ((1ull << 44) - 1) + ((b >> 45) & 1);
  b &= ~((1ull << 45) - 1);
  const float f = (float)__longlong_as_double((long long)b);  // exact: 8 significant bits
  return __ushort_as_bfloat16((unsigned short)(__float_as_uint(f) >> 16));
}

template <typename T>
__device__ __forceinline__ T conv_weight(double x);
template <>
__device__ __forceinline__ float conv_weight<float>(double x) { return (float)x; }
template <>
__device__ __forceinline__ __nv_bfloat16 conv_weight<__nv_bfloat16>(double x) { return d2bf16(x); }

// Element n of tensor with stream state st: pairs (2j, 2j+1) from outputs 2j, 2j+1.
template <typename T>
__global__ void init_kernel(T* __restrict__ dst, int64_t rows, int64_t cols, uint64_t st, int64_t grp,
                            int64_t grp_stride, int64_t grp_off, int64_t pair_hd) {
  const int64_t n = rows * cols;
  const int64_t npairs = (n + 1) / 2;
  for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < npairs; j += (int64_t)gridDim.x * blockDim.x) {
    const uint64_t u0 = mix64(st + (uint64_t)(2 * j + 1) * GAMMA);
    const uint64_t u1 = mix64(st + (uint64_t)(2 * j + 2) * GAMMA);
    const double a = (double)((u0 >> 11) + 1) * 0x1p-53;
    const double b = (double)(u1 >> 11) * 0x1p-53;
    const double r = sqrt(-2.0 * log(a));
    const double t = 6.283185307179586 * b;
    const double z[2] = {r * cos(t), r * sin(t)};
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int64_t idx = 2 * j + e;
      if (idx >= n) break;
      int64_t rr = idx / cols;
      const int64_t cc = idx % cols;
      if (pair_hd) {  // head row i -> 2i (i < hd/2) or 2(i - hd/2) + 1
        const int64_t h = rr / pair_hd, i = rr % pair_hd, half = pair_hd / 2;
        rr = h * pair_hd + (i < half ? 2 * i : 2 * (i - half) + 1);
      }
      const int64_t drow = (rr / grp) * grp_stride + grp_off + rr % grp;
      dst[drow * cols + cc] = conv_weight<T>(0.02 * z[e]);
    }
  }
}

__global__ void fill_f32(float* p, int64_t n, float v) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) p[i] = v;
}

static uint64_t tensor_state(uint64_t seed, uint64_t tid) { return mix64(seed + (tid + 1) * GAMMA); }

template <typename T>
static int init_tensor(void* dst, int64_t rows, int64_t cols, uint64_t seed, uint64_t tid, int64_t grp,
                       int64_t grp_stride, int64_t grp_off, int64_t pair_hd) {
  const int64_t npairs = (rows * cols + 1) / 2;
  int64_t blocks = (npairs + 255) / 256;
  if (blocks > 65536) blocks = 65536;
  if (blocks < 1) blocks = 1;
  init_kernel<T><<<(unsigned)blocks, 256>>>(reinterpret_cast<T*>(dst), rows, cols, tensor_state(seed, tid),
                                            grp > 0 ? grp : rows, grp > 0 ? grp_stride : 0, grp_off, pair_hd);
  return launch_status();
}

static uint64_t fnv1a(const uint8_t* p, size_t n) {
  uint64_t h = 0xCBF29CE484222325ull;
  for (size_t i = 0; i < n; ++i) {
    h ^= p[i];
    h *= 0x100000001B3ull;
  }
  return h;
}

static uint64_t config_fingerprint(const dlmz_model_config& c) {
  uint8_t buf[7 * 4 + 2 * 4 + 8];
  uint32_t u[7] = {c.n_layers, c.d, c.n_heads, c.n_kv_heads, c.ffn, c.vocab, c.dtype};
  size_t o = 0;
  for (int i = 0; i < 7; ++i)
    for (int b = 0; b < 4; ++b) buf[o++] = (uint8_t)(u[i] >> (8 * b));
  uint32_t f[2];
  memcpy(&f[0], &c.rope_theta, 4);
  memcpy(&f[1], &c.norm_eps, 4);
  for (int i = 0; i < 2; ++i)
    for (int b = 0; b < 4; ++b) buf[o++] = (uint8_t)(f[i] >> (8 * b));
  for (int b = 0; b < 8; ++b) buf[o++] = (uint8_t)(c.seed >> (8 * b));
  return fnv1a(buf, o);
}

size_t model_workspace_per_token(const dlmz_model* m) {
  const size_t d = m->cfg.d, F = m->cfg.ffn;
  size_t b = 4 * d + m->esz * (2 * d + m->nqkv + F + m->dkv + 16 * m->cfg.n_kv_heads) + 4 * (d / 128);
  if (!m->tc) b += 4 * 2 * F;  // float32 gate/up buffer of the CUDA-core path
  return b;
}

template <typename T>
static int gemm(const T* A, const T* B, int M, int N, int K, int epi, const GemmEpilogue& ep, cudaStream_t s) {
  if constexpr (sizeof(T) == 2) {
    if (gemm_tc_supported(M, N, K) && epi != EPI_ROPE_BF16 && epi != EPI_SWIGLU_BF16)
      return gemm_bf16_tc(A, K, B, K, M, N, K, epi, ep, s);
  }
  return gemm_simt<T>(A, K, B, K, M, N, K, epi, ep, s);
}

// The layers of the forward (embedding through the last residual add) of nc
// windows of L positions; the float32 residual stream is left in ws.x for the
// LM head.  maps (optional): every layer's head-averaged attention
// [n_layers][nc][L][L].
template <typename T>
static int layers_impl(dlmz_model* m, const int32_t* state, int nc, int L, cudaStream_t s, float* maps = nullptr) {
  const dlmz_model_config& c = m->cfg;
  const int d = c.d, F = c.ffn, hd = m->hd, nq = m->nqkv;
  const int Tt = nc * L;
  ForwardWorkspace& w = m->ws;
  DLMZ_TRY(w.x.ensure((size_t)Tt * d * 4));
  DLMZ_TRY(w.h.ensure((size_t)Tt * d * sizeof(T)));
  DLMZ_TRY(w.qkv.ensure((size_t)Tt * nq * sizeof(T)));
  DLMZ_TRY(w.attn.ensure((size_t)Tt * d * sizeof(T)));
  DLMZ_TRY(w.act.ensure((size_t)Tt * F * sizeof(T)));
  if (!m->tc) DLMZ_TRY(w.gu.ensure((size_t)Tt * 2 * F * 4));
  // tensor-core attention reads V transposed (keys contiguous), written by the QKV epilogue
  const bool tc_attn = m->tc && attention_tc_supported(L, hd);
  if (tc_attn) {
    const int vrows = attention_vt_rows(hd), blocks = nc * (int)c.n_kv_heads;
    DLMZ_TRY(w.vt.ensure((size_t)blocks * vrows * L * 2));
  }
  if (w.rope_L < L) {  // (cos, sin) of pos * theta^(-2i/hd), from double precision
    const int half = hd / 2;
    std::vector<float2> cs((size_t)L * half);
    for (int p = 0; p < L; ++p)
      for (int i = 0; i < half; ++i) {
        const double ang = (double)p * pow((double)c.rope_theta, -2.0 * i / hd);
        cs[(size_t)p * half + i] = make_float2((float)cos(ang), (float)sin(ang));
      }
    DLMZ_TRY(w.rope.ensure(cs.size() * sizeof(float2)));
    DLMZ_CUDA_TRY(cudaMemcpy(w.rope.p, cs.data(), cs.size() * sizeof(float2), cudaMemcpyHostToDevice));
    w.rope_L = L;
  }
  float* x = w.x.as<float>();
  T* h = w.h.as<T>();
  T* qkv = w.qkv.as<T>();
  T* attn = w.attn.as<T>();
  T* act = w.act.as<T>();
  const float2* cs = w.rope.as<float2>();
  auto epi = [&](void* out, int ldo) {
    GemmEpilogue e{};
    e.out = out;
    e.ldo = ldo;
    e.rope_cs = cs;
    e.L = L;
    e.head_dim = hd;
    e.gu_block = m->gu_block;
    e.n_kv = (int)c.n_kv_heads;
    e.d_model = d;
    e.eps = c.norm_eps;
    return e;
  };
  GemmEpilogue ep{};
  if (m->tc) {
    // Tensor-core path with RMSNorm fused into the GEMM epilogues: h holds
    // bf16(x) and ssq the per-row partial sums of x^2 (unit norm gains).
    const int np = d / 128;
    DLMZ_TRY(w.ssq.ensure((size_t)Tt * np * 4));
    float* ssq = w.ssq.as<float>();
    bf16* y = reinterpret_cast<bf16*>(h);
    DLMZ_TRY(embed_norm(state, Tt, reinterpret_cast<const bf16*>(m->E), d, x, y, ssq, np, s));
    for (uint32_t l = 0; l < c.n_layers; ++l) {
      ep = epi(qkv, nq);
      ep.rope_cols = d + m->dkv;
      ep.ssq_in = ssq;
      ep.n_part = np;
      if (tc_attn) {
        ep.vt = w.vt.p;
        ep.v_col0 = d + m->dkv;
        ep.vt_rows = attention_vt_rows(hd);
      }
      DLMZ_TRY(gemm_bf16_tc(y, d, reinterpret_cast<const bf16*>(m->wqkv[l]), d, Tt, nq, d, EPI_ROPE_BF16, ep, s));
      if (maps)
        DLMZ_TRY(attention_maps<bf16>(reinterpret_cast<const bf16*>(qkv), nq, nc, L, c.n_heads, c.n_kv_heads, hd, d,
                                      maps + (size_t)l * Tt * L, s));
      if (tc_attn)
        DLMZ_TRY(attention_bf16_tc(reinterpret_cast<const bf16*>(qkv), nq, w.vt.p, nc, L, c.n_heads,
                                   c.n_kv_heads, hd, d, reinterpret_cast<bf16*>(attn), s));
      else if (hd == 64 || hd == 128)
        DLMZ_TRY(attention_bf16_mma(reinterpret_cast<const bf16*>(qkv), nq, nc, L, c.n_heads, c.n_kv_heads, hd, d,
                                    reinterpret_cast<bf16*>(attn), s));
      else
        DLMZ_TRY(attention_simt<bf16>(reinterpret_cast<const bf16*>(qkv), nq, nc, L, c.n_heads, c.n_kv_heads, hd, d,
                                      reinterpret_cast<bf16*>(attn), s));
      ep = epi(x, d);
      ep.y_out = y;
      ep.ssq_out = ssq;
      ep.n_part = np;
      DLMZ_TRY(gemm_bf16_tc(reinterpret_cast<const bf16*>(attn), d, reinterpret_cast<const bf16*>(m->wo[l]), d, Tt, d,
                            d, EPI_RESID_F32, ep, s));
      ep = epi(act, F);
      ep.ssq_in = ssq;
      ep.n_part = np;
      DLMZ_TRY(gemm_bf16_tc(y, d, reinterpret_cast<const bf16*>(m->wgu[l]), d, Tt, 2 * F, d, EPI_SWIGLU_BF16, ep, s));
      ep = epi(x, d);
      ep.y_out = y;
      ep.ssq_out = ssq;
      ep.n_part = np;
      DLMZ_TRY(gemm_bf16_tc(reinterpret_cast<const bf16*>(act), F, reinterpret_cast<const bf16*>(m->wdown[l]), F, Tt,
                            d, F, EPI_RESID_F32, ep, s));
    }
  } else {
    DLMZ_TRY(embed<T>(state, Tt, reinterpret_cast<const T*>(m->E), d, x, s));
    for (uint32_t l = 0; l < c.n_layers; ++l) {
      DLMZ_TRY(rmsnorm<T>(x, Tt, d, m->gains, c.norm_eps, h, L, 0, 0, s));
      ep = epi(qkv, nq);
      DLMZ_TRY(gemm<T>(h, reinterpret_cast<const T*>(m->wqkv[l]), Tt, nq, d, sizeof(T) == 2 ? EPI_BF16 : EPI_F32, ep,
                       s));
      DLMZ_TRY(rope_inplace<T>(qkv, Tt, nq, c.n_heads + c.n_kv_heads, hd, L, cs, s));
      if (maps) DLMZ_TRY(attention_maps<T>(qkv, nq, nc, L, c.n_heads, c.n_kv_heads, hd, d, maps + (size_t)l * Tt * L, s));
      if constexpr (sizeof(T) == 2) {
        if (hd == 64 || hd == 128)
          DLMZ_TRY(attention_bf16_mma(qkv, nq, nc, L, c.n_heads, c.n_kv_heads, hd, d, attn, s));
        else
          DLMZ_TRY(attention_simt<T>(qkv, nq, nc, L, c.n_heads, c.n_kv_heads, hd, d, attn, s));
      } else {
        DLMZ_TRY(attention_simt<T>(qkv, nq, nc, L, c.n_heads, c.n_kv_heads, hd, d, attn, s));
      }
      ep = epi(x, d);
      DLMZ_TRY(gemm<T>(attn, reinterpret_cast<const T*>(m->wo[l]), Tt, d, d, EPI_RESID_F32, ep, s));
      DLMZ_TRY(rmsnorm<T>(x, Tt, d, m->gains, c.norm_eps, h, L, 0, 0, s));
      ep = epi(w.gu.p, 2 * F);
      DLMZ_TRY(gemm<T>(h, reinterpret_cast<const T*>(m->wgu[l]), Tt, 2 * F, d, EPI_F32, ep, s));
      DLMZ_TRY(swiglu<T>(w.gu.as<float>(), Tt, F, m->gu_block, act, s));
      ep = epi(x, d);
      DLMZ_TRY(gemm<T>(act, reinterpret_cast<const T*>(m->wdown[l]), Tt, d, F, EPI_RESID_F32, ep, s));
    }
  }
  m->ws.x_tokens = Tt;
  return DLMZ_OK;
}

// LM head on R rows of the residual stream left by the last layers_impl:
// final RMSNorm of x rows (idx[r] when idx is given, else
// (r / rpc) * L + row0 + r % rpc) and f32 logits [R x V].
template <typename T>
static int head_impl(dlmz_model* m, const int32_t* idx, int R, int L, int row0, int rpc, float* logits,
                     cudaStream_t s, float* pmax = nullptr, float* pmin = nullptr, bool* parts = nullptr) {
  const dlmz_model_config& c = m->cfg;
  const int d = c.d, V = c.vocab;
  if (R == 0) return DLMZ_OK;
  ForwardWorkspace& w = m->ws;
  DLMZ_TRY(w.hc.ensure((size_t)R * d * sizeof(T)));
  T* hc = w.hc.as<T>();
  if (idx) DLMZ_TRY(rmsnorm_gather<T>(w.x.as<float>(), idx, R, d, m->gains, c.norm_eps, hc, s));
  else DLMZ_TRY(rmsnorm<T>(w.x.as<float>(), R, d, m->gains, c.norm_eps, hc, L, row0, rpc, s));
  GemmEpilogue ep{};
  ep.out = logits;
  ep.ldo = V;
  // the tensor-core epilogue can also leave each row's maxima and minima per 128 columns
  const bool tc = sizeof(T) == 2 && gemm_tc_supported(R, V, d);
  if (parts) *parts = tc && pmax && pmin;
  if (tc && pmax && pmin) {
    ep.pmax = pmax;
    ep.pmin = pmin;
    ep.n_part = V / 128;
  }
  return gemm<T>(hc, reinterpret_cast<const T*>(m->head), R, V, d, EPI_F32, ep, s);
}

int model_attention_maps(dlmz_model* m, const int32_t* state, int nc, int L, float* maps, cudaStream_t s) {
  if (nc <= 0 || L <= 0 || !maps) return DLMZ_EINVAL;
  if (m->bf16) return layers_impl<bf16>(m, state, nc, L, s, maps);
  return layers_impl<float>(m, state, nc, L, s, maps);
}

int model_layers(dlmz_model* m, const int32_t* state, int nc, int L, cudaStream_t s) {
  if (nc <= 0 || L <= 0) return DLMZ_EINVAL;
  if (m->bf16) return layers_impl<bf16>(m, state, nc, L, s);
  return layers_impl<float>(m, state, nc, L, s);
}

int model_head(dlmz_model* m, const int32_t* idx, int n, float* logits, cudaStream_t s, float* pmax, float* pmin,
               bool* parts) {
  if (parts) *parts = false;
  if (n < 0 || (n > 0 && (!idx || !logits))) return DLMZ_EINVAL;
  if (m->bf16) return head_impl<bf16>(m, idx, n, 0, 0, 0, logits, s, pmax, pmin, parts);
  return head_impl<float>(m, idx, n, 0, 0, 0, logits, s);
}

int model_forward(dlmz_model* m, const int32_t* state, int nc, int L, int row0, int rpc, float* logits,
                  cudaStream_t s) {
  if (nc <= 0 || L <= 0 || rpc <= 0 || row0 < 0 || row0 + rpc > L) return DLMZ_EINVAL;
  DLMZ_TRY(model_layers(m, state, nc, L, s));
  if (m->bf16) return head_impl<bf16>(m, nullptr, nc * rpc, L, row0, rpc, logits, s);
  return head_impl<float>(m, nullptr, nc * rpc, L, row0, rpc, logits, s);
}

}  // namespace dlmz

using namespace dlmz;

extern "C" int dlmz_model_create(const dlmz_model_config* cfg, dlmz_model** out) {
  if (!out) return DLMZ_EINVAL;
  *out = nullptr;
  if (!cfg) return DLMZ_EINVAL;
  const dlmz_model_config c = *cfg;
  if (!c.n_layers || !c.d || !c.n_heads || !c.n_kv_heads || !c.ffn || c.vocab < 2) return DLMZ_EINVAL;
  if (c.d % c.n_heads || c.n_heads % c.n_kv_heads) return DLMZ_EINVAL;
  if (c.dtype != DLMZ_FP32 && c.dtype != DLMZ_BF16) return DLMZ_EINVAL;
  if (c.vocab >= (1u << 24)) return DLMZ_EINVAL;
  const int hd = c.d / c.n_heads;
  if (hd % 2 || hd > 128) return DLMZ_EINVAL;
  if (!(c.rope_theta > 1.0f) || !(c.norm_eps >= 0.0f)) return DLMZ_EINVAL;
  dlmz_model* m = new dlmz_model();
  m->cfg = c;
  m->hd = hd;
  m->dkv = c.n_kv_heads * hd;
  m->nqkv = c.d + 2 * m->dkv;
  m->gu_block = (c.ffn % 128 == 0) ? 128 : (int)c.ffn;
  m->bf16 = c.dtype == DLMZ_BF16;
  m->esz = m->bf16 ? 2 : 4;
  m->tc = m->bf16 && c.d % 256 == 0 && m->nqkv % 256 == 0 && c.ffn % 128 == 0 && (hd == 32 || hd == 64 || hd == 128);
  if (!m->tc && !m->bf16 && hd > 64) {
    delete m;
    return DLMZ_EINVAL;
  }
  if (!m->bf16 && hd != 8 && hd != 16 && hd != 32 && hd != 64) {
    delete m;
    return DLMZ_EINVAL;
  }
  if (m->bf16 && !(hd == 64 || hd == 128) && hd != 8 && hd != 16 && hd != 32) {
    delete m;
    return DLMZ_EINVAL;
  }
  const size_t d = c.d, F = c.ffn, V = c.vocab, nl = c.n_layers;
  const size_t per_layer = (size_t)m->nqkv * d + d * d + 2 * F * d + d * F;
  const size_t elems = (V + 1) * d + V * d + nl * per_layer;
  const size_t align = 256;
  size_t bytes = 0;
  auto carve = [&](size_t n) {
    size_t off = bytes;
    bytes += (n * m->esz + align - 1) / align * align;
    return off;
  };
  std::vector<size_t> offs;
  offs.push_back(carve((V + 1) * d));
  offs.push_back(carve(V * d));
  for (size_t l = 0; l < nl; ++l) {
    offs.push_back(carve((size_t)m->nqkv * d));
    offs.push_back(carve(d * d));
    offs.push_back(carve(2 * F * d));
    offs.push_back(carve(d * F));
  }
  (void)elems;
  if (cudaMalloc(&m->weights, bytes) != cudaSuccess || cudaMalloc((void**)&m->gains, d * 4) != cudaSuccess) {
    cudaGetLastError();
    dlmz_model_destroy(m);
    return DLMZ_ENOMEM;
  }
  uint8_t* base = reinterpret_cast<uint8_t*>(m->weights);
  m->E = base + offs[0];
  m->head = base + offs[1];
  for (size_t l = 0; l < nl; ++l) {
    m->wqkv.push_back(base + offs[2 + 4 * l]);
    m->wo.push_back(base + offs[3 + 4 * l]);
    m->wgu.push_back(base + offs[4 + 4 * l]);
    m->wdown.push_back(base + offs[5 + 4 * l]);
  }
  const uint64_t seed = c.seed;
  const int64_t gb = m->gu_block;
  const size_t es = m->esz;
  int rc = DLMZ_OK;
  auto init = [&](void* dst, int64_t rows, int64_t cols, uint64_t tid, int64_t grp, int64_t gs, int64_t go,
                  int64_t pair_hd = 0) {
    if (rc != DLMZ_OK) return;
    rc = m->bf16 ? init_tensor<bf16>(dst, rows, cols, seed, tid, grp, gs, go, pair_hd)
                 : init_tensor<float>(dst, rows, cols, seed, tid, grp, gs, go, pair_hd);
  };
  const int64_t pair_hd = m->tc ? hd : 0;
  init(m->E, V + 1, d, 0, 0, 0, 0);
  init(m->head, V, d, 1, 0, 0, 0);
  for (size_t l = 0; l < nl; ++l) {
    const uint64_t t0 = 2 + 8 * l;
    uint8_t* q = reinterpret_cast<uint8_t*>(m->wqkv[l]);
    init(q, d, d, t0 + 0, 0, 0, 0, pair_hd);
    init(q + d * d * es, m->dkv, d, t0 + 1, 0, 0, 0, pair_hd);
    init(q + (d + m->dkv) * d * es, m->dkv, d, t0 + 2, 0, 0, 0);
    init(m->wo[l], d, d, t0 + 3, 0, 0, 0);
    init(m->wgu[l], F, d, t0 + 4, gb, 2 * gb, 0);
    init(m->wgu[l], F, d, t0 + 5, gb, 2 * gb, gb);
    init(m->wdown[l], d, F, t0 + 6, 0, 0, 0);
  }
  if (rc == DLMZ_OK) {
    fill_f32<<<(unsigned)((d + 255) / 256), 256>>>(m->gains, (int64_t)d, 1.0f);
    rc = launch_status();
  }
  if (rc == DLMZ_OK && cudaDeviceSynchronize() != cudaSuccess) rc = DLMZ_ECUDA;
  if (rc != DLMZ_OK) {
    dlmz_model_destroy(m);
    return rc;
  }
  m->fingerprint = config_fingerprint(c);
  *out = m;
  return DLMZ_OK;
}

extern "C" void dlmz_model_destroy(dlmz_model* m) {
  if (!m) return;
  if (m->weights) cudaFree(m->weights);
  if (m->gains) cudaFree(m->gains);
  m->ws.x.release();
  m->ws.h.release();
  m->ws.qkv.release();
  m->ws.attn.release();
  m->ws.act.release();
  m->ws.gu.release();
  m->ws.hc.release();
  m->ws.rope.release();
  m->ws.vt.release();
  m->ws.ssq.release();
  pipeline_release(m);
  delete m;
}

extern "C" uint64_t dlmz_model_fingerprint(const dlmz_model* m) { return m ? m->fingerprint : 0; }

extern "C" int dlmz_model_set_logits_budget(dlmz_model* m, size_t bytes) {
  if (!m) return DLMZ_EINVAL;
  m->logits_budget = bytes;
  return DLMZ_OK;
}

extern "C" int dlmz_model_get_config(const dlmz_model* m, dlmz_model_config* cfg) {
  if (!m || !cfg) return DLMZ_EINVAL;
  *cfg = m->cfg;
  return DLMZ_OK;
}
