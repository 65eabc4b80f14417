// Launch helpers shared between the translation units of libdlmz.
#pragma once

#include "common.cuh"

namespace dlmz {

typedef __nv_bfloat16 bf16;

// ---- GEMM epilogues --------------------------------------------------------
enum {
  EPI_BF16 = 0,        // out = bf16(acc)
  EPI_F32 = 1,         // out = acc (float32)
  EPI_RESID_F32 = 2,   // out += acc (float32 residual stream, in place)
  EPI_SWIGLU_BF16 = 3, // out[:, f] = bf16(silu(g_f) * u_f), gate/up interleaved in blocks
  EPI_ROPE_BF16 = 4,   // out = bf16(RoPE(acc)) on columns < rope_cols, bf16(acc) beyond; the
                       // head dimensions are stored as rotation pairs (2t, 2t+1)
};

struct GemmEpilogue {
  void* out;
  int ldo;               // output leading dimension (elements)
  const float2* rope_cs; // [L x head_dim/2] (cos, sin) for EPI_ROPE_BF16
  int L;                 // window length (position = row % L)
  int head_dim;
  int rope_cols;         // columns [0, rope_cols) get RoPE (Q and K heads)
  int gu_block;          // SwiGLU: gate/up interleave block (columns)
  void* vt;              // RoPE epilogue: if set, columns >= v_col0 (the V heads) go to
  int v_col0;            //   vt [window][kv head][vt_rows][L] as f16 (keys contiguous) instead of `out`
  int n_kv;
  int vt_rows;           //   head_dim + the attention kernel's extra rows
  // Fused RMSNorm.  Producer (residual epilogue): y_out = bf16(x) and per-row
  // partial sums of x^2, one per 128 columns, into ssq_out [rows x n_part].
  // Consumer (RoPE / SwiGLU epilogues): each row of the product is scaled by
  // rsqrt(sum of the row's n_part partials / d_model + eps) (unit norm gains).
  bf16* y_out;
  float* ssq_out;
  const float* ssq_in;
  int n_part;
  int d_model;
  float eps;
  // Float32 epilogue (LM head): if set, each row's maximum (NaN-propagating) and minimum over
  // every 128 output columns, into [rows x N / 128] each -- the quantiser's first pass.
  float* pmax;
  float* pmin;
};

// tcgen05 path: N % 256 == 0, K % 64 == 0, 16-byte aligned operands.
bool gemm_tc_supported(int M, int N, int K);
int gemm_bf16_tc(const bf16* A, int lda, const bf16* B, int ldb, int M, int N, int K, int epi,
                 const GemmEpilogue& ep, cudaStream_t s);
// CUDA-core path (any shape; float32 or bf16 inputs, float32 accumulation).
template <typename T>
int gemm_simt(const T* A, int lda, const T* B, int ldb, int M, int N, int K, int epi,
              const GemmEpilogue& ep, cudaStream_t s);

// ---- layers -------------------------------------------------------------------
// x[t] = E[state[t]] (f32), y[t] = bf16(x[t]), ssq[t] = {sum x^2, 0, ...} (n_part entries)
int embed_norm(const int32_t* state, int n, const bf16* E, int d, float* x, bf16* y, float* ssq, int n_part,
               cudaStream_t s);
template <typename T>
int embed(const int32_t* state, int T_tokens, const T* E, int d, float* x, cudaStream_t s);
// h[r] = OutT(x[row(r)] * g / sqrt(mean(x^2) + eps)); row(r) = (r / rpc) * L + row0 + r % rpc
// when rpc > 0, else r.
template <typename OutT>
int rmsnorm(const float* x, int rows, int d, const float* g, float eps, OutT* h, int L, int row0,
            int rpc, cudaStream_t s);
// h[r] = OutT(x[idx[r]] * g / sqrt(mean(x^2) + eps)) (rows gathered by token index).
template <typename OutT>
int rmsnorm_gather(const float* x, const int32_t* idx, int rows, int d, const float* g, float eps, OutT* h,
                   cudaStream_t s);
template <typename T>
int rope_inplace(T* qkv, int T_tokens, int ld, int n_heads_rot, int head_dim, int L,
                 const float2* cs, cudaStream_t s);
template <typename T>
int swiglu(const float* gu, int T_tokens, int F, int gu_block, T* out, cudaStream_t s);
template <typename T>
int attention_simt(const T* qkv, int ld, int n_chunks, int L, int n_heads, int n_kv_heads,
                   int head_dim, int d, T* out, cudaStream_t s);
// Head-averaged attention probabilities of every window [n_chunks][L][L] from the
// RoPE'd Q and K of one layer (attention-based context, Sec. 3.4).
template <typename T>
int attention_maps(const T* qkv, int ld, int n_chunks, int L, int n_heads, int n_kv_heads, int head_dim, int d,
                   float* maps, cudaStream_t s);
bool attention_tc_supported(int L, int hd);
int attention_bf16_tc(const bf16* qkv, int ld, const void* vt, int n_chunks, int L, int n_heads, int n_kv_heads,
                      int head_dim, int d, bf16* out, cudaStream_t s);
// Rows per (window, kv head) of the attention kernel's V^T buffer.
int attention_vt_rows(int head_dim);
// Writes that buffer (f16) from the V columns [v_col, v_col + n_kv_heads * head_dim) of bf16 rows.
int attention_vt_from_rows(const bf16* qkv, int ld, int v_col, int n_chunks, int L, int n_kv_heads, int head_dim,
                           void* vt, cudaStream_t s);
int attention_bf16_mma(const bf16* qkv, int ld, int n_chunks, int L, int n_heads, int n_kv_heads,
                       int head_dim, int d, bf16* out, cudaStream_t s);

// ---- quantiser / selector / coder --------------------------------------------------
int quantize_rows(const float* logits, int rows, int V, int P, uint32_t* cdf, uint64_t* W,
                  uint64_t* A, int32_t* Hq, int32_t* top, float* mx, cudaStream_t s,
                  const float* pmax = nullptr, const float* pmin = nullptr);

}  // namespace dlmz
