// Model object: device weights of the masked DLM and its forward workspace.
#pragma once

#include <vector>

#include "kernels.cuh"

namespace dlmz {

// Grow-only device buffer.
struct DevBuf {
  void* p = nullptr;
  size_t bytes = 0;
  int ensure(size_t n) {
    if (n <= bytes) return DLMZ_OK;
    if (p) cudaFree(p);
    p = nullptr;
    bytes = 0;
    if (n == 0) return DLMZ_OK;
    if (cudaMalloc(&p, n) != cudaSuccess) {
      cudaGetLastError();
      return DLMZ_ENOMEM;
    }
    bytes = n;
    return DLMZ_OK;
  }
  void release() {
    if (p) cudaFree(p);
    p = nullptr;
    bytes = 0;
  }
  template <typename T>
  T* as() const { return reinterpret_cast<T*>(p); }
};

struct ForwardWorkspace {
  DevBuf x, h, qkv, attn, act, gu, hc, rope, vt, ssq;
  int rope_L = 0;
  int64_t x_tokens = 0;  // rows of x written by the last model_layers
};

}  // namespace dlmz

struct dlmz_model {
  dlmz_model_config cfg;
  int hd, dkv, nqkv, gu_block;
  bool bf16;
  bool tc;  // tensor-core GEMM path usable for every projection
  size_t esz;
  void* weights = nullptr;  // one allocation
  void* E = nullptr;
  std::vector<void*> wqkv, wo, wgu, wdown;
  void* head = nullptr;
  float* gains = nullptr;  // ones [d]
  uint64_t fingerprint = 0;
  dlmz::ForwardWorkspace ws;
  void* pipe = nullptr;  // pipeline workspace (owned, see pipeline.cu)
  size_t logits_budget = 0;  // bytes of candidate logits a step holds at once (0: the default)
};

namespace dlmz {
// Forward of a batch (Definition 3): logits [n_chunks*rpc x V] for positions
// [row0, row0+rpc) of every window.
int model_forward(dlmz_model* m, const int32_t* state, int n_chunks, int L, int row0, int rpc, float* logits,
                  cudaStream_t s);
// The layers of the forward (embedding through the last residual add) of a
// batch; the float32 residual stream stays in the model's workspace until the
// next call, for model_head.
int model_layers(dlmz_model* m, const int32_t* state, int n_chunks, int L, cudaStream_t s);
// LM head on n rows of the last model_layers batch: final RMSNorm of the
// residual rows idx[0..n) (token index = window * L + position) and float32
// logits [n x V].  Each row's logits depend only on that row, so a row gives
// bit-identical logits in any call and at any place in idx.  pmax / pmin (optional,
// [n x V / 128]): on the tensor-core path each row's maximum (NaN-propagating) and
// minimum per 128 logits, for the quantiser; *parts tells whether they were written.
int model_head(dlmz_model* m, const int32_t* idx, int n, float* logits, cudaStream_t s, float* pmax = nullptr,
               float* pmin = nullptr, bool* parts = nullptr);
// Every layer's head-averaged attention probabilities [n_layers][n_chunks][L][L]
// for the windows' states (no LM head).
int model_attention_maps(dlmz_model* m, const int32_t* state, int n_chunks, int L, float* maps, cudaStream_t s);
// Attention-based context scores [n_chunks][L] of the windows' symbols (Sec. 3.4):
// two masked passes, Attention Rollout; maps and state are scratch.
int context_attention_scores(dlmz_model* m, const int32_t* symbols, int n_chunks, int L, float* scores, DevBuf& maps,
                             DevBuf& state, cudaStream_t s);
// Frees the pipeline workspace attached to the model (pipeline.cu).
void pipeline_release(dlmz_model* m);
// Bytes of forward workspace per token (for batch sizing).
size_t model_workspace_per_token(const dlmz_model* m);
}  // namespace dlmz
