/*
 * dlmz.h -- C ABI of the GB300 (sm_103a) diffusion-LM lossless compressor.
 *
 * Method: "Diffuse to Compress: Leveraging Diffusion LMs for Lossless
 * Compression".  A masked, bidirectional diffusion LM (Definition 3,
 * Sec. 3.1) predicts a distribution for every masked position of a window
 * in one forward pass; a commitment schedule (Sec. 3.3) picks positions;
 * their true symbols are entropy coded under the predicted distributions
 * and revealed as context (iterative pipeline, Sec. 3.2); the input is cut
 * into non-overlapping windows of size w stored in the header (Sec. 4).
 *
 * Conventions for every entry point:
 *  - Return 0 on success or a negative DLMZ_E* code; dlmz_strerror() names it.
 *  - "d_" pointers are device pointers (CUDA global memory of the current
 *    device); other pointers are host pointers.  The caller owns every
 *    buffer it passes in; the library never frees them.
 *  - "stream" is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Step-level calls are asynchronous on that stream; whole-file
 *    calls synchronise it before returning.
 *  - Device kernels never wait unboundedly: a pipeline wait that exceeds its
 *    time limit makes the call return DLMZ_ETIMEOUT.
 *  - A model is immutable after creation and may be shared by sequential
 *    calls; calls on one model are not thread-safe.
 */
#ifndef DLMZ_H
#define DLMZ_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define DLMZ_API __attribute__((visibility("default")))
#else
#define DLMZ_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* ---- error codes ------------------------------------------------------ */
#define DLMZ_OK 0
#define DLMZ_EINVAL (-1)      /* bad argument (NULL pointer, zero size, unsupported shape) */
#define DLMZ_EBADINPUT (-2)   /* input symbols invalid (token id >= V, length not a multiple of 4) */
#define DLMZ_ECORRUPT (-3)    /* container damaged: magic, version, lengths, stream or checksum */
#define DLMZ_EMODEL (-4)      /* container written by a different model (fingerprint mismatch) */
#define DLMZ_ENOMEM (-5)      /* host or device allocation failed */
#define DLMZ_ECUDA (-6)       /* a CUDA runtime or driver call failed */
#define DLMZ_ETIMEOUT (-7)    /* a device-side pipeline wait exceeded its limit */
#define DLMZ_ECAPACITY (-8)   /* caller-provided output buffer too small */

/* ---- model -------------------------------------------------------------- */
#define DLMZ_FP32 0u
#define DLMZ_BF16 1u

typedef struct dlmz_model dlmz_model; /* opaque; owns the device weights */

/* LLaDA-style masked DLM (Definition 3): pre-norm blocks of RMSNorm ->
 * GQA/MHA attention with RoPE (rotate-half, applied to Q and K), no causal
 * mask -> residual -> RMSNorm -> SwiGLU FFN -> residual; final RMSNorm and
 * an untied LM head over V symbols.  The embedding has V+1 rows; row V is
 * [MASK].  d must be a multiple of n_heads, n_heads of n_kv_heads, and the
 * head dimension even. */
typedef struct {
  uint32_t n_layers, d, n_heads, n_kv_heads, ffn, vocab;
  uint32_t dtype;      /* DLMZ_FP32: all storage float32; DLMZ_BF16: bf16 weights and
                          activations between kernels, float32 residual stream and logits */
  float rope_theta;    /* RoPE base (10000) */
  float norm_eps;      /* RMSNorm epsilon (1e-5) */
  uint64_t seed;       /* weights ~ N(0, 0.02) from SplitMix64 + Box-Muller of (seed, tensor, index) */
} dlmz_model_config;

/* Create a randomly initialised model on the current device (trained
 * weights stand in: Sec. 4 uses LLaDA-8B).  *out receives the handle; on
 * error *out is NULL.  Errors: EINVAL (shape), ENOMEM, ECUDA. */
DLMZ_API int dlmz_model_create(const dlmz_model_config* cfg, dlmz_model** out);
/* Release the model and its device memory.  NULL is accepted. */
DLMZ_API void dlmz_model_destroy(dlmz_model* m);
/* FNV-1a 64 of the packed configuration; stored in every container header. */
DLMZ_API uint64_t dlmz_model_fingerprint(const dlmz_model* m);
/* Copy the model configuration into *cfg. */
DLMZ_API int dlmz_model_get_config(const dlmz_model* m, dlmz_model_config* cfg);
/* Memory budget of one denoising step's logits.  A step's LM head and
 * quantiser run on its candidate rows only -- the masked positions of the
 * active block of each window, the rows that get a distribution
 * (Definition 3).  When the candidates' float32 logits [rows x V] exceed
 * `bytes`, the head and the quantiser's scores run in slabs of rows, and
 * after the selection the selected rows' logits are computed once more for
 * the coder (bit-identical: a row's logits depend only on that row).
 * 0 restores the default (24 GiB).  Streams do not depend on the budget.
 * Errors: EINVAL (NULL model). */
DLMZ_API int dlmz_model_set_logits_budget(dlmz_model* m, size_t bytes);

/* ---- commitment schedule (Sec. 3.3) and initial context (Sec. 3.4) ---- */
#define DLMZ_TOPK_CONF 0u   /* k most confident masked positions of the leftmost incomplete block */
#define DLMZ_ENTROPY 1u     /* all masked positions with entropy <= tau; at least k_min, at most k_max */
#define DLMZ_UNIFORM 2u     /* uniform block (Sec. 3.3 par. 1): K = k steps of floor(n/K) masked positions,
                               left to right, the last step taking the remainder */
#define DLMZ_PROGRESSIVE 3u /* progressive (Sec. 3.3 par. 2): u_k = round(u_1 r^(k-1)) left to right,
                               u_1 = k, r = growth_q16 / 65536 (exact 16.16 fixed-point sequence) */

#define DLMZ_CODER_RANGE 0u /* range coder, minimal termination: ideal length + at most ~1 bit per window */
#define DLMZ_CODER_RANS 1u  /* rANS, 64-bit state, 32-bit words: ideal length + at most 96 bits per window */
#define DLMZ_CODER_RANKS 2u /* symbol ranking: each symbol's rank (frequency descending, ties by index) as an
                               LEB128 varint -- the paper's ranking pipeline before its back-end compressor */

#define DLMZ_CONTEXT_NONE 0u       /* every position starts masked (c = 0) */
#define DLMZ_CONTEXT_CONTIGUOUS 1u /* the first c symbols of each window stay visible */
#define DLMZ_CONTEXT_RANDOM 2u     /* c positions per window drawn from context_seed (SplitMix64,
                                      partial Fisher-Yates); symbols stored raw in the file */
#define DLMZ_CONTEXT_ATTENTION 3u  /* attention-based (Sec. 3.4, policy 4): the c positions that masked tokens
                                      attend to most (two complementary masked forwards, Attention Rollout);
                                      positions and symbols stored in the file */

typedef struct {
  uint32_t kind;
  uint32_t k;            /* TOPK_CONF: positions per step; UNIFORM: K steps; PROGRESSIVE: u_1 (all >= 1) */
  uint32_t block;        /* TOPK_CONF: block length; 0 = the whole window */
  float tau_bits;        /* ENTROPY: threshold tau in bits (entropy base 2) */
  uint32_t k_min;        /* ENTROPY: m, minimum positions per step (>= 1) */
  uint32_t k_max;        /* ENTROPY: cap per step; 0 = no cap */
  uint32_t growth_q16;   /* PROGRESSIVE: growth ratio r in 16.16 fixed point, 1 .. 64 * 65536 */
  uint32_t context;      /* DLMZ_CONTEXT_*: initial context of every window (compress only; the
                            decompressor reads it from the file) */
  uint32_t context_c;    /* c, symbols per window left visible (0 exactly when context is NONE) */
  uint32_t coder;        /* DLMZ_CODER_RANGE (default), DLMZ_CODER_RANS (the paper's rANS, Sec. 2.1) or
                            DLMZ_CODER_RANKS (symbol ranking, varint ranks) */
  uint64_t context_seed; /* RANDOM: seed of the positions */
} dlmz_k_policy;

/* ---- whole-file API, host buffers ------------------------------------ */
/* Compress in[0, in_bytes) with windows of chunk_len symbols (w, Sec. 4).
 * Symbols are bytes when V <= 256, otherwise little-endian uint32 token ids
 * (in_bytes % 4 == 0, each id < V) -- else EBADINPUT.  On success *out is a
 * malloc'd container of *out_bytes bytes, released with dlmz_free; on error
 * *out is NULL.  batch_chunks = 0 picks the default batch (<= 1024 windows
 * per forward batch, bounded by device memory); the value used is stored in
 * the header so the decoder replays the same batches.  The policy's context
 * fields select an initial context (Sec. 3.4): those symbols are stored raw
 * in the file and not coded. */
DLMZ_API int dlmz_compress(const dlmz_model* m, const void* in, size_t in_bytes, uint32_t chunk_len,
                  const dlmz_k_policy* policy, uint8_t** out, size_t* out_bytes);
DLMZ_API int dlmz_compress_ex(const dlmz_model* m, const void* in, size_t in_bytes, uint32_t chunk_len,
                     const dlmz_k_policy* policy, uint32_t batch_chunks, uint8_t** out,
                     size_t* out_bytes);
/* Decompress a container; *out is malloc'd (release with dlmz_free).
 * Errors: ECORRUPT (header, lengths, streams or CRC-32), EMODEL (fingerprint). */
DLMZ_API int dlmz_decompress(const dlmz_model* m, const uint8_t* stream, size_t stream_bytes,
                    uint8_t** out, size_t* out_bytes);
/* Free a buffer returned by the library.  NULL is accepted. */
DLMZ_API void dlmz_free(void* p);
/* Static description of an error code. */
DLMZ_API const char* dlmz_strerror(int code);

/* ---- whole-file API, device-resident --------------------------------- */
/* Upper bound of the container size for in_bytes of input. */
DLMZ_API size_t dlmz_compress_bound(const dlmz_model* m, size_t in_bytes, uint32_t chunk_len);
/* As dlmz_compress_ex with d_in / d_out in device memory; out_cap is d_out's
 * capacity (ECAPACITY if too small); *out_bytes is the container size. */
DLMZ_API int dlmz_compress_device(const dlmz_model* m, const void* d_in, size_t in_bytes, uint32_t chunk_len,
                         const dlmz_k_policy* policy, uint32_t batch_chunks, uint8_t* d_out,
                         size_t out_cap, size_t* out_bytes, void* stream);
/* As dlmz_decompress with d_in / d_out in device memory. */
DLMZ_API int dlmz_decompress_device(const dlmz_model* m, const uint8_t* d_in, size_t in_bytes,
                           uint8_t* d_out, size_t out_cap, size_t* out_bytes, void* stream);

/* ---- step-level API (device pointers) ---------------------------------
 * A batch holds n_chunks windows of equal length L.  "state" is int32
 * [n_chunks x L] with symbol ids in [0, V] (V = [MASK]).  The LM-head rows
 * of a step are the positions [row0, row0 + rows_per_chunk) of every window,
 * row r belonging to window r / rows_per_chunk. */

/* Masked-DLM forward (Definition 3): float32 logits [n_chunks*rows_per_chunk x V]
 * for positions [row0, row0+rows_per_chunk) of every window of d_state. */
DLMZ_API int dlmz_forward_logits(const dlmz_model* m, const int32_t* d_state, uint32_t n_chunks,
                        uint32_t L, uint32_t row0, uint32_t rows_per_chunk, float* d_logits,
                        void* stream);
/* Attention-based context scores (Sec. 3.4, policy 4) of n_chunks windows of L
 * symbols d_symbols [n_chunks x L] (int32, each < V): two forwards, one with
 * the even and one with the odd positions masked; every layer's attention
 * averaged over heads, A_l, and rolled out (Attention Rollout: R = Ã_N ... Ã_1,
 * Ã_l = A_l / 2 + I / 2); d_scores [n_chunks x L] (float32) receives, for each
 * position j, sum over the masked i of R[i, j] from the pass in which j is
 * visible.  Compression keeps the c highest (ties: lower position).  Uses
 * n_layers * n_chunks * L^2 * 4 bytes of device scratch.  Errors: EINVAL. */
DLMZ_API int dlmz_context_scores(const dlmz_model* m, const int32_t* d_symbols, uint32_t n_chunks, uint32_t L,
                                 float* d_scores, void* stream);

/* Dense contraction of the forward (Definition 3's projections and LM head):
 * d_D [M x N] float32 = d_A [M x K] bf16 . d_B [N x K]^T bf16, all row-major
 * and contiguous.  Runs on the tcgen05 tensor cores when N % 256 == 0 and
 * K % 64 == 0 (16-byte aligned operands), else on CUDA cores.  Each output
 * element's K order is fixed, so results do not depend on M. */
DLMZ_API int dlmz_gemm_bf16(const void* d_A, const void* d_B, float* d_D, uint32_t M, uint32_t N, uint32_t K,
                            void* stream);

/* Bidirectional grouped-query attention of one layer (Definition 3: every
 * position attends to every position of its window; no mask), on its own:
 * for window w, query head h and its KV head g = h / (n_heads / n_kv_heads),
 *   out[w L + i, h hd + e] = sum_j softmax_j(q_i . k_j / sqrt(hd)) v_j[e].
 * d_qkv: bf16 [n_chunks L x ld] device rows (window-major, L rows per window),
 *   columns [Q heads | K heads | V heads]: query head h at h*hd, key head g at
 *   n_heads*hd + g*hd, value head g at (n_heads + n_kv_heads)*hd + g*hd;
 *   ld >= (n_heads + 2 n_kv_heads) hd and a multiple of 8.
 * d_out: bf16 [n_chunks L x n_heads hd] device.  Both 16-byte aligned; the
 *   caller owns both.
 * head_dim one of 8, 16, 32, 64, 128; n_chunks <= 65535.  Runs on the tcgen05
 * tensor cores when L % 128 == 0 and head_dim is 64 or 128 (V is converted to
 * f16 there, so |v| < 65504), else on CUDA cores; P is rounded to f16 (tensor
 * cores) or kept in float32 (CUDA cores) before P V.  The tensor-core path
 * converts V into a library-owned V^T scratch buffer (grown with cudaMalloc
 * as needed, kept until exit): calls that overlap on the GPU race on it;
 * sequential calls are independent.  DLMZ_EINVAL on bad sizes or alignment,
 * DLMZ_ENOMEM if the V^T scratch cannot be allocated. */
DLMZ_API int dlmz_attention_bf16(const void* d_qkv, uint32_t ld, uint32_t n_chunks, uint32_t L, uint32_t n_heads,
                                 uint32_t n_kv_heads, uint32_t head_dim, void* d_out, void* stream);

/* Integer quantiser (one rule shared by encoder and decoder): per row of
 * float32 logits [rows x V], with P CDF bits (V < 2^P, P <= 24):
 *   m = max, top = lowest argmax; q_v = rint(min(fl(fl(m - l_v) * C), 8191)),
 *   C = fl32(256 log2 e); w_v = T[q_v & 255] >> (q_v >> 8), T[j] = round(2^31 2^(-j/256));
 *   W = sum w_v; A = sum w_v q_v; f_v = 1 + floor(w_v (2^P - V) / W), remainder to top;
 *   Hq = entropy (Sec. 3.3, bits) of w/W in units of 2^-16 bit.
 * Outputs (any may be NULL except d_W and d_Hq): d_cdf [rows x (V+1)] uint32,
 * d_W uint64, d_A uint64, d_Hq int32, d_top int32.  Non-finite logits give
 * EBADINPUT (checked on the device, reported after synchronising). */
DLMZ_API int dlmz_quantize(const float* d_logits, uint32_t rows, uint32_t V, uint32_t P, uint32_t* d_cdf,
                  uint64_t* d_W, uint64_t* d_A, int32_t* d_Hq, int32_t* d_top, void* stream);

/* Per group of group_size consecutive rows, the k rows with the smallest
 * (key, index), written ascending as in-group indices to d_out [groups x k]
 * (k <= group_size <= 4096).  With keys = Hq this is the entropy top-k of the
 * isolated quantise+select workload. */
DLMZ_API int dlmz_select_smallest(const uint64_t* d_keys, uint32_t groups, uint32_t group_size, uint32_t k,
                         int32_t* d_out, void* stream);

/* Allocation-free dlmz_select_smallest (the paper has no counterpart: this is
 * a deployment entry point).  For callers that cannot call cudaMalloc -- code
 * whose device memory belongs to another allocator, latency-critical paths
 * that cannot take cudaMalloc's implicit device synchronisation, hosts with a
 * fixed device-memory budget.  Same arguments and results as
 * dlmz_select_smallest; the kernel's scratch (one count per group) is a
 * static device array of 65536 int32 (256 KiB, held by every GPU that loads
 * the library until exit), so groups > 65536 returns DLMZ_EINVAL.  The first
 * call on a device looks up the array's device address (cudaGetSymbolAddress)
 * and must come before any stream capture.  Calls share the array: calls that
 * overlap on the GPU race; sequential calls need no clearing between them.
 * It calls no cudaMalloc or cudaFree. */
DLMZ_API int dlmz_select_smallest_noalloc(const uint64_t* d_keys, uint32_t groups, uint32_t group_size, uint32_t k,
                                          int32_t* d_out, void* stream);

/* Opaque per-batch coder state (range coder, one stream per window). */
typedef struct dlmz_coder dlmz_coder;
/* Allocate coder state for n_chunks windows of length L with P-bit tables. */
DLMZ_API int dlmz_coder_create(uint32_t n_chunks, uint32_t L, uint32_t V, uint32_t P, dlmz_coder** out);
/* As dlmz_coder_create with the statistical coder chosen (DLMZ_CODER_*); the
 * policies given to its steps must name the same coder (else EINVAL).  rANS
 * keeps each window's (c, f) pairs until dlmz_coder_finish codes them. */
DLMZ_API int dlmz_coder_create_ex(uint32_t n_chunks, uint32_t L, uint32_t V, uint32_t P, uint32_t coder,
                                  dlmz_coder** out);
DLMZ_API void dlmz_coder_destroy(dlmz_coder* c);
/* Encoder: reset every stream to the empty state.  Decoder: read stream c
 * from d_bytes + d_offsets[c] (big-endian 16-bit units, d_bits[c] bits long;
 * bytes past the length read as zero and are never accessed).  The device
 * buffers must stay valid while decode steps run. */
DLMZ_API int dlmz_coder_reset_encoder(dlmz_coder* c, void* stream);
DLMZ_API int dlmz_coder_load_decoder(dlmz_coder* c, const uint8_t* d_bytes, const uint64_t* d_offsets,
                            const uint32_t* d_bits, void* stream);
/* One commitment step (Sec. 3.2 / 3.3) on logits of the step's rows:
 * quantise, select with the policy, code the selected positions in ascending
 * order into each window's stream (encoder: true symbols from d_symbols
 * [n_chunks x L]; decoder: decoded) and reveal them in d_state.
 * d_committed (may be NULL) receives the number of positions committed per
 * window [n_chunks].  For UNIFORM and PROGRESSIVE the caller runs the
 * schedule: policy->k is this step's u_k, and the step commits the u_k
 * leftmost masked positions inside the rows (the logits' scores are not used).
 * The policy's context fields are ignored here (the caller sets d_state). */
DLMZ_API int dlmz_encode_step(dlmz_coder* c, const dlmz_k_policy* policy, const float* d_logits,
                     uint32_t row0, uint32_t rows_per_chunk, const int32_t* d_symbols,
                     int32_t* d_state, int32_t* d_committed, void* stream);
DLMZ_API int dlmz_decode_step(dlmz_coder* c, const dlmz_k_policy* policy, const float* d_logits,
                     uint32_t row0, uint32_t rows_per_chunk, int32_t* d_state,
                     int32_t* d_committed, void* stream);
/* One denoising step with the model's own distributions (Sec. 3.2), over
 * the coder's batch (n_chunks windows of L positions, d_state [n_chunks x L],
 * [MASK] = V): the forward pass of the batch (Definition 3), the LM head and
 * the quantiser on the candidate rows only -- the masked positions of
 * [row0, row0 + rows_per_chunk) in each window -- the selection of the policy
 * (Sec. 3.3; confidence or entropy keys, or the k leftmost masked positions
 * for UNIFORM / PROGRESSIVE with k = the step's size), then the coding
 * (encode: the true symbols d_symbols [n_chunks x L]) or decoding of the
 * selected positions, which are revealed in d_state.  d_committed (optional,
 * [n_chunks]) receives the count per window.  The model's V must be the
 * coder's and P the library's precision for it (16 for V <= 4096, else 24);
 * policy->coder must be the coder's kind and policy->context NONE (a caller
 * that wants an initial context reveals it in d_state itself).  Synchronises
 * once with the host per call (the candidate count sizes the LM head).
 * Errors: EINVAL, ENOMEM, ECUDA; stream corruption shows at dlmz_check. */
DLMZ_API int dlmz_model_encode_step(dlmz_model* m, dlmz_coder* c, const dlmz_k_policy* policy, uint32_t row0,
                                    uint32_t rows_per_chunk, const int32_t* d_symbols, int32_t* d_state,
                                    int32_t* d_committed, void* stream);
DLMZ_API int dlmz_model_decode_step(dlmz_model* m, dlmz_coder* c, const dlmz_k_policy* policy, uint32_t row0,
                                    uint32_t rows_per_chunk, int32_t* d_state, int32_t* d_committed, void* stream);
/* Terminate every stream (call once per encoded batch): bit lengths to
 * d_bits [n_chunks]; if d_bytes is not NULL each stream's ceil(bits/8) bytes
 * are copied to d_bytes + d_offsets[c], or to d_bytes + c * 2 *
 * dlmz_coder_capacity_units() when d_offsets is NULL. */
DLMZ_API int dlmz_coder_finish(dlmz_coder* c, uint32_t* d_bits, uint8_t* d_bytes, const uint64_t* d_offsets,
                      void* stream);
/* Maximum stream size in units per window for this coder. */
DLMZ_API uint32_t dlmz_coder_capacity_units(const dlmz_coder* c);
/* Synchronise and report any device-side error flag (ECORRUPT for a stream
 * that cannot come from the encoder, ETIMEOUT, EBADINPUT). */
DLMZ_API int dlmz_check(void* stream);

/* Failure-detection self-test (not part of the method): launches a kernel
 * whose bounded mbarrier wait (the kind every pipeline kernel uses) gives up
 * after limit_us microseconds (1 .. 1e6) because nothing arrives.  Returns
 * DLMZ_ETIMEOUT when the timeout was detected and reported the way a stuck
 * pipeline wait is; the device error word is cleared and the context stays
 * usable.  Errors: EINVAL (limit), ECUDA. */
DLMZ_API int dlmz_selftest_wait_timeout(uint32_t limit_us, void* stream);
/* The same for the cluster-scope wait of the quantiser's CTA pairs: a cluster
 * of two CTAs, CTA 0 waits (limit_us, 1 .. 1e6) on its mbarrier for one
 * arrival that CTA 1 makes through distributed shared memory only when
 * peer_arrives is 1.  Returns DLMZ_OK when the wait completed (peer_arrives
 * 1), DLMZ_ETIMEOUT when it gave up (peer_arrives 0); the device error word
 * is cleared and the context stays usable.  Errors: EINVAL (limit,
 * peer_arrives > 1), ECUDA. */
DLMZ_API int dlmz_selftest_cluster_wait(uint32_t limit_us, uint32_t peer_arrives, void* stream);

/* ---- live profiling (not part of the method) ------------------------------
 * Between dlmz_profile_begin and dlmz_profile_end the library records CUDA
 * events on each launch's stream around every kernel and counts launches.
 * Classes: 0 tensor-core GEMM, 1 CUDA-core GEMM, 2 attention, 3 quantiser,
 * 4 selector, 5 coder, 6 embedding/norm/RoPE/SwiGLU, 7 other.  flops and
 * bytes are the algorithmic work of the timed launches (2MNK for a GEMM,
 * 4 L^2 hd per window-head for attention, logits read for the quantiser). */
typedef struct {
  uint64_t launches;     /* every kernel launched by the library */
  uint64_t n[8];         /* timed launches per class */
  double ms[8];          /* summed launch durations per class (ms) */
  double flops[8];
  double bytes[8];
} dlmz_profile;
DLMZ_API int dlmz_profile_begin(void);
/* Number of kernels the library has launched since it was loaded (all
 * devices and streams; counted whether or not profiling is on, at no device
 * cost), so a caller can count the launches of a timed region without the
 * per-launch events of dlmz_profile_begin. */
DLMZ_API uint64_t dlmz_launch_count(void);
/* Synchronises the device and fills *out. */
DLMZ_API int dlmz_profile_end(dlmz_profile* out);

#ifdef __cplusplus
}
#endif
#endif /* DLMZ_H */
