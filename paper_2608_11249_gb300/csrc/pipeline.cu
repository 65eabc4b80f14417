// Iterative DLM compression pipeline (Sec. 3.2) and the C ABI.
//
// compress: the input is cut into non-overlapping windows of chunk_len
// symbols (w, Sec. 4); windows of equal length run as a batch.  Each batch
// starts masked -- fully, or with c context symbols per window left visible
// (Sec. 3.4) -- and repeats forward -> quantise -> select -> code -> reveal
// until every masked position is committed (coverage sum u_k = n, Sec. 3.3).  Each window owns one range-coder stream.  decompress replays
// the same batches and schedule from the header alone (Sec. 3.3, last
// paragraph): the selection of a step never depends on the symbols that
// step codes, so the decoder sees the same logits at every step.
//
// Container (little-endian): 64-byte header (magic "DLMZ", version, P,
// policy kind, model fingerprint, V, chunk_len, batch_chunks, k, block,
// tau_q, k_min, k_max, n_symbols, n_chunks, checksum), one LEB128 varint per
// window with its stream's bit length, then the streams (ceil(bits/8) bytes
// each).  The checksum is the CRC-32 (IEEE) of the windows' CRC-32s.
// Version 2 (a context, Sec. 3.4) extends the header by 16 bytes (context
// kind, c, seed) and puts the context symbols (min(c, window) per window,
// ascending position, 1 or 4 bytes each) between the header and the lengths.
// For the progressive schedule the block field holds r in 16.16 fixed point.
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <vector>

#include "coder.cuh"
#include "model.cuh"

namespace dlmz {

// ---- error word -------------------------------------------------------------------------
static int* g_err[kMaxDevices] = {};
int* device_error_word() {
  const int dev = device_ordinal();
  if (dev < 0) return nullptr;
  if (!g_err[dev]) {
    int* p = nullptr;
    if (cudaMalloc(&p, sizeof(int)) != cudaSuccess) return nullptr;
    cudaMemset(p, 0, sizeof(int));
    g_err[dev] = p;
  }
  return g_err[dev];
}

static int clear_device_error(cudaStream_t s) {
  DLMZ_CUDA_TRY(cudaMemsetAsync(device_error_word(), 0, sizeof(int), s));
  return DLMZ_OK;
}

static int check_device(cudaStream_t s) {
  DLMZ_CUDA_TRY(cudaStreamSynchronize(s));
  int* e = device_error_word();
  int h = 0;
  DLMZ_CUDA_TRY(cudaMemcpy(&h, e, sizeof(int), cudaMemcpyDeviceToHost));
  if (h) DLMZ_CUDA_TRY(cudaMemset(e, 0, sizeof(int)));
  if (h & ERR_TIMEOUT) return DLMZ_ETIMEOUT;
  if (h & ERR_LAUNCH) return DLMZ_ECUDA;
  if (h & ERR_NONFINITE) return DLMZ_EBADINPUT;
  if (h & (ERR_CORRUPT | ERR_CAPACITY)) return DLMZ_ECORRUPT;
  return DLMZ_OK;
}

// ---- small kernels ---------------------------------------------------------------------
__global__ void fill_i32(int32_t* p, int64_t n, int32_t v) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) p[i] = v;
}

// input symbols of windows [c0, c0+nc) (each Lb long) -> int32
__global__ void symbols_in_kernel(const uint8_t* in, int64_t sym0, int64_t n, int tok, int V, int32_t* out, int* err) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    int64_t v;
    if (tok) {
      const uint8_t* p = in + 4 * (sym0 + i);
      v = (int64_t)p[0] | ((int64_t)p[1] << 8) | ((int64_t)p[2] << 16) | ((int64_t)p[3] << 24);
      if (v >= V) {
        atomicOr(err, ERR_NONFINITE);  // reported as EBADINPUT
        v = 0;
      }
    } else {
      v = in[sym0 + i];
    }
    out[i] = (int32_t)v;
  }
}

__global__ void symbols_out_kernel(const int32_t* sym, int64_t sym0, int64_t n, int tok, uint8_t* out) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t v = (uint32_t)sym[i];
    if (tok) {
      uint8_t* p = out + 4 * (sym0 + i);
      p[0] = (uint8_t)v;
      p[1] = (uint8_t)(v >> 8);
      p[2] = (uint8_t)(v >> 16);
      p[3] = (uint8_t)(v >> 24);
    } else {
      out[sym0 + i] = (uint8_t)v;
    }
  }
}

// CRC-32 (IEEE, reflected polynomial 0xEDB88320) of each window, one thread per window.
__global__ void window_crc_kernel(const uint8_t* data, uint64_t nbytes, uint64_t wbytes, int nwin, uint32_t* out) {
  __shared__ uint32_t T[256];
  for (int i = threadIdx.x; i < 256; i += blockDim.x) {
    uint32_t c = (uint32_t)i;
    for (int k = 0; k < 8; ++k) c = (c >> 1) ^ (0xEDB88320u & (0u - (c & 1u)));
    T[i] = c;
  }
  __syncthreads();
  const int w = blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= nwin) return;
  const uint64_t b0 = (uint64_t)w * wbytes;
  const uint64_t b1 = b0 + wbytes < nbytes ? b0 + wbytes : nbytes;
  uint32_t crc = 0xFFFFFFFFu;
  for (uint64_t i = b0; i < b1; ++i) crc = T[(crc ^ data[i]) & 0xFF] ^ (crc >> 8);
  out[w] = ~crc;
}

__global__ void gather_streams_kernel(const uint8_t* staging, uint64_t cap, const uint32_t* bits,
                                      const uint64_t* offsets, int n, uint8_t* out) {
  const int c = blockIdx.x;
  if (c >= n) return;
  const uint64_t nb = (bits[c] + 7) / 8;
  const uint8_t* src = staging + (size_t)c * cap;
  uint8_t* dst = out + offsets[c];
  for (uint64_t i = threadIdx.x; i < nb; i += blockDim.x) dst[i] = src[i];
}

__global__ void sum_i32_kernel(const int32_t* v, int n, unsigned long long* out) {
  unsigned long long s = 0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) s += (unsigned long long)v[i];
  for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  __shared__ unsigned long long red[32];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long t = 0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) t += red[i];
    *out = t;
  }
}

// Initial context (Sec. 3.4) of windows [0, nc) (each L long): the ce context
// positions of window w (pos[w*ce + i], or i itself when pos is null) take their
// symbol -- from `symbols` when compressing (also written to out_syms, sb bytes
// little-endian each, for the file) or from the file's bytes when decompressing
// (a symbol >= V there marks the file corrupt and is replaced by 0).
__global__ void context_kernel(int32_t* state, int nc, int L, int ce, const int32_t* pos, const int32_t* symbols,
                               const uint8_t* file_syms, uint8_t* out_syms, int sb, int V, int* err) {
  const int64_t n = (int64_t)nc * ce;
  for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < n; idx += (int64_t)gridDim.x * blockDim.x) {
    const int64_t w = idx / ce;
    const int p = pos ? pos[idx] : (int)(idx % ce);
    int32_t v;
    if (symbols) {
      v = symbols[w * L + p];
    } else {
      uint32_t u = 0;
      for (int b = 0; b < sb; ++b) u |= (uint32_t)file_syms[idx * sb + b] << (8 * b);
      if (u >= (uint32_t)V) {
        atomicOr(err, ERR_CORRUPT);
        u = 0;
      }
      v = (int32_t)u;
    }
    state[w * L + p] = v;
    if (out_syms)
      for (int b = 0; b < sb; ++b) out_syms[idx * sb + b] = (uint8_t)((uint32_t)v >> (8 * b));
  }
}

static unsigned grid_for(int64_t n, int threads = 256) {
  int64_t b = (n + threads - 1) / threads;
  if (b < 1) b = 1;
  if (b > 65535) b = 65535;
  return (unsigned)b;
}

static uint32_t crc32_host(const uint8_t* p, size_t n) {
  uint32_t crc = 0xFFFFFFFFu;
  for (size_t i = 0; i < n; ++i) {
    crc ^= p[i];
    for (int k = 0; k < 8; ++k) crc = (crc >> 1) ^ (0xEDB88320u & (0u - (crc & 1u)));
  }
  return ~crc;
}

// ---- left-to-right schedules (Sec. 3.3, paragraphs 1-2) --------------------------------
// Uniform block: K = min(k, n) steps of floor(n / K), the last taking the remainder.
// Progressive: x_1 = u_1 2^16, x_(k+1) = floor(x_k r_q / 2^16) (capped at n 2^16, which
// changes no step), u_k = max(1, floor((x_k + 2^15) / 2^16)), at most what remains.
static std::vector<int> schedule_sizes(int n, const dlmz_k_policy& p) {
  std::vector<int> u;
  if (n <= 0) return u;
  if (p.kind == DLMZ_UNIFORM) {
    const int K = (int64_t)p.k < n ? (int)p.k : n;
    const int q = n / K;
    u.assign(K - 1, q);
    u.push_back(n - (K - 1) * q);
    return u;
  }
  unsigned __int128 x = (unsigned __int128)p.k << 16;
  const unsigned __int128 cap = (unsigned __int128)n << 16;
  for (int rem = n; rem > 0;) {
    unsigned __int128 v = (x + (1u << 15)) >> 16;
    if (v < 1) v = 1;
    const int take = v < (unsigned __int128)rem ? (int)v : rem;
    u.push_back(take);
    rem -= take;
    x = (x * p.growth_q16) >> 16;
    if (x > cap) x = cap;
  }
  return u;
}

// ---- initial context positions (Sec. 3.4) ----------------------------------------------
// Random: partial Fisher-Yates (Durstenfeld) of [0, n) with output i of the
// SplitMix64 stream (Steele, Lea & Flood 2014) whose state is output `window` of
// the stream seeded by `seed`; output j of a stream with state s is mix(s + (j+1) gamma).
static uint64_t sm64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
static constexpr uint64_t SM64_GAMMA = 0x9E3779B97F4A7C15ull;

static int context_count(const dlmz_k_policy& p, int n) {
  return p.context == DLMZ_CONTEXT_NONE ? 0 : ((int64_t)p.context_c < n ? (int)p.context_c : n);
}

static void context_positions(const dlmz_k_policy& p, int n, uint64_t window, int32_t* out) {
  const int ce = context_count(p, n);
  if (p.context == DLMZ_CONTEXT_CONTIGUOUS) {
    for (int i = 0; i < ce; ++i) out[i] = i;
    return;
  }
  if (ce == 0) return;
  const uint64_t st = sm64_mix(p.context_seed + (window + 1) * SM64_GAMMA);
  std::vector<int32_t> slot(n);
  for (int i = 0; i < n; ++i) slot[i] = i;
  for (int i = 0; i < ce; ++i) {
    const uint64_t o = sm64_mix(st + (uint64_t)(i + 1) * SM64_GAMMA);
    const int j = i + (int)(o % (uint64_t)(n - i));
    const int32_t t = slot[i];
    slot[i] = slot[j];
    slot[j] = t;
  }
  std::sort(slot.begin(), slot.begin() + ce);
  for (int i = 0; i < ce; ++i) out[i] = slot[i];
}

// Context of one batch: ce positions per window (host and device copies).
struct BatchContext {
  int ce = 0;                   // context symbols per window of this batch
  std::vector<int32_t> pos;     // nc x ce, ascending per window (empty when contiguous)
  const int32_t* d_pos = nullptr;
  const uint8_t* file_syms = nullptr;  // decompress: the batch's symbols in the file
  uint8_t* out_syms = nullptr;         // compress: where the batch's symbols go
  int sb = 1;                          // bytes per stored symbol
};

// ---- per-batch step state ---------------------------------------------------------
struct StepBufs {
  DevBuf logits, W, Hq, top, mx, sel_count, sel_pos, committed, sum, pairs;
  DevBuf rowcf, segcum, rowK, rowD;  // row-parallel coder scratch, one entry per selected row
  DevBuf pmax, pmin;                 // LM-head rows' maxima / minima per 128 logits (the quantiser's first pass)
  // candidate rows of a model step: per-window counts, offsets [nc + 1], token index of
  // each candidate, the candidate row of each position of [row0, row0 + rpc) (-1: none),
  // token index of each selected row and the stats of the recomputed selected rows
  DevBuf cand_count, cand_off, cand_total, cand_tok, row_map, sel_tok, sW, sHq, stop, smx;
  int64_t* host_total = nullptr;  // pinned: candidate count of the step, read while the layers run
  cudaEvent_t total_ready = nullptr;
  int ensure(size_t rows, int V, int nc, int kcap) {
    DLMZ_TRY(logits.ensure(rows * (size_t)V * 4));
    DLMZ_TRY(W.ensure(rows * 8));
    DLMZ_TRY(Hq.ensure(rows * 4));
    DLMZ_TRY(top.ensure(rows * 4));
    DLMZ_TRY(mx.ensure(rows * 4));
    DLMZ_TRY(sel_count.ensure((size_t)nc * 4));
    DLMZ_TRY(sel_pos.ensure((size_t)nc * kcap * 4));
    DLMZ_TRY(committed.ensure((size_t)nc * 4));
    DLMZ_TRY(sum.ensure(8));
    return DLMZ_OK;
  }
  int ensure_cand(int nc, int rpc, int kcap) {
    DLMZ_TRY(cand_count.ensure((size_t)nc * 4));
    DLMZ_TRY(cand_off.ensure((size_t)nc * 4 + 4));
    DLMZ_TRY(cand_tok.ensure((size_t)nc * rpc * 4));
    DLMZ_TRY(row_map.ensure((size_t)nc * rpc * 4));
    DLMZ_TRY(sel_tok.ensure((size_t)nc * kcap * 4));
    DLMZ_TRY(cand_total.ensure(8));
    if (!host_total) {
      void* h = nullptr;
      if (cudaMallocHost(&h, 8) != cudaSuccess) {
        (void)cudaGetLastError();
        return DLMZ_ENOMEM;
      }
      host_total = reinterpret_cast<int64_t*>(h);
    }
    if (!total_ready) DLMZ_CUDA_TRY(cudaEventCreateWithFlags(&total_ready, cudaEventDisableTiming));
    return DLMZ_OK;
  }
  int ensure_sel_stats(size_t rows) {
    DLMZ_TRY(sW.ensure(rows * 8));
    DLMZ_TRY(sHq.ensure(rows * 4));
    DLMZ_TRY(stop.ensure(rows * 4));
    DLMZ_TRY(smx.ensure(rows * 4));
    return DLMZ_OK;
  }
  void release() {
    logits.release(); W.release(); Hq.release(); top.release(); mx.release();
    sel_count.release(); sel_pos.release(); committed.release(); sum.release(); pairs.release();
    cand_count.release(); cand_off.release(); cand_total.release(); cand_tok.release(); row_map.release(); sel_tok.release();
    sW.release(); sHq.release(); stop.release(); smx.release();
    if (host_total) cudaFreeHost(host_total);
    host_total = nullptr;
    if (total_ready) cudaEventDestroy(total_ready);
    total_ready = nullptr;
  }
};

// ---- candidate rows of a model step ------------------------------------------------
// The candidates of a step are the masked positions of [row0, row0 + rpc) in each
// window (Definition 3: one distribution per masked position); only they go
// through the LM head and the quantiser.
__device__ __forceinline__ int block_sum_i32(int v, int* red) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  int t = 0;
  for (int i = 0; i < (int)(blockDim.x >> 5); ++i) t += red[i];
  return t;
}

__global__ void cand_count_kernel(const int32_t* __restrict__ state, int L, int mask_id, int row0, int rpc,
                                  int32_t* __restrict__ counts) {
  __shared__ int red[32];
  const int c = blockIdx.x;
  int n = 0;
  for (int i = threadIdx.x; i < rpc; i += blockDim.x) n += state[(size_t)c * L + row0 + i] == mask_id;
  n = block_sum_i32(n, red);
  if (threadIdx.x == 0) counts[c] = n;
}

// offsets[i] = counts[0] + ... + counts[i - 1] for i <= nc, and *total = offsets[nc]; one CTA.
__global__ void cand_scan_kernel(const int32_t* __restrict__ counts, int nc, int32_t* __restrict__ offsets,
                                 int64_t* __restrict__ total) {
  __shared__ int wsum[32];
  __shared__ int carry;
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int b = 0; b < nc; b += blockDim.x) {
    const int i = b + threadIdx.x;
    const int v = i < nc ? counts[i] : 0;
    int inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += t;
    }
    if (lane == 31) wsum[w] = inc;
    __syncthreads();
    if (w == 0) {
      int x = lane < nw ? wsum[lane] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += t;
      }
      if (lane < nw) wsum[lane] = x;  // inclusive over warps
    }
    __syncthreads();
    const int pre = carry + (w > 0 ? wsum[w - 1] : 0) + inc - v;
    if (i < nc) offsets[i] = pre;
    __syncthreads();
    if (threadIdx.x == 0) carry += wsum[nw - 1];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    offsets[nc] = carry;
    *total = carry;
  }
}

// Candidates of window c in ascending position: token index (c * L + position) at
// offsets[c] + rank, and row_map[c * rpc + i] = that row (or -1 for a committed position).
__global__ void cand_write_kernel(const int32_t* __restrict__ state, int L, int mask_id, int row0, int rpc,
                                  const int32_t* __restrict__ offsets, int32_t* __restrict__ cand_tok,
                                  int32_t* __restrict__ row_map) {
  __shared__ int wcount[32];
  const int c = blockIdx.x, lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int base = offsets[c];
  for (int i0 = 0; i0 < rpc; i0 += blockDim.x) {
    const int i = i0 + threadIdx.x;
    const bool ok = i < rpc && state[(size_t)c * L + row0 + i] == mask_id;
    const unsigned bal = __ballot_sync(0xffffffffu, ok);
    if (lane == 0) wcount[w] = __popc(bal);
    __syncthreads();
    int off = base, tot = 0;
    for (int j = 0; j < nw; ++j) {
      if (j < w) off += wcount[j];
      tot += wcount[j];
    }
    if (i < rpc) {
      const int r = ok ? off + __popc(bal & ((1u << lane) - 1)) : -1;
      row_map[(size_t)c * rpc + i] = r;
      if (ok) cand_tok[r] = c * L + row0 + i;
    }
    base += tot;
    __syncthreads();
  }
}

// Token index of the j-th selected position of each window (row c * kcap + j); rows
// past a window's count repeat its position 0 (their logits are never read).
__global__ void sel_tok_kernel(const int32_t* __restrict__ sel_count, const int32_t* __restrict__ sel_pos, int nc,
                               int L, int kcap, int32_t* __restrict__ tok) {
  const int64_t n = (int64_t)nc * kcap;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const int c = (int)(i / kcap), j = (int)(i % kcap);
    tok[i] = c * L + (j < sel_count[c] ? sel_pos[i] : 0);
  }
}

static int kcap_for(const dlmz_k_policy& p, int rpc) {
  int k = p.kind != DLMZ_ENTROPY ? (int)p.k : (p.k_max ? (int)p.k_max : rpc);
  if (p.kind == DLMZ_ENTROPY && (int)p.k_min > k) k = (int)p.k_min;
  return k < rpc ? k : rpc;
}

static int64_t tau_q_of(float tau) { return (int64_t)floor((double)tau * 65536.0); }

static int precision_for(uint32_t V) { return V <= 4096 ? 16 : 24; }

// Where a step's symbols come from and go to (encoder: symbols, streams; decoder: the
// file's streams), and the coder state of the batch's windows.
struct StepIO {
  const int32_t* symbols;
  int32_t* state;
  CoderState* cst;
  uint8_t* ebytes;
  uint64_t cap_bytes;
  const uint8_t* in_bytes;
  const uint64_t* in_off;
  const uint32_t* in_bits;
  bool decode;
  int32_t* committed;
};

// Selection (Sec. 3.3) on the keys in sb.W (confidence) / sb.Hq (entropy); a key row is
// found through row_map when given.
static int select_step(StepBufs& sb, const int32_t* state, int nc, int L, int V, const dlmz_k_policy& pol, int row0,
                       int rpc, int kcap, const int32_t* row_map, cudaStream_t s) {
  if (pol.kind != DLMZ_ENTROPY)  // left-to-right schedules: the k leftmost masked rows (keys ignored)
    return select_rows<uint64_t>(state, nc, L, V, row0, rpc, pol.kind == DLMZ_TOPK_CONF ? sb.W.as<uint64_t>() : nullptr,
                                 0, (int)pol.k, 0, 0, 0, kcap, sb.sel_count.as<int32_t>(), sb.sel_pos.as<int32_t>(), s,
                                 row_map);
  return select_rows<int32_t>(state, nc, L, V, row0, rpc, sb.Hq.as<int32_t>(), 1, 0, tau_q_of(pol.tau_bits),
                              (int)pol.k_min, (int)pol.k_max, kcap, sb.sel_count.as<int32_t>(),
                              sb.sel_pos.as<int32_t>(), s, row_map);
}

// Frequency of the selected rows, code (or decode) and reveal (Sec. 3.2).
static int code_rows(StepBufs& sb, const StepIO& io, const float* logits, const float* mx, const uint64_t* W,
                     const int32_t* top, const int32_t* row_map, bool sel_major, int nc, int L, int V, int P,
                     const dlmz_k_policy& pol, int row0, int rpc, int kcap, cudaStream_t s) {
  CodeArgs a{};
  a.logits = logits;
  a.mx = mx;
  a.W = W;
  a.top = top;
  a.row_map = row_map;
  a.sel_major = sel_major ? 1 : 0;
  a.sel_count = sb.sel_count.as<int32_t>();
  a.sel_pos = sb.sel_pos.as<int32_t>();
  a.symbols = io.symbols;
  a.state = io.state;
  a.state_c = io.cst;
  a.bytes = io.ebytes;
  a.cap_bytes = io.cap_bytes;
  a.in_bytes = io.in_bytes;
  a.in_offsets = io.in_off;
  a.in_bits = io.in_bits;
  a.committed = io.committed;
  a.err = device_error_word();
  a.V = V;
  a.P = P;
  a.L = L;
  a.row0 = row0;
  a.rpc = rpc;
  a.kcap = kcap;
  a.coder = (int)pol.coder;
  if (pol.coder == DLMZ_CODER_RANS && !io.decode) {  // one (c, f) pair per position of every window
    DLMZ_TRY(sb.pairs.ensure((size_t)nc * L * 8));
    a.pairs = sb.pairs.as<uint64_t>();
    a.pair_cap = L;
  }
  if (pol.coder != DLMZ_CODER_RANKS) {
    const size_t nrows = (size_t)nc * kcap;
    a.nseg = (V + CODE_SEG - 1) / CODE_SEG;
    if (io.decode) {
      DLMZ_TRY(sb.segcum.ensure(nrows * (a.nseg + 1) * 4));
      DLMZ_TRY(sb.rowK.ensure(nrows * 8));
      DLMZ_TRY(sb.rowD.ensure(nrows * 4));
      a.segcum = sb.segcum.as<uint32_t>();
      a.rowK = sb.rowK.as<uint64_t>();
      a.rowD = sb.rowD.as<uint32_t>();
    } else {
      DLMZ_TRY(sb.rowcf.ensure(nrows * 8));
      a.rowcf = sb.rowcf.as<uint64_t>();
    }
  }
  return code_step(a, io.decode, nc, s);
}

// quantise + select + code one step on caller-given logits of rows [row0, row0+rpc) of each window
static int run_step(StepBufs& sb, const float* logits, int nc, int L, int V, int P, const dlmz_k_policy& pol,
                    int row0, int rpc, const int32_t* symbols, int32_t* state, CoderState* cst, uint8_t* ebytes,
                    uint64_t cap_bytes, const uint8_t* in_bytes, const uint64_t* in_off, const uint32_t* in_bits,
                    bool decode, int32_t* committed, cudaStream_t s) {
  const int rows = nc * rpc;
  const int kcap = kcap_for(pol, rpc);
  DLMZ_TRY(sb.ensure(rows, 1, nc, kcap));
  DLMZ_TRY(quantize_rows(logits, rows, V, P, nullptr, sb.W.as<uint64_t>(), nullptr, sb.Hq.as<int32_t>(),
                         sb.top.as<int32_t>(), sb.mx.as<float>(), s));
  DLMZ_TRY(select_step(sb, state, nc, L, V, pol, row0, rpc, kcap, nullptr, s));
  const StepIO io{symbols, state, cst, ebytes, cap_bytes, in_bytes, in_off, in_bits, decode, committed};
  return code_rows(sb, io, logits, sb.mx.as<float>(), sb.W.as<uint64_t>(), sb.top.as<int32_t>(), nullptr, false, nc,
                   L, V, P, pol, row0, rpc, kcap, s);
}

// Bytes of float32 logits one model step may hold at once (rows beyond it go through
// the LM head in slabs).
static size_t logits_budget(const dlmz_model* m) {
  return m->logits_budget ? m->logits_budget : ((size_t)24 << 30);
}

// One step of the iterative pipeline with the model's own distributions: the
// forward over the batch, the LM head and the quantiser on the candidate rows
// only (the masked positions of [row0, row0 + rpc) in each window), selection,
// and the coding of the selected symbols.  When the candidates' logits exceed the
// budget, the head and the quantiser's scores run in slabs of rows, and after
// the selection the selected rows' logits are computed once more for the coder
// (bit-identical: a row's logits depend only on that row).
static int model_step(dlmz_model* m, StepBufs& sb, const dlmz_k_policy& pol, int nc, int L, int row0, int rpc,
                      const StepIO& io, cudaStream_t s) {
  const int V = (int)m->cfg.vocab, P = precision_for(m->cfg.vocab);
  const int kcap = kcap_for(pol, rpc);
  DLMZ_TRY(sb.ensure_cand(nc, rpc, kcap));
  // the candidates depend only on the state: list them first, so their number reaches
  // the host while the layers run
  int32_t* off = sb.cand_off.as<int32_t>();
  int32_t* cand = sb.cand_tok.as<int32_t>();
  int32_t* row_map = sb.row_map.as<int32_t>();
  cand_count_kernel<<<nc, 256, 0, s>>>(io.state, L, V, row0, rpc, sb.cand_count.as<int32_t>());
  DLMZ_TRY(launch_status());
  cand_scan_kernel<<<1, 1024, 0, s>>>(sb.cand_count.as<int32_t>(), nc, off, sb.cand_total.as<int64_t>());
  DLMZ_TRY(launch_status());
  cand_write_kernel<<<nc, 256, 0, s>>>(io.state, L, V, row0, rpc, off, cand, row_map);
  DLMZ_TRY(launch_status());
  DLMZ_CUDA_TRY(cudaMemcpyAsync(sb.host_total, sb.cand_total.p, 8, cudaMemcpyDeviceToHost, s));
  DLMZ_CUDA_TRY(cudaEventRecord(sb.total_ready, s));
  DLMZ_TRY(model_layers(m, io.state, nc, L, s));
  DLMZ_CUDA_TRY(cudaEventSynchronize(sb.total_ready));
  const int64_t M = *sb.host_total;
  if (M < 0 || M > (int64_t)nc * rpc) return DLMZ_ECORRUPT;
  const int64_t sel_rows = (int64_t)nc * kcap;
  int64_t slab = (int64_t)(logits_budget(m) / ((size_t)V * 4));
  if (slab < sel_rows) slab = sel_rows;
  if (slab < 1) slab = 1;
  const bool slabbed = M > slab;
  const size_t mrows = (size_t)(M > 0 ? M : 1);
  DLMZ_TRY(sb.ensure(mrows, 0, nc, kcap));  // scores of every candidate, selection buffers
  DLMZ_TRY(sb.logits.ensure((slabbed ? (size_t)slab : mrows) * V * 4));
  float* logits = sb.logits.as<float>();
  // the head's epilogue leaves each row's maxima per 128 logits, so the quantiser reads each logit
  // once (large vocabularies: V > 512 takes the persistent kernel)
  const bool want_parts = V > 512 && V % 128 == 0;
  const size_t head_rows = slabbed ? (size_t)slab : mrows;
  if (want_parts) {
    const size_t np = head_rows < (size_t)sel_rows ? (size_t)sel_rows : head_rows;
    DLMZ_TRY(sb.pmax.ensure(np * (V / 128) * 4));
    DLMZ_TRY(sb.pmin.ensure(np * (V / 128) * 4));
  }
  float* pmx = want_parts ? sb.pmax.as<float>() : nullptr;
  float* pmn = want_parts ? sb.pmin.as<float>() : nullptr;
  for (int64_t r0 = 0; r0 < M; r0 += slab) {
    const int n = (int)(M - r0 < slab ? M - r0 : slab);
    bool parts = false;
    DLMZ_TRY(model_head(m, cand + r0, n, logits, s, pmx, pmn, &parts));
    DLMZ_TRY(quantize_rows(logits, n, V, P, nullptr, sb.W.as<uint64_t>() + r0, nullptr, sb.Hq.as<int32_t>() + r0,
                           sb.top.as<int32_t>() + r0, sb.mx.as<float>() + r0, s, parts ? pmx : nullptr,
                           parts ? pmn : nullptr));
  }
  DLMZ_TRY(select_step(sb, io.state, nc, L, V, pol, row0, rpc, kcap, row_map, s));
  if (!slabbed)
    return code_rows(sb, io, logits, sb.mx.as<float>(), sb.W.as<uint64_t>(), sb.top.as<int32_t>(), row_map, false, nc,
                     L, V, P, pol, row0, rpc, kcap, s);
  // the selected rows once more, row c * kcap + j for the j-th selected position of window c
  DLMZ_TRY(sb.ensure_sel_stats((size_t)sel_rows));
  int32_t* stok = sb.sel_tok.as<int32_t>();
  sel_tok_kernel<<<grid_for(sel_rows), 256, 0, s>>>(sb.sel_count.as<int32_t>(), sb.sel_pos.as<int32_t>(), nc, L, kcap,
                                                   stok);
  DLMZ_TRY(launch_status());
  bool parts = false;
  DLMZ_TRY(model_head(m, stok, (int)sel_rows, logits, s, pmx, pmn, &parts));
  DLMZ_TRY(quantize_rows(logits, (int)sel_rows, V, P, nullptr, sb.sW.as<uint64_t>(), nullptr, sb.sHq.as<int32_t>(),
                         sb.stop.as<int32_t>(), sb.smx.as<float>(), s, parts ? pmx : nullptr, parts ? pmn : nullptr));
  return code_rows(sb, io, logits, sb.smx.as<float>(), sb.sW.as<uint64_t>(), sb.stop.as<int32_t>(), nullptr, true, nc,
                   L, V, P, pol, row0, rpc, kcap, s);
}

static int validate_policy(const dlmz_k_policy* p) {
  if (!p) return DLMZ_EINVAL;
  if (p->context > DLMZ_CONTEXT_ATTENTION || (p->context == DLMZ_CONTEXT_NONE) != (p->context_c == 0) ||
      p->coder > DLMZ_CODER_RANKS)
    return DLMZ_EINVAL;
  if (p->kind == DLMZ_TOPK_CONF || p->kind == DLMZ_UNIFORM) return p->k >= 1 ? DLMZ_OK : DLMZ_EINVAL;
  if (p->kind == DLMZ_PROGRESSIVE)
    return p->k >= 1 && p->growth_q16 >= 1 && p->growth_q16 <= (64u << 16) ? DLMZ_OK : DLMZ_EINVAL;
  if (p->kind == DLMZ_ENTROPY) {
    if (p->k_min < 1) return DLMZ_EINVAL;
    if (p->k_max && p->k_max < p->k_min) return DLMZ_EINVAL;
    if (!(p->tau_bits >= 0.0f) || p->tau_bits > 30000.0f) return DLMZ_EINVAL;
    return DLMZ_OK;
  }
  return DLMZ_EINVAL;
}


static uint64_t cap_bytes_for(uint32_t L, int P) {
  const uint64_t units = ((uint64_t)L * P + 80) / 16 + 4;
  return 2 * units;
}

// One batch of nc windows of length Lb through all steps.
static int run_batch(dlmz_model* m, StepBufs& sb, const dlmz_k_policy& pol, int nc, int Lb, const int32_t* symbols,
                     int32_t* state, CoderState* cst, uint8_t* ebytes, uint64_t cap_bytes, const uint8_t* in_bytes,
                     const uint64_t* in_off, const uint32_t* in_bits, bool decode, const BatchContext& bx,
                     cudaStream_t s) {
  const int V = (int)m->cfg.vocab;
  const int ce = bx.ce;
  const StepIO io{symbols, state, cst, ebytes, cap_bytes, in_bytes, in_off, in_bits, decode, nullptr};
  fill_i32<<<grid_for((int64_t)nc * Lb), 256, 0, s>>>(state, (int64_t)nc * Lb, V);
  DLMZ_TRY(launch_status());
  if (ce > 0) {
    context_kernel<<<grid_for((int64_t)nc * ce), 256, 0, s>>>(state, nc, Lb, ce, bx.d_pos, decode ? nullptr : symbols,
                                                             bx.file_syms, decode ? nullptr : bx.out_syms, bx.sb, V,
                                                             device_error_word());
    DLMZ_TRY(launch_status());
  }
  if (decode) DLMZ_TRY(coder_load(cst, nc, in_bytes, in_off, in_bits, (int)pol.coder, s));
  else DLMZ_TRY(coder_reset(cst, nc, s));
  // context positions of window w inside [a, b)
  auto ctx_in = [&](int w, int a, int b) -> int {
    if (ce == 0) return 0;
    if (bx.pos.empty()) return std::max(0, std::min(b, ce) - a);  // contiguous: [0, ce)
    const int32_t* p = bx.pos.data() + (size_t)w * ce;
    return (int)(std::lower_bound(p, p + ce, b) - std::lower_bound(p, p + ce, a));
  };
  if (pol.kind == DLMZ_TOPK_CONF) {
    const int B = pol.block ? (int)pol.block : Lb;
    for (int b0 = 0; b0 < Lb; b0 += B) {
      const int Bl = B < Lb - b0 ? B : Lb - b0;
      // steps for this block: the window with the most masked positions in it decides
      int most = 0;
      for (int w = 0; w < (bx.pos.empty() ? 1 : nc); ++w) most = std::max(most, Bl - ctx_in(w, b0, b0 + Bl));
      const int steps = (most + (int)pol.k - 1) / (int)pol.k;
      if (steps == 0) continue;
      for (int t = 0; t < steps; ++t) DLMZ_TRY(model_step(m, sb, pol, nc, Lb, b0, Bl, io, s));
    }
  } else if (pol.kind == DLMZ_UNIFORM || pol.kind == DLMZ_PROGRESSIVE) {
    // every window has n = Lb - ce masked positions, so one schedule serves the batch; step k
    // commits masked positions [t, t + u_k) of each window, whose rows span [lo, hi) over the batch
    const int n = Lb - ce;
    const std::vector<int> sizes = schedule_sizes(n, pol);
    std::vector<int32_t> masked;  // nc x n masked positions, ascending (random context only)
    if (!bx.pos.empty()) {
      masked.resize((size_t)nc * n);
      for (int w = 0; w < nc; ++w) {
        const int32_t* p = bx.pos.data() + (size_t)w * ce;
        int q = 0, j = 0;
        for (int x = 0; x < Lb; ++x) {
          if (j < ce && p[j] == x) ++j;
          else masked[(size_t)w * n + q++] = x;
        }
      }
    }
    auto mpos = [&](int w, int t) -> int { return masked.empty() ? ce + t : masked[(size_t)w * n + t]; };
    int t = 0;
    for (const int u : sizes) {
      int lo = Lb, hi = 0;
      for (int w = 0; w < (masked.empty() ? 1 : nc); ++w) {
        lo = std::min(lo, mpos(w, t));
        hi = std::max(hi, mpos(w, t + u - 1) + 1);
      }
      dlmz_k_policy sp = pol;
      sp.k = (uint32_t)u;
      DLMZ_TRY(model_step(m, sb, sp, nc, Lb, lo, hi - lo, io, s));
      t += u;
    }
  } else {
    DLMZ_TRY(sb.ensure(1, 0, nc, kcap_for(pol, Lb)));
    StepIO eio = io;
    eio.committed = sb.committed.as<int32_t>();
    int64_t remaining = (int64_t)nc * (Lb - ce);
    for (int64_t step = 0; remaining > 0; ++step) {
      if (step > (int64_t)Lb) return DLMZ_ECORRUPT;  // every step commits >= 1 per live window
      DLMZ_TRY(model_step(m, sb, pol, nc, Lb, 0, Lb, eio, s));
      sum_i32_kernel<<<1, 256, 0, s>>>(sb.committed.as<int32_t>(), nc, sb.sum.as<unsigned long long>());
      DLMZ_TRY(launch_status());
      unsigned long long done = 0;
      DLMZ_CUDA_TRY(cudaMemcpyAsync(&done, sb.sum.p, 8, cudaMemcpyDeviceToHost, s));
      DLMZ_CUDA_TRY(cudaStreamSynchronize(s));
      if (done == 0) return DLMZ_ECORRUPT;
      remaining -= (int64_t)done;
    }
  }
  return DLMZ_OK;
}

struct PipeWs {
  StepBufs sb;
  DevBuf symbols, state, cst, staging, bits, crcs, offsets, hin, hout, ctxpos, ctxsyms;
  DevBuf ctxscore, ctxkeys, ctxsel, ctxmaps, ctxstate;  // attention-based context
  void release() {
    sb.release(); symbols.release(); state.release(); cst.release(); staging.release(); bits.release();
    crcs.release(); offsets.release(); hin.release(); hout.release(); ctxpos.release(); ctxsyms.release();
    ctxscore.release(); ctxkeys.release(); ctxsel.release(); ctxmaps.release(); ctxstate.release();
  }
};

static PipeWs& pipe_of(dlmz_model* m) {
  if (!m->pipe) m->pipe = new PipeWs();
  return *reinterpret_cast<PipeWs*>(m->pipe);
}

static int default_batch(const dlmz_model* m, uint32_t L, uint32_t n_chunks) {
  size_t freeb = 0, total = 0;
  cudaMemGetInfo(&freeb, &total);
  const size_t lb = logits_budget(m);
  size_t budget = (freeb > lb ? freeb - lb : 0) / 2;
  const size_t cap = (size_t)48 << 30;
  if (budget > cap) budget = cap;
  // forward workspace and per-position step state; the candidate logits have their own budget
  const size_t per_chunk = (size_t)L * (model_workspace_per_token(m) + 64);
  size_t b = per_chunk ? budget / per_chunk : 1;
  if (b > 1024) b = 1024;
  if (b < 1) b = 1;
  if (b > n_chunks) b = n_chunks ? n_chunks : 1;
  return (int)b;
}

struct Header {
  uint32_t P, kind, vocab, chunk_len, batch_chunks, k, block, tau_q, k_min, k_max, n_chunks, crc;
  uint64_t fingerprint, n_symbols;
  uint32_t coder = 0;                // 0: range coder, 1: rANS, 2: symbol ranks
  uint32_t ctx_kind = 0, ctx_c = 0;  // version 2: initial context (Sec. 3.4)
  uint64_t ctx_seed = 0;
  size_t size() const { return ctx_c ? 80 : 64; }
  // context symbols over all windows
  uint64_t ctx_count() const {
    if (!ctx_c || !chunk_len) return 0;
    const uint64_t full = n_symbols / chunk_len, tail = n_symbols % chunk_len;
    const uint64_t per = ctx_c < chunk_len ? ctx_c : chunk_len;
    return full * per + (ctx_c < tail ? ctx_c : tail);
  }
  // bytes of the stored context positions (attention-based context only) and symbols, after the header
  uint64_t ctx_pos_bytes() const { return ctx_kind == DLMZ_CONTEXT_ATTENTION ? 4 * ctx_count() : 0; }
  uint64_t ctx_bytes() const { return ctx_pos_bytes() + ctx_count() * (vocab > 256 ? 4 : 1); }
};

static void put32(uint8_t* p, uint32_t v) { for (int i = 0; i < 4; ++i) p[i] = (uint8_t)(v >> (8 * i)); }
static void put64(uint8_t* p, uint64_t v) { for (int i = 0; i < 8; ++i) p[i] = (uint8_t)(v >> (8 * i)); }
static uint32_t get32(const uint8_t* p) { uint32_t v = 0; for (int i = 0; i < 4; ++i) v |= (uint32_t)p[i] << (8 * i); return v; }
static uint64_t get64(const uint8_t* p) { uint64_t v = 0; for (int i = 0; i < 8; ++i) v |= (uint64_t)p[i] << (8 * i); return v; }

static void write_header(uint8_t* o, const Header& h) {
  memcpy(o, "DLMZ", 4);
  o[4] = h.ctx_c ? 2 : 1;
  o[5] = (uint8_t)h.coder;
  o[6] = (uint8_t)h.P;
  o[7] = (uint8_t)h.kind;
  put64(o + 8, h.fingerprint);
  put32(o + 16, h.vocab);
  put32(o + 20, h.chunk_len);
  put32(o + 24, h.batch_chunks);
  put32(o + 28, h.k);
  put32(o + 32, h.block);
  put32(o + 36, h.tau_q);
  put32(o + 40, h.k_min);
  put32(o + 44, h.k_max);
  put64(o + 48, h.n_symbols);
  put32(o + 56, h.n_chunks);
  put32(o + 60, h.crc);
  if (h.ctx_c) {
    put32(o + 64, h.ctx_kind);
    put32(o + 68, h.ctx_c);
    put64(o + 72, h.ctx_seed);
  }
}

// o holds the first min(n, 80) bytes of the file
static int read_header(const uint8_t* o, size_t n, Header& h) {
  if (n < 64) return DLMZ_ECORRUPT;
  if (memcmp(o, "DLMZ", 4) || (o[4] != 1 && o[4] != 2) || o[5] > 2) return DLMZ_ECORRUPT;
  h.coder = o[5];
  h.P = o[6];
  h.kind = o[7];
  h.fingerprint = get64(o + 8);
  h.vocab = get32(o + 16);
  h.chunk_len = get32(o + 20);
  h.batch_chunks = get32(o + 24);
  h.k = get32(o + 28);
  h.block = get32(o + 32);
  h.tau_q = get32(o + 36);
  h.k_min = get32(o + 40);
  h.k_max = get32(o + 44);
  h.n_symbols = get64(o + 48);
  h.n_chunks = get32(o + 56);
  h.crc = get32(o + 60);
  if (h.chunk_len == 0 && h.n_symbols) return DLMZ_ECORRUPT;
  const uint64_t exp = h.chunk_len ? (h.n_symbols + h.chunk_len - 1) / h.chunk_len : 0;
  if (exp != h.n_chunks) return DLMZ_ECORRUPT;
  if (o[4] == 2) {
    if (n < 80) return DLMZ_ECORRUPT;
    h.ctx_kind = get32(o + 64);
    h.ctx_c = get32(o + 68);
    h.ctx_seed = get64(o + 72);
    if (h.ctx_kind < DLMZ_CONTEXT_CONTIGUOUS || h.ctx_kind > DLMZ_CONTEXT_ATTENTION || h.ctx_c == 0)
      return DLMZ_ECORRUPT;
  }
  return DLMZ_OK;
}

// The batch's context: positions (host + device) and where its symbols are in the file.
static int batch_context(const dlmz_k_policy& pol, int c0, int nc, int Lb, int sb, DevBuf& dpos, uint64_t sym_off,
                         const uint8_t* file, uint8_t* out, cudaStream_t s, BatchContext& bx,
                         const int32_t* attn_pos = nullptr) {
  bx = BatchContext{};
  bx.ce = context_count(pol, Lb);
  bx.sb = sb;
  if (bx.ce == 0) return DLMZ_OK;
  bx.file_syms = file ? file + sym_off * sb : nullptr;
  bx.out_syms = out ? out + sym_off * sb : nullptr;
  if (pol.context == DLMZ_CONTEXT_RANDOM || pol.context == DLMZ_CONTEXT_ATTENTION) {
    bx.pos.resize((size_t)nc * bx.ce);
    if (pol.context == DLMZ_CONTEXT_RANDOM) {
      for (int w = 0; w < nc; ++w) context_positions(pol, Lb, (uint64_t)(c0 + w), bx.pos.data() + (size_t)w * bx.ce);
    } else {  // attention-based: given by the caller (chosen on the device, or read from the file)
      if (!attn_pos) return DLMZ_EINVAL;
      std::copy(attn_pos, attn_pos + bx.pos.size(), bx.pos.begin());
    }
    DLMZ_TRY(dpos.ensure(bx.pos.size() * 4));
    DLMZ_CUDA_TRY(cudaMemcpyAsync(dpos.p, bx.pos.data(), bx.pos.size() * 4, cudaMemcpyHostToDevice, s));
    bx.d_pos = dpos.as<int32_t>();
  }
  return DLMZ_OK;
}

static void put_varint(std::vector<uint8_t>& o, uint64_t v) {
  do {
    uint8_t b = v & 0x7F;
    v >>= 7;
    o.push_back(v ? (b | 0x80) : b);
  } while (v);
}

// Batches: full windows in groups of bc, then the ragged tail window alone.
struct BatchPlan {
  int c0, nc, L;
};
static std::vector<BatchPlan> plan_batches(uint64_t n_sym, uint32_t L, int bc) {
  std::vector<BatchPlan> v;
  const uint64_t nfull = n_sym / L;
  for (uint64_t c = 0; c < nfull; c += bc) v.push_back({(int)c, (int)(nfull - c < (uint64_t)bc ? nfull - c : bc), (int)L});
  if (n_sym % L) v.push_back({(int)nfull, 1, (int)(n_sym % L)});
  return v;
}

// larger score -> smaller key (scores are >= 0), equal scores -> equal keys (the lower position wins)
__global__ void score_keys_kernel(const float* scores, int64_t n, uint64_t* keys) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    keys[i] = (uint64_t)(~(__float_as_uint(fmaxf(scores[i], 0.f)) | 0x80000000u));
}

// Attention-based context of windows [0, nc) of length Lb: the ce highest-scoring
// positions of each, ascending, to host `pos` [nc x ce].  Scored in sub-batches so
// the attention maps stay near 2 GB.
static int attention_context(dlmz_model* m, const int32_t* symbols, int nc, int Lb, int ce, PipeWs& w,
                             std::vector<int32_t>& pos, cudaStream_t s) {
  pos.assign((size_t)nc * ce, 0);
  if (ce == 0 || nc == 0) return DLMZ_OK;
  const size_t per = (size_t)m->cfg.n_layers * Lb * Lb * 4;
  int sub = (int)std::max<size_t>(1, ((size_t)2 << 30) / per);
  if (sub > nc) sub = nc;
  DLMZ_TRY(w.ctxscore.ensure((size_t)nc * Lb * 4));
  DLMZ_TRY(w.ctxkeys.ensure((size_t)nc * Lb * 8));
  DLMZ_TRY(w.ctxsel.ensure((size_t)nc * ce * 4 + (size_t)nc * 4));
  for (int c0 = 0; c0 < nc; c0 += sub) {
    const int n = std::min(sub, nc - c0);
    DLMZ_TRY(context_attention_scores(m, symbols + (size_t)c0 * Lb, n, Lb, w.ctxscore.as<float>() + (size_t)c0 * Lb,
                                      w.ctxmaps, w.ctxstate, s));
  }
  const int64_t n = (int64_t)nc * Lb;
  score_keys_kernel<<<grid_for(n), 256, 0, s>>>(w.ctxscore.as<float>(), n, w.ctxkeys.as<uint64_t>());
  DLMZ_TRY(launch_status());
  int32_t* sel = w.ctxsel.as<int32_t>();
  DLMZ_TRY(select_rows<uint64_t>(nullptr, nc, Lb, -1, 0, Lb, w.ctxkeys.as<uint64_t>(), 0, ce, 0, 0, 0, ce,
                                 sel + (size_t)nc * ce, sel, s));
  DLMZ_CUDA_TRY(cudaMemcpyAsync(pos.data(), sel, pos.size() * 4, cudaMemcpyDeviceToHost, s));
  DLMZ_CUDA_TRY(cudaStreamSynchronize(s));
  return DLMZ_OK;
}

static int compress_device(dlmz_model* m, const uint8_t* d_in, size_t in_bytes, uint32_t L, const dlmz_k_policy* pol,
                           uint32_t batch_chunks, uint8_t* d_out, size_t out_cap, size_t* out_bytes, cudaStream_t s) {
  if (!m || !pol || !out_bytes || L == 0) return DLMZ_EINVAL;
  if (in_bytes && !d_in) return DLMZ_EINVAL;
  DLMZ_TRY(validate_policy(pol));
  const uint32_t V = m->cfg.vocab;
  const int tok = V > 256;
  if (tok && in_bytes % 4) return DLMZ_EBADINPUT;
  const uint64_t n_sym = tok ? in_bytes / 4 : in_bytes;
  const uint64_t n_chunks64 = (n_sym + L - 1) / L;
  if (n_chunks64 > 0x7fffffff) return DLMZ_EINVAL;
  const int n_chunks = (int)n_chunks64;
  const int P = precision_for(V);
  const uint64_t cap = cap_bytes_for(L, P);
  const int bc = batch_chunks ? (int)batch_chunks : default_batch(m, L, (uint32_t)n_chunks);
  PipeWs& w = pipe_of(m);
  DLMZ_TRY(device_error_word() ? DLMZ_OK : DLMZ_ENOMEM);
  DLMZ_TRY(clear_device_error(s));
  DLMZ_TRY(w.staging.ensure((size_t)n_chunks * cap + 16));
  DLMZ_TRY(w.bits.ensure((size_t)n_chunks * 4 + 4));
  DLMZ_TRY(w.crcs.ensure((size_t)n_chunks * 4 + 4));
  DLMZ_TRY(w.offsets.ensure((size_t)n_chunks * 8 + 8));
  const size_t bl = (size_t)bc * L;
  DLMZ_TRY(w.symbols.ensure(bl * 4));
  DLMZ_TRY(w.state.ensure(bl * 4));
  DLMZ_TRY(w.cst.ensure((size_t)bc * sizeof(CoderState)));
  const uint64_t wbytes = (uint64_t)L * (tok ? 4 : 1);
  if (n_chunks) {
    window_crc_kernel<<<(n_chunks + 127) / 128, 128, 0, s>>>(d_in, in_bytes, wbytes, n_chunks, w.crcs.as<uint32_t>());
    DLMZ_TRY(launch_status());
  }
  Header h{};
  h.coder = pol->coder;
  h.ctx_kind = pol->context_c ? pol->context : 0;
  h.ctx_c = pol->context_c;
  h.ctx_seed = pol->context_seed;
  h.chunk_len = L;
  h.n_symbols = n_sym;
  h.vocab = V;
  const uint64_t ctx_bytes = h.ctx_bytes(), ctx_pos_bytes = h.ctx_pos_bytes();
  const int sbytes = tok ? 4 : 1;
  DLMZ_TRY(w.ctxsyms.ensure(ctx_bytes + 16));
  const uint64_t ce_full = (uint64_t)context_count(*pol, (int)L);
  std::vector<uint8_t> all_pos(ctx_pos_bytes);  // attention-based context: positions of every window, u32 LE
  for (const BatchPlan& b : plan_batches(n_sym, L, bc)) {
    const int64_t nsym_b = (int64_t)b.nc * b.L;
    symbols_in_kernel<<<grid_for(nsym_b), 256, 0, s>>>(d_in, (int64_t)b.c0 * L, nsym_b, tok, (int)V,
                                                       w.symbols.as<int32_t>(), device_error_word());
    DLMZ_TRY(launch_status());
    uint8_t* eb = w.staging.as<uint8_t>() + (size_t)b.c0 * cap;
    BatchContext bx;
    std::vector<int32_t> apos;
    if (pol->context == DLMZ_CONTEXT_ATTENTION) {
      DLMZ_TRY(attention_context(m, w.symbols.as<int32_t>(), b.nc, b.L, context_count(*pol, b.L), w, apos, s));
      for (size_t i = 0; i < apos.size(); ++i) put32(all_pos.data() + 4 * ((uint64_t)b.c0 * ce_full + i), (uint32_t)apos[i]);
    }
    DLMZ_TRY(batch_context(*pol, b.c0, b.nc, b.L, sbytes, w.ctxpos, (uint64_t)b.c0 * ce_full, nullptr,
                           w.ctxsyms.as<uint8_t>() + ctx_pos_bytes, s, bx, apos.data()));
    DLMZ_TRY(run_batch(m, w.sb, *pol, b.nc, b.L, w.symbols.as<int32_t>(), w.state.as<int32_t>(),
                       w.cst.as<CoderState>(), eb, cap, nullptr, nullptr, nullptr, false, bx, s));
    DLMZ_TRY(coder_finish(w.cst.as<CoderState>(), b.nc, eb, cap, w.bits.as<uint32_t>() + b.c0, nullptr, nullptr,
                          (int)pol->coder, w.sb.pairs.as<uint64_t>(), b.L, P, s));
  }
  DLMZ_TRY(check_device(s));
  std::vector<uint32_t> bits(n_chunks), crcs(n_chunks);
  if (n_chunks) {
    DLMZ_CUDA_TRY(cudaMemcpy(bits.data(), w.bits.p, (size_t)n_chunks * 4, cudaMemcpyDeviceToHost));
    DLMZ_CUDA_TRY(cudaMemcpy(crcs.data(), w.crcs.p, (size_t)n_chunks * 4, cudaMemcpyDeviceToHost));
  }
  std::vector<uint8_t> crcb((size_t)n_chunks * 4);
  for (int c = 0; c < n_chunks; ++c) put32(crcb.data() + 4 * c, crcs[c]);
  h.P = P;
  h.kind = pol->kind;
  h.batch_chunks = bc;
  h.k = pol->k;
  h.block = pol->kind == DLMZ_PROGRESSIVE ? pol->growth_q16 : pol->block;
  h.tau_q = (uint32_t)tau_q_of(pol->tau_bits);
  h.k_min = pol->k_min;
  h.k_max = pol->k_max;
  h.n_chunks = n_chunks;
  h.crc = crc32_host(crcb.data(), crcb.size());
  h.fingerprint = m->fingerprint;
  std::vector<uint8_t> head(h.size());
  write_header(head.data(), h);
  std::vector<uint8_t> lens;
  for (int c = 0; c < n_chunks; ++c) put_varint(lens, bits[c]);
  std::vector<uint64_t> offs(n_chunks);
  uint64_t pos = head.size() + ctx_bytes + lens.size();
  for (int c = 0; c < n_chunks; ++c) {
    offs[c] = pos;
    pos += (bits[c] + 7) / 8;
  }
  *out_bytes = pos;
  if (pos > out_cap) return DLMZ_ECAPACITY;
  if (!d_out) return DLMZ_EINVAL;
  DLMZ_CUDA_TRY(cudaMemcpyAsync(d_out, head.data(), head.size(), cudaMemcpyHostToDevice, s));
  if (ctx_pos_bytes)
    DLMZ_CUDA_TRY(cudaMemcpyAsync(d_out + head.size(), all_pos.data(), ctx_pos_bytes, cudaMemcpyHostToDevice, s));
  if (ctx_bytes > ctx_pos_bytes)
    DLMZ_CUDA_TRY(cudaMemcpyAsync(d_out + head.size() + ctx_pos_bytes, w.ctxsyms.as<uint8_t>() + ctx_pos_bytes,
                                  ctx_bytes - ctx_pos_bytes, cudaMemcpyDeviceToDevice, s));
  if (!lens.empty())
    DLMZ_CUDA_TRY(cudaMemcpyAsync(d_out + head.size() + ctx_bytes, lens.data(), lens.size(), cudaMemcpyHostToDevice, s));
  if (n_chunks) {
    DLMZ_CUDA_TRY(cudaMemcpyAsync(w.offsets.p, offs.data(), (size_t)n_chunks * 8, cudaMemcpyHostToDevice, s));
    gather_streams_kernel<<<n_chunks, 128, 0, s>>>(w.staging.as<uint8_t>(), cap, w.bits.as<uint32_t>(),
                                                   w.offsets.as<uint64_t>(), n_chunks, d_out);
    DLMZ_TRY(launch_status());
  }
  return check_device(s);
}

static int decompress_device(dlmz_model* m, const uint8_t* d_in, size_t in_bytes, uint8_t* d_out, size_t out_cap,
                             size_t* out_bytes, cudaStream_t s) {
  if (!m || !d_in || !out_bytes) return DLMZ_EINVAL;
  DLMZ_TRY(device_error_word() ? DLMZ_OK : DLMZ_ENOMEM);
  DLMZ_TRY(clear_device_error(s));
  uint8_t hb[80];
  if (in_bytes < 64) return DLMZ_ECORRUPT;
  DLMZ_CUDA_TRY(cudaMemcpy(hb, d_in, in_bytes < 80 ? in_bytes : 80, cudaMemcpyDeviceToHost));
  Header h{};
  DLMZ_TRY(read_header(hb, in_bytes, h));
  if (h.fingerprint != m->fingerprint) return DLMZ_EMODEL;
  if (h.vocab != m->cfg.vocab || (int)h.P != precision_for(h.vocab)) return DLMZ_ECORRUPT;
  dlmz_k_policy pol{};
  pol.kind = h.kind;
  pol.k = h.k;
  pol.block = h.kind == DLMZ_PROGRESSIVE ? 0 : h.block;
  pol.growth_q16 = h.kind == DLMZ_PROGRESSIVE ? h.block : 65536;
  pol.tau_bits = (float)(h.tau_q / 65536.0);
  pol.k_min = h.k_min;
  pol.k_max = h.k_max;
  pol.coder = h.coder;
  pol.context = h.ctx_kind;
  pol.context_c = h.ctx_c;
  pol.context_seed = h.ctx_seed;
  if (validate_policy(&pol) != DLMZ_OK) return DLMZ_ECORRUPT;
  const uint64_t hsize = h.size(), ctx_bytes = h.ctx_bytes();
  if (hsize + ctx_bytes > in_bytes) return DLMZ_ECORRUPT;
  if (h.n_symbols && h.batch_chunks == 0) return DLMZ_ECORRUPT;
  const int tok = h.vocab > 256;
  const uint64_t out_need = h.n_symbols * (tok ? 4 : 1);
  *out_bytes = out_need;
  if (out_need > out_cap) return DLMZ_ECAPACITY;
  if (out_need && !d_out) return DLMZ_EINVAL;
  const int n_chunks = (int)h.n_chunks;
  const uint64_t lens0 = hsize + ctx_bytes;  // the length table follows the context symbols
  const size_t vmax = (size_t)n_chunks * 5 < in_bytes - lens0 ? (size_t)n_chunks * 5 : in_bytes - lens0;
  std::vector<uint8_t> vb(vmax);
  if (vmax) DLMZ_CUDA_TRY(cudaMemcpy(vb.data(), d_in + lens0, vmax, cudaMemcpyDeviceToHost));
  std::vector<uint32_t> bits(n_chunks);
  size_t p = 0;
  for (int c = 0; c < n_chunks; ++c) {
    uint64_t v = 0;
    int sh = 0;
    for (;;) {
      if (p >= vmax || sh > 35) return DLMZ_ECORRUPT;
      const uint8_t b = vb[p++];
      v |= (uint64_t)(b & 0x7F) << sh;
      sh += 7;
      if (!(b & 0x80)) break;
    }
    if (v > 0xFFFFFFFFull) return DLMZ_ECORRUPT;
    bits[c] = (uint32_t)v;
  }
  std::vector<uint64_t> offs(n_chunks);
  uint64_t pos = lens0 + p;
  for (int c = 0; c < n_chunks; ++c) {
    offs[c] = pos;
    pos += (bits[c] + 7) / 8;
  }
  if (pos != in_bytes) return DLMZ_ECORRUPT;
  const uint32_t L = h.chunk_len;
  const int bc = (int)h.batch_chunks;
  PipeWs& w = pipe_of(m);
  DLMZ_TRY(w.bits.ensure((size_t)n_chunks * 4 + 4));
  DLMZ_TRY(w.offsets.ensure((size_t)n_chunks * 8 + 8));
  DLMZ_TRY(w.crcs.ensure((size_t)n_chunks * 4 + 4));
  if (n_chunks) {
    DLMZ_CUDA_TRY(cudaMemcpyAsync(w.bits.p, bits.data(), (size_t)n_chunks * 4, cudaMemcpyHostToDevice, s));
    DLMZ_CUDA_TRY(cudaMemcpyAsync(w.offsets.p, offs.data(), (size_t)n_chunks * 8, cudaMemcpyHostToDevice, s));
  }
  const size_t bl = (size_t)(bc < n_chunks ? bc : (n_chunks ? n_chunks : 1)) * L;
  DLMZ_TRY(w.state.ensure(bl * 4));
  DLMZ_TRY(w.cst.ensure((size_t)bc * sizeof(CoderState)));
  const uint64_t ce_full = (uint64_t)context_count(pol, (int)L);
  const uint64_t ctx_pos_bytes = h.ctx_pos_bytes();
  std::vector<uint8_t> all_pos(ctx_pos_bytes);
  if (ctx_pos_bytes) DLMZ_CUDA_TRY(cudaMemcpy(all_pos.data(), d_in + hsize, ctx_pos_bytes, cudaMemcpyDeviceToHost));
  for (const BatchPlan& b : plan_batches(h.n_symbols, L, bc)) {
    BatchContext bx;
    std::vector<int32_t> apos;
    if (ctx_pos_bytes) {  // positions of the batch's windows: ascending, inside the window
      const int ce = context_count(pol, b.L);
      apos.resize((size_t)b.nc * ce);
      for (size_t i = 0; i < apos.size(); ++i) {
        const uint32_t p = get32(all_pos.data() + 4 * ((uint64_t)b.c0 * ce_full + i));
        if (p >= (uint32_t)b.L || (i % ce && (int32_t)p <= apos[i - 1])) return DLMZ_ECORRUPT;
        apos[i] = (int32_t)p;
      }
    }
    DLMZ_TRY(batch_context(pol, b.c0, b.nc, b.L, tok ? 4 : 1, w.ctxpos, (uint64_t)b.c0 * ce_full,
                           d_in + hsize + ctx_pos_bytes, nullptr, s, bx, apos.data()));
    DLMZ_TRY(run_batch(m, w.sb, pol, b.nc, b.L, nullptr, w.state.as<int32_t>(), w.cst.as<CoderState>(), nullptr, 0,
                       d_in, w.offsets.as<uint64_t>() + b.c0, w.bits.as<uint32_t>() + b.c0, true, bx, s));
    const int64_t nsym_b = (int64_t)b.nc * b.L;
    symbols_out_kernel<<<grid_for(nsym_b), 256, 0, s>>>(w.state.as<int32_t>(), (int64_t)b.c0 * L, nsym_b, tok, d_out);
    DLMZ_TRY(launch_status());
  }
  int rc = check_device(s);
  if (rc != DLMZ_OK) return rc;
  std::vector<uint32_t> crcs(n_chunks);
  if (n_chunks) {
    window_crc_kernel<<<(n_chunks + 127) / 128, 128, 0, s>>>(d_out, out_need, (uint64_t)L * (tok ? 4 : 1), n_chunks,
                                                             w.crcs.as<uint32_t>());
    DLMZ_TRY(launch_status());
    DLMZ_CUDA_TRY(cudaMemcpyAsync(crcs.data(), w.crcs.p, (size_t)n_chunks * 4, cudaMemcpyDeviceToHost, s));
    DLMZ_CUDA_TRY(cudaStreamSynchronize(s));
  }
  std::vector<uint8_t> crcb((size_t)n_chunks * 4);
  for (int c = 0; c < n_chunks; ++c) put32(crcb.data() + 4 * c, crcs[c]);
  if (crc32_host(crcb.data(), crcb.size()) != h.crc) return DLMZ_ECORRUPT;
  return DLMZ_OK;
}

void pipeline_release(dlmz_model* m) {
  if (m && m->pipe) {
    PipeWs* w = reinterpret_cast<PipeWs*>(m->pipe);
    w->release();
    delete w;
    m->pipe = nullptr;
  }
}

}  // namespace dlmz

using namespace dlmz;

extern "C" {

const char* dlmz_strerror(int code) {
  switch (code) {
    case DLMZ_OK: return "ok";
    case DLMZ_EINVAL: return "invalid argument";
    case DLMZ_EBADINPUT: return "invalid input symbols";
    case DLMZ_ECORRUPT: return "corrupt container";
    case DLMZ_EMODEL: return "container written by another model";
    case DLMZ_ENOMEM: return "out of memory";
    case DLMZ_ECUDA: return "CUDA error";
    case DLMZ_ETIMEOUT: return "device wait timed out";
    case DLMZ_ECAPACITY: return "output buffer too small";
  }
  return "unknown error";
}

void dlmz_free(void* p) { free(p); }

size_t dlmz_compress_bound(const dlmz_model* m, size_t in_bytes, uint32_t chunk_len) {
  if (!m || !chunk_len) return 0;
  const uint64_t n_sym = m->cfg.vocab > 256 ? in_bytes / 4 : in_bytes;
  const uint64_t nc = (n_sym + chunk_len - 1) / chunk_len;
  return 64 + nc * 5 + nc * cap_bytes_for(chunk_len, precision_for(m->cfg.vocab));
}

int dlmz_compress_device(const dlmz_model* m, const void* d_in, size_t in_bytes, uint32_t chunk_len,
                         const dlmz_k_policy* policy, uint32_t batch_chunks, uint8_t* d_out, size_t out_cap,
                         size_t* out_bytes, void* stream) {
  return compress_device(const_cast<dlmz_model*>(m), reinterpret_cast<const uint8_t*>(d_in), in_bytes, chunk_len,
                         policy, batch_chunks, d_out, out_cap, out_bytes, reinterpret_cast<cudaStream_t>(stream));
}

int dlmz_decompress_device(const dlmz_model* m, const uint8_t* d_in, size_t in_bytes, uint8_t* d_out, size_t out_cap,
                           size_t* out_bytes, void* stream) {
  return decompress_device(const_cast<dlmz_model*>(m), d_in, in_bytes, d_out, out_cap, out_bytes,
                           reinterpret_cast<cudaStream_t>(stream));
}

int dlmz_compress_ex(const dlmz_model* mc, const void* in, size_t in_bytes, uint32_t chunk_len,
                     const dlmz_k_policy* policy, uint32_t batch_chunks, uint8_t** out, size_t* out_bytes) {
  if (out) *out = nullptr;
  if (!mc || !out || !out_bytes || (in_bytes && !in)) return DLMZ_EINVAL;
  dlmz_model* m = const_cast<dlmz_model*>(mc);
  PipeWs& w = pipe_of(m);
  const size_t bound = dlmz_compress_bound(m, in_bytes, chunk_len);
  if (!bound) return DLMZ_EINVAL;
  DLMZ_TRY(w.hin.ensure(in_bytes + 16));
  DLMZ_TRY(w.hout.ensure(bound));
  if (in_bytes) DLMZ_CUDA_TRY(cudaMemcpy(w.hin.p, in, in_bytes, cudaMemcpyHostToDevice));
  size_t n = 0;
  DLMZ_TRY(compress_device(m, w.hin.as<uint8_t>(), in_bytes, chunk_len, policy, batch_chunks, w.hout.as<uint8_t>(),
                           bound, &n, 0));
  uint8_t* o = (uint8_t*)malloc(n ? n : 1);
  if (!o) return DLMZ_ENOMEM;
  if (cudaMemcpy(o, w.hout.p, n, cudaMemcpyDeviceToHost) != cudaSuccess) {
    free(o);
    return DLMZ_ECUDA;
  }
  *out = o;
  *out_bytes = n;
  return DLMZ_OK;
}

int dlmz_compress(const dlmz_model* m, const void* in, size_t in_bytes, uint32_t chunk_len, const dlmz_k_policy* policy,
                  uint8_t** out, size_t* out_bytes) {
  return dlmz_compress_ex(m, in, in_bytes, chunk_len, policy, 0, out, out_bytes);
}

int dlmz_decompress(const dlmz_model* mc, const uint8_t* stream, size_t stream_bytes, uint8_t** out, size_t* out_bytes) {
  if (out) *out = nullptr;
  if (!mc || !stream || !out || !out_bytes) return DLMZ_EINVAL;
  if (stream_bytes < 64) return DLMZ_ECORRUPT;
  dlmz_model* m = const_cast<dlmz_model*>(mc);
  Header h{};
  DLMZ_TRY(read_header(stream, stream_bytes, h));
  const uint64_t need = h.n_symbols * (h.vocab > 256 ? 4 : 1);
  if (need > ((uint64_t)1 << 40)) return DLMZ_ECORRUPT;
  PipeWs& w = pipe_of(m);
  DLMZ_TRY(w.hin.ensure(stream_bytes + 16));
  DLMZ_TRY(w.hout.ensure(need + 16));
  DLMZ_CUDA_TRY(cudaMemcpy(w.hin.p, stream, stream_bytes, cudaMemcpyHostToDevice));
  size_t n = 0;
  DLMZ_TRY(decompress_device(m, w.hin.as<uint8_t>(), stream_bytes, w.hout.as<uint8_t>(), need, &n, 0));
  uint8_t* o = (uint8_t*)malloc(n ? n : 1);
  if (!o) return DLMZ_ENOMEM;
  if (n && cudaMemcpy(o, w.hout.p, n, cudaMemcpyDeviceToHost) != cudaSuccess) {
    free(o);
    return DLMZ_ECUDA;
  }
  *out = o;
  *out_bytes = n;
  return DLMZ_OK;
}

int dlmz_check(void* stream) { return check_device(reinterpret_cast<cudaStream_t>(stream)); }

// ---- step-level API ---------------------------------------------------------------------

int dlmz_forward_logits(const dlmz_model* m, const int32_t* d_state, uint32_t n_chunks, uint32_t L, uint32_t row0,
                        uint32_t rows_per_chunk, float* d_logits, void* stream) {
  if (!m || !d_state || !d_logits) return DLMZ_EINVAL;
  if (!device_error_word()) return DLMZ_ENOMEM;
  return model_forward(const_cast<dlmz_model*>(m), d_state, (int)n_chunks, (int)L, (int)row0, (int)rows_per_chunk,
                       d_logits, reinterpret_cast<cudaStream_t>(stream));
}

int dlmz_context_scores(const dlmz_model* mc, const int32_t* d_symbols, uint32_t n_chunks, uint32_t L,
                        float* d_scores, void* stream) {
  dlmz_model* m = const_cast<dlmz_model*>(mc);
  if (!m || !d_symbols || !d_scores || !L || n_chunks > 0x7fffffffu) return DLMZ_EINVAL;
  PipeWs& w = pipe_of(m);
  return context_attention_scores(m, d_symbols, (int)n_chunks, (int)L, d_scores, w.ctxmaps, w.ctxstate,
                                  reinterpret_cast<cudaStream_t>(stream));
}

int dlmz_gemm_bf16(const void* d_A, const void* d_B, float* d_D, uint32_t M, uint32_t N, uint32_t K, void* stream) {
  if (!d_A || !d_B || !d_D || !M || !N || !K) return DLMZ_EINVAL;
  if (!device_error_word()) return DLMZ_ENOMEM;
  GemmEpilogue ep{};
  ep.out = d_D;
  ep.ldo = (int)N;
  const bf16* A = reinterpret_cast<const bf16*>(d_A);
  const bf16* B = reinterpret_cast<const bf16*>(d_B);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (gemm_tc_supported((int)M, (int)N, (int)K) && !((reinterpret_cast<uintptr_t>(d_A) | reinterpret_cast<uintptr_t>(d_B)) & 15))
    return gemm_bf16_tc(A, (int)K, B, (int)K, (int)M, (int)N, (int)K, EPI_F32, ep, s);
  return gemm_simt<bf16>(A, (int)K, B, (int)K, (int)M, (int)N, (int)K, EPI_F32, ep, s);
}

int dlmz_attention_bf16(const void* d_qkv, uint32_t ld, uint32_t n_chunks, uint32_t L, uint32_t n_heads,
                        uint32_t n_kv_heads, uint32_t head_dim, void* d_out, void* stream) {
  if (!d_qkv || !d_out || !n_heads || !n_kv_heads || n_heads % n_kv_heads || !head_dim || head_dim % 8 ||
      head_dim > 128)
    return DLMZ_EINVAL;
  const uint64_t d = (uint64_t)n_heads * head_dim, width = d + 2ull * n_kv_heads * head_dim;
  if (ld < width || ld % 8 || ((reinterpret_cast<uintptr_t>(d_qkv) | reinterpret_cast<uintptr_t>(d_out)) & 15))
    return DLMZ_EINVAL;
  if (n_chunks > 65535 || (uint64_t)n_chunks * L * ld >= (1ull << 31) || (uint64_t)n_chunks * L * d >= (1ull << 31))
    return DLMZ_EINVAL;
  if (!n_chunks || !L) return DLMZ_OK;
  if (!device_error_word()) return DLMZ_ENOMEM;
  const bf16* qkv = reinterpret_cast<const bf16*>(d_qkv);
  bf16* out = reinterpret_cast<bf16*>(d_out);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int nc = (int)n_chunks, l = (int)L, nh = (int)n_heads, nkv = (int)n_kv_heads, hd = (int)head_dim;
  if (attention_tc_supported(l, hd)) {
    static DevBuf vt_dev[kMaxDevices];  // V^T scratch of the tensor-core kernel, one per device
    const int dev = device_ordinal();
    if (dev < 0) return DLMZ_ECUDA;
    DevBuf& vt = vt_dev[dev];
    DLMZ_TRY(vt.ensure((size_t)nc * nkv * attention_vt_rows(hd) * l * 2));
    DLMZ_TRY(attention_vt_from_rows(qkv, (int)ld, (int)(d + (uint64_t)nkv * hd), nc, l, nkv, hd, vt.p, s));
    return attention_bf16_tc(qkv, (int)ld, vt.p, nc, l, nh, nkv, hd, (int)d, out, s);
  }
  if (hd == 64 || hd == 128) return attention_bf16_mma(qkv, (int)ld, nc, l, nh, nkv, hd, (int)d, out, s);
  return attention_simt<bf16>(qkv, (int)ld, nc, l, nh, nkv, hd, (int)d, out, s);
}

int dlmz_quantize(const float* d_logits, uint32_t rows, uint32_t V, uint32_t P, uint32_t* d_cdf, uint64_t* d_W,
                  uint64_t* d_A, int32_t* d_Hq, int32_t* d_top, void* stream) {
  if (!d_logits || !d_W || !d_Hq || V < 2 || P > 24 || (1ull << P) <= V) return DLMZ_EINVAL;
  if (!device_error_word()) return DLMZ_ENOMEM;
  return quantize_rows(d_logits, (int)rows, (int)V, (int)P, d_cdf, d_W, d_A, d_Hq, d_top, nullptr,
                       reinterpret_cast<cudaStream_t>(stream));
}

int dlmz_select_smallest(const uint64_t* d_keys, uint32_t groups, uint32_t group_size, uint32_t k, int32_t* d_out,
                         void* stream) {
  if (!d_keys || !d_out || k == 0 || k > group_size || group_size > 4096) return DLMZ_EINVAL;
  static DevBuf counts_dev[kMaxDevices];  // one count per group, one buffer per device
  const int dev = device_ordinal();
  if (dev < 0) return DLMZ_ECUDA;
  DevBuf& counts = counts_dev[dev];
  DLMZ_TRY(counts.ensure((size_t)groups * 4 + 4));
  return select_rows<uint64_t>(nullptr, (int)groups, (int)group_size, -1, 0, (int)group_size, d_keys, 0, (int)k, 0, 0,
                               0, (int)k, counts.as<int32_t>(), d_out, reinterpret_cast<cudaStream_t>(stream));
}

struct dlmz_coder {
  int nc, L, V, P, coder;
  uint64_t cap;
  DevBuf cst, bytes;
  StepBufs sb;
  const uint8_t* in_bytes = nullptr;
  const uint64_t* in_off = nullptr;
  const uint32_t* in_bits = nullptr;
};

int dlmz_coder_create_ex(uint32_t n_chunks, uint32_t L, uint32_t V, uint32_t P, uint32_t coder, dlmz_coder** out) {
  if (!out) return DLMZ_EINVAL;
  *out = nullptr;
  if (!n_chunks || !L || V < 2 || P > 24 || (1ull << P) <= V || coder > DLMZ_CODER_RANKS) return DLMZ_EINVAL;
  if (!device_error_word()) return DLMZ_ENOMEM;
  dlmz_coder* c = new dlmz_coder();
  c->coder = (int)coder;
  c->nc = (int)n_chunks;
  c->L = (int)L;
  c->V = (int)V;
  c->P = (int)P;
  c->cap = cap_bytes_for(L, (int)P);
  if (c->cst.ensure((size_t)n_chunks * sizeof(CoderState)) || c->bytes.ensure((size_t)n_chunks * c->cap)) {
    dlmz_coder_destroy(c);
    return DLMZ_ENOMEM;
  }
  *out = c;
  return DLMZ_OK;
}

int dlmz_coder_create(uint32_t n_chunks, uint32_t L, uint32_t V, uint32_t P, dlmz_coder** out) {
  return dlmz_coder_create_ex(n_chunks, L, V, P, DLMZ_CODER_RANGE, out);
}

void dlmz_coder_destroy(dlmz_coder* c) {
  if (!c) return;
  c->cst.release();
  c->bytes.release();
  c->sb.release();
  delete c;
}

uint32_t dlmz_coder_capacity_units(const dlmz_coder* c) { return c ? (uint32_t)(c->cap / 2) : 0; }

int dlmz_coder_reset_encoder(dlmz_coder* c, void* stream) {
  if (!c) return DLMZ_EINVAL;
  return coder_reset(c->cst.as<CoderState>(), c->nc, reinterpret_cast<cudaStream_t>(stream));
}

int dlmz_coder_load_decoder(dlmz_coder* c, const uint8_t* d_bytes, const uint64_t* d_offsets, const uint32_t* d_bits,
                            void* stream) {
  if (!c || !d_bytes || !d_offsets || !d_bits) return DLMZ_EINVAL;
  c->in_bytes = d_bytes;
  c->in_off = d_offsets;
  c->in_bits = d_bits;
  return coder_load(c->cst.as<CoderState>(), c->nc, d_bytes, d_offsets, d_bits, c->coder,
                    reinterpret_cast<cudaStream_t>(stream));
}

static int step_common(dlmz_coder* c, const dlmz_k_policy* pol, const float* d_logits, uint32_t row0, uint32_t rpc,
                       const int32_t* d_symbols, int32_t* d_state, int32_t* d_committed, bool decode, void* stream) {
  if (!c || !d_logits || !d_state || validate_policy(pol) != DLMZ_OK) return DLMZ_EINVAL;
  if ((int)pol->coder != c->coder) return DLMZ_EINVAL;  // the coder's kind decides
  if (rpc == 0 || row0 + rpc > (uint32_t)c->L) return DLMZ_EINVAL;
  if (!decode && !d_symbols) return DLMZ_EINVAL;
  if (decode && !c->in_bytes) return DLMZ_EINVAL;
  return run_step(c->sb, d_logits, c->nc, c->L, c->V, c->P, *pol, (int)row0, (int)rpc, d_symbols, d_state,
                  c->cst.as<CoderState>(), c->bytes.as<uint8_t>(), c->cap, c->in_bytes, c->in_off, c->in_bits, decode,
                  d_committed, reinterpret_cast<cudaStream_t>(stream));
}

static int model_step_common(dlmz_model* m, dlmz_coder* c, const dlmz_k_policy* pol, uint32_t row0, uint32_t rpc,
                             const int32_t* d_symbols, int32_t* d_state, int32_t* d_committed, bool decode,
                             void* stream) {
  if (!m || !c || !d_state || validate_policy(pol) != DLMZ_OK) return DLMZ_EINVAL;
  if ((int)pol->coder != c->coder || pol->context != DLMZ_CONTEXT_NONE) return DLMZ_EINVAL;
  if ((int)m->cfg.vocab != c->V || precision_for(m->cfg.vocab) != c->P) return DLMZ_EINVAL;
  if (rpc == 0 || row0 + rpc > (uint32_t)c->L) return DLMZ_EINVAL;
  if (!decode && !d_symbols) return DLMZ_EINVAL;
  if (decode && !c->in_bytes) return DLMZ_EINVAL;
  const StepIO io{d_symbols, d_state, c->cst.as<CoderState>(), c->bytes.as<uint8_t>(), c->cap, c->in_bytes,
                  c->in_off, c->in_bits, decode, d_committed};
  return model_step(m, c->sb, *pol, c->nc, c->L, (int)row0, (int)rpc, io, reinterpret_cast<cudaStream_t>(stream));
}

int dlmz_model_encode_step(dlmz_model* m, dlmz_coder* c, const dlmz_k_policy* policy, uint32_t row0,
                           uint32_t rows_per_chunk, const int32_t* d_symbols, int32_t* d_state, int32_t* d_committed,
                           void* stream) {
  return model_step_common(m, c, policy, row0, rows_per_chunk, d_symbols, d_state, d_committed, false, stream);
}

int dlmz_model_decode_step(dlmz_model* m, dlmz_coder* c, const dlmz_k_policy* policy, uint32_t row0,
                           uint32_t rows_per_chunk, int32_t* d_state, int32_t* d_committed, void* stream) {
  return model_step_common(m, c, policy, row0, rows_per_chunk, nullptr, d_state, d_committed, true, stream);
}

int dlmz_encode_step(dlmz_coder* c, const dlmz_k_policy* policy, const float* d_logits, uint32_t row0,
                     uint32_t rows_per_chunk, const int32_t* d_symbols, int32_t* d_state, int32_t* d_committed,
                     void* stream) {
  return step_common(c, policy, d_logits, row0, rows_per_chunk, d_symbols, d_state, d_committed, false, stream);
}

int dlmz_decode_step(dlmz_coder* c, const dlmz_k_policy* policy, const float* d_logits, uint32_t row0,
                     uint32_t rows_per_chunk, int32_t* d_state, int32_t* d_committed, void* stream) {
  return step_common(c, policy, d_logits, row0, rows_per_chunk, nullptr, d_state, d_committed, true, stream);
}

int dlmz_coder_finish(dlmz_coder* c, uint32_t* d_bits, uint8_t* d_bytes, const uint64_t* d_offsets, void* stream) {
  if (!c || !d_bits) return DLMZ_EINVAL;
  return coder_finish(c->cst.as<CoderState>(), c->nc, c->bytes.as<uint8_t>(), c->cap, d_bits, d_bytes, d_offsets,
                      c->coder, c->sb.pairs.as<uint64_t>(), c->L, c->P, reinterpret_cast<cudaStream_t>(stream));
}

}  // extern "C"
