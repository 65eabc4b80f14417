// Coder state and launch helpers of the selection / range-coding step.
#pragma once

#include "kernels.cuh"

namespace dlmz {

// Per-window coder state.  Range coder -- encoder: low/rng and the count of
// emitted 16-bit units; decoder: `low` holds val = code - low, `n_units` the
// next unit to read.  rANS -- encoder: `n_units` counts the buffered (c, f)
// pairs; decoder: `low` is the state x, `n_units` the next 32-bit word.
// Ranks -- `n_units` is the byte position in the window's varint stream.
struct CoderState {
  uint64_t low;
  uint64_t rng;
  uint32_t n_units;
  uint32_t pad;
};

struct CodeArgs {
  const float* logits;       // [n_chunks * rpc x V], or rows found through row_map / sel_major
  const float* mx;           // per row: max logit
  const uint64_t* W;         // per row: W
  const int32_t* top;        // per row: lowest argmax
  const int32_t* sel_count;  // [n_chunks]
  const int32_t* sel_pos;    // [n_chunks x kcap], ascending
  const int32_t* symbols;    // encoder: true symbols [n_chunks x L]
  int32_t* state;            // [n_chunks x L]
  CoderState* state_c;       // [n_chunks]
  uint8_t* bytes;            // encoder streams [n_chunks x cap_bytes]
  uint64_t cap_bytes;
  const uint8_t* in_bytes;   // decoder streams
  const uint64_t* in_offsets;
  const uint32_t* in_bits;
  int32_t* committed;        // optional [n_chunks]
  int* err;
  int V, P, L, row0, rpc, kcap;
  int coder;                 // 0: range coder, 1: rANS, 2: symbol ranks (varints)
  uint64_t* pairs;           // rANS encoder: (c << 32 | f) per coded symbol [n_chunks x pair_cap]
  int pair_cap;
  const int32_t* row_map;    // optional [n_chunks x rpc]: row of logits / mx / W / top of each candidate
  int sel_major;             // without row_map: row of the j-th selected position = c * kcap + j
  // scratch of the row-parallel range / rANS path, [n_chunks x kcap] selected rows:
  uint64_t* rowcf;           // encoder: (c_s << 32) | f_s of each selected row
  uint32_t* segcum;          // decoder: per row nseg + 1 prefix sums of 1 + floor(w R / W) at segment starts
  uint64_t* rowK;            // decoder: floor(R 2^64 / W) of each selected row
  uint32_t* rowD;            // decoder: the remainder D of each selected row
  int nseg;                  // decoder: segments of CODE_SEG elements per row
};

constexpr int CODE_SEG = 512;  // elements per segment of a row's coarse CDF (decoder)

// keys of window c's position row0 + i: keys[row_map[c * rpc + i]] when row_map is
// given (candidates only), else keys[c * rpc + i].
template <typename K>
int select_rows(const int32_t* state, int n_chunks, int L, int mask_id, int row0, int rpc, const K* keys, int n_rule,
                int k, int64_t tau_q, int k_min, int k_max, int kcap, int32_t* sel_count, int32_t* sel_pos,
                cudaStream_t s, const int32_t* row_map = nullptr);
int code_step(const CodeArgs& a, bool decode, int n_chunks, cudaStream_t s);
int coder_reset(CoderState* st, int n, cudaStream_t s);
int coder_load(CoderState* st, int n, const uint8_t* bytes, const uint64_t* offsets, const uint32_t* bits, int coder,
               cudaStream_t s);
// Terminates every stream (range coder) or codes every window's buffered pairs
// in reverse (rANS: pairs, pair_cap, P), then bit lengths / copies as documented
// at dlmz_coder_finish.
int coder_finish(CoderState* st, int n, uint8_t* bytes, uint64_t cap_bytes, uint32_t* bits, uint8_t* out,
                 const uint64_t* offsets, int coder, const uint64_t* pairs, int pair_cap, int P, cudaStream_t s);

}  // namespace dlmz
