// Commitment schedule (Sec. 3.3) and per-window range coding of the
// committed symbols (statistical coding, Sec. 2.1 / Sec. 4), one
// independent stream per window.
//
// Selection: every schedule here commits the n smallest candidates under
// (key, position): top-k confidence (key W, n = min(k, #candidates) of the
// leftmost incomplete block), the entropy threshold (key H_q, n = #{H_q <=
// tau} or m if fewer, capped by k_max), and the left-to-right uniform-block and
// progressive schedules (no key: the n = u_k leftmost masked positions).  A CTA per window ranks its
// candidates, so the result does not depend on thread order.
//
// Range coder: 64-bit low/range, 16-bit output units stored big-endian,
// renormalisation below 2^48, carries propagated into the emitted units,
// minimal termination.  The decoder keeps val = code - low and reads units
// beyond the stream's length as zero (never past its buffer).
// rANS (the paper's coder, Sec. 2.1): 64-bit state in [2^31, 2^63), 32-bit
// words; encode x = floor(x/f) 2^P + x mod f + c after emitting the low word
// when x >= 2^(63-P) f.  Last in, first out: the steps buffer a window's
// (c, f) pairs and the finish kernel codes them in reverse; the stream is the
// final state (8 bytes big-endian) then the words in reverse emission order.
// Symbol ranks (the paper's ranking pipeline): each coded symbol becomes
// #{v : f_v > f_s} + #{v < s : f_v = f_s} (integer frequencies of the step's
// table), written as an LEB128 varint; the decoder finds the frequency level
// holding rank r by binary search (block counts), then the symbol by index.
#include "kernels.cuh"
#include "coder.cuh"
#include "exp_table.inc"
#include "intq.cuh"

namespace dlmz {

static __constant__ uint32_t c_exp_table_c[256] = DLMZ_EXP_TABLE_INIT;

// ---- selection ----------------------------------------------------------------------
// CTA per window.  The n smallest candidates under (key, position) are those with key < K* plus
// the lowest-position ones with key == K*, where K* is the n-th smallest key: a most-significant-
// digit-first radix select (8 passes of 8-bit digits, a shared histogram each) finds K* and how
// many of its ties are taken, then one ordered pass writes the selected positions ascending.
constexpr int SEL_T = 256;  // threads per window (one histogram bin per thread)

// exclusive prefix sum over the CTA of one value per thread (SEL_T threads); *total gets the sum
__device__ __forceinline__ int sel_block_scan(int v, int* wtot, int* total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int inc = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += t;
  }
  if (lane == 31) wtot[w] = inc;
  __syncthreads();
  const int tv = lane < SEL_T / 32 ? wtot[lane] : 0;
  const int pre = __reduce_add_sync(0xffffffffu, lane < w ? tv : 0);
  *total = __reduce_add_sync(0xffffffffu, tv);
  __syncthreads();  // wtot may be rewritten by the next scan
  return pre + inc - v;
}

template <typename K>
__global__ void __launch_bounds__(SEL_T) select_kernel(const int32_t* __restrict__ state, int L, int mask_id, int row0,
                                                       int rpc, const K* __restrict__ keys,
                                                       const int32_t* __restrict__ row_map, int n_rule, int k,
                                                       int64_t tau_q, int k_min, int k_max, int kcap,
                                                       int32_t* __restrict__ sel_count, int32_t* __restrict__ sel_pos) {
  extern __shared__ uint64_t skey[];  // rpc keys, then rpc flags (as bytes)
  uint8_t* valid = reinterpret_cast<uint8_t*>(skey + rpc);
  __shared__ int hist[SEL_T];
  __shared__ int wtot[SEL_T / 32];
  __shared__ int s_bin, s_below;
  const int c = blockIdx.x;
  int nv = 0, nb = 0;
  for (int i = threadIdx.x; i < rpc; i += SEL_T) {
    const bool ok = state ? state[(size_t)c * L + row0 + i] == mask_id : true;
    // null keys: position order; with a row map only candidates have a key row
    const int64_t kr = row_map ? (ok ? row_map[(size_t)c * rpc + i] : -1) : (int64_t)c * rpc + i;
    const uint64_t key = keys && kr >= 0 ? (uint64_t)(int64_t)keys[kr] : 0;
    skey[i] = key;
    valid[i] = ok;
    nv += ok;
    nb += ok && (int64_t)key <= tau_q;
  }
  int tv, tb;
  sel_block_scan(nv, wtot, &tv);
  sel_block_scan(nb, wtot, &tb);
  int n;
  if (n_rule == 0) {
    n = min(k, tv);
  } else {
    n = tb < k_min ? min(k_min, tv) : tb;
    if (k_max > 0 && n > k_max) n = k_max;
  }
  const int nsel = min(n, kcap);
  // K* = the nsel-th smallest key; `need` of its ties (lowest positions first) are taken
  uint64_t kstar = ~0ull;
  int need = 0x7fffffff;
  if (nsel > 0 && nsel < tv) {
    uint64_t prefix = 0, pmask = 0;
    int rank = nsel - 1;  // 0-based rank of K* among the candidates still matching the prefix
#pragma unroll 1
    for (int shift = 56; shift >= 0; shift -= 8) {
      hist[threadIdx.x] = 0;
      __syncthreads();
      for (int i = threadIdx.x; i < rpc; i += SEL_T) {
        const uint64_t key = skey[i];
        if (valid[i] && (key & pmask) == prefix) atomicAdd(&hist[(int)(key >> shift) & 255], 1);
      }
      __syncthreads();
      const int cnt = hist[threadIdx.x];
      int tot;
      const int below = sel_block_scan(cnt, wtot, &tot);
      if (below <= rank && rank < below + cnt) {  // exactly one bin holds the rank
        s_bin = threadIdx.x;
        s_below = below;
      }
      __syncthreads();
      prefix |= (uint64_t)s_bin << shift;
      pmask |= 0xFFull << shift;
      rank -= s_below;
    }
    kstar = prefix;
    need = rank + 1;
  }
  // ordered pass: candidate i is selected iff key < K*, or key == K* and fewer than `need` ties
  // precede it (with nsel >= #candidates every candidate is selected)
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int ties = 0, base = 0;
  for (int i0 = 0; i0 < rpc; i0 += SEL_T) {
    const int i = i0 + threadIdx.x;
    const bool ok = i < rpc && valid[i] && nsel > 0;
    const uint64_t key = ok ? skey[i] : 0;
    const bool tie = ok && key == kstar;
    int tot;
    const int tie_before = ties + sel_block_scan(tie ? 1 : 0, wtot, &tot);
    ties += tot;
    const bool sel = ok && (nsel >= tv || key < kstar || (tie && tie_before < need));
    const int off = base + sel_block_scan(sel ? 1 : 0, wtot, &tot);
    if (sel) sel_pos[(size_t)c * kcap + off] = row0 + i;
    base += tot;
    (void)lane;
    (void)w;
  }
  if (threadIdx.x == 0) sel_count[c] = nsel;
}

template <typename K>
int select_rows(const int32_t* state, int n_chunks, int L, int mask_id, int row0, int rpc, const K* keys, int n_rule,
                int k, int64_t tau_q, int k_min, int k_max, int kcap, int32_t* sel_count, int32_t* sel_pos,
                cudaStream_t s, const int32_t* row_map) {
  if (n_chunks == 0) return DLMZ_OK;
  const size_t smem = (size_t)rpc * 9 + 16;
  if (smem > 200 * 1024) return DLMZ_EINVAL;
  static PerDeviceOnce attr;
  DLMZ_TRY(attr.run(
      [] { return cudaFuncSetAttribute(select_kernel<K>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024); }));
  ProfScope prof(PROF_SELECT, s, 0, (double)n_chunks * rpc * (sizeof(K) + 4));
  select_kernel<K><<<n_chunks, SEL_T, smem, s>>>(state, L, mask_id, row0, rpc, keys, row_map, n_rule, k, tau_q, k_min,
                                               k_max, kcap, sel_count, sel_pos);
  return launch_status();
}
template int select_rows<uint64_t>(const int32_t*, int, int, int, int, int, const uint64_t*, int, int, int64_t, int,
                                   int, int, int32_t*, int32_t*, cudaStream_t, const int32_t*);
template int select_rows<int32_t>(const int32_t*, int, int, int, int, int, const int32_t*, int, int, int64_t, int,
                                  int, int, int32_t*, int32_t*, cudaStream_t, const int32_t*);

// ---- range coder -----------------------------------------------------------------------
constexpr uint64_t RENORM = 1ull << 48;
constexpr int CT = 256;  // threads per window in the coding kernel

__device__ __forceinline__ uint32_t unit_at(const uint8_t* b, uint64_t nbytes, uint32_t i) {
  const uint64_t o = 2ull * i;
  uint32_t hi = o < nbytes ? b[o] : 0u;
  uint32_t lo = o + 1 < nbytes ? b[o + 1] : 0u;
  return (hi << 8) | lo;
}

// big-endian 32-bit word at byte offset o (bytes at or past nbytes read as 0)
__device__ __forceinline__ uint64_t word_at(const uint8_t* b, uint64_t nbytes, uint64_t o) {
  uint64_t w = 0;
  for (int i = 0; i < 4; ++i) w = (w << 8) | (o + i < nbytes ? b[o + i] : 0u);
  return w;
}

constexpr uint64_t RANS_L = 1ull << 31;

__device__ __forceinline__ void put_unit(uint8_t* b, uint32_t i, uint32_t u) {
  b[2 * i] = (uint8_t)(u >> 8);
  b[2 * i + 1] = (uint8_t)u;
}

__device__ void enc_symbol(CoderState& st, uint8_t* buf, uint32_t cap_units, int P, uint64_t cs, uint64_t fs,
                           int* err) {
  const uint64_t r = st.rng >> P;
  const uint64_t nl = st.low + r * cs;
  if (nl < st.low) {  // carry into the emitted units
    int i = (int)st.n_units - 1;
    for (; i >= 0; --i) {
      const uint32_t u = ((unit_at(buf, 2ull * cap_units, i) + 1) & 0xFFFFu);
      put_unit(buf, i, u);
      if (u) break;
    }
    if (i < 0) atomicOr(err, ERR_CORRUPT);
  }
  st.low = nl;
  st.rng = r * fs;
  while (st.rng < RENORM) {
    if (st.n_units < cap_units) put_unit(buf, st.n_units, (uint32_t)(st.low >> 48));
    else atomicOr(err, ERR_CAPACITY);
    st.n_units++;
    st.low <<= 16;
    st.rng <<= 16;
  }
}

__device__ __forceinline__ uint64_t block_excl_scan(uint64_t v, uint64_t* wsum, uint64_t* total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  uint64_t inc = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint64_t t = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += t;
  }
  __syncthreads();
  if (lane == 31) wsum[w] = inc;
  __syncthreads();
  uint64_t pre = 0, tot = 0;
  for (int i = 0; i < nw; ++i) {
    if (i < w) pre += wsum[i];
    tot += wsum[i];
  }
  *total = tot;
  return pre + inc - v;
}

template <bool DECODE>
__global__ void __launch_bounds__(CT) code_kernel(CodeArgs a) {
  __shared__ uint32_t T[256];
  __shared__ uint32_t tabf[QW0 + 1];  // floor(w(q) R / W) of the current row (0 from QW0 on)
  __shared__ uint64_t wsum[CT / 32];
  __shared__ uint64_t s_slot, s_cs, s_fs;
  __shared__ int s_sym;
  __shared__ CoderState st;
  for (int i = threadIdx.x; i < 256; i += CT) T[i] = c_exp_table_c[i];
  const int c = blockIdx.x;
  const int n = a.sel_count[c];
  if (threadIdx.x == 0) st = a.state_c[c];
  __syncthreads();
  const int V = a.V, P = a.P;
  const uint64_t R = (1ull << P) - (uint64_t)V;
  const int segl = (V + CT - 1) / CT;
  const int v0 = threadIdx.x * segl, v1 = min(V, v0 + segl);
  uint8_t* ebuf = a.bytes + (size_t)c * a.cap_bytes;  // encoder stream
  const uint8_t* dbuf = DECODE ? a.in_bytes + (a.in_offsets ? a.in_offsets[c] : 0) : nullptr;
  const uint64_t dn = DECODE ? (a.in_bits[c] + 7) / 8 : 0;
  for (int j = 0; j < n; ++j) {
    const int pos = a.sel_pos[(size_t)c * a.kcap + j];
    // the row of this position's logits and stats: through the candidate map, the j-th
    // selected row of the window, or the dense row of [row0, row0 + rpc)
    const size_t row = a.row_map ? (size_t)a.row_map[(size_t)c * a.rpc + (pos - a.row0)]
                     : a.sel_major ? (size_t)c * a.kcap + j
                                   : (size_t)c * a.rpc + (pos - a.row0);
    const float* lr = a.logits + row * V;
    const float m = a.mx[row];
    const uint64_t Wr = a.W[row];
    const int top = a.top[row];
    // this row's floor(w(q) R / W) for every code (division-free, K = floor(R 2^64 / W)); the
    // barrier at the end of the previous symbol leaves the table free
    {
      uint64_t K = 0;
      if ((threadIdx.x & 31) == 0) K = recip_scaled((uint32_t)R, Wr);
      K = __shfl_sync(0xffffffffu, K, 0);
      for (int b = threadIdx.x; b <= QW0; b += CT) tabf[b] = b < QW0 ? floor_wr_over_w(quant_w(T, b), (uint32_t)R, Wr, K) : 0u;
      __syncthreads();
    }
    // floor(w_v R / W) of element v (codes from QW0 on weigh nothing, non-finite values land there)
    auto flo_of = [&](int v) -> uint64_t { return tabf[code_index(__fsub_rn(m, lr[v]))]; };
    uint64_t sseg = 0;
    for (int v = v0; v < v1; ++v) sseg += 1 + flo_of(v);
    uint64_t total;
    const uint64_t pre = block_excl_scan(sseg, wsum, &total);
    const uint64_t D = (1ull << P) - total;
    // f_v of this row (the same integer table the coders use)
#define FREQ(v_) (1 + flo_of(v_) + ((v_) == top ? D : 0))
    const uint64_t lo = pre + (v0 > top ? D : 0);
    const uint64_t hi = lo + sseg + (top >= v0 && top < v1 ? D : 0);
    if (!DECODE) {
      const int sym = a.symbols[(size_t)c * a.L + pos];
      if (sym >= v0 && sym < v1) {
        uint64_t cum = lo;
        for (int v = v0; v < v1; ++v) {
          const uint64_t f = FREQ(v);
          if (v == sym) {
            s_cs = cum;
            s_fs = f;
            break;
          }
          cum += f;
        }
      }
      __syncthreads();
      uint64_t rank = 0;
      if (a.coder == 2) {  // rank of sym: frequencies above f_s, then equal ones with a smaller index
        uint64_t cnt = 0;
        for (int v = v0; v < v1; ++v) {
          const uint64_t f = FREQ(v);
          cnt += f > s_fs || (f == s_fs && v < sym);
        }
        block_excl_scan(cnt, wsum, &rank);
      }
      if (threadIdx.x == 0) {
        CoderState t = st;
        if (a.coder == 2) {
          uint64_t r = rank;
          do {
            const uint8_t b = (uint8_t)((r & 0x7F) | (r >= 0x80 ? 0x80 : 0));
            if (t.n_units < a.cap_bytes) ebuf[t.n_units] = b;
            else atomicOr(a.err, ERR_CAPACITY);
            t.n_units++;
            r >>= 7;
          } while (r);
        } else if (a.coder == 1) {  // buffered; coded in reverse when the window is finished
          if (t.n_units < (uint32_t)a.pair_cap) a.pairs[(size_t)c * a.pair_cap + t.n_units] = (s_cs << 32) | s_fs;
          else atomicOr(a.err, ERR_CAPACITY);
          t.n_units++;
        } else {
          enc_symbol(t, ebuf, a.cap_bytes / 2, P, s_cs, s_fs, a.err);
        }
        st = t;
        a.state[(size_t)c * a.L + pos] = sym;
      }
      __syncthreads();
    } else {
      if (threadIdx.x == 0) {
        if (a.coder == 2) {  // next varint of the window's rank stream
          uint64_t r = 0, pos = st.n_units;
          int sh = 0;
          bool done = false;
          while (!done) {
            const uint8_t b = pos < dn ? dbuf[pos] : 0x80;
            ++pos;
            if (sh < 63) r |= (uint64_t)(b & 0x7F) << sh;
            sh += 7;
            done = !(b & 0x80) || sh > 35;
            if (pos > dn) done = true;
          }
          if (pos > dn || sh > 35 || r >= (uint64_t)V) {
            atomicOr(a.err, ERR_CORRUPT);
            r = 0;
          }
          st.n_units = (uint32_t)pos;
          s_slot = r;
        } else if (a.coder == 1) {
          s_slot = st.low & ((1ull << P) - 1);  // x mod 2^P
        } else {
          const uint64_t r = st.rng >> P;
          uint64_t slot = st.low / r;  // decoder keeps val in .low
          if (slot >= (1ull << P)) {
            atomicOr(a.err, ERR_CORRUPT);
            slot = (1ull << P) - 1;
          }
          s_slot = slot;
        }
      }
      __syncthreads();
      const uint64_t slot = s_slot;
      if (a.coder == 2) {  // slot holds the rank r: find the frequency level, then the symbol by index
        uint64_t flo = 1, fhi = (1ull << P) + 1, tot;  // count(f >= flo) > r >= count(f >= fhi)
        while (fhi - flo > 1) {
          const uint64_t mid = (flo + fhi) / 2;
          uint64_t cnt = 0;
          for (int v = v0; v < v1; ++v) cnt += FREQ(v) >= mid;
          block_excl_scan(cnt, wsum, &tot);
          if (tot > slot) flo = mid;
          else fhi = mid;
        }
        uint64_t above = 0, eq = 0;
        for (int v = v0; v < v1; ++v) {
          const uint64_t f = FREQ(v);
          above += f > flo;
          eq += f == flo;
        }
        block_excl_scan(above, wsum, &tot);
        const uint64_t t = slot - tot;  // index of the symbol among those with f == flo
        const uint64_t pre = block_excl_scan(eq, wsum, &tot);
        if (t >= pre && t < pre + eq) {
          uint64_t k = pre;
          for (int v = v0; v < v1; ++v) {
            if (FREQ(v) == flo) {
              if (k == t) {
                s_sym = v;
                s_fs = flo;
                break;
              }
              ++k;
            }
          }
        }
      } else if (slot >= lo && slot < hi) {
        uint64_t cum = lo;
        for (int v = v0; v < v1; ++v) {
          const uint64_t f = FREQ(v);
          if (slot < cum + f) {
            s_sym = v;
            s_cs = cum;
            s_fs = f;
            break;
          }
          cum += f;
        }
      }
      __syncthreads();
      if (threadIdx.x == 0) {
        CoderState t = st;
        if (a.coder == 2) {
          // the rank stream advanced when it was read
        } else if (a.coder == 1) {
          t.low = s_fs * (t.low >> P) + slot - s_cs;
          if (t.low < RANS_L) {
            t.low = (t.low << 32) | word_at(dbuf, dn, 8 + 4ull * t.n_units);
            t.n_units++;
          }
        } else {
          const uint64_t r = t.rng >> P;
          t.low -= r * s_cs;
          t.rng = r * s_fs;
          while (t.rng < RENORM) {
            t.low = (t.low << 16) | unit_at(dbuf, dn, t.n_units++);
            t.rng <<= 16;
          }
        }
        st = t;
        a.state[(size_t)c * a.L + pos] = s_sym;
      }
      __syncthreads();
    }
  }
#undef FREQ
  if (threadIdx.x == 0) {
    a.state_c[c] = st;
    if (a.committed) a.committed[c] = n;
  }
}

// ---- row-parallel range / rANS coding ----------------------------------------------------------
// The frequencies of the selected rows do not depend on one another: one CTA per selected row
// (grid kcap x windows) computes them from the row's logits in one pass, and only the coder itself,
// which is sequential within a window, runs per window afterwards.
constexpr int RT_ROWS = 256;

__device__ __forceinline__ size_t selected_row(const CodeArgs& a, int c, int j, int pos) {
  return a.row_map ? (size_t)a.row_map[(size_t)c * a.rpc + (pos - a.row0)]
       : a.sel_major ? (size_t)c * a.kcap + j
                     : (size_t)c * a.rpc + (pos - a.row0);
}

// shared table floor(w(q) R / W) of one row for every code (0 from QW0 on); all threads call it
__device__ void build_floor_table(uint32_t* tabf, const uint32_t* T, uint32_t R, uint64_t Wr) {
  uint64_t K = 0;
  if ((threadIdx.x & 31) == 0) K = recip_scaled(R, Wr);
  K = __shfl_sync(0xffffffffu, K, 0);
  for (int b = threadIdx.x; b <= QW0; b += blockDim.x) tabf[b] = b < QW0 ? floor_wr_over_w(quant_w(T, b), R, Wr, K) : 0u;
  __syncthreads();
}

// floor(w R / W) of one element: from the shared table for large vocabularies; directly (K) for
// vocabularies below the table's 7938 entries, where building the table would cost more than the row
struct RowFloor {
  const uint32_t* tabf;
  const uint32_t* T;
  uint32_t R;
  uint64_t W, K;
  bool table;
  __device__ __forceinline__ uint32_t operator()(float m, float x) const {
    const uint32_t q = code_index(__fsub_rn(m, x));
    if (table) return tabf[q];
    return q < (uint32_t)QW0 ? floor_wr_over_w(quant_w(T, (int)q), R, W, K) : 0u;
  }
};

__device__ RowFloor row_floor(uint32_t* tabf, const uint32_t* T, uint32_t R, uint64_t Wr, int V) {
  RowFloor rf{tabf, T, R, Wr, 0, V > QW0};
  if (rf.table) {
    build_floor_table(tabf, T, R, Wr);
  } else {
    uint64_t K = 0;
    if ((threadIdx.x & 31) == 0) K = recip_scaled(R, Wr);
    rf.K = __shfl_sync(0xffffffffu, K, 0);
  }
  return rf;
}

// block sum of one u32 per thread (RT_ROWS threads); every thread gets the total
__device__ __forceinline__ uint32_t rows_block_sum(uint32_t v, uint32_t* red) {
  v = __reduce_add_sync(0xffffffffu, v);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  const uint32_t t = __reduce_add_sync(0xffffffffu, (threadIdx.x & 31) < RT_ROWS / 32 ? red[threadIdx.x & 31] : 0u);
  __syncthreads();
  return t;
}

// Encoder: (c_s, f_s) of the true symbol s of selected row j of window c:
// c_s = s + sum_{v<s} floor(w_v R / W) + (top < s ? D : 0), f_s = 1 + floor(w_s R / W) + (s == top ? D : 0),
// D = R - sum_v floor(w_v R / W).
__global__ void __launch_bounds__(RT_ROWS) enc_rows_kernel(CodeArgs a) {
  __shared__ uint32_t T[256];
  __shared__ uint32_t tabf[QW0 + 1];
  __shared__ uint32_t red[RT_ROWS / 32];
  const int c = blockIdx.y, j = blockIdx.x;
  if (j >= a.sel_count[c]) return;
  for (int i = threadIdx.x; i < 256; i += RT_ROWS) T[i] = c_exp_table_c[i];
  const int pos = a.sel_pos[(size_t)c * a.kcap + j];
  const size_t row = selected_row(a, c, j, pos);
  const int V = a.V, sym = a.symbols[(size_t)c * a.L + pos];
  const float* lr = a.logits + row * V;
  const float m = a.mx[row];
  const uint64_t Wr = a.W[row];
  const int top = a.top[row];
  const uint32_t R = (1u << a.P) - (uint32_t)V;
  __syncthreads();
  const RowFloor flo = row_floor(tabf, T, R, Wr, V);
  uint32_t s_all = 0, s_lt = 0;
  if ((V & 3) == 0 && (reinterpret_cast<uintptr_t>(lr) & 15) == 0) {
    const float4* l4 = reinterpret_cast<const float4*>(lr);
    for (int i = threadIdx.x; i < (V >> 2); i += RT_ROWS) {
      const float4 x = l4[i];
      const int v = 4 * i;
      const uint32_t f0 = flo(m, x.x), f1 = flo(m, x.y), f2 = flo(m, x.z), f3 = flo(m, x.w);
      s_all += f0 + f1 + f2 + f3;
      s_lt += (v < sym ? f0 : 0u) + (v + 1 < sym ? f1 : 0u) + (v + 2 < sym ? f2 : 0u) + (v + 3 < sym ? f3 : 0u);
    }
  } else {
    for (int v = threadIdx.x; v < V; v += RT_ROWS) {
      const uint32_t f = flo(m, lr[v]);
      s_all += f;
      s_lt += v < sym ? f : 0u;
    }
  }
  s_all = rows_block_sum(s_all, red);
  s_lt = rows_block_sum(s_lt, red);
  if (threadIdx.x == 0) {
    const uint32_t D = R - s_all;
    const uint64_t cs = (uint64_t)sym + s_lt + (top < sym ? D : 0u);
    const uint64_t fs = 1ull + flo(m, lr[sym]) + (sym == top ? D : 0u);
    a.rowcf[(size_t)c * a.kcap + j] = (cs << 32) | fs;
  }
}

// Encoder, per window (one thread): code the window's selected symbols in ascending position.
__global__ void enc_seq_kernel(CodeArgs a, int n_chunks) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= n_chunks) return;
  const int n = a.sel_count[c];
  CoderState t = a.state_c[c];
  uint8_t* ebuf = a.bytes + (size_t)c * a.cap_bytes;
  for (int j = 0; j < n; ++j) {
    const int pos = a.sel_pos[(size_t)c * a.kcap + j];
    const uint64_t cf = a.rowcf[(size_t)c * a.kcap + j];
    const uint64_t cs = cf >> 32, fs = cf & 0xFFFFFFFFull;
    if (a.coder == 1) {  // buffered; coded in reverse when the window is finished
      if (t.n_units < (uint32_t)a.pair_cap) a.pairs[(size_t)c * a.pair_cap + t.n_units] = (cs << 32) | fs;
      else atomicOr(a.err, ERR_CAPACITY);
      t.n_units++;
    } else {
      enc_symbol(t, ebuf, a.cap_bytes / 2, a.P, cs, fs, a.err);
    }
    a.state[(size_t)c * a.L + pos] = a.symbols[(size_t)c * a.L + pos];
  }
  a.state_c[c] = t;
  if (a.committed) a.committed[c] = n;
}

// Decoder, per selected row: the row's coarse CDF (prefix sums of 1 + floor(w R / W) at the starts
// of its segments of CODE_SEG elements, without D), D and K = floor(R 2^64 / W).
__global__ void __launch_bounds__(RT_ROWS) dec_rows_kernel(CodeArgs a) {
  __shared__ uint32_t T[256];
  __shared__ uint32_t tabf[QW0 + 1];
  __shared__ uint32_t wtot[RT_ROWS / 32];
  const int c = blockIdx.y, j = blockIdx.x;
  if (j >= a.sel_count[c]) return;
  for (int i = threadIdx.x; i < 256; i += RT_ROWS) T[i] = c_exp_table_c[i];
  const int pos = a.sel_pos[(size_t)c * a.kcap + j];
  const size_t row = selected_row(a, c, j, pos);
  const int V = a.V, nseg = a.nseg;
  const float* lr = a.logits + row * V;
  const float m = a.mx[row];
  const uint64_t Wr = a.W[row];
  const uint32_t R = (1u << a.P) - (uint32_t)V;
  const size_t cj = (size_t)c * a.kcap + j;
  uint32_t* cum = a.segcum + cj * (nseg + 1);
  __syncthreads();
  const RowFloor flo = row_floor(tabf, T, R, Wr, V);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool vec = (V & 3) == 0 && (reinterpret_cast<uintptr_t>(lr) & 15) == 0;
  // segment sums, one warp per segment (coalesced)
  for (int sg = warp; sg < nseg; sg += RT_ROWS / 32) {
    const int base = sg * CODE_SEG;
    uint32_t sum = 0;
    if (vec) {
      const float4* l4 = reinterpret_cast<const float4*>(lr + base);
#pragma unroll
      for (int i = 0; i < CODE_SEG / 128; ++i) {
        const int e = 4 * (lane + 32 * i);
        if (base + e < V) {  // V % 4 == 0: the float4 is wholly in the row
          const float4 x = l4[lane + 32 * i];
          sum += 4u + flo(m, x.x) + flo(m, x.y) + flo(m, x.z) + flo(m, x.w);
        }
      }
    } else {
      for (int e = lane; e < CODE_SEG; e += 32)
        if (base + e < V) sum += 1u + flo(m, lr[base + e]);
    }
    sum = __reduce_add_sync(0xffffffffu, sum);
    if (lane == 0) cum[sg] = sum;
  }
  __syncthreads();  // the segment sums are visible to the block
  // exclusive prefix over the segments, RT_ROWS at a time
  uint32_t carry = 0;
  for (int s0 = 0; s0 < nseg; s0 += RT_ROWS) {
    const int sg = s0 + threadIdx.x;
    const uint32_t v = sg < nseg ? cum[sg] : 0u;
    uint32_t inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t t = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += t;
    }
    if (lane == 31) wtot[warp] = inc;
    __syncthreads();
    const uint32_t tv = lane < RT_ROWS / 32 ? wtot[lane] : 0u;
    const uint32_t pre = carry + __reduce_add_sync(0xffffffffu, lane < warp ? tv : 0u) + inc - v;
    carry += __reduce_add_sync(0xffffffffu, tv);
    if (sg < nseg) cum[sg] = pre;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    cum[nseg] = carry;                      // V + sum_v floor(w_v R / W)
    a.rowD[cj] = (1u << a.P) - carry;       // = R - sum_v floor(w_v R / W)
    a.rowK[cj] = flo.table ? recip_scaled(R, Wr) : flo.K;
  }
}

// Decoder, one warp per window: for each selected row in ascending position, the slot from the
// coder state, the segment holding it (a search over the coarse CDF), the symbol inside that
// segment (a warp scan of its frequencies), then the coder update.
constexpr int DEC_WARPS = 4;
__global__ void __launch_bounds__(32 * DEC_WARPS) dec_seq_kernel(CodeArgs a, int n_chunks) {
  __shared__ uint32_t T[256];
  for (int i = threadIdx.x; i < 256; i += blockDim.x) T[i] = c_exp_table_c[i];
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int c = blockIdx.x * DEC_WARPS + (threadIdx.x >> 5);
  if (c >= n_chunks) return;  // warp-uniform
  const int n = a.sel_count[c], V = a.V, P = a.P, nseg = a.nseg;
  const uint32_t R = (1u << P) - (uint32_t)V;
  const uint8_t* dbuf = a.in_bytes + (a.in_offsets ? a.in_offsets[c] : 0);
  const uint64_t dn = (a.in_bits[c] + 7) / 8;
  CoderState st = a.state_c[c];  // every lane keeps a copy; lane 0's updates are broadcast
  for (int j = 0; j < n; ++j) {
    const int pos = a.sel_pos[(size_t)c * a.kcap + j];
    const size_t row = selected_row(a, c, j, pos);
    const size_t cj = (size_t)c * a.kcap + j;
    const float* lr = a.logits + row * V;
    const float m = a.mx[row];
    const uint64_t Wr = a.W[row], K = a.rowK[cj];
    const uint32_t D = a.rowD[cj];
    const int top = a.top[row];
    const uint32_t* cum = a.segcum + cj * (nseg + 1);
    uint64_t slot;
    if (a.coder == 1) {
      slot = st.low & ((1ull << P) - 1);  // x mod 2^P
    } else {
      slot = st.low / (st.rng >> P);     // the decoder keeps val = code - low in .low
      if (slot >= (1ull << P)) {
        if (lane == 0) atomicOr(a.err, ERR_CORRUPT);
        slot = (1ull << P) - 1;
      }
    }
    // CDF at the start of segment s: cum[s] + D when the top element lies before it
    auto start = [&](int sg) -> uint64_t { return (uint64_t)cum[sg] + ((int64_t)sg * CODE_SEG > top ? D : 0u); };
    int lo = 0, hi = nseg;  // start(lo) <= slot; the answer is in [lo, hi)
    while (hi - lo > 1) {
      const int step = (hi - lo + 31) / 32;
      const int sg = lo + lane * step;
      const bool le = sg < hi && start(sg) <= slot;
      const unsigned b = __ballot_sync(0xffffffffu, le);
      const int l = 31 - __clz(b);  // lane 0 always qualifies (start(lo) <= slot)
      lo = lo + l * step;
      hi = min(hi, lo + step);
    }
    // the symbol inside segment lo
    const int base = lo * CODE_SEG;
    uint64_t cb = start(lo);
    int sym = -1;
    uint64_t cs = 0, fs = 1;
    for (int e0 = 0; e0 < CODE_SEG && sym < 0; e0 += 32) {
      const int v = base + e0 + lane;
      uint32_t f = 0;
      if (v < V) {
        const uint32_t q = code_index(__fsub_rn(m, lr[v]));
        f = 1u + (q < (uint32_t)QW0 ? floor_wr_over_w(quant_w(T, (int)q), R, Wr, K) : 0u) + (v == top ? D : 0u);
      }
      uint32_t inc = f;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += t;
      }
      const unsigned hit = __ballot_sync(0xffffffffu, v < V && cb + inc > slot);
      if (hit) {
        const int l = __ffs(hit) - 1;
        const uint32_t incl = __shfl_sync(0xffffffffu, inc, l), fl = __shfl_sync(0xffffffffu, f, l);
        sym = base + e0 + l;
        cs = cb + incl - fl;
        fs = fl;
      }
      cb += __shfl_sync(0xffffffffu, inc, 31);
    }
    if (sym < 0) {  // only for a damaged stream: the slot lies beyond the row's total
      if (lane == 0) atomicOr(a.err, ERR_CORRUPT);
      sym = 0;
      cs = 0;
      fs = 1;
    }
    if (a.coder == 1) {
      st.low = fs * (st.low >> P) + slot - cs;
      if (st.low < RANS_L) {
        st.low = (st.low << 32) | word_at(dbuf, dn, 8 + 4ull * st.n_units);
        st.n_units++;
      }
    } else {
      const uint64_t r = st.rng >> P;
      st.low -= r * cs;
      st.rng = r * fs;
      while (st.rng < RENORM) {
        st.low = (st.low << 16) | unit_at(dbuf, dn, st.n_units++);
        st.rng <<= 16;
      }
    }
    if (lane == 0) a.state[(size_t)c * a.L + pos] = sym;
  }
  if (lane == 0) {
    a.state_c[c] = st;
    if (a.committed) a.committed[c] = n;
  }
}

int code_step(const CodeArgs& a, bool decode, int n_chunks, cudaStream_t s) {
  if (n_chunks == 0) return DLMZ_OK;
  ProfScope prof(PROF_CODE, s, 0, 0);
  const bool rows = a.coder != 2 && a.kcap > 0 && a.kcap <= 65535 && (decode ? (a.segcum && a.rowK && a.rowD) : a.rowcf != nullptr);
  if (!rows) {  // symbol ranks: one CTA per window does everything
    if (decode) code_kernel<true><<<n_chunks, CT, 0, s>>>(a);
    else code_kernel<false><<<n_chunks, CT, 0, s>>>(a);
    return launch_status();
  }
  const dim3 grid((unsigned)a.kcap, (unsigned)n_chunks);
  if (n_chunks > 65535) return DLMZ_EINVAL;
  if (!decode) {
    enc_rows_kernel<<<grid, RT_ROWS, 0, s>>>(a);
    DLMZ_TRY(launch_status());
    enc_seq_kernel<<<(n_chunks + 127) / 128, 128, 0, s>>>(a, n_chunks);
  } else {
    dec_rows_kernel<<<grid, RT_ROWS, 0, s>>>(a);
    DLMZ_TRY(launch_status());
    dec_seq_kernel<<<(n_chunks + DEC_WARPS - 1) / DEC_WARPS, 32 * DEC_WARPS, 0, s>>>(a, n_chunks);
  }
  return launch_status();
}

__global__ void coder_reset_kernel(CoderState* st, int n) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c < n) {
    st[c].low = 0;
    st[c].rng = ~0ull;
    st[c].n_units = 0;
  }
}

__global__ void coder_load_kernel(CoderState* st, int n, const uint8_t* bytes, const uint64_t* offsets,
                                  const uint32_t* bits, int coder) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= n) return;
  const uint8_t* b = bytes + (offsets ? offsets[c] : 0);
  const uint64_t nb = (bits[c] + 7) / 8;
  uint64_t v = 0;
  if (coder == 1) {  // the final state of the encoder leads the stream
    v = (word_at(b, nb, 0) << 32) | word_at(b, nb, 4);
    st[c].n_units = 0;
  } else if (coder == 2) {  // ranks: read from byte 0
    st[c].n_units = 0;
  } else {
    for (int i = 0; i < 4; ++i) v = (v << 16) | unit_at(b, nb, i);
    st[c].n_units = 4;
  }
  st[c].low = v;
  st[c].rng = ~0ull;
}

// rANS: code window c's buffered pairs in reverse.  Words go down from the end
// of the window's buffer; the state goes below them; the stream is then moved
// to the front of the buffer.
__global__ void rans_finish_kernel(CoderState* st, int n, const uint64_t* pairs, int pair_cap, int P, uint8_t* bytes,
                                   uint64_t cap_bytes, uint32_t* bits_out, uint8_t* out, const uint64_t* offsets,
                                   int* err) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= n) return;
  uint8_t* buf = bytes + (size_t)c * cap_bytes;
  const uint32_t np = st[c].n_units < (uint32_t)pair_cap ? st[c].n_units : (uint32_t)pair_cap;
  const uint64_t* pr = pairs + (size_t)c * pair_cap;
  uint64_t x = RANS_L, pos = cap_bytes & ~3ull;  // next word ends at pos
  bool ok = true;
  for (int i = (int)np - 1; i >= 0; --i) {
    const uint64_t cs = pr[i] >> 32, fs = pr[i] & 0xFFFFFFFFull;
    if (x >= ((RANS_L >> P) << 32) * fs) {
      if (pos >= 12) {  // room for this word and the 8-byte state
        pos -= 4;
        for (int b = 0; b < 4; ++b) buf[pos + b] = (uint8_t)(x >> (8 * (3 - b)));
      } else {
        ok = false;
      }
      x >>= 32;
    }
    x = ((x / fs) << P) + (x % fs) + cs;
  }
  if (!ok) {
    atomicOr(err, ERR_CAPACITY);
    bits_out[c] = 0;
    return;
  }
  const uint64_t words = ((cap_bytes & ~3ull) - pos) / 4;
  pos -= 8;
  for (int b = 0; b < 8; ++b) buf[pos + b] = (uint8_t)(x >> (8 * (7 - b)));
  const uint64_t nbytes = 8 + 4 * words;
  for (uint64_t i = 0; i < nbytes; ++i) buf[i] = buf[pos + i];  // front of the buffer (pos >= 0, ascending copy)
  bits_out[c] = (uint32_t)(8 * nbytes);
  if (out) {
    uint8_t* dst = out + (offsets ? offsets[c] : (uint64_t)c * cap_bytes);
    for (uint64_t i = 0; i < nbytes; ++i) dst[i] = buf[i];
  }
}

// Minimal termination: shortest t with a multiple of 2^(64-t) in [low, low+rng).
__global__ void coder_finish_kernel(CoderState* st, int n, uint8_t* bytes, uint64_t cap_bytes, uint32_t* bits_out,
                                    uint8_t* out, const uint64_t* offsets, int* err) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= n) return;
  CoderState t = st[c];
  uint8_t* buf = bytes + (size_t)c * cap_bytes;
  const unsigned __int128 low = t.low;
  const unsigned __int128 hi = low + t.rng - 1;
  unsigned __int128 v = 0;
  int tb = 0;
  for (tb = 0; tb <= 64; ++tb) {
    const unsigned __int128 g = (unsigned __int128)1 << (64 - tb);
    v = (low + g - 1) / g * g;
    if (v <= hi) break;
  }
  if (v >> 64) {  // carry into the emitted units
    int i = (int)t.n_units - 1;
    for (; i >= 0; --i) {
      const uint32_t u = (unit_at(buf, cap_bytes, i) + 1) & 0xFFFFu;
      put_unit(buf, i, u);
      if (u) break;
    }
    if (i < 0) atomicOr(err, ERR_CORRUPT);
  }
  const uint64_t v64 = (uint64_t)v;
  const uint32_t nb = (tb + 7) / 8;
  const uint64_t tail = tb ? (v64 >> (64 - tb)) << (8 * nb - tb) : 0;
  const uint64_t base = 2ull * t.n_units;
  if (base + nb > cap_bytes) {
    atomicOr(err, ERR_CAPACITY);
  } else {
    for (uint32_t i = 0; i < nb; ++i) buf[base + i] = (uint8_t)(tail >> (8 * (nb - 1 - i)));
  }
  const uint64_t total_bits = 16ull * t.n_units + tb;
  bits_out[c] = (uint32_t)total_bits;
  if (out && base + nb <= cap_bytes) {  // copy out: at offsets[c], or at c * cap_bytes
    const uint64_t nbytes = (total_bits + 7) / 8;
    uint8_t* dst = out + (offsets ? offsets[c] : (uint64_t)c * cap_bytes);
    for (uint64_t i = 0; i < nbytes; ++i) dst[i] = buf[i];
  }
}

int coder_reset(CoderState* st, int n, cudaStream_t s) {
  if (!n) return DLMZ_OK;
  coder_reset_kernel<<<(n + 255) / 256, 256, 0, s>>>(st, n);
  return launch_status();
}
int coder_load(CoderState* st, int n, const uint8_t* bytes, const uint64_t* offsets, const uint32_t* bits, int coder,
               cudaStream_t s) {
  if (!n) return DLMZ_OK;
  coder_load_kernel<<<(n + 255) / 256, 256, 0, s>>>(st, n, bytes, offsets, bits, coder);
  return launch_status();
}

// Ranks: the varint stream is complete as written; report its length and copy it out.
__global__ void ranks_finish_kernel(const CoderState* st, int n, const uint8_t* bytes, uint64_t cap_bytes,
                                    uint32_t* bits_out, uint8_t* out, const uint64_t* offsets, int* err) {
  const int c = blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= n) return;
  const uint64_t nbytes = st[c].n_units;
  if (nbytes > cap_bytes) {
    atomicOr(err, ERR_CAPACITY);
    bits_out[c] = 0;
    return;
  }
  bits_out[c] = (uint32_t)(8 * nbytes);
  if (out) {
    const uint8_t* buf = bytes + (size_t)c * cap_bytes;
    uint8_t* dst = out + (offsets ? offsets[c] : (uint64_t)c * cap_bytes);
    for (uint64_t i = 0; i < nbytes; ++i) dst[i] = buf[i];
  }
}
int coder_finish(CoderState* st, int n, uint8_t* bytes, uint64_t cap_bytes, uint32_t* bits, uint8_t* out,
                 const uint64_t* offsets, int coder, const uint64_t* pairs, int pair_cap, int P, cudaStream_t s) {
  if (!n) return DLMZ_OK;
  if (coder == 2)
    ranks_finish_kernel<<<(n + 127) / 128, 128, 0, s>>>(st, n, bytes, cap_bytes, bits, out, offsets,
                                                        device_error_word());
  else if (coder == 1)
    rans_finish_kernel<<<(n + 127) / 128, 128, 0, s>>>(st, n, pairs, pair_cap, P, bytes, cap_bytes, bits, out, offsets,
                                                       device_error_word());
  else
    coder_finish_kernel<<<(n + 127) / 128, 128, 0, s>>>(st, n, bytes, cap_bytes, bits, out, offsets,
                                                        device_error_word());
  return launch_status();
}

}  // namespace dlmz
