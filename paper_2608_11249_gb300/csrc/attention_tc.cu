// Bidirectional attention on the 5th-generation tensor cores (Definition 3:
// every position attends to every position of its window, no mask).
//
// Persistent CTAs (two per SM at head dim 64, one at 128) walk work items
// (128 queries, head, window); 6 warps:
//   warp 0      TMA: Q once per item (2-stage ring, so the next item's Q is
//               in flight during this item); per key tile of 128: K and V^T
//               (keys contiguous, written so by the QKV epilogue), each
//               through a 2-stage ring, K requested one tile ahead of V.
//   warp 1      allocates TMEM (S: 128 columns, P: 64, O: head_dim) and
//               issues S_j = Q K_j^T (A and B in shared memory) and
//               O += P_j V_j (A = P_j in TMEM) with tcgen05.mma from one thread.
//   warps 2-5   softmax, one thread per query row (its TMEM lane): the row of
//               S_j in one 128-column TMEM load, its max, P_j = 2^(S_j - m) by
//               ex2.approx.f16x2, stored back to TMEM as f16 pairs (the A
//               operand of P V), and the row sum l of those f16 values; the
//               running max is raised (and O and l rescaled) only when it grows
//               by more than 8 (log2 units), so P <= 2^8; finally O / l -> bf16,
//               deferred into the next item's first tile so the next S is
//               taken (and the MMA warp goes on) before the last P V is waited for.
// At head dim 128 the item's output is drained from TMEM in 32-column chunks
// after P has been handed over (the 128 S registers and O never coexist).
// GQA: query head h reads KV head h / (n_heads / n_kv_heads).  Requires the
// window length to be a multiple of 128.  All waits are bounded.
#include "kernels.cuh"
#include "tcgen05.cuh"

namespace dlmz {
namespace fat {

constexpr int BQ = 128, BK = 128;
constexpr int THREADS = 192;
constexpr float RESCALE_THRESHOLD = 8.0f;

// TMEM columns: S [0, 128), P [128, 192) (f16 pairs), O from O_COL (a multiple of head_dim).
template <int HD>
struct Tmem {
  static constexpr int O_COL = HD == 64 ? 192 : 256;
  static constexpr int COLS = HD == 64 ? 256 : 512;
  static constexpr int CTAS_PER_SM = HD == 64 ? 2 : 1;
};

template <int HD>
struct Smem {
  static_assert(HD == 64 || HD == 128, "Q / K rows of one or two 128-byte swizzle blocks");
  static constexpr int QT = BQ * HD * 2;             // one query tile: HD / 64 blocks of [128 x 64] bf16
  static constexpr int Q = 0;                        // 2 query tiles
  static constexpr int KT = BK * HD * 2;             // one key tile: HD / 64 blocks of [128 x 64] bf16
  static constexpr int K = Q + 2 * QT;               // 2 key tiles
  static constexpr int VTT = HD * BK * 2;            // one V^T tile: 2 blocks of [HD x 64] f16 (keys 0-63, 64-127)
  static constexpr int VT = K + 2 * KT;              // 2 V^T tiles
  static constexpr int BARS = VT + 2 * VTT;
  static constexpr int TOTAL = BARS + 256 + 1024;    // + barriers + alignment slack
};

__device__ __forceinline__ uint32_t hadd2(uint32_t a, uint32_t b) {
  uint32_t y;
  asm("add.rn.f16x2 %0, %1, %2;" : "=r"(y) : "r"(a), "r"(b));
  return y;
}
// Row sum of 128 f16 values held as 64 pairs: a pairwise f16x2 tree (every
// partial sum <= 128 * 2^8 stays finite in f16), the last two lanes in f32.
__device__ __forceinline__ float row_sum_f16x2(const uint32_t* p) {
  uint32_t t[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) t[i] = hadd2(p[i], p[i + 32]);
#pragma unroll
  for (int w = 16; w >= 1; w >>= 1)
#pragma unroll
    for (int i = 0; i < w; ++i) t[i] = hadd2(t[i], t[i + w]);
  const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&t[0]));
  return f.x + f.y;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
  float y;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(y) : "f"(a), "f"(b), "f"(c));
  return y;
}
// (x0, x1) * (a0, a1) + (b0, b1) in one packed f32x2 FMA; each lane rounds as fmaf.
__device__ __forceinline__ void fma2(float& y0, float& y1, float x0, float x1, float a0, float a1, float b0, float b1) {
  uint64_t x, a, b, y;
  asm("mov.b64 %0, {%1, %2};" : "=l"(x) : "f"(x0), "f"(x1));
  asm("mov.b64 %0, {%1, %2};" : "=l"(a) : "f"(a0), "f"(a1));
  asm("mov.b64 %0, {%1, %2};" : "=l"(b) : "f"(b0), "f"(b1));
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(y) : "l"(x), "l"(a), "l"(b));
  asm("mov.b64 {%0, %1}, %2;" : "=f"(y0), "=f"(y1) : "l"(y));
}

// N values of one query row of an item's output: O / l -> bf16, from 16-byte stores.
template <int N>
__device__ __forceinline__ void write_row(bf16* __restrict__ dst, const uint32_t* o, float l) {
  const float inv = 1.0f / l;
  uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int t = 0; t < N / 8; ++t) {
    uint32_t u[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      __nv_bfloat162 p2 = __floats2bfloat162_rn(__uint_as_float(o[8 * t + 2 * e]) * inv,
                                                __uint_as_float(o[8 * t + 2 * e + 1]) * inv);
      u[e] = *reinterpret_cast<uint32_t*>(&p2);
    }
    d4[t] = make_uint4(u[0], u[1], u[2], u[3]);
  }
}

// This thread's output row of the item (TMEM lane) drained from O in chunks of 32
// columns (head dim 128: the S registers are dead here, so the chunks stay small).
template <int HD>
__device__ __forceinline__ void drain_row(uint32_t tO_lane, bf16* __restrict__ dst, float l) {
#pragma unroll 1
  for (int c = 0; c < HD / 32; ++c) {
    float v[32];
    t5::tmem_ld32(tO_lane + c * 32, v);
    write_row<32>(dst + c * 32, reinterpret_cast<const uint32_t*>(v), l);
  }
}

template <int HD>
__global__ void __launch_bounds__(THREADS, Tmem<HD>::CTAS_PER_SM)  // head dim 64: two CTAs per SM, <= 168 registers
    fa_tc_kernel(const __grid_constant__ CUtensorMap tmQK, const __grid_constant__ CUtensorMap tmVt, int n_chunks,
                 int L, int nh, int nkv, int d, bf16* __restrict__ out, float scale_log2, int* err) {
  using S = Smem<HD>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  const uint32_t base = (smem_u32(smem_raw) + 1023) & ~1023u;
  const uint32_t sQ = base + S::Q, sK = base + S::K, sVt = base + S::VT;
  const uint32_t bar = base + S::BARS;
  const uint32_t s_full = bar + 80, s_free = bar + 88, p_ready = bar + 96, o_done = bar + 104, o_free = bar + 112;
  auto q_full = [&](int st) { return bar + 128 + 8 * st; };  // per query stage
  auto q_empty = [&](int st) { return bar + 144 + 8 * st; };
  auto k_full = [&](int st) { return bar + 16 + 8 * st; };   // per key stage
  auto k_empty = [&](int st) { return bar + 32 + 8 * st; };
  auto v_full = [&](int st) { return bar + 48 + 8 * st; };   // per V^T stage
  auto v_empty = [&](int st) { return bar + 64 + 8 * st; };
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nt = L / BK, nqt = L / BQ;
  // work items (query tile, head, window), query tile fastest; this CTA takes
  // items blockIdx.x, blockIdx.x + gridDim.x, ...  Tiles are counted across
  // items (J), so every barrier's phase is a function of J or of the item count.
  const int items = n_chunks * nh * nqt;
  const int n_my = blockIdx.x < items ? (items - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
  const int total = n_my * nt;
  auto item_of = [&](int it, int& w, int& h, int& q0) {
    const int id = (int)blockIdx.x + it * (int)gridDim.x;
    q0 = (id % nqt) * BQ;
    h = (id / nqt) % nh;
    w = id / (nqt * nh);
  };

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int st = 0; st < 2; ++st) {
      mbar_init(q_full(st), 1);
      mbar_init(q_empty(st), 1);
      mbar_init(k_full(st), 1);
      mbar_init(k_empty(st), 1);
      mbar_init(v_full(st), 1);
      mbar_init(v_empty(st), 1);
    }
    mbar_init(s_full, 1);
    mbar_init(s_free, 4 * 32);
    mbar_init(p_ready, 4 * 32);
    mbar_init(o_done, 1);
    mbar_init(o_free, 4 * 32);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) t5::tmem_alloc(smem_u32(&tmem_slot), Tmem<HD>::COLS);
  t5::fence_before();
  __syncthreads();
  t5::fence_after();
  const uint32_t tmem = tmem_slot;
  const uint32_t tS = tmem, tP = tmem + BK, tO = tmem + Tmem<HD>::O_COL;

  if (warp == 0) {
    if (lane == 0) {
      uint32_t kpend = 0, vpend = 0, kpar = 0, vpar = 0;  // per stage (bit): copy issued, its phase
      uint32_t qpend = 0, qpar = 0;
      // per global tile J: (item's Q when J starts an item), K_J, then V_{J-1}
      for (int J = 0; J <= total && !abort_flag; ++J) {
        if (J < total) {
          const int it = J / nt, j = J % nt;
          int w, h, q0;
          item_of(it, w, h, q0);
          const int g = h / (nh / nkv);
          if (j == 0) {  // item it - 2's last QK^T has read this Q stage
            const int qs = it & 1;
            const uint32_t qph = (it >> 1) & 1;
            if (!mbar_wait_bounded(q_empty(qs), qph ^ 1, &abort_flag, err)) break;
            mbar_arrive_expect_tx(q_full(qs), BQ * HD * 2);
            for (int kb = 0; kb < HD / 64; ++kb)
              t5::tma_load_2d(sQ + qs * S::QT + kb * BQ * 128, &tmQK, h * HD + kb * 64, w * L + q0, q_full(qs));
            qpend |= 1u << qs;
            qpar = (qpar & ~(1u << qs)) | (qph << qs);
          }
          const int st = J & 1;
          const uint32_t ph = (J >> 1) & 1;
          if (!mbar_wait_bounded(k_empty(st), ph ^ 1, &abort_flag, err)) break;
          mbar_arrive_expect_tx(k_full(st), BK * HD * 2);
          for (int kb = 0; kb < HD / 64; ++kb)
            t5::tma_load_2d(sK + st * S::KT + kb * BK * 128, &tmQK, d + g * HD + kb * 64, w * L + j * BK, k_full(st));
          kpend |= 1u << st;
          kpar = (kpar & ~(1u << st)) | (ph << st);
        }
        if (J >= 1) {
          const int Jv = J - 1, it = Jv / nt, j = Jv % nt;
          int w, h, q0;
          item_of(it, w, h, q0);
          const int g = h / (nh / nkv);
          const int st = Jv & 1;
          const uint32_t ph = (Jv >> 1) & 1;
          if (!mbar_wait_bounded(v_empty(st), ph ^ 1, &abort_flag, err)) break;
          mbar_arrive_expect_tx(v_full(st), BK * HD * 2);
          for (int kk = 0; kk < 2; ++kk)
            t5::tma_load_2d(sVt + st * S::VTT + kk * HD * 128, &tmVt, j * BK + kk * 64, (w * nkv + g) * HD,
                            v_full(st));
          vpend |= 1u << st;
          vpar = (vpar & ~(1u << st)) | (ph << st);
        }
      }
      if (abort_flag) {  // let our own copies land before the CTA can exit
        volatile int never = 0;
        for (int st = 0; st < 2; ++st) {
          if (qpend & (1u << st)) mbar_wait_bounded(q_full(st), (qpar >> st) & 1, &never, err, 100000000ull);
          if (kpend & (1u << st)) mbar_wait_bounded(k_full(st), (kpar >> st) & 1, &never, err, 100000000ull);
          if (vpend & (1u << st)) mbar_wait_bounded(v_full(st), (vpar >> st) & 1, &never, err, 100000000ull);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t ID_S = t5::idesc_bf16(BQ, BK);
      constexpr uint32_t ID_O = t5::idesc_f16(BQ, HD);
      bool issued = false;
      // descriptors of the operand stages (the K = 16 steps add 32 bytes to the start address)
      const uint64_t dQ0 = t5::sw128_desc(sQ), dK0 = t5::sw128_desc(sK), dV0 = t5::sw128_desc(sVt);
      constexpr uint64_t QT16 = S::QT >> 4, KT16 = S::KT >> 4, VT16 = S::VTT >> 4;
      // S_J = Q K_J^T (it = J / nt, j = J % nt); the first tile of an item waits for that item's Q,
      // the last one releases Q to the next item's load
      auto issue_s = [&](int J, int it, int j) -> bool {
        const int st = J & 1, qs = it & 1;
        if (j == 0 && !mbar_wait_bounded(q_full(qs), (it >> 1) & 1, &abort_flag, err)) return false;
        if (!mbar_wait_bounded(k_full(st), (J >> 1) & 1, &abort_flag, err)) return false;
        t5::fence_after();
        const uint64_t dq = dQ0 + (uint64_t)qs * QT16, dk = dK0 + (uint64_t)st * KT16;
#pragma unroll
        for (int kb = 0; kb < HD / 64; ++kb)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            t5::mma_bf16(tS, dq + (uint64_t)((kb * BQ * 128 + 32 * k) >> 4), dk + (uint64_t)((kb * BK * 128 + 32 * k) >> 4),
                         ID_S, (kb | k) != 0);
        t5::commit(s_full);
        t5::commit(k_empty(st));
        if (j == nt - 1) t5::commit(q_empty(qs));
        issued = true;
        return true;
      };
      bool ok = total == 0 || issue_s(0, 0, 0);
      int it = 0, j = 0;  // J = it * nt + j
      for (int J = 0; ok && J < total; ++J) {
        const int st = J & 1;
        const int it1 = j + 1 == nt ? it + 1 : it, j1 = j + 1 == nt ? 0 : j + 1;  // of J + 1
        // S_{J+1} goes as soon as the softmax has S_J in registers, so it runs under P_J's exponentials
        // (across items too: the next item's first QK^T overlaps this item's last softmax and epilogue)
        if (J + 1 < total) {
          if (!mbar_wait_bounded(s_free, J & 1, &abort_flag, err)) break;
          if (!issue_s(J + 1, it1, j1)) break;
        }
        if (!mbar_wait_bounded(p_ready, J & 1, &abort_flag, err)) break;
        if (!mbar_wait_bounded(v_full(st), (J >> 1) & 1, &abort_flag, err)) break;
        // the first PV of an item overwrites O: the softmax warps must have read the previous item's O
        if (j == 0 && it > 0 && !mbar_wait_bounded(o_free, (it - 1) & 1, &abort_flag, err)) break;
        t5::fence_after();
        // 8 steps of 16 keys: P_j columns 8k..8k+7, V^T block k / 4 at byte offset 32 (k % 4)
        const uint64_t dv = dV0 + (uint64_t)st * VT16;
#pragma unroll
        for (int k = 0; k < BK / 16; ++k)
          t5::mma_tmem_a(tO, tP + 8 * k, dv + (uint64_t)(((k >> 2) * HD * 128 + 32 * (k & 3)) >> 4), ID_O,
                         (j | k) != 0);
        t5::commit(v_empty(st));
        t5::commit(o_done);
        it = it1;
        j = j1;
      }
      if (abort_flag && issued) {
        volatile int never = 0;
        const uint32_t drain = bar + 120;
        mbar_init(drain, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        t5::commit(drain);
        mbar_wait_bounded(drain, 0, &never, err, 100000000ull);
      }
    }
  } else {
    const int q = warp & 3;
    const int r = q * 32 + lane;  // query row within the tile (= TMEM lane)
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    auto row_of = [&](int it) {  // this thread's output row of item `it`
      int w, h, q0;
      item_of(it, w, h, q0);
      return out + ((size_t)w * L + q0 + r) * d + (size_t)h * HD;
    };
    float m = -INFINITY, l = 0.0f;
    // An item's epilogue is deferred into the next item's first tile: that tile's S is loaded
    // (so the MMA warp can go on) and exponentiated first; O is read where the P store has to
    // wait for the last P V anyway, and written out after P_J is handed over.
    bool pend = false;
    float l_pend = 0.0f;
    for (int J = 0; J < total; ++J) {
      const int j = J % nt;
      // waits are made warp-uniform: tcgen05.ld/st below are warp-collective
      if (!__all_sync(0xffffffffu, mbar_wait_bounded(s_full, J & 1, &abort_flag, err))) break;
      t5::fence_after();
      uint32_t sr[BK];
      t5::tmem_ld128(tS + lane_off, sr);
      t5::fence_before();
      mbar_arrive(s_free);  // S_J is in registers: the MMA warp may overwrite it with S_{J+1}
      float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};  // 4 independent chains
#pragma unroll
      for (int i = 0; i < BK / 2; ++i)
        m4[i & 3] = max3(m4[i & 3], __uint_as_float(sr[2 * i]), __uint_as_float(sr[2 * i + 1]));
      float mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
      mx *= scale_log2;
      // the running max first (P needs only m); P_J is computed in registers while PV_{J-1} may still run
      float f = 1.0f;
      bool need = false;
      if (j == 0) {  // a new item: fresh running max and row sum
        m = mx;
        l = 0.0f;
      } else if (mx > m + RESCALE_THRESHOLD) {
        need = true;
        f = t5::ex2(m - mx);
        m = mx;
      }
      // P = 2^(s * scale - m) as f16 pairs (in place of S): pair c holds keys 2c, 2c + 1
#pragma unroll
      for (int c = 0; c < BK / 2; ++c) {
        float x0, x1;
        fma2(x0, x1, __uint_as_float(sr[2 * c]), __uint_as_float(sr[2 * c + 1]), scale_log2, scale_log2, -m, -m);
        sr[c] = t5::ex2_f16x2(t5::pack_f16x2(x0, x1));
      }
      l = l * f + row_sum_f16x2(sr);
      bool p_stored = false;
      if (j > 0 || pend) {
        // PV_{J-1} done: P's columns free, O stable (at an item's first tile: the previous item's O is final)
        if (!__all_sync(0xffffffffu, mbar_wait_bounded(o_done, (J - 1) & 1, &abort_flag, err))) break;
        t5::fence_after();
        if (j == 0) {
          if constexpr (HD == 64) {
            uint32_t o[HD];
            t5::tmem_ld64(tO + lane_off, o);
            t5::tmem_st64(tP + lane_off, sr);
            t5::fence_before();
            mbar_arrive(o_free);  // O is in registers: this item's first PV may overwrite it
            mbar_arrive(p_ready);
            write_row<HD>(row_of(J / nt - 1), o, l_pend);  // the previous item's output, off the MMA warp's path
          } else {
            // P first (the MMA warp still waits for o_free before this item's first PV), then O in chunks
            t5::tmem_st64(tP + lane_off, sr);
            t5::fence_before();
            mbar_arrive(p_ready);
            drain_row<HD>(tO + lane_off, row_of(J / nt - 1), l_pend);
            t5::fence_before();
            mbar_arrive(o_free);
          }
          p_stored = true;
          pend = false;
        } else if (__any_sync(0xffffffffu, need)) {  // the whole warp rescales its O rows (f = 1 where not needed)
#pragma unroll 1
          for (int c = 0; c < HD / 16; ++c) {
            uint32_t oc[16];
            t5::tmem_ld16(tO + lane_off + c * 16, oc);
#pragma unroll
            for (int i = 0; i < 16; ++i) oc[i] = __float_as_uint(__uint_as_float(oc[i]) * f);
            t5::tmem_st16(tO + lane_off + c * 16, oc);
          }
        }
      }
      if (!p_stored) {
        t5::tmem_st64(tP + lane_off, sr);
        t5::fence_before();
        mbar_arrive(p_ready);
      }
      if (j == nt - 1) {
        pend = true;
        l_pend = l;
      }
    }
    if (pend && !abort_flag) {  // the last item's epilogue
      if (__all_sync(0xffffffffu, mbar_wait_bounded(o_done, (total - 1) & 1, &abort_flag, err))) {
        t5::fence_after();
        drain_row<HD>(tO + lane_off, row_of((total - 1) / nt), l_pend);
        t5::fence_before();
      }
    }
  }
  t5::fence_before();
  __syncthreads();
  if (warp == 1) {
    t5::fence_after();
    t5::tmem_dealloc(tmem, Tmem<HD>::COLS);
  }
}

}  // namespace fat

// ---- two query tiles per CTA --------------------------------------------------------------
// Persistent, one CTA per SM, work items (256 queries = query tiles A and B, head, window):
// each K and V^T tile brought into shared memory serves both query tiles, so the bytes
// moved from L2 per tensor-core FLOP are half those of one query tile per CTA.  10 warps:
//   warp 0      TMA: per key tile K_j then V^T_{j-1} (2-stage rings), Q_A and Q_B once per
//               item (each released as soon as the item's last S of that tile is issued).
//   warp 1      allocates all 512 TMEM columns -- S_A [0,128), S_B [128,256),
//               O_A [256, 256+HD), O_B [256+HD, 256+2HD); P_X is written over the first 64
//               columns of S_X -- and issues, per key tile j,
//                  PV_A(j), S_A(j+1), PV_B(j), S_B(j+1)
//               so each softmax group works on its tile while the tensor core runs the
//               other tile's two products.  The tcgen05.mma operations of one thread run
//               in issue order, so S_X(j+1) overwrites P_X(j) only after PV_X(j) has read
//               it, and the commit after S_X(j+1) also covers PV_X(j): a softmax group that
//               sees S_X(j+1) may rescale or read O_X.
//   warps 2-5   softmax of query tile A (one thread per row, as in fat::fa_tc_kernel);
//   warps 6-9   the same for query tile B.
// An item's output (O_X / l) is written at the next item's first tile of X, before the
// first P V of that item overwrites O_X.  Requires the window length to be a multiple of
// 256; used at head dim 128.  All waits are bounded.
namespace fa2 {

constexpr int BQ = 128, BK = 128;
constexpr int THREADS = 320;
constexpr float RESCALE_THRESHOLD = 8.0f;

template <int HD>
struct Smem {
  static_assert(HD == 64 || HD == 128, "Q / K rows of one or two 128-byte swizzle blocks");
  static constexpr int QT = BQ * HD * 2;   // one query tile
  static constexpr int Q = 0;              // Q_A, Q_B
  static constexpr int KT = BK * HD * 2;   // one key tile
  static constexpr int K = Q + 2 * QT;     // 2 key stages
  static constexpr int VTT = HD * BK * 2;  // one V^T tile (f16)
  static constexpr int VT = K + 2 * KT;    // 2 V^T stages
  static constexpr int BARS = VT + 2 * VTT;
  // + barriers + alignment slack; at least 116 KB so that one CTA holds an SM (it takes all of TMEM)
  static constexpr int TOTAL = BARS + 256 + 1024 > 116 * 1024 ? BARS + 256 + 1024 : 116 * 1024;
};

template <int HD>
__global__ void __launch_bounds__(THREADS, 1)
    fa2_kernel(const __grid_constant__ CUtensorMap tmQK, const __grid_constant__ CUtensorMap tmVt, int n_chunks,
               int L, int nh, int nkv, int d, bf16* __restrict__ out, float scale_log2, int* err) {
  using S = Smem<HD>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;
  const uint32_t base = (smem_u32(smem_raw) + 1023) & ~1023u;
  const uint32_t sQ = base + S::Q, sK = base + S::K, sVt = base + S::VT;
  const uint32_t bar = base + S::BARS;
  auto k_full = [&](int st) { return bar + 8 * st; };
  auto k_empty = [&](int st) { return bar + 16 + 8 * st; };
  auto v_full = [&](int st) { return bar + 32 + 8 * st; };
  auto v_empty = [&](int st) { return bar + 48 + 8 * st; };
  auto q_full = [&](int x) { return bar + 64 + 8 * x; };
  auto q_empty = [&](int x) { return bar + 80 + 8 * x; };
  auto s_full = [&](int x) { return bar + 96 + 8 * x; };
  auto p_ready = [&](int x) { return bar + 112 + 8 * x; };
  auto o_free = [&](int x) { return bar + 128 + 8 * x; };
  auto fin = [&](int x) { return bar + 144 + 8 * x; };
  const uint32_t drain_bar = bar + 160;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nt = L / BK, npair = L / (2 * BQ);
  const int items = n_chunks * nh * npair;
  const int n_my = blockIdx.x < items ? (items - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
  const int total = n_my * nt;
  auto item_of = [&](int it, int& w, int& h, int& q0) {  // q0: first query of tile A
    const int id = (int)blockIdx.x + it * (int)gridDim.x;
    q0 = (id % npair) * 2 * BQ;
    h = (id / npair) % nh;
    w = id / (npair * nh);
  };

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int x = 0; x < 2; ++x) {
      mbar_init(k_full(x), 1);
      mbar_init(k_empty(x), 1);
      mbar_init(v_full(x), 1);
      mbar_init(v_empty(x), 1);
      mbar_init(q_full(x), 1);
      mbar_init(q_empty(x), 1);
      mbar_init(s_full(x), 1);
      mbar_init(p_ready(x), 4 * 32);
      mbar_init(o_free(x), 4 * 32);
      mbar_init(fin(x), 1);
    }
    mbar_init(drain_bar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) t5::tmem_alloc(smem_u32(&tmem_slot), 512);
  t5::fence_before();
  __syncthreads();
  t5::fence_after();
  const uint32_t tmem = tmem_slot;
  auto tS = [&](int x) { return tmem + x * BK; };
  auto tO = [&](int x) { return tmem + 2 * BK + x * HD; };

  if (warp == 0) {
    if (lane == 0) {
      uint32_t kpend = 0, vpend = 0, kpar = 0, vpar = 0, qpend = 0, qpar = 0;
      for (int J = 0; J <= total && !abort_flag; ++J) {
        if (J < total) {
          const int it = J / nt, j = J % nt;
          int w, h, q0;
          item_of(it, w, h, q0);
          const int g = h / (nh / nkv);
          const int st = J & 1;
          const uint32_t ph = (J >> 1) & 1;
          if (!mbar_wait_bounded(k_empty(st), ph ^ 1, &abort_flag, err)) break;
          mbar_arrive_expect_tx(k_full(st), BK * HD * 2);
          for (int kb = 0; kb < HD / 64; ++kb)
            t5::tma_load_2d(sK + st * S::KT + kb * BK * 128, &tmQK, d + g * HD + kb * 64, w * L + j * BK, k_full(st));
          kpend |= 1u << st;
          kpar = (kpar & ~(1u << st)) | (ph << st);
        }
        if (J >= 1) {  // V^T_{J-1}: the P V products of tile J-1 come before the S products of tile J
          const int Jv = J - 1, it = Jv / nt, j = Jv % nt;
          int w, h, q0;
          item_of(it, w, h, q0);
          const int g = h / (nh / nkv);
          const int st = Jv & 1;
          const uint32_t ph = (Jv >> 1) & 1;
          if (!mbar_wait_bounded(v_empty(st), ph ^ 1, &abort_flag, err)) break;
          mbar_arrive_expect_tx(v_full(st), BK * HD * 2);
          for (int kk = 0; kk < 2; ++kk)
            t5::tma_load_2d(sVt + st * S::VTT + kk * HD * 128, &tmVt, j * BK + kk * 64, (w * nkv + g) * HD,
                            v_full(st));
          vpend |= 1u << st;
          vpar = (vpar & ~(1u << st)) | (ph << st);
        }
        if (J < total && J % nt == 0) {  // the item's query tiles, each once the previous item's last S_X is issued
          const int it = J / nt;
          int w, h, q0;
          item_of(it, w, h, q0);
          const uint32_t ph = it & 1;
          bool ok = true;
          for (int x = 0; x < 2 && ok; ++x) {
            if (!mbar_wait_bounded(q_empty(x), ph ^ 1, &abort_flag, err)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(q_full(x), BQ * HD * 2);
            for (int kb = 0; kb < HD / 64; ++kb)
              t5::tma_load_2d(sQ + x * S::QT + kb * BQ * 128, &tmQK, h * HD + kb * 64, w * L + q0 + x * BQ, q_full(x));
            qpend |= 1u << x;
            qpar = (qpar & ~(1u << x)) | (ph << x);
          }
          if (!ok) break;
        }
      }
      if (abort_flag) {  // let our own copies land before the CTA can exit
        volatile int never = 0;
        for (int st = 0; st < 2; ++st) {
          if (qpend & (1u << st)) mbar_wait_bounded(q_full(st), (qpar >> st) & 1, &never, err, 100000000ull);
          if (kpend & (1u << st)) mbar_wait_bounded(k_full(st), (kpar >> st) & 1, &never, err, 100000000ull);
          if (vpend & (1u << st)) mbar_wait_bounded(v_full(st), (vpar >> st) & 1, &never, err, 100000000ull);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t ID_S = t5::idesc_bf16(BQ, BK);
      constexpr uint32_t ID_O = t5::idesc_f16(BQ, HD);
      bool issued = false;
      // descriptors of the operand stages (the K = 16 steps add 32 bytes to the start address)
      const uint64_t dQ0 = t5::sw128_desc(sQ), dK0 = t5::sw128_desc(sK), dV0 = t5::sw128_desc(sVt);
      constexpr uint64_t QT16 = S::QT >> 4, KT16 = S::KT >> 4, VT16 = S::VTT >> 4;
      // S_X(J) = Q_X K_J^T (it = J / nt, j = J % nt); tile A waits for K_J (and, at an item's first
      // tile, each tile for its Q)
      auto issue_s = [&](int x, int J, int it, int j) -> bool {
        const int st = J & 1;
        if (j == 0 && !mbar_wait_bounded(q_full(x), it & 1, &abort_flag, err)) return false;
        if (x == 0 && !mbar_wait_bounded(k_full(st), (J >> 1) & 1, &abort_flag, err)) return false;
        t5::fence_after();
        const uint64_t dq = dQ0 + (uint64_t)x * QT16, dk = dK0 + (uint64_t)st * KT16;
#pragma unroll
        for (int kb = 0; kb < HD / 64; ++kb)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            t5::mma_bf16(tS(x), dq + (uint64_t)((kb * BQ * 128 + 32 * k) >> 4), dk + (uint64_t)((kb * BK * 128 + 32 * k) >> 4),
                         ID_S, (kb | k) != 0);
        t5::commit(s_full(x));
        if (x == 1) t5::commit(k_empty(st));
        if (j == nt - 1) t5::commit(q_empty(x));
        issued = true;
        return true;
      };
      // O_X (+)= P_X(J) V_J, P_X in the first 64 columns of S_X (8 columns per 16 keys)
      auto issue_pv = [&](int x, int J, int it, int j) -> bool {
        const int st = J & 1;
        if (!mbar_wait_bounded(p_ready(x), J & 1, &abort_flag, err)) return false;
        if (x == 0 && !mbar_wait_bounded(v_full(st), (J >> 1) & 1, &abort_flag, err)) return false;
        // the first P V of an item overwrites O_X: the softmax group must have read the previous item's O_X
        if (j == 0 && it > 0 && !mbar_wait_bounded(o_free(x), (it - 1) & 1, &abort_flag, err)) return false;
        t5::fence_after();
        const uint64_t dv = dV0 + (uint64_t)st * VT16;
#pragma unroll
        for (int k = 0; k < BK / 16; ++k)
          t5::mma_tmem_a(tO(x), tS(x) + 8 * k, dv + (uint64_t)(((k >> 2) * HD * 128 + 32 * (k & 3)) >> 4), ID_O,
                         (j | k) != 0);
        if (x == 1) t5::commit(v_empty(st));
        if (J == total - 1) t5::commit(fin(x));
        return true;
      };
      bool ok = total == 0 || (issue_s(0, 0, 0, 0) && issue_s(1, 0, 0, 0));
      int it = 0, j = 0;  // J = it * nt + j
      for (int J = 0; ok && J < total; ++J) {
        const int it1 = j + 1 == nt ? it + 1 : it, j1 = j + 1 == nt ? 0 : j + 1;  // of J + 1
        if (!issue_pv(0, J, it, j)) break;
        if (J + 1 < total && !issue_s(0, J + 1, it1, j1)) break;
        if (!issue_pv(1, J, it, j)) break;
        if (J + 1 < total && !issue_s(1, J + 1, it1, j1)) break;
        it = it1;
        j = j1;
      }
      if (abort_flag && issued) {
        volatile int never = 0;
        t5::commit(drain_bar);
        mbar_wait_bounded(drain_bar, 0, &never, err, 100000000ull);
      }
    }
  } else {
    const int x = (warp - 2) >> 2;  // query tile of this softmax group
    const int q = warp & 3;         // TMEM lane quadrant of this warp
    const int r = q * 32 + lane;    // query row within the tile (= TMEM lane)
    const uint32_t lane_off = (uint32_t)(q * 32) << 16;
    const uint32_t tSx = tS(x) + lane_off, tOx = tO(x) + lane_off;
    auto row_of = [&](int it) {
      int w, h, q0;
      item_of(it, w, h, q0);
      return out + ((size_t)w * L + q0 + x * BQ + r) * d + (size_t)h * HD;
    };
    float m = -INFINITY, l = 0.0f, l_pend = 0.0f;
    bool pend = false;
    for (int J = 0; J < total; ++J) {
      const int j = J % nt;
      if (!__all_sync(0xffffffffu, mbar_wait_bounded(s_full(x), J & 1, &abort_flag, err))) break;
      t5::fence_after();
      uint32_t sr[BK];
      t5::tmem_ld128(tSx, sr);
      float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
      for (int i = 0; i < BK / 2; ++i)
        m4[i & 3] = fat::max3(m4[i & 3], __uint_as_float(sr[2 * i]), __uint_as_float(sr[2 * i + 1]));
      float mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
      mx *= scale_log2;
      float f = 1.0f;
      bool need = false;
      if (j == 0) {
        m = mx;
        l = 0.0f;
      } else if (mx > m + RESCALE_THRESHOLD) {
        need = true;
        f = t5::ex2(m - mx);
        m = mx;
      }
#pragma unroll
      for (int c = 0; c < BK / 2; ++c) {
        float x0, x1;
        fat::fma2(x0, x1, __uint_as_float(sr[2 * c]), __uint_as_float(sr[2 * c + 1]), scale_log2, scale_log2, -m, -m);
        sr[c] = t5::ex2_f16x2(t5::pack_f16x2(x0, x1));
      }
      l = l * f + fat::row_sum_f16x2(sr);
      // S_X(J) complete means every earlier product is too: O_X holds the sum through tile J - 1
      if (j == 0 && pend) {  // the previous item's output, before this item's first P V overwrites O_X
        fat::drain_row<HD>(tOx, row_of(J / nt - 1), l_pend);
        t5::fence_before();
        mbar_arrive(o_free(x));
        pend = false;
      } else if (j > 0 && __any_sync(0xffffffffu, need)) {  // the whole warp rescales its O rows (f = 1 elsewhere)
#pragma unroll 1
        for (int c = 0; c < HD / 16; ++c) {
          uint32_t oc[16];
          t5::tmem_ld16(tOx + c * 16, oc);
#pragma unroll
          for (int i = 0; i < 16; ++i) oc[i] = __float_as_uint(__uint_as_float(oc[i]) * f);
          t5::tmem_st16(tOx + c * 16, oc);
        }
      }
      t5::tmem_st64(tSx, sr);  // P_X(J) over the first 64 columns of S_X
      t5::fence_before();
      mbar_arrive(p_ready(x));
      if (j == nt - 1) {
        pend = true;
        l_pend = l;
      }
    }
    if (pend && !abort_flag) {  // the last item's output
      if (__all_sync(0xffffffffu, mbar_wait_bounded(fin(x), 0, &abort_flag, err))) {
        t5::fence_after();
        fat::drain_row<HD>(tOx, row_of((total - 1) / nt), l_pend);
        t5::fence_before();
      }
    }
  }
  t5::fence_before();
  __syncthreads();
  if (warp == 1) {
    t5::fence_after();
    t5::tmem_dealloc(tmem, 512);
  }
}

}  // namespace fa2

bool attention_tc_supported(int L, int hd) { return L > 0 && L % fat::BK == 0 && (hd == 64 || hd == 128); }

int attention_vt_rows(int hd) { return hd; }

// V^T (f16, [window][kv head][hd][L]) from the V columns of [Q | K | V] rows,
// through a 32 x 32 shared-memory tile so reads and writes are both coalesced.
__global__ void vt_from_rows_kernel(const bf16* __restrict__ qkv, int ld, int v_col, int L, int nkv, int hd, int wg0,
                                    __half* __restrict__ vt) {
  __shared__ float t[32][33];
  const int wg = wg0 + (int)blockIdx.z, w = wg / nkv, g = wg % nkv;
  const int p0 = blockIdx.x * 32, d0 = blockIdx.y * 32;
  for (int i = threadIdx.y; i < 32; i += blockDim.y) {
    const int p = p0 + i, dim = d0 + threadIdx.x;
    t[i][threadIdx.x] =
        p < L && dim < hd ? __bfloat162float(qkv[(size_t)(w * L + p) * ld + v_col + g * hd + dim]) : 0.0f;
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += blockDim.y) {
    const int dim = d0 + i, p = p0 + threadIdx.x;
    if (p < L && dim < hd) vt[((size_t)wg * hd + dim) * L + p] = __float2half(t[threadIdx.x][i]);
  }
}

int attention_vt_from_rows(const bf16* qkv, int ld, int v_col, int n_chunks, int L, int nkv, int hd, void* vt,
                           cudaStream_t s) {
  const int blocks = n_chunks * nkv;
  for (int wg0 = 0; wg0 < blocks; wg0 += 65535) {
    const int nz = blocks - wg0 < 65535 ? blocks - wg0 : 65535;
    vt_from_rows_kernel<<<dim3((L + 31) / 32, (hd + 31) / 32, nz), dim3(32, 8), 0, s>>>(
        qkv, ld, v_col, L, nkv, hd, wg0, reinterpret_cast<__half*>(vt));
    DLMZ_TRY(launch_status());
  }
  return DLMZ_OK;
}

int attention_bf16_tc(const bf16* qkv, int ld, const void* vt, int n_chunks, int L, int nh, int nkv, int hd, int d,
                      bf16* out, cudaStream_t s) {
  if (n_chunks == 0) return DLMZ_OK;
  if (!attention_tc_supported(L, hd) || (ld % 8) || (reinterpret_cast<uintptr_t>(qkv) & 15) ||
      (reinterpret_cast<uintptr_t>(vt) & 15))
    return DLMZ_EINVAL;
  CUtensorMap mqk, mvt;
  DLMZ_TRY(t5::make_map_bf16(&mqk, qkv, (uint64_t)n_chunks * L, ld, ld, 128, 64));
  DLMZ_TRY(t5::make_map_f16(&mvt, vt, (uint64_t)n_chunks * nkv * hd, L, L, hd, 64));
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)hd);
  // persistent: two CTAs (head dim 64) or one (128) per SM walk the work items
  const int64_t items = (int64_t)n_chunks * nh * (L / fat::BQ);
  if (items > 0x7fffffff) return DLMZ_EINVAL;
  ProfScope prof(PROF_ATTN, s, 4.0 * n_chunks * nh * (double)L * L * hd, 2.0 * n_chunks * L * (double)(ld + d));
  if (hd == 128 && L % (2 * fa2::BQ) == 0) {
    // two query tiles per CTA, one CTA per SM (at head dim 64 the one-tile kernel, two CTAs per SM,
    // measured faster: 38.9 against 39.2 ms per byte-model forward over 1024 windows of 512)
    const int64_t items2 = items / 2;
    const int grid = items2 < num_sms() ? (int)items2 : num_sms();
    constexpr int SM = fa2::Smem<128>::TOTAL;
    static PerDeviceOnce attr;
    DLMZ_TRY(attr.run(
        [] { return cudaFuncSetAttribute(fa2::fa2_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, SM); }));
    fa2::fa2_kernel<128><<<grid, fa2::THREADS, SM, s>>>(mqk, mvt, n_chunks, L, nh, nkv, d, out, scale_log2,
                                                       device_error_word());
  } else if (hd == 64) {
    constexpr int SM = fat::Smem<64>::TOTAL;
    static PerDeviceOnce attr;
    DLMZ_TRY(attr.run(
        [] { return cudaFuncSetAttribute(fat::fa_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, SM); }));
    const int cap = fat::Tmem<64>::CTAS_PER_SM * num_sms();
    const int grid = items < cap ? (int)items : cap;
    fat::fa_tc_kernel<64><<<grid, fat::THREADS, SM, s>>>(mqk, mvt, n_chunks, L, nh, nkv, d, out, scale_log2,
                                                        device_error_word());
  } else {
    constexpr int SM = fat::Smem<128>::TOTAL;
    static PerDeviceOnce attr;
    DLMZ_TRY(attr.run(
        [] { return cudaFuncSetAttribute(fat::fa_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, SM); }));
    const int cap = fat::Tmem<128>::CTAS_PER_SM * num_sms();
    const int grid = items < cap ? (int)items : cap;
    fat::fa_tc_kernel<128><<<grid, fat::THREADS, SM, s>>>(mqk, mvt, n_chunks, L, nh, nkv, d, out, scale_log2,
                                                         device_error_word());
  }
  return launch_status();
}

}  // namespace dlmz
