// Dense bf16 GEMM on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
//   D[m, n] = sum_k A[m, k] * B[n, k]      A: [M x K] bf16, B: [N x K] bf16 (both K-major)
//
// This is every dense contraction of the masked-DLM forward (Definition 3):
// the fused QKV projection (with RoPE in the epilogue), the attention output
// projection and the FFN down projection (residual add into the float32
// stream), the gate/up projection (SwiGLU in the epilogue) and the LM head
// (float32 logits).
//
// Design (one CTA per SM, persistent over output tiles of 128 x 256 taken in
// grouped order: a group of G row blocks is swept column block by column
// block, so the G A-slices stay in L2 while B streams through it once per
// group; G is sized from K so the group's A fits in a fraction of L2):
//   warp 0      TMA producer: 128B-swizzled A/B K-slices (64 elements) into a
//               4-stage shared-memory ring, completion on mbarriers.
//   warp 1      allocates 512 TMEM columns (two 128x256 fp32 accumulators) and
//               issues tcgen05.mma (M=128, N=256, K=16) from one thread;
//               tcgen05.commit frees a ring slot / publishes an accumulator.
//   warps 2-9   epilogue, two warps per TMEM lane quadrant (one column half
//               each): tcgen05.ld 32 lanes x 32 columns (each thread owns one
//               output row), fused op, staged through shared memory so global
//               accesses are row-contiguous.
// Two accumulators let the epilogue of tile i overlap the MMAs of tile i+1.
// Every mbarrier wait is bounded; on timeout the CTA sets the error word,
// waits (bounded) for its own outstanding copies and MMAs, frees TMEM and
// returns.  Output values depend only on (m, n) and K (fixed K order, no
// split-K), so results are independent of M and of the batch composition.
#include "common.cuh"
#include "kernels.cuh"
#include "tcgen05.cuh"

namespace dlmz {
namespace tc {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;  // bf16 elements = 128 bytes = one swizzle row
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int BM_ALIGN_VT = 128;  // transposed V needs whole windows per 128-row tile
constexpr int THREADS = 320;  // TMA warp, MMA warp, 8 epilogue warps
constexpr int TMEM_COLS = 512;
constexpr int STG_BYTES = 8 * 32 * 128;  // epilogue staging, 8 warps x 32 x 32 float32
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + 256 + STG_BYTES;

constexpr uint32_t IDESC = t5::idesc_bf16(BM, BN);  // D f32, A/B bf16, both K-major

using t5::fence_after;
using t5::fence_before;
using t5::tmem_ld32;

// Epilogue staging: each epilogue warp owns a 32 x 32 float32 buffer; 16-byte
// chunks are XOR-swizzled by row so both the row-per-thread writes and the
// row-contiguous read-out are free of bank conflicts.
__device__ __forceinline__ uint32_t stg_off(int row, int chunk) {
  return (uint32_t)(row * 128 + ((chunk ^ (row & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack2_f16(float a, float b) {
  __half2 p = __floats2half2_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&p);
}

__device__ __forceinline__ uint32_t pack2_bf16(float a, float b) {
  __nv_bfloat162 p = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&p);
}

// The value a bfloat16 store of x would hold (V is kept in f16 for the
// attention kernel, after the same bf16 rounding as every stored tensor).
__device__ __forceinline__ float bf16_round(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

// silu(g) = g / (1 + e^-g): ex2-based exponential and reciprocal, a few ulp
// of float32 (the product is then stored in bf16).
__device__ __forceinline__ float silu_f32(float g) { return __fdividef(g, 1.0f + __expf(-g)); }

// Global data an epilogue chunk needs besides the accumulator (residual
// values or RoPE (cos, sin) pairs), loaded one chunk ahead to hide latency.
struct EpiAux {
  float4 x[8];
};

template <int EPI>
__device__ __forceinline__ void epi_load_aux(EpiAux& a, int c, int lane, int row0, int M, int n0,
                                             const GemmEpilogue& ep) {
  if constexpr (EPI == EPI_RESID_F32) {
    const int col0 = n0 + c * 32;
#pragma unroll
    for (int it = 0; it < 8; ++it) {
      const int r = it * 4 + (lane >> 3), m = row0 + r;
      a.x[it] = m < M ? *reinterpret_cast<const float4*>(reinterpret_cast<const float*>(ep.out) + (size_t)m * ep.ldo +
                                                         col0 + (lane & 7) * 4)
                      : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  } else if constexpr (EPI == EPI_ROPE_BF16) {  // this lane's (cos, sin) pairs: 4 rows x 4 rotation pairs
    const int col = n0 + c * 32 + 8 * (lane & 3);
    if (col < ep.rope_cols) {
      const int half = ep.head_dim >> 1;
      const int t0 = (col % ep.head_dim) >> 1;
#pragma unroll
      for (int it = 0; it < 4; ++it) {
        const int m = row0 + it * 8 + (lane >> 2);
        const float4* cs = reinterpret_cast<const float4*>(ep.rope_cs + (size_t)((m < M ? m : 0) % ep.L) * half + t0);
        a.x[2 * it] = cs[0];
        a.x[2 * it + 1] = cs[1];
      }
    }
  }
}

// Drain one accumulator tile.  Epilogue warp e (0..7) reads TMEM lane quadrant
// q = warp % 4 (tile rows [32q, 32q+32)) and the column half e / 4.  Per
// 32-column chunk: tcgen05.ld (thread = row), optional SwiGLU, stage, then
// row-contiguous global accesses (8 lanes x 16 B per float32 row segment, 4
// lanes x 16 B per bf16 row segment) with the residual add, RoPE rotation or
// bf16 conversion.
// Fused RMSNorm, consumer side: sum of the row's partial sums of x^2 (the
// caller loads it one tile ahead so the loads overlap the previous tile).
__device__ __forceinline__ float row_ssq(const GemmEpilogue& ep, int m, int M) {
  float ss = 0.f;
  if (ep.ssq_in && m < M)
    for (int i = 0; i < ep.n_part; ++i) ss += ep.ssq_in[(size_t)m * ep.n_part + i];
  return ss;
}

template <int EPI>
__device__ __forceinline__ void epilogue_tile(uint32_t tacc, int q, int half, int lane, int m0, int M, int n0,
                                              const GemmEpilogue& ep, uint8_t* stg, float row_ss) {
  const uint32_t tbase = tacc + ((uint32_t)(q * 32) << 16);
  const int row0 = m0 + q * 32;
  constexpr int NCH = (EPI == EPI_SWIGLU_BF16 ? BN / 64 : BN / 32) / 2;  // chunks per column half
  const int c0 = half * NCH;
  // fused RMSNorm, consumer side: this thread's accumulator row is scaled by rsqrt(mean x^2 + eps)
  float rs = 1.0f;
  if constexpr (EPI == EPI_ROPE_BF16 || EPI == EPI_SWIGLU_BF16) {
    if (ep.ssq_in) rs = rsqrtf(row_ss / (float)ep.d_model + ep.eps);
  }
  // fused RMSNorm, producer side: sums of x^2 of the rows this lane stores
  float rowsum[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  // float32 epilogue: this thread's row maximum (NaN-propagating) and minimum over its 128 columns
  float pmx = -INFINITY, pmn = INFINITY;
  EpiAux cur, nxt;
  if constexpr (EPI == EPI_RESID_F32) epi_load_aux<EPI>(cur, c0, lane, row0, M, n0, ep);
  // RoPE: a warp takes every other chunk (c = half, half + 2, ...), so with head_dim 64 all its
  // chunks rotate the same pairs and the (cos, sin) table is loaded once per tile
  int rope_t = -1;
#pragma unroll 1
  for (int ci = 0; ci < NCH; ++ci) {
    const int c = EPI == EPI_ROPE_BF16 ? half + 2 * ci : c0 + ci;
    if constexpr (EPI == EPI_RESID_F32) {
      if (ci + 1 < NCH) epi_load_aux<EPI>(nxt, c + 1, lane, row0, M, n0, ep);
    } else if constexpr (EPI == EPI_ROPE_BF16) {
      const int t = (n0 + c * 32) % ep.head_dim;
      if (t != rope_t && n0 + c * 32 < ep.rope_cols) {
        epi_load_aux<EPI>(cur, c, lane, row0, M, n0, ep);
        rope_t = t;
      }
    }
    float v[32];
    tmem_ld32(tbase + c * 32, v);
    if constexpr (EPI == EPI_F32) {
      if (ep.pmax) {
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
          asm("max.NaN.f32 %0, %1, %2, %3;" : "=f"(pmx) : "f"(pmx), "f"(v[i]), "f"(v[i + 1]));
          asm("min.f32 %0, %1, %2, %3;" : "=f"(pmn) : "f"(pmn), "f"(v[i]), "f"(v[i + 1]));
        }
      }
    }
    if constexpr (EPI == EPI_SWIGLU_BF16) {  // columns [0,128) gate, [128,256) up of the same features
      float u[32];
      tmem_ld32(tbase + BN / 2 + c * 32, u);
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = silu_f32(rs * v[i]) * (rs * u[i]);
    } else if constexpr (EPI == EPI_ROPE_BF16) {
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] *= rs;
    }
    const int col0 = (EPI == EPI_SWIGLU_BF16 ? n0 / 2 : n0) + c * 32;
    // V heads of the QKV projection are staged transposed ([dim][token], a
    // thread writes its token down a column, each dim row rotated by
    // 4 * (dim mod 8) floats so both the 4-byte writes and the 16-byte reads of
    // token runs are free of bank conflicts); everything else is staged
    // [token][dim] with 16-byte chunks swizzled by row.
    const bool vt_chunk = EPI == EPI_ROPE_BF16 && ep.vt && col0 >= ep.v_col0;
    if (vt_chunk) {
#pragma unroll
      for (int j = 0; j < 32; ++j) reinterpret_cast<float*>(stg)[j * 32 + ((lane + 4 * (j & 7)) & 31)] = v[j];
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j)
        *reinterpret_cast<float4*>(stg + stg_off(lane, j)) = make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
    }
    __syncwarp();
    if constexpr (EPI == EPI_F32 || EPI == EPI_RESID_F32) {
#pragma unroll
      for (int it = 0; it < 8; ++it) {
        const int r = it * 4 + (lane >> 3), ch = lane & 7;
        const int m = row0 + r;
        float4 val = *reinterpret_cast<const float4*>(stg + stg_off(r, ch));
        if constexpr (EPI == EPI_RESID_F32) {
          val.x += cur.x[it].x;
          val.y += cur.x[it].y;
          val.z += cur.x[it].z;
          val.w += cur.x[it].w;
          if (ep.y_out) {  // warp-uniform: shuffles below
            float sq = val.x * val.x + val.y * val.y + val.z * val.z + val.w * val.w;
            sq += __shfl_xor_sync(0xffffffffu, sq, 1);
            sq += __shfl_xor_sync(0xffffffffu, sq, 2);
            sq += __shfl_xor_sync(0xffffffffu, sq, 4);
            rowsum[it] += sq;
            if (m < M)
              *reinterpret_cast<uint2*>(ep.y_out + (size_t)m * ep.ldo + col0 + ch * 4) =
                  make_uint2(pack2_bf16(val.x, val.y), pack2_bf16(val.z, val.w));
          }
        }
        if (m < M)
          *reinterpret_cast<float4*>(reinterpret_cast<float*>(ep.out) + (size_t)m * ep.ldo + col0 + ch * 4) = val;
      }
    } else if (vt_chunk) {
      // V heads, transposed and f16: vt[window][kv head][vt_rows][pos]; 32 positions of a dim are contiguous
      const int win = row0 / ep.L, pos0 = row0 % ep.L;
      const int vi = col0 - ep.v_col0, gh = vi / ep.head_dim, dim0 = vi % ep.head_dim;
      __half* vb = reinterpret_cast<__half*>(ep.vt) + ((size_t)(win * ep.n_kv + gh) * ep.vt_rows + dim0) * ep.L + pos0;
#pragma unroll
      for (int it = 0; it < 4; ++it) {
        const int j = it * 8 + (lane >> 2), p0 = 8 * (lane & 3);
        const float4 a = *reinterpret_cast<const float4*>(stg + (j * 32 + ((p0 + 4 * (j & 7)) & 31)) * 4);
        const float4 b = *reinterpret_cast<const float4*>(stg + (j * 32 + ((p0 + 4 + 4 * (j & 7)) & 31)) * 4);
        const float w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
        float r[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) r[e] = bf16_round(w[e]);
        *reinterpret_cast<uint4*>(vb + (size_t)j * ep.L + p0) =
            make_uint4(pack2_f16(r[0], r[1]), pack2_f16(r[2], r[3]), pack2_f16(r[4], r[5]), pack2_f16(r[6], r[7]));
      }
    } else {
#pragma unroll
      for (int it = 0; it < 4; ++it) {
        const int r = it * 8 + (lane >> 2), qd = lane & 3;
        const int m = row0 + r;
        const float4 a = *reinterpret_cast<const float4*>(stg + stg_off(r, 2 * qd));
        const float4 b = *reinterpret_cast<const float4*>(stg + stg_off(r, 2 * qd + 1));
        float w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
        const int col = col0 + 8 * qd;
        if constexpr (EPI == EPI_ROPE_BF16) {
          if (col < ep.rope_cols) {  // head dims stored as rotation pairs (2t, 2t+1)
            const float4 c01 = cur.x[2 * it], c23 = cur.x[2 * it + 1];
            const float cr[4] = {c01.x, c01.z, c23.x, c23.z}, sr[4] = {c01.y, c01.w, c23.y, c23.w};
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              const float x0 = w[2 * t], x1 = w[2 * t + 1];
              w[2 * t] = x0 * cr[t] - x1 * sr[t];
              w[2 * t + 1] = x1 * cr[t] + x0 * sr[t];
            }
          }
        }
        if (m < M)
          *reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(ep.out) + (size_t)m * ep.ldo + col) =
              make_uint4(pack2_bf16(w[0], w[1]), pack2_bf16(w[2], w[3]), pack2_bf16(w[4], w[5]), pack2_bf16(w[6], w[7]));
      }
    }
    __syncwarp();
    if constexpr (EPI == EPI_RESID_F32) cur = nxt;
  }
  if constexpr (EPI == EPI_F32) {
    const int m = row0 + lane;
    if (ep.pmax && m < M) {  // this thread's row; part = 128-column block of the output
      const int n_part = ep.n_part, part = n0 / 128 + half;
      ep.pmax[(size_t)m * n_part + part] = pmx;
      ep.pmin[(size_t)m * n_part + part] = pmn;
    }
  }
  if constexpr (EPI == EPI_RESID_F32) {
    if (ep.ssq_out && (lane & 7) == 0) {
      const int part = n0 / 128 + half;
#pragma unroll
      for (int it = 0; it < 8; ++it) {
        const int m = row0 + it * 4 + (lane >> 3);
        if (m < M) ep.ssq_out[(size_t)m * ep.n_part + part] = rowsum[it];
      }
    }
  }
}

// Tile t of the grouped order: groups of `group` row blocks, column blocks in
// order inside a group, row blocks fastest (the last group may be shorter).
__device__ __forceinline__ void grouped_tile(int t, int m_tiles, int n_tiles, int group, int& m0, int& n0) {
  const int per_group = group * n_tiles;
  const int g = t / per_group, r = t % per_group;
  const int gm0 = g * group;
  const int gs = m_tiles - gm0 < group ? m_tiles - gm0 : group;
  m0 = (gm0 + r % gs) * BM;
  n0 = (r / gs) * BN;
}

template <int EPI>
__global__ void __launch_bounds__(THREADS, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                int M, int N, int K, int group, GemmEpilogue ep, int* err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * A_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint8_t* stg_all = smem + STAGES * STAGE_BYTES + 256;
  // bars: full[STAGES], empty[STAGES], tfull[2], tempty[2], drain
  __shared__ uint32_t tmem_slot;
  __shared__ volatile int abort_flag;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t full0 = smem_u32(bars);
  const uint32_t empty0 = full0 + 8 * STAGES;
  const uint32_t tfull0 = empty0 + 8 * STAGES;
  const uint32_t tempty0 = tfull0 + 16;
  const uint32_t drain = tempty0 + 16;

  if (threadIdx.x == 0) {
    abort_flag = 0;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull0 + 8 * a, 1);
      mbar_init(tempty0 + 8 * a, 8 * 32);
    }
    mbar_init(drain, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_slot)),
                 "r"(TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = tmem_slot;

  const int num_k = K / BK;
  const int n_tiles = N / BN;
  const int m_tiles = (M + BM - 1) / BM;
  const int total = m_tiles * n_tiles;
  const int cid = (int)blockIdx.x, n_ctas = (int)gridDim.x;
  auto tile_of = [&](int t, int& m0, int& n0) { grouped_tile(t, m_tiles, n_tiles, group, m0, n0); };

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued_mask = 0, issued_phase = 0;  // per stage: issued at least once / its last phase
      for (int tile = cid; tile < total && !abort_flag; tile += n_ctas) {
        int m0, n0;
        tile_of(tile, m0, n0);
        for (int kb = 0; kb < num_k; ++kb) {
          if (!mbar_wait_bounded(empty0 + 8 * stage, phase ^ 1, &abort_flag, err)) break;
          mbar_arrive_expect_tx(full0 + 8 * stage, STAGE_BYTES);  // rows past M read as zero, full byte count
          t5::tma_load_2d(smem_u32(sA + stage * A_BYTES), &tmA, kb * BK, m0, full0 + 8 * stage);
          t5::tma_load_2d(smem_u32(sB + stage * B_BYTES), &tmB, kb * BK, n0, full0 + 8 * stage);
          issued_mask |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (abort_flag) {  // drain our own copies before the CTA may exit
        volatile int never = 0;
        for (int s = 0; s < STAGES; ++s)
          if (issued_mask & (1u << s))
            mbar_wait_bounded(full0 + 8 * s, (issued_phase >> s) & 1, &never, err, 100000000ull);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool issued_any = false;
      // descriptors of the ring's stages (the K = 16 steps add 32 bytes to the start address)
      const uint64_t dA0 = t5::sw128_desc(smem_u32(sA)), dB0 = t5::sw128_desc(smem_u32(sB));
      for (int tile = cid; tile < total && !abort_flag; tile += n_ctas) {
        if (!mbar_wait_bounded(tempty0 + 8 * acc, acc_phase ^ 1, &abort_flag, err)) break;
        fence_after();
        const uint32_t d_tmem = tmem + acc * BN;
        bool ok = true;
        for (int kb = 0; kb < num_k; ++kb) {
          if (!mbar_wait_bounded(full0 + 8 * stage, phase, &abort_flag, err)) {
            ok = false;
            break;
          }
          fence_after();
          const uint64_t da = dA0 + (uint64_t)stage * (A_BYTES >> 4), db = dB0 + (uint64_t)stage * (B_BYTES >> 4);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            t5::mma_bf16(d_tmem, da + (uint64_t)(2 * k), db + (uint64_t)(2 * k), IDESC, (kb | k) != 0);
          issued_any = true;
          t5::commit(empty0 + 8 * stage);  // the stage is free once the products have read it
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        t5::commit(tfull0 + 8 * acc);
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1;
        }
      }
      if (abort_flag && issued_any) {  // wait for our MMAs before TMEM is freed
        volatile int never = 0;
        t5::commit(drain);
        mbar_wait_bounded(drain, 0, &never, err, 100000000ull);
      }
    }
  } else {
    const int q = warp & 3;  // TMEM lane quadrant this warp may access
    const int half = (warp - 2) >> 2;
    uint8_t* stg = stg_all + (warp - 2) * 32 * 128;
    int acc = 0;
    uint32_t acc_phase = 0;
    constexpr bool kScale = EPI == EPI_ROPE_BF16 || EPI == EPI_SWIGLU_BF16;
    float ss_next = 0.f;
    if (kScale && cid < total) {
      int m1, n1;
      tile_of(cid, m1, n1);
      ss_next = row_ssq(ep, m1 + q * 32 + lane, M);
    }
    for (int tile = cid; tile < total; tile += n_ctas) {
      const float ss_cur = ss_next;
      if (kScale && tile + n_ctas < total) {  // next tile's row, loaded while this tile drains
        int m1, n1;
        tile_of(tile + n_ctas, m1, n1);
        ss_next = row_ssq(ep, m1 + q * 32 + lane, M);
      }
      // warp-uniform outcome: the epilogue's tcgen05.ld is warp-collective
      if (!__all_sync(0xffffffffu, mbar_wait_bounded(tfull0 + 8 * acc, acc_phase, &abort_flag, err))) break;
      fence_after();
      int m0, n0;
      tile_of(tile, m0, n0);
      epilogue_tile<EPI>(tmem + acc * BN, q, half, lane, m0, M, n0, ep, stg, ss_cur);
      fence_before();
      mbar_arrive(tempty0 + 8 * acc);
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1;
      }
    }
  }
  fence_before();
  __syncthreads();
  if (warp == 1) {
    fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
  }
}

// ---- host side ------------------------------------------------------------

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

}  // namespace tc

static int make_map_2d(CUtensorMap* map, CUtensorMapDataType dt, const void* base, uint64_t rows, uint64_t cols,
                       uint64_t ld, uint32_t box_rows, uint32_t box_cols) {
  tc::EncodeTiledFn fn = tc::encode_fn();
  if (!fn) return DLMZ_ECUDA;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    fprintf(stderr, "dlmz: cuTensorMapEncodeTiled failed (%d)\n", (int)r);
    return DLMZ_ECUDA;
  }
  return DLMZ_OK;
}

int t5::make_map_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t ld,
                      uint32_t box_rows, uint32_t box_cols) {
  return make_map_2d(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, base, rows, cols, ld, box_rows, box_cols);
}

int t5::make_map_f16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint64_t ld,
                     uint32_t box_rows, uint32_t box_cols) {
  return make_map_2d(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, base, rows, cols, ld, box_rows, box_cols);
}

namespace tc {

// Row blocks per group of the tile order: the group's A slices (BM x K bf16
// each) take at most ~48 MB of the 129 MB L2, and at least one block.
static int group_for(int m_tiles, int K) {
  const long a_tile = (long)BM * K * 2;
  long g = (48l << 20) / a_tile;
  if (g < 1) g = 1;
  if (g > m_tiles) g = m_tiles;
  return (int)g;
}

template <int EPI>
static int launch(const CUtensorMap& a, const CUtensorMap& b, int M, int N, int K, const GemmEpilogue& ep,
                  cudaStream_t s) {
  static PerDeviceOnce attr;
  DLMZ_TRY(attr.run([] {
    return cudaFuncSetAttribute(gemm_kernel<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  }));
  // persistent: one CTA per SM (shared memory and all 512 TMEM columns) walks the tiles
  const int m_tiles = (M + BM - 1) / BM;
  const long tiles = (long)m_tiles * (N / BN);
  if (tiles > 0x7fffffffl) return DLMZ_EINVAL;
  const int grid = tiles < num_sms() ? (int)tiles : num_sms();
  const double out_b = EPI == EPI_F32 ? 4.0 * M * N : EPI == EPI_RESID_F32 ? 8.0 * M * N
                     : EPI == EPI_SWIGLU_BF16 ? 1.0 * M * N : 2.0 * M * N;
  ProfScope prof(PROF_GEMM_TC, s, 2.0 * M * N * K, 2.0 * M * K + 2.0 * N * K + out_b);
  gemm_kernel<EPI><<<grid, THREADS, SMEM_BYTES, s>>>(a, b, M, N, K, group_for(m_tiles, K), ep, device_error_word());
  return launch_status();
}

}  // namespace tc

bool gemm_tc_supported(int M, int N, int K) { return M > 0 && N % tc::BN == 0 && K % tc::BK == 0 && K > 0; }

int gemm_bf16_tc(const __nv_bfloat16* A, int lda, const __nv_bfloat16* B, int ldb, int M, int N, int K,
                 int epi, const GemmEpilogue& ep, cudaStream_t s) {
  if (!gemm_tc_supported(M, N, K)) return DLMZ_EINVAL;
  if ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(B)) & 15) return DLMZ_EINVAL;
  if ((lda | ldb) & 7) return DLMZ_EINVAL;
  CUtensorMap ma, mb;
  DLMZ_TRY(t5::make_map_bf16(&ma, A, M, K, lda, tc::BM, tc::BK));
  DLMZ_TRY(t5::make_map_bf16(&mb, B, N, K, ldb, tc::BN, tc::BK));
  switch (epi) {
    case EPI_BF16: return tc::launch<EPI_BF16>(ma, mb, M, N, K, ep, s);
    case EPI_F32: return tc::launch<EPI_F32>(ma, mb, M, N, K, ep, s);
    case EPI_RESID_F32: return tc::launch<EPI_RESID_F32>(ma, mb, M, N, K, ep, s);
    case EPI_SWIGLU_BF16: return tc::launch<EPI_SWIGLU_BF16>(ma, mb, M, N, K, ep, s);
    case EPI_ROPE_BF16:
      if (ep.head_dim % 8 || !ep.rope_cs || (reinterpret_cast<uintptr_t>(ep.rope_cs) & 15)) return DLMZ_EINVAL;
      if (ep.vt && (ep.L % tc::BM_ALIGN_VT || M % ep.L || ep.v_col0 % 32 || (reinterpret_cast<uintptr_t>(ep.vt) & 15)))
        return DLMZ_EINVAL;
      return tc::launch<EPI_ROPE_BF16>(ma, mb, M, N, K, ep, s);
  }
  return DLMZ_EINVAL;
}

}  // namespace dlmz
