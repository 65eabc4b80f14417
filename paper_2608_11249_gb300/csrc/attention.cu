// Bidirectional flash attention for bf16 windows (Definition 3: every masked
// position attends to every position of its window, no causal mask).
//
// CTA = (64 queries, head, window), 4 warps x 16 query rows.  Q stays in
// registers as mma A-fragments; K/V tiles of 64 keys stream through a
// double-buffered, XOR-swizzled shared-memory ring (cp.async); S = Q K^T and
// O += P V run on m16n8k16 bf16 tensor-core MMAs with float32 accumulators;
// the softmax is online (running max / sum per row) in float32, with P
// rounded to bf16 only as the MMA operand.  GQA: query head h reads KV head
// h / (n_heads / n_kv_heads).
#include "kernels.cuh"

namespace dlmz {
namespace fa {

constexpr int BMQ = 64;
constexpr int BNK = 64;

__device__ __forceinline__ uint32_t swz(int row, int chunk, int chunks_per_row) {
  return (uint32_t)(row * chunks_per_row + (chunk ^ (row & 7))) * 16u;
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int bytes = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(bytes) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ void ldm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&p);
}

// Load `rows` rows x HD bf16 (row stride ld) starting at window row r0 into a
// swizzled tile; rows >= L are zero-filled.
template <int HD>
__device__ __forceinline__ void load_tile(uint32_t sbase, const bf16* __restrict__ g, size_t ld, int r0, int L) {
  constexpr int CPR = HD / 8;  // 16-byte chunks per row
  for (int i = threadIdx.x; i < 64 * CPR; i += 128) {
    const int r = i / CPR, c = i % CPR;
    const bool ok = r0 + r < L;
    const bf16* src = g + (size_t)(ok ? r0 + r : 0) * ld + c * 8;
    cp_async16(sbase + swz(r, c, CPR), src, ok);
  }
}

template <int HD>
__global__ void __launch_bounds__(128) flash_kernel(const bf16* __restrict__ qkv, int ld, int L, int nh, int nkv,
                                                    int d, bf16* __restrict__ out, float scale_log2) {
  extern __shared__ __align__(128) uint8_t sm[];
  constexpr int CPR = HD / 8;
  constexpr int TILE = 64 * HD * 2;  // bytes per 64-row tile
  const uint32_t sQ = smem_u32(sm);
  const uint32_t sK = sQ + TILE;      // 2 buffers
  const uint32_t sV = sK + 2 * TILE;  // 2 buffers

  const int chunk = blockIdx.z, h = blockIdx.y, q0 = blockIdx.x * BMQ;
  const int g = h / (nh / nkv);
  const int dkv = nkv * HD;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bf16* base = qkv + (size_t)chunk * L * ld;
  const bf16* Qg = base + h * HD;
  const bf16* Kg = base + d + g * HD;
  const bf16* Vg = base + d + dkv + g * HD;

  load_tile<HD>(sQ, Qg, ld, q0, L);
  load_tile<HD>(sK, Kg, ld, 0, L);
  load_tile<HD>(sV, Vg, ld, 0, L);
  cp_commit();

  uint32_t qf[HD / 16][4];
  float o[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};

  const int ntiles = (L + BNK - 1) / BNK;
  for (int t = 0; t < ntiles; ++t) {
    const int buf = t & 1;
    if (t + 1 < ntiles) {
      load_tile<HD>(sK + (buf ^ 1) * TILE, Kg, ld, (t + 1) * BNK, L);
      load_tile<HD>(sV + (buf ^ 1) * TILE, Vg, ld, (t + 1) * BNK, L);
    }
    cp_commit();
    cp_wait<1>();
    __syncthreads();
    if (t == 0) {
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk) {
        const int r = warp * 16 + (lane & 15), c = 2 * kk + (lane >> 4);
        ldm_x4(sQ + swz(r, c, CPR), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
      }
    }
    // S = Q K^T for 16 rows x 64 keys per warp
    float s[8][4];
#pragma unroll
    for (int j = 0; j < 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
    const uint32_t kb = sK + buf * TILE;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int j = 0; j < 8; j += 2) {
        const int key = j * 8 + ((lane >> 4) << 3) + (lane & 7);
        const int c = 2 * kk + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldm_x4(kb + swz(key, c, CPR), b0, b1, b2, b3);
        mma16816(s[j], qf[kk], b0, b1);
        mma16816(s[j + 1], qf[kk], b2, b3);
      }
    }
    // mask keys beyond the window, online softmax (base 2)
    const int kbase = t * BNK;
    float mnew[2] = {mrow[0], mrow[1]};
#pragma unroll
    for (int j = 0; j < 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kbase + j * 8 + 2 * (lane & 3) + (e & 1);
        s[j][e] = key < L ? s[j][e] * scale_log2 : -INFINITY;
      }
      mnew[0] = fmaxf(mnew[0], fmaxf(s[j][0], s[j][1]));
      mnew[1] = fmaxf(mnew[1], fmaxf(s[j][2], s[j][3]));
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      mnew[r] = fmaxf(mnew[r], __shfl_xor_sync(0xffffffffu, mnew[r], 1));
      mnew[r] = fmaxf(mnew[r], __shfl_xor_sync(0xffffffffu, mnew[r], 2));
    }
    float corr[2], psum[2] = {0.f, 0.f};
#pragma unroll
    for (int r = 0; r < 2; ++r) corr[r] = exp2f(mrow[r] - mnew[r]);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      s[j][0] = exp2f(s[j][0] - mnew[0]);
      s[j][1] = exp2f(s[j][1] - mnew[0]);
      s[j][2] = exp2f(s[j][2] - mnew[1]);
      s[j][3] = exp2f(s[j][3] - mnew[1]);
      psum[0] += s[j][0] + s[j][1];
      psum[1] += s[j][2] + s[j][3];
    }
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      psum[r] += __shfl_xor_sync(0xffffffffu, psum[r], 1);
      psum[r] += __shfl_xor_sync(0xffffffffu, psum[r], 2);
      lrow[r] = lrow[r] * corr[r] + psum[r];
      mrow[r] = mnew[r];
    }
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) {
      o[i][0] *= corr[0];
      o[i][1] *= corr[0];
      o[i][2] *= corr[1];
      o[i][3] *= corr[1];
    }
    // O += P V
    const uint32_t vb = sV + buf * TILE;
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {  // 16 keys per step
      uint32_t a[4];
      a[0] = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
      a[1] = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
      a[2] = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      a[3] = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
      for (int n = 0; n < HD / 8; n += 2) {
        const int key = 16 * kk + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int c = n + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldm_x4_t(vb + swz(key, c, CPR), b0, b1, b2, b3);
        mma16816(o[n], a, b0, b1);
        mma16816(o[n + 1], a, b2, b3);
      }
    }
    __syncthreads();  // buffer `buf` is refilled by the next iteration's prefetch
  }
  // normalise and store rows q0 + warp*16 + {g, g+8}
  const float inv0 = 1.0f / lrow[0], inv1 = 1.0f / lrow[1];
  const int r0 = q0 + warp * 16 + (lane >> 2);
  bf16* ob = out + (size_t)chunk * L * d + h * HD;
#pragma unroll
  for (int n = 0; n < HD / 8; ++n) {
    const int col = n * 8 + 2 * (lane & 3);
    if (r0 < L)
      *reinterpret_cast<uint32_t*>(ob + (size_t)r0 * d + col) = pack_bf16(o[n][0] * inv0, o[n][1] * inv0);
    if (r0 + 8 < L)
      *reinterpret_cast<uint32_t*>(ob + (size_t)(r0 + 8) * d + col) = pack_bf16(o[n][2] * inv1, o[n][3] * inv1);
  }
}

}  // namespace fa

int attention_bf16_mma(const bf16* qkv, int ld, int n_chunks, int L, int nh, int nkv, int hd, int d, bf16* out,
                       cudaStream_t s) {
  if (n_chunks == 0 || L == 0) return DLMZ_OK;
  if ((ld % 8) || (d % 8) || (reinterpret_cast<uintptr_t>(qkv) & 15)) return DLMZ_EINVAL;
  dim3 grid((L + fa::BMQ - 1) / fa::BMQ, nh, n_chunks);
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)hd);
  ProfScope prof(PROF_ATTN, s, 4.0 * n_chunks * nh * (double)L * L * hd, 2.0 * n_chunks * L * (double)(ld + d));
  if (hd == 64) {
    constexpr int SM = 5 * 64 * 64 * 2;
    fa::flash_kernel<64><<<grid, 128, SM, s>>>(qkv, ld, L, nh, nkv, d, out, scale_log2);
  } else if (hd == 128) {
    constexpr int SM = 5 * 64 * 128 * 2;
    static PerDeviceOnce attr;
    DLMZ_TRY(attr.run(
        [] { return cudaFuncSetAttribute(fa::flash_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, SM); }));
    fa::flash_kernel<128><<<grid, 128, SM, s>>>(qkv, ld, L, nh, nkv, d, out, scale_log2);
  } else {
    return DLMZ_EINVAL;
  }
  return launch_status();
}

}  // namespace dlmz
