// Shared device/host helpers of the dlmz CUDA library (sm_103a).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>

#include "../../include/dlmz.h"

namespace dlmz {

// Device-side error word (one per device, zeroed by dlmz_check).
// Bits: 1 = wait timed out, 2 = corrupt stream, 4 = non-finite logits,
// 8 = stream capacity exceeded.
enum : int { ERR_TIMEOUT = 1, ERR_CORRUPT = 2, ERR_NONFINITE = 4, ERR_CAPACITY = 8, ERR_LAUNCH = 16 };

int* device_error_word();  // lazily allocated device int

#define DLMZ_CUDA_TRY(expr)                                                      \
  do {                                                                           \
    cudaError_t e_ = (expr);                                                     \
    if (e_ != cudaSuccess) {                                                     \
      fprintf(stderr, "dlmz: %s failed: %s (%s:%d)\n", #expr,                    \
              cudaGetErrorString(e_), __FILE__, __LINE__);                       \
      return DLMZ_ECUDA;                                                         \
    }                                                                            \
  } while (0)

#define DLMZ_TRY(expr)          \
  do {                          \
    int r_ = (expr);            \
    if (r_ != DLMZ_OK) return r_; \
  } while (0)

// ---- live per-kernel-class profiler (CUDA events on the launch stream) ----------
enum ProfClass { PROF_GEMM_TC = 0, PROF_GEMM_SIMT, PROF_ATTN, PROF_QUANT, PROF_SELECT, PROF_CODE, PROF_LAYER,
                 PROF_OTHER, PROF_NCLASS };
bool prof_on();
void prof_count_launch();
void prof_record(int cls, cudaStream_t s, bool start, double flops, double bytes);

// Records CUDA events around the launches of one kernel class while
// profiling is enabled (dlmz_profile_begin / dlmz_profile_end).
struct ProfScope {
  int cls;
  cudaStream_t s;
  double flops, bytes;
  ProfScope(int c, cudaStream_t st, double f, double b) : cls(c), s(st), flops(f), bytes(b) {
    if (prof_on()) prof_record(cls, s, true, 0, 0);
  }
  ~ProfScope() {
    if (prof_on()) prof_record(cls, s, false, flops, bytes);
  }
};

inline int launch_status() {
  prof_count_launch();
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    fprintf(stderr, "dlmz: kernel launch failed: %s\n", cudaGetErrorString(e));
    return DLMZ_ECUDA;
  }
  return DLMZ_OK;
}

// ---- per-device caches ------------------------------------------------------
// Kernel attributes, occupancy limits, SM counts and scratch buffers belong to
// one device, so every cache of the library is indexed by the ordinal of the
// current device (at most kMaxDevices devices per process).
constexpr int kMaxDevices = 64;

// Ordinal of the current device, or -1 when it cannot be used as an index.
inline int device_ordinal() {
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return -1;
  return d;
}

// Runs a set-up step (returning cudaError_t) once per device: the first call
// on each device runs it, later calls on that device return DLMZ_OK at once.
struct PerDeviceOnce {
  bool done[kMaxDevices] = {};
  template <class F>
  int run(F f) {
    const int d = device_ordinal();
    if (d < 0) return DLMZ_ECUDA;
    if (done[d]) return DLMZ_OK;
    const cudaError_t e = f();
    if (e != cudaSuccess) {
      fprintf(stderr, "dlmz: per-device set-up failed: %s\n", cudaGetErrorString(e));
      return DLMZ_ECUDA;
    }
    done[d] = true;
    return DLMZ_OK;
  }
};

inline int num_sms() {
  static int n[kMaxDevices] = {};
  const int dev = device_ordinal();
  if (dev < 0) return 1;
  if (!n[dev]) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
    n[dev] = v > 0 ? v : 1;
  }
  return n[dev];
}

// ---- device helpers -------------------------------------------------------

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(bar)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile(
      "{\n\t.reg .b64 st;\n\tmbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(bar),
      "r"(bytes)
      : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait on an mbarrier phase.  Gives up after `limit_ns` (or when
// *abort is set by another role), raising ERR_TIMEOUT in the global error
// word and *abort; returns false then.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity,
                                                  volatile int* abort, int* err,
                                                  uint64_t limit_ns = 2000000000ull) {
  if (mbar_try_wait(bar, parity)) return true;
  uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((it & 63) == 0) {
      if (*abort) return false;
      if (globaltimer_ns() - t0 > limit_ns) {
        *abort = 1;
        atomicOr(err, ERR_TIMEOUT);
        return false;
      }
    }
  }
}

// ---- thread-block clusters: rank, distributed shared memory, cluster-scope mbarriers ----

__device__ __forceinline__ uint32_t cluster_nctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

// shared::cluster address of the variable at shared::cta address `addr` in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}

__device__ __forceinline__ void st_cluster_u32(uint32_t caddr, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(caddr), "r"(v) : "memory");
}

__device__ __forceinline__ void st_cluster_u64(uint32_t caddr, uint64_t v) {
  asm volatile("st.shared::cluster.u64 [%0], %1;" ::"r"(caddr), "l"(v) : "memory");
}

// one arrival on an mbarrier of another CTA of the cluster; release at cluster scope orders this
// thread's earlier shared::cluster stores before it
__device__ __forceinline__ void mbar_arrive_remote(uint32_t caddr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(caddr) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// bounded wait (as mbar_wait_bounded) for arrivals from other CTAs of the cluster
__device__ __forceinline__ bool mbar_wait_cluster_bounded(uint32_t bar, uint32_t parity, int* err,
                                                          uint64_t limit_ns = 2000000000ull) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if ((it & 63) == 0 && globaltimer_ns() - t0 > limit_ns) {
      atomicOr(err, ERR_TIMEOUT);
      return false;
    }
  }
}

// all threads of every CTA of the cluster (a hardware barrier; each CTA must reach it the same
// number of times)
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ void fence_mbarrier_init_cluster() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ float bf16_to_f(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T>
__device__ __forceinline__ float to_f(T v);
template <>
__device__ __forceinline__ float to_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

}  // namespace dlmz
