// Self-test of the bounded device waits (failure detection without a GPU fault).
//
// Every wait of the library's kernels on an mbarrier is bounded: when a phase
// does not complete within the limit, the waiting role sets ERR_TIMEOUT in the
// device error word and the kernel winds down, so the host reports
// DLMZ_ETIMEOUT and the context stays usable.  This kernel makes such a wait
// run out on purpose: one thread initialises an mbarrier that expects one
// arrival nobody makes and waits on it with the caller's limit.
#include "kernels.cuh"

namespace dlmz {

__global__ void wait_timeout_kernel(uint64_t limit_ns, int* err, int* done) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ volatile int abort_flag;
  if (threadIdx.x != 0) return;
  abort_flag = 0;
  const uint32_t b = smem_u32(&bar);
  mbar_init(b, 1);
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  const bool ok = mbar_wait_bounded(b, 0, &abort_flag, err, limit_ns);
  *done = ok ? 1 : 2;  // 2: gave up after the limit, as intended
}

// The same across a cluster of two CTAs, as in the quantiser's exchanges: CTA 0 waits (cluster
// scope, bounded) for one arrival that CTA 1 makes on CTA 0's mbarrier only if `peer_arrives`.
// Both CTAs meet at a cluster barrier at the end, which CTA 0 reaches after its wait returns.
__global__ void cluster_wait_kernel(uint64_t limit_ns, int peer_arrives, int* err, int* done) {
  __shared__ __align__(8) uint64_t bar;
  if (cluster_nctarank() != 2) {  // launched without its cluster shape: no cluster operation runs
    if (threadIdx.x == 0) atomicOr(err, ERR_LAUNCH);
    return;
  }
  const uint32_t rank = cluster_ctarank();
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    fence_mbarrier_init_cluster();
  }
  cluster_sync_all();  // CTA 0's barrier is initialised before CTA 1 may arrive on it
  if (threadIdx.x == 0) {
    if (rank == 1 && peer_arrives) mbar_arrive_remote(mapa_shared(smem_u32(&bar), 0));
    if (rank == 0) *done = mbar_wait_cluster_bounded(smem_u32(&bar), 0, err, limit_ns) ? 1 : 2;
  }
  cluster_sync_all();  // neither CTA leaves while the other may still touch its shared memory
}

}  // namespace dlmz

using namespace dlmz;

extern "C" int dlmz_selftest_cluster_wait(uint32_t limit_us, uint32_t peer_arrives, void* stream) {
  if (limit_us == 0 || limit_us > 1000000 || peer_arrives > 1) return DLMZ_EINVAL;
  int* err = device_error_word();
  if (!err) return DLMZ_ENOMEM;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int* done = nullptr;
  DLMZ_CUDA_TRY(cudaMallocAsync(reinterpret_cast<void**>(&done), sizeof(int), s));
  DLMZ_CUDA_TRY(cudaMemsetAsync(done, 0, sizeof(int), s));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2);
  cfg.blockDim = dim3(32);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaLaunchKernelEx(&cfg, cluster_wait_kernel, (uint64_t)limit_us * 1000ull, (int)peer_arrives, err, done);
  int rc = launch_status();
  int h = 0;
  if (cudaMemcpyAsync(&h, done, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    rc = DLMZ_ECUDA;
  cudaFreeAsync(done, s);
  if (rc != DLMZ_OK) return rc;
  if (h != (peer_arrives ? 1 : 2)) return DLMZ_ECUDA;  // completed exactly when the peer arrived
  return dlmz_check(stream);                            // ETIMEOUT when the wait gave up (bit cleared)
}

extern "C" int dlmz_selftest_wait_timeout(uint32_t limit_us, void* stream) {
  if (limit_us == 0 || limit_us > 1000000) return DLMZ_EINVAL;
  int* err = device_error_word();
  if (!err) return DLMZ_ENOMEM;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int* done = nullptr;
  DLMZ_CUDA_TRY(cudaMallocAsync(reinterpret_cast<void**>(&done), sizeof(int), s));
  DLMZ_CUDA_TRY(cudaMemsetAsync(done, 0, sizeof(int), s));
  wait_timeout_kernel<<<1, 32, 0, s>>>((uint64_t)limit_us * 1000ull, err, done);
  int rc = launch_status();
  int h = 0;
  if (cudaMemcpyAsync(&h, done, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    rc = DLMZ_ECUDA;
  cudaFreeAsync(done, s);
  if (rc != DLMZ_OK) return rc;
  if (h != 2) return DLMZ_ECUDA;  // the wait must have given up, not completed
  return dlmz_check(stream);      // reports the timeout bit (and clears it)
}
