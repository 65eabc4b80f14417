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

}  // namespace dlmz

using namespace dlmz;

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
