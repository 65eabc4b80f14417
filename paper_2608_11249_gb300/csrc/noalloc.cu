// Allocation-free variant of dlmz_select_smallest.
//
// Some callers cannot call cudaMalloc: code whose device memory is owned by
// another allocator (a caching or pooled allocator that has reserved the free
// memory), latency-critical paths that cannot accept cudaMalloc's implicit
// device-wide synchronisation, and hosts that enforce a fixed device-memory
// budget at start-up.  This entry point serves them: the selection kernel's
// scratch (the per-group count it writes besides the caller's output) lives
// in a file-scope __device__ array, so the call allocates nothing.
//
// The array holds at most kMaxGroups counts (256 KiB); every GPU that loads
// the library keeps it until the process exits.  Host code cannot use the
// array's name as a device address: on the first call on each device (with
// that device current) its address is fetched once with
// cudaGetSymbolAddress and then passed to the kernel.  Make that first call
// before any stream capture.  All calls share the array; the kernel
// overwrites every count it uses before reading it, so nothing has to be
// cleared between calls, but calls that overlap on the GPU race on it.
#include <mutex>

#include "coder.cuh"

namespace {

constexpr uint32_t kMaxGroups = 65536;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) int32_t g_select_counts[kMaxGroups];

std::mutex g_mu;
int32_t* g_counts_ptr[kMaxDevices] = {};

// Device address of g_select_counts on the current device (set up once per device).
int counts_address(int32_t** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return DLMZ_ECUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_counts_ptr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_select_counts);
    if (e != cudaSuccess || !p) {
      fprintf(stderr, "dlmz: cudaGetSymbolAddress failed: %s\n", cudaGetErrorString(e));
      return DLMZ_ECUDA;
    }
    g_counts_ptr[dev] = static_cast<int32_t*>(p);
  }
  *out = g_counts_ptr[dev];
  return DLMZ_OK;
}

}  // namespace

extern "C" int dlmz_select_smallest_noalloc(const uint64_t* d_keys, uint32_t groups, uint32_t group_size, uint32_t k,
                                            int32_t* d_out, void* stream) {
  if (!d_keys || !d_out || k == 0 || k > group_size || group_size > 4096) return DLMZ_EINVAL;
  if (groups > kMaxGroups) {
    fprintf(stderr, "dlmz_select_smallest_noalloc: %u groups exceed the maximum of %u\n", groups, kMaxGroups);
    return DLMZ_EINVAL;
  }
  int32_t* counts = nullptr;
  const int rc = counts_address(&counts);
  if (rc != DLMZ_OK) return rc;
  return dlmz::select_rows<uint64_t>(nullptr, (int)groups, (int)group_size, -1, 0, (int)group_size, d_keys, 0, (int)k,
                                     0, 0, 0, (int)k, counts, d_out, reinterpret_cast<cudaStream_t>(stream));
}
