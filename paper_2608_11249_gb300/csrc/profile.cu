// Live per-kernel-class profiler: CUDA event pairs recorded on each launch's
// stream while enabled, summed at dlmz_profile_end.
#include <atomic>
#include <vector>

#include "common.cuh"

namespace dlmz {

namespace {
struct Pending {
  int cls;
  cudaEvent_t a, b;
  double flops, bytes;
};
bool g_on = false;
uint64_t g_launches = 0;
std::atomic<uint64_t> g_total{0};  // every launch since the library was loaded
std::vector<Pending> g_pending;
std::vector<cudaEvent_t> g_pool;
cudaEvent_t g_open[PROF_NCLASS];

cudaEvent_t take_event() {
  if (!g_pool.empty()) {
    cudaEvent_t e = g_pool.back();
    g_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}
}  // namespace

bool prof_on() { return g_on; }

void prof_count_launch() {
  g_total.fetch_add(1, std::memory_order_relaxed);
  if (g_on) ++g_launches;
}

void prof_record(int cls, cudaStream_t s, bool start, double flops, double bytes) {
  if (start) {
    g_open[cls] = take_event();
    cudaEventRecord(g_open[cls], s);
  } else if (g_open[cls]) {
    cudaEvent_t b = take_event();
    cudaEventRecord(b, s);
    g_pending.push_back({cls, g_open[cls], b, flops, bytes});
    g_open[cls] = nullptr;
  }
}

}  // namespace dlmz

using namespace dlmz;

extern "C" uint64_t dlmz_launch_count(void) { return g_total.load(std::memory_order_relaxed); }

extern "C" int dlmz_profile_begin(void) {
  for (auto& p : g_pending) {
    g_pool.push_back(p.a);
    g_pool.push_back(p.b);
  }
  g_pending.clear();
  for (int i = 0; i < PROF_NCLASS; ++i) g_open[i] = nullptr;
  g_launches = 0;
  g_on = true;
  return DLMZ_OK;
}

extern "C" int dlmz_profile_end(dlmz_profile* out) {
  g_on = false;
  if (!out) return DLMZ_EINVAL;
  *out = dlmz_profile{};
  DLMZ_CUDA_TRY(cudaDeviceSynchronize());
  out->launches = g_launches;
  for (auto& p : g_pending) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, p.a, p.b) == cudaSuccess) {
      out->n[p.cls] += 1;
      out->ms[p.cls] += ms;
      out->flops[p.cls] += p.flops;
      out->bytes[p.cls] += p.bytes;
    }
    g_pool.push_back(p.a);
    g_pool.push_back(p.b);
  }
  g_pending.clear();
  return DLMZ_OK;
}
