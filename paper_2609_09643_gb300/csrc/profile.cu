// Measurement support: CUDA-event timing of the library's main kernels and
// a launch counter (see unison_profile_enable in include/unison.h).
#include <atomic>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "common.cuh"
#include "profile.cuh"

namespace {
struct Rec {
  std::string name;
  cudaEvent_t a, b;
};
std::mutex g_mu;
std::vector<Rec> g_recs;
bool g_on = false;
std::atomic<uint64_t> g_launches{0};
}  // namespace

namespace unison {

void count_launches(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

ProfSpan::ProfSpan(const char *name, cudaStream_t s) : stream_(s) {
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_on || !name || !*name) return;
  if (cudaEventCreate(&a_) != cudaSuccess || cudaEventCreate(&b_) != cudaSuccess) {
    cudaGetLastError();
    return;
  }
  name_ = name;
  active_ = true;
  cudaEventRecord(a_, s);
}

ProfSpan::~ProfSpan() {
  if (!active_) return;
  cudaEventRecord(b_, stream_);
  std::lock_guard<std::mutex> lk(g_mu);
  g_recs.push_back({name_, a_, b_});
}

}  // namespace unison

extern "C" int unison_profile_enable(int on) {
  std::lock_guard<std::mutex> lk(g_mu);
  g_on = on != 0;
  return UNISON_OK;
}

extern "C" int unison_profile_read(const char *kernel, double *total_ms, uint64_t *launches, int reset) {
  if (!kernel) return UNISON_ERR_ARG;
  std::lock_guard<std::mutex> lk(g_mu);
  double tot = 0;
  uint64_t n = 0;
  std::vector<Rec> keep;
  for (auto &r : g_recs) {
    if (r.name == kernel) {
      float ms = 0;
      if (cudaEventSynchronize(r.b) != cudaSuccess || cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) {
        cudaGetLastError();
        return UNISON_ERR_CUDA;
      }
      tot += ms;
      n++;
      if (reset) {
        cudaEventDestroy(r.a);
        cudaEventDestroy(r.b);
        continue;
      }
    }
    keep.push_back(r);
  }
  g_recs.swap(keep);
  if (total_ms) *total_ms = tot;
  if (launches) *launches = n;
  return UNISON_OK;
}

extern "C" uint64_t unison_launch_count(void) { return g_launches.load(); }
