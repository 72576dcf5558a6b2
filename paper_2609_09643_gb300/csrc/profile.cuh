// Internal measurement helpers (CUDA-event spans, launch counter).
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

namespace unison {

void count_launches(uint64_t n);

// Records CUDA events around the enclosed launches when profiling is on.
class ProfSpan {
 public:
  ProfSpan(const char *name, cudaStream_t s);
  ~ProfSpan();
  ProfSpan(const ProfSpan &) = delete;
  ProfSpan &operator=(const ProfSpan &) = delete;

 private:
  cudaStream_t stream_;
  cudaEvent_t a_{}, b_{};
  std::string name_;
  bool active_ = false;
};

}  // namespace unison
