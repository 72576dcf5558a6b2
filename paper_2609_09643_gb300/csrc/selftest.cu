// Library self-checks and fault injection (see unison.h).
//
// unison_selftest_division checks, on the device, the division every score
// of eq. (t1) uses: floor(x / s) computed as the high word of x * magic_for(s)
// (Granlund and Montgomery, PLDI 1994), valid for x < 2^43 and 2 <= s < 2^12.
// Each x is checked against the definition of the quotient, q*s <= x <
// (q+1)*s, with multiplications only.
#include <atomic>
#include <cstdint>

#include "common.cuh"

using namespace unison;

namespace {

__device__ unsigned long long g_division_mismatches;

constexpr uint64_t kXLimit = 1ull << 43;
constexpr uint32_t kDense = 1u << 20;    // every x below this
constexpr uint32_t kQuotients = 1u << 16;  // sampled quotients per divisor

__device__ __forceinline__ bool quotient_ok(uint64_t x, uint32_t s, uint64_t mg) {
  const uint64_t q = __umul64hi(x, mg);
  return q * s <= x && x - q * s < s;
}

// One CTA per divisor s = 2 + blockIdx.x.
__global__ void __launch_bounds__(256) division_check_kernel() {
  const uint32_t s = 2 + blockIdx.x;
  const uint64_t mg = magic_for(s);
  unsigned long long bad = 0;
  for (uint32_t x = threadIdx.x; x < kDense; x += blockDim.x) bad += !quotient_ok(x, s, mg);
  // quotient boundaries q*s - 1, q*s, q*s + s - 1, for quotients spread over
  // [1, qmax] with qmax the largest such that qmax*s + s - 1 < 2^43
  const uint64_t qmax = (kXLimit - s) / s;
  for (uint32_t i = threadIdx.x; i < kQuotients; i += blockDim.x) {
    const uint64_t q = 1 + (qmax - 1) * i / (kQuotients - 1);
    bad += !quotient_ok(q * s - 1, s, mg);
    bad += !quotient_ok(q * s, s, mg);
    bad += !quotient_ok(q * s + s - 1, s, mg);
  }
  if (bad) atomicAdd(&g_division_mismatches, bad);
}

std::atomic<int> g_fail_allocs{0};

}  // namespace

namespace unison {
bool unison_fault_alloc() {
  int n = g_fail_allocs.load();
  while (n > 0)
    if (g_fail_allocs.compare_exchange_weak(n, n - 1)) return true;
  return false;
}
}  // namespace unison

extern "C" void unison_debug_fail_allocations(int n) { g_fail_allocs.store(n > 0 ? n : 0); }

extern "C" int unison_selftest_division(uint64_t *mismatches, void *cuda_stream) {
  if (!mismatches) return UNISON_ERR_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const unsigned long long zero = 0;
  unsigned long long got = 0;
  if (cudaMemcpyToSymbolAsync(g_division_mismatches, &zero, sizeof(zero), 0, cudaMemcpyHostToDevice, st) !=
      cudaSuccess)
    return UNISON_ERR_CUDA;
  division_check_kernel<<<4094, 256, 0, st>>>();
  if (cudaGetLastError() != cudaSuccess) return UNISON_ERR_CUDA;
  if (cudaMemcpyFromSymbolAsync(&got, g_division_mismatches, sizeof(got), 0, cudaMemcpyDeviceToHost, st) !=
          cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return UNISON_ERR_CUDA;
  *mismatches = got;
  return UNISON_OK;
}
