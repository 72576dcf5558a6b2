// Internal helpers shared by the library's translation units (not part of
// the C ABI).  Nothing here is shared with the CPU oracle.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/unison.h"

namespace unison {

// Locked integer format, eq. (lock): b_h = 12 (Lambda = 2^12 - 1), b_g = 32,
// b_s = 64, tau = 1e3 (microseconds), eps_q = floor(0.01 * Lambda + 1/2).
constexpr uint32_t kLambda = 4095u;
constexpr uint32_t kEpsQ = 41u;
constexpr uint32_t kTMax = 50u;   // hazard table covers turns 0..50, eq. (hazard)
constexpr uint32_t kLutN = 51u;

// A policy key is at most 40 bits (a SPEAR score of a live session is below
// 2^39 under the documented input limits: g_q < 2^31 gives T1 < 2^38 and
// P_Z < 2^32 gives T2 < 2^32).  A completed session, or a session with no
// next arrival under Belady, takes the maximal key 2^40 - 1.  Packing the
// key above the inverted 24-bit session id gives one 64-bit word whose
// unsigned order is the ranking order: larger key first, then smaller id.
constexpr uint64_t kKeyMax40 = (1ull << 40) - 1;
constexpr uint32_t kIdMask = 0xFFFFFFu;

// floor(x / s) for x < 2^43 and 2 <= s < 2^12 by one multiply-high
// (Granlund and Montgomery, PLDI 1994, Thm 4.2 with N = 43): with
// l = ceil(log2 s) and m = ceil(2^(43+l) / s), floor(x/s) = floor(x m / 2^(43+l));
// storing m << (21 - l) turns that into the high word of a 64x64 product.
__host__ __device__ inline uint64_t magic_for(uint32_t s) {
  uint32_t l = 0;
  while ((1u << l) < s) l++;
  // m = ceil(2^(43+l) / s) fits 44 bits; compute without 128-bit division.
  const uint64_t num = 1ull << (43 + l);  // 43 + l <= 55
  const uint64_t m = (num + s - 1) / s;
  return m << (21 - l);
}

// Fault injection (unison_debug_fail_allocations): true, once per pending
// fault, at a device allocation that should then fail as out of memory.
bool unison_fault_alloc();

__host__ __device__ __forceinline__ uint64_t pack_key(uint64_t key40, uint32_t id) {
  return (key40 << 24) | ((~id) & kIdMask);
}
__host__ __device__ __forceinline__ uint32_t packed_id(uint64_t pk) {
  return (~(uint32_t)pk) & kIdMask;
}

// Event word 1 layout: session in bits 0..23, bit 30 = first turn (arrival)
// or final turn (completion), bit 31 = arrival.
constexpr uint32_t kEvArrival = 1u << 31;
constexpr uint32_t kEvEdge = 1u << 30;
constexpr uint32_t kNoRef = 0xFFFFFFFFu;

constexpr uint64_t kFnvOffset = 0xCBF29CE484222325ull;
constexpr uint64_t kFnvPrime = 0x100000001B3ull;

}  // namespace unison

// Internal view of a trace (host staging + device copies).
struct unison_trace {
  uint32_t n_sessions = 0;
  uint64_t n_turns = 0;
  uint64_t n_events = 0;
  uint32_t min_out_tok = 0;

  // One page-locked host block holding every array below, copied to the
  // device with a single cudaMemcpyAsync.
  void *h_block = nullptr;
  bool h_pinned = false;
  void *d_block = nullptr;
  size_t block_bytes = 0;
  int device = -1;
  cudaStream_t last_stream = nullptr;

  // Offsets (bytes) of each array inside the block.
  size_t off_ev = 0;        // uint4[E]: time32, session|flags, in_tok, out_tok
  size_t off_prev_out = 0;  // u32[E]: l^out of the previous turn (arrivals)
  size_t off_nref = 0;      // u32[E]: event index of the next arrival (arrivals)
  size_t off_prev_ev = 0;   // u32[E]: event index of the previous completion (arrivals of turn >= 1)
  size_t off_turn_ev = 0;   // u32[2T]: arrival and completion event of each turn
  size_t off_turn_t = 0;    // u32[2T]: arrival and completion time32 of each turn
  size_t off_turn_off = 0;  // u32[S+1]: session turn offsets
  size_t off_tps = 0;       // u32[S]: turns per session

  template <typename T>
  T *h(size_t off) const { return reinterpret_cast<T *>(static_cast<char *>(h_block) + off); }
  template <typename T>
  T *d(size_t off) const { return reinterpret_cast<T *>(static_cast<char *>(d_block) + off); }
};
