// Standalone ranking of large live sets (the scan of Sec. IV-D, eqs. pipe and
// scan, generalised from one argmax to a top-k) and the TIDE fill of
// Sec. III-C (eqs. budget, promote, demote) over the same ranking.
//
// Every record gets a packed comparable key ck = score40 << 24 | ~index24:
// unsigned order on ck is the ranking order (larger score first, ties to
// the smaller index).  Three ordered selections are needed per live set:
//   V  victims: unpinned resident records, largest ck first (top-k);
//   D  fast-tier demotion candidates: unpinned fast-tier records, largest first;
//   P  HBM promotion candidates: unpinned HBM records, smallest ck first.
// Kernels, in launch order:
//   rank_sample_kernel   16 CTAs per set: order statistics of a jittered
//                        stratified sample give each list a threshold, turned
//                        into per-turn thresholds on the gap average (the
//                        score is monotone in the gap for a fixed turn, so
//                        the streaming test needs no division).
//   rank_filter_kernel   one pass over every record (8 B each: gap average,
//                        turn, flags, tier), emitting the exact values of the
//                        records that pass a threshold.
//   rank_finish_kernel   one CTA per (list, set): exact top-M of the list's
//                        candidates by radix select and a bitonic sort; if
//                        the candidates overflowed or fell short, the CTA
//                        re-selects the list exactly by streaming the whole
//                        set.  The set's last CTA writes the victims and runs
//                        the fill as warp prefix scans.
#include <algorithm>
#include <map>
#include <cstring>
#include <mutex>
#include <type_traits>
#include <vector>

#include "common.cuh"
#include "profile.cuh"

using namespace unison;

namespace {

constexpr int kLists = 3;  // 0 = V, 1 = D, 2 = P
constexpr uint32_t kSample = 16384;
constexpr uint32_t kSmemCand = 16384;
constexpr uint32_t kCandCap = 65536;
constexpr uint32_t kMaxSel = 4096;
constexpr uint32_t kFinishThreads = 1024;
constexpr uint32_t kFull = 0xFFFFFFFFu;

struct RankWork {
  unsigned int cand[kLists];  // candidates emitted per list
  unsigned int status;        // UNISON_ERR_TIMEOUT if a bounded wait gave up
  unsigned int got[kLists];   // selected entries per list (finish)
  unsigned int ticket;        // finish CTAs done with their list
  unsigned int sticket;       // sample CTAs done
};

constexpr uint32_t kSampleCtas = 16;     // sample CTAs per set
constexpr uint32_t kSampleThreads = 1024;
constexpr uint32_t kMaxR = 256;          // largest sample rank used for a threshold

struct RankSet {
  const uint32_t *gap;
  const uint16_t *turn;
  const uint32_t *kv;
  const uint8_t *tier;
  const uint8_t *flags;
  uint32_t n, k, max_moves, kvb;
  uint64_t penalty, budget, free_s, free_h;
  uint32_t *victims, *promote, *demote, *counts;
  uint64_t *moved, *keys;
  uint32_t tile0, ntiles;
  uint32_t sigma[kLutN];
  // per-set constants, computed on the host
  uint32_t ns, nruns, sq, srem;  // sample size, its runs of 8, n = sq * nruns + srem
  uint32_t sctas;                // sample CTAs (at most kSampleCtas)
  uint32_t cta0, nctas;           // filter, group mode: CTAs [cta0, cta0 + nctas) stream this set
  uint32_t act;                  // active lists (bit L)
  uint32_t rL[kLists];           // sample rank of each list's threshold
  uint64_t t2v[kLutN];           // eq. (t2) per turn index
  uint64_t mgv[kLutN];           // division magic of sigma per turn index
  // scratch (per set)
  RankWork *work;
  uint64_t *cand;    // [3][kCandCap]
  uint64_t *sorted;  // [3][kMaxSel]
  uint32_t *ssz;     // [3][kMaxSel] KV tokens of the sorted entries (D and P)
  uint2 *gthr;       // [3][51] (gA, gB)
  uint64_t *thr;     // [3] threshold in list-value space; [3+L] = active flag
  uint32_t *part;    // [3][kSampleCtas][kMaxR] per-CTA top summaries of the sample
  uint32_t *part_n;  // [3][kSampleCtas] entries in each
};

// ---------------------------------------------------------------- keys ----
__device__ __forceinline__ uint64_t score_of(uint32_t g, uint32_t t, bool done, const uint64_t *t2,
                                             const uint64_t *magic) {
  if (done) return ~0ull;
  return __umul64hi((uint64_t)g * kLambda, magic[t]) + t2[t];
}

__device__ __forceinline__ uint64_t ck_of(uint64_t score, uint32_t idx) {
  const uint64_t k40 = score == ~0ull ? kKeyMax40 : score;
  return (k40 << 24) | ((~idx) & kIdMask);
}

__device__ __forceinline__ uint32_t elig_mask(uint8_t fl, uint8_t tr) {
  if (fl & 1) return 0;  // pinned: never ranked for eviction or migration
  uint32_t m = 0;
  if (tr == 1) m = 1u | 2u;
  if (tr == 2) m = 1u | 4u;
  return m;
}

// Smallest gap average whose score reaches K at turn index t.
__device__ __forceinline__ uint32_t g_at_least(uint64_t K, uint32_t sigma, uint64_t t2) {
  if (K <= t2) return 0;
  const uint64_t m = K - t2;
  const uint64_t g = (m * sigma + kLambda - 1) / kLambda;
  return g > 0xFFFFFFFFull ? 0xFFFFFFFFu : (uint32_t)g;
}

// -------------------------------------------------------- block helpers ----
// Value with the given rank (1 = largest) among get(0..n-1) -- MSB-first
// radix select, 8 bits per pass.  All threads of the block call it and get
// the same value.  hist[2][256] and pick[2][2] are double-buffered, so a
// pass takes two barriers.
template <typename Get>
__device__ uint64_t block_select_rank(Get get, uint32_t n, uint32_t rank, unsigned int (*hist)[256],
                                      unsigned int (*pick)[2], unsigned long long *bcast) {
  // bytes on which every value agrees need no pass: start at the highest
  // byte where some two values differ
  unsigned long long a = ~0ull, o = 0ull;
  for (uint32_t i = threadIdx.x; i < n; i += blockDim.x) {
    const uint64_t v = get(i);
    a &= v;
    o |= v;
  }
  for (int s = 16; s; s >>= 1) {
    a &= __shfl_xor_sync(0xFFFFFFFFu, a, s);
    o |= __shfl_xor_sync(0xFFFFFFFFu, o, s);
  }
  if (threadIdx.x == 0) {
    bcast[0] = ~0ull;
    bcast[1] = 0ull;
  }
  for (uint32_t i = threadIdx.x; i < 2 * 256; i += blockDim.x) (&hist[0][0])[i] = 0;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) {
    atomicAnd(&bcast[0], a);
    atomicOr(&bcast[1], o);
  }
  __syncthreads();
  const uint64_t same = ~(bcast[0] ^ bcast[1]);  // bits equal in every value
  const uint64_t common = bcast[0] & same;
  int top = 7;
  while (top > 0 && ((same >> (8 * top)) & 0xFF) == 0xFF) top--;
  uint64_t mask = top < 7 ? (~0ull << (8 * (top + 1))) : 0ull;
  uint64_t prefix = common & mask;
  uint32_t need = rank;
  for (int b = top; b >= 0; b--) {
    const int pb = b & 1;
    for (uint32_t base = 0; base < n; base += blockDim.x) {
      const uint32_t i = base + threadIdx.x;
      bool in = false;
      uint32_t d = 0;
      if (i < n) {
        const uint64_t v = get(i);
        in = (v & mask) == prefix;
        d = (uint32_t)(v >> (8 * b)) & 0xFF;
      }
      // lanes with the same digit add once per group
      const unsigned act = __ballot_sync(0xFFFFFFFFu, in);
      if (in) {
        const unsigned grp = __match_any_sync(act, d);
        if ((__ffs(grp) - 1) == (int)(threadIdx.x & 31)) atomicAdd(&hist[pb][d], (unsigned)__popc(grp));
      }
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      // lane l owns digits 255-8l .. 248-8l (descending); find the digit where
      // the count of larger-or-equal values first reaches `need`
      const int l = threadIdx.x;
      uint32_t c[8], tot = 0;
#pragma unroll
      for (int q = 0; q < 8; q++) {
        c[q] = hist[pb][255 - 8 * l - q];
        tot += c[q];
      }
      uint32_t incl = tot;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (l >= o) incl += y;
      }
      const uint32_t excl = incl - tot;
      const unsigned hit = __ballot_sync(0xFFFFFFFFu, excl < need && incl >= need);
      if (l == __ffs(hit) - 1) {
        uint32_t cum = excl;
#pragma unroll
        for (int q = 0; q < 8; q++) {
          if (cum + c[q] >= need) {
            pick[pb][0] = 255 - 8 * l - q;
            pick[pb][1] = need - cum;
            cum = 0xFFFFFFFFu;  // found: no later digit matches
            break;
          }
          cum += c[q];
        }
      }
    }
    // the other histogram was last read before the barrier above
    for (uint32_t i = threadIdx.x; i < 256; i += blockDim.x) hist[pb ^ 1][i] = 0;
    __syncthreads();
    prefix |= (uint64_t)pick[pb][0] << (8 * b);
    mask |= 0xFFull << (8 * b);
    need = pick[pb][1];
  }
  __syncthreads();  // hist, pick and bcast free for the caller
  return prefix;
}

// Sort, descending, of a[0..n) padded with zeros to a power of two p >= 32
// (tmp: p more entries of scratch).  Each warp sorts runs of 32 in registers
// (bitonic network over shuffles); then runs are merged pairwise, log2(p/32)
// levels of one barrier each: an element of the left run lands at its index
// plus the number of right-run elements above it, an element of the right
// run at its index plus the number of left-run elements at or above it, both
// counts by binary search in the other (sorted) run.
__device__ void block_sort_desc(uint64_t *a, uint32_t n, uint64_t *tmp) {
  if (n <= 1) return;
  uint32_t p = 32;
  while (p < n) p <<= 1;
  for (uint32_t i = n + threadIdx.x; i < p; i += blockDim.x) a[i] = 0;
  __syncthreads();
  const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  for (uint32_t r = warp; r < p / 32; r += nw) {
    uint64_t x = a[r * 32 + lane];
#pragma unroll
    for (uint32_t k = 2; k <= 32; k <<= 1) {
      const bool desc = (lane & k) == 0;
#pragma unroll
      for (uint32_t j = k >> 1; j > 0; j >>= 1) {
        const uint64_t y = __shfl_xor_sync(0xFFFFFFFFu, x, j);
        const bool lower = (lane & j) == 0;
        x = (lower == desc) ? (x > y ? x : y) : (x < y ? x : y);
      }
    }
    a[r * 32 + lane] = x;
  }
  __syncthreads();
  uint64_t *src = a, *dst = tmp;
  for (uint32_t m = 32; m < p; m <<= 1) {
    for (uint32_t i = threadIdx.x; i < p; i += blockDim.x) {
      const uint64_t v = src[i];
      const uint32_t run0 = i & ~(2 * m - 1);
      const bool left = (i & m) == 0;
      const uint64_t *other = src + run0 + (left ? m : 0);
      uint32_t lo = 0, hi = m;  // other-run elements placed before v: a prefix
      while (lo < hi) {
        const uint32_t mid = (lo + hi) >> 1;
        const uint64_t w = other[mid];
        if (left ? (w > v) : (w >= v)) lo = mid + 1; else hi = mid;
      }
      dst[run0 + (i & (m - 1)) + lo] = v;
    }
    __syncthreads();
    uint64_t *t = src;
    src = dst;
    dst = t;
  }
  if (src != a) {
    for (uint32_t i = threadIdx.x; i < p; i += blockDim.x) a[i] = src[i];
    __syncthreads();
  }
}

__device__ __forceinline__ uint64_t list_val(uint64_t ck, int L) { return L == 2 ? ~ck : ck; }

// ------------------------------------------------------------- sample ----
// Sample size and per-list ranks: ns records (ns/8 runs of 8, one run per
// stratum) and rank r_L = ceil(target_L * ns / n), with ns about kSampleRank
// times n over the largest target, capped at kSample; the sample is split over
// ceil(ns / 1024) CTAs.  Candidates above the rank-r_L sample value number
// about target_L / r_L * Gamma(r_L), and fall short of M_L with probability
// P(Gamma(r_L) < r_L M_L / target_L).  Targets: 2 M + 1024 while the sample
// is not capped (r = 32 for the largest list: below 1e-6), else 6 M + 2048
// (r >= 8 at 2^24 records: about 1e-5).  A shortfall costs time, never
// exactness (the finish re-selects the list).
constexpr uint32_t kSampleRank = 32;
__host__ __device__ __forceinline__ uint64_t umin64(uint64_t a, uint64_t b) { return a < b ? a : b; }
__host__ __device__ __forceinline__ bool list_active(const RankSet &S, int L) {
  const uint32_t M = (L == 0) ? S.k : S.max_moves;
  return M > 0 && (L == 0 || S.budget > 0);
}
__host__ __device__ __forceinline__ uint64_t list_target_of(const RankSet &S, int L, bool wide) {
  const uint32_t M = (L == 0) ? S.k : S.max_moves;
  return wide ? 6ull * M + 2048 : 2ull * M + 1024;
}
// q samples per thread (1 or 4: more samples per CTA make a CTA slower but
// let many sets' sample CTAs fit in one wave).
__host__ __device__ __forceinline__ uint32_t sample_ctas(uint32_t ns, uint32_t q) {
  return ns ? (ns + kSampleThreads * q - 1) / (kSampleThreads * q) : 1u;
}
// Sample size for the given targets (0: no sample, the whole set qualifies).
__host__ __device__ __forceinline__ uint64_t sample_size_raw(const RankSet &S, bool wide) {
  if (S.n <= kSample) return 0;
  uint64_t tmax = 0;
  for (int L = 0; L < kLists; L++)
    if (list_active(S, L) && list_target_of(S, L, wide) > tmax) tmax = list_target_of(S, L, wide);
  if (tmax == 0) return 0;
  return ((uint64_t)kSampleRank * S.n) / tmax;
}
// The narrow targets unless their sample would exceed the cap.
__host__ __device__ __forceinline__ bool wide_targets(const RankSet &S) { return sample_size_raw(S, false) > kSample; }
__host__ __device__ __forceinline__ uint64_t list_target(const RankSet &S, int L) {
  return list_target_of(S, L, wide_targets(S));
}
__host__ __device__ __forceinline__ uint32_t sample_size(const RankSet &S, uint32_t q) {
  uint64_t ns = umin64(sample_size_raw(S, wide_targets(S)), kSample);
  const uint32_t step = 8 * sample_ctas((uint32_t)ns, q);
  ns -= ns % step;  // whole runs, evenly split over the CTAs
  return (uint32_t)ns;
}

// 32-bit order-preserving summary of a list value v = key40 << 24 | low24:
// key40 >> 9 below the maximal key, and 2^31 | low24 on it (completed
// sessions all carry the maximal key, so only their index orders them).
// summary(a) <= summary(b) whenever a <= b; summary_floor(f) is the smallest
// list value whose summary is f.
__device__ __forceinline__ uint32_t summary_of(uint64_t v) {
  const uint64_t K = v >> 24;
  return K == kKeyMax40 ? (0x80000000u | (uint32_t)(v & kIdMask)) : (uint32_t)(K >> 9);
}
__device__ __forceinline__ uint64_t summary_floor(uint32_t f) {
  return (f & 0x80000000u) ? ((kKeyMax40 << 24) | (f & kIdMask)) : ((uint64_t)f << 33);
}

// Joint MSB-first radix select over the block, 8-bit digits: for every list
// L in `sel`, the value of rank need[L] (1 = largest) among the values
// v[L][q] whose bit L * Q + q of `has` is set (Q values per thread per list).
// All threads get the results in out[L].  Histograms and digit picks are
// double-buffered (hist[2][kLists][256], pick[2][2 * kLists]), so a pass
// takes two barriers.
template <int Q>
__device__ void joint_select32(const uint32_t (&v)[kLists][Q], uint32_t has, uint32_t sel,
                               const uint32_t (&need_in)[kLists], uint32_t (&out)[kLists],
                               unsigned int (*hist)[kLists][256], unsigned int (*pick)[2 * kLists]) {
  const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t need[kLists], prefix[kLists];
#pragma unroll
  for (int L = 0; L < kLists; L++) {
    need[L] = need_in[L];
    prefix[L] = 0;
  }
  for (uint32_t i = threadIdx.x; i < 2 * kLists * 256; i += blockDim.x) (&hist[0][0][0])[i] = 0;
  __syncthreads();
  for (int b = 3; b >= 0; b--) {
    const int pb = b & 1;
    const uint32_t mask = b == 3 ? 0u : (~0u << (8 * (b + 1)));
#pragma unroll
    for (int L = 0; L < kLists; L++) {
      if (!((sel >> L) & 1)) continue;  // block-uniform
#pragma unroll
      for (int q = 0; q < Q; q++) {
        const bool in = ((has >> (L * Q + q)) & 1) && (v[L][q] & mask) == prefix[L];
        const uint32_t d = (v[L][q] >> (8 * b)) & 0xFF;
        // lanes with the same digit add once per group
        const unsigned ain = __ballot_sync(kFull, in);
        if (in) {
          const unsigned grp = __match_any_sync(ain, d);
          if ((__ffs(grp) - 1) == (int)lane) atomicAdd(&hist[pb][L][d], (unsigned)__popc(grp));
        }
      }
    }
    __syncthreads();
    if (warp < (uint32_t)kLists && ((sel >> warp) & 1)) {
      // lane l owns digits 255-8l .. 248-8l (descending): find the digit where
      // the count of larger-or-equal values first reaches need
      const int L = warp;
      uint32_t nd = 0;
#pragma unroll
      for (int LL = 0; LL < kLists; LL++)
        if (LL == L) nd = need[LL];
      uint32_t c[8], tot = 0;
#pragma unroll
      for (int qq = 0; qq < 8; qq++) {
        c[qq] = hist[pb][L][255 - 8 * lane - qq];
        tot += c[qq];
      }
      uint32_t incl = tot;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(kFull, incl, o);
        if ((int)lane >= o) incl += y;
      }
      const uint32_t excl = incl - tot;
      const unsigned hit = __ballot_sync(kFull, excl < nd && incl >= nd);
      if ((int)lane == __ffs(hit) - 1) {
        uint32_t cum = excl;
#pragma unroll
        for (int qq = 0; qq < 8; qq++) {
          if (cum + c[qq] >= nd) {
            pick[pb][L] = 255 - 8 * lane - qq;
            pick[pb][kLists + L] = nd - cum;
            cum = 0xFFFFFFFFu;  // found: no later digit matches
            break;
          }
          cum += c[qq];
        }
      }
    }
    // the other histogram was last read before the barrier above: clear it
    // for the next pass
    for (uint32_t i = threadIdx.x; i < kLists * 256; i += blockDim.x) (&hist[pb ^ 1][0][0])[i] = 0;
    __syncthreads();
#pragma unroll
    for (int L = 0; L < kLists; L++) {
      if (!((sel >> L) & 1)) continue;
      prefix[L] |= pick[pb][L] << (8 * b);
      need[L] = pick[pb][kLists + L];
    }
  }
  __syncthreads();  // hist and pick free for the caller
#pragma unroll
  for (int L = 0; L < kLists; L++) out[L] = prefix[L];
}

// S.sctas <= kSampleCtas CTAs per set.  1. One sample per thread: run j of ns/8 covers
// stratum j (records [j n / (ns/8), (j+1) n / (ns/8))), 8 consecutive
// records at a hashed offset inside it.  2. Per list, each CTA keeps the top
// r_L summaries of its eligible samples (all of them when it has fewer).
// 3. The last CTA to finish selects the summary of rank r_L among those
// partial lists -- the rank-r_L summary of the whole sample -- and turns it
// into the list's threshold: the smallest list value with that summary (at
// least r_L samples reach it), plus, per turn index, the smallest gap whose
// key reaches the threshold's key (gA) or exceeds it (gB).
// Programmatic dependent launch: the filter is launched while the sample
// runs, and the finish while the filter runs.  A kernel lets its dependent
// start once all its CTAs are running (launch_dependents), and a dependent
// waits for its prerequisite grid to complete, with that grid's memory
// visible, before it reads what that grid wrote (wait).  Without the launch
// attribute both are no-ops.
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <int Q>
__global__ void __launch_bounds__(kSampleThreads) rank_sample_kernel(const RankSet *sets) {
  pdl_launch_dependents();
  const RankSet &S = sets[blockIdx.y];
  const uint32_t c = blockIdx.x;  // this CTA's share of the sample
  const uint32_t nct = S.sctas;
  if (c >= nct) return;           // the set needs fewer CTAs
  __shared__ uint64_t t2s[kLutN], mgs[kLutN];
  __shared__ unsigned int hist[2][kLists][256];
  __shared__ unsigned int pick[2][2 * kLists];
  __shared__ unsigned int ecount[kLists], wpos[kLists];
  __shared__ unsigned int is_last;
  const uint32_t tid = threadIdx.x, lane = tid & 31;
  if (tid < kLutN) {
    t2s[tid] = S.t2v[tid];
    mgs[tid] = S.mgv[tid];
  }
  if (tid < kLists) {
    ecount[tid] = 0;
    wpos[tid] = 0;
  }
  __syncthreads();
  const uint32_t ns = S.ns, act = S.act;
  const uint32_t per = ns / nct;  // samples of this CTA (<= 1024 Q, a multiple of 8)
  uint32_t rL[kLists];
#pragma unroll
  for (int L = 0; L < kLists; L++) rL[L] = S.rL[L];
  // 1. this thread's samples j = tid + 1024 q: run j / 8 of the CTA's share
  uint32_t f[kLists][Q];
  uint32_t m = 0;  // bit L * Q + q: sample q is eligible for list L
  // the sampled records' indices first, then all their loads at once (they
  // are independent random reads), then their keys
  uint32_t rr[Q];
  bool ok[Q];
#pragma unroll
  for (int q = 0; q < Q; q++) {
    const uint32_t jt = tid + kSampleThreads * q;
    ok[q] = jt < per;
    rr[q] = 0;
    if (ok[q]) {
      // stratum bounds floor(run n / nruns) with n = sq nruns + srem, in 32 bits
      const uint32_t nruns = S.nruns, run = c * (per / 8) + jt / 8, o = jt % 8;
      const uint32_t lo = run * S.sq + (run * S.srem) / nruns;
      const uint32_t hi = (run + 1) * S.sq + ((run + 1) * S.srem) / nruns;
      uint32_t h = run * 0x9E3779B1u;
      h ^= h >> 16;
      h *= 0x85EBCA6Bu;
      h ^= h >> 13;
      const uint32_t span = hi - lo - 8;  // strata hold at least 8 records
      rr[q] = lo + (h % (span + 1)) + o;
    }
  }
  uint8_t fl[Q], tr[Q];
  uint16_t tu[Q];
  uint32_t gg[Q];
#pragma unroll
  for (int q = 0; q < Q; q++) {  // index 0 for an unused slot: a valid record
    fl[q] = S.flags[rr[q]];
    tr[q] = S.tier[rr[q]];
    tu[q] = S.turn[rr[q]];
    gg[q] = S.gap[rr[q]];
  }
#pragma unroll
  for (int q = 0; q < Q; q++) {
#pragma unroll
    for (int L = 0; L < kLists; L++) f[L][q] = 0;
    if (ok[q]) {
      const uint32_t t = min((uint32_t)tu[q], kTMax);
      const uint64_t ck = ck_of(score_of(gg[q], t, (fl[q] & 2) != 0, t2s, mgs), rr[q]);
      const uint32_t em = elig_mask(fl[q], tr[q]) & act;
#pragma unroll
      for (int L = 0; L < kLists; L++) {
        f[L][q] = summary_of(list_val(ck, L));
        m |= ((em >> L) & 1u) << (L * Q + q);
      }
    }
  }
#pragma unroll
  for (int L = 0; L < kLists; L++) {
    uint32_t cnt = 0;
#pragma unroll
    for (int q = 0; q < Q; q++) cnt += __popc(__ballot_sync(kFull, (m >> (L * Q + q)) & 1));
    if (lane == 0 && cnt) atomicAdd(&ecount[L], cnt);
  }
  __syncthreads();
  // 2. per list: this CTA's top r_L (the summary of rank r_L, then the values
  // above it and enough copies of it)
  uint32_t sel = 0, need[kLists], T[kLists] = {0, 0, 0};
#pragma unroll
  for (int L = 0; L < kLists; L++) {
    need[L] = rL[L];
    if (rL[L] && ecount[L] > rL[L]) sel |= 1u << L;
  }
  if (sel) joint_select32<Q>(f, m, sel, need, T, hist, pick);
#pragma unroll
  for (int L = 0; L < kLists; L++) {
    if (!rL[L]) continue;
    const bool all = !((sel >> L) & 1);  // keep every eligible sample
    uint32_t *dst = S.part + ((size_t)L * kSampleCtas + c) * kMaxR;
#pragma unroll
    for (int q = 0; q < Q; q++) {
      const bool has = (m >> (L * Q + q)) & 1;
      const bool above = has && (all || f[L][q] > T[L]);
      const unsigned bal = __ballot_sync(kFull, above);
      unsigned wbase = 0;
      if (lane == 0 && bal) wbase = atomicAdd(&wpos[L], (unsigned)__popc(bal));
      wbase = __shfl_sync(kFull, wbase, 0);
      if (above) dst[wbase + __popc(bal & ((1u << lane) - 1))] = f[L][q];
    }
  }
  __syncthreads();
  // ties at the rank-r_L summary fill each partial list up to r_L entries
#pragma unroll
  for (int L = 0; L < kLists; L++) {
    if (!rL[L]) continue;
    const bool all = !((sel >> L) & 1);
    const uint32_t nab = wpos[L], total = all ? nab : rL[L];
    uint32_t *dst = S.part + ((size_t)L * kSampleCtas + c) * kMaxR;
    for (uint32_t q = nab + tid; q < total; q += kSampleThreads) dst[q] = T[L];
    if (tid == 0) S.part_n[L * kSampleCtas + c] = total;
  }
  // 3. the last CTA to finish merges the partial lists and sets the thresholds
  __threadfence();
  __syncthreads();
  if (tid == 0) is_last = (atomicAdd(&S.work->sticket, 1u) == nct - 1);
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  // entry counts of the partial lists, then kSampleCtas * r_L <= 4096
  // entries per list: one per thread when they fit, else four per thread
  __shared__ unsigned int pn[kLists * kSampleCtas];
  if (tid < kLists * kSampleCtas) pn[tid] = (tid % kSampleCtas) < nct ? __ldcg(&S.part_n[tid]) : 0u;
  __syncthreads();
  uint32_t rmax = 0, sel2 = 0;
#pragma unroll
  for (int L = 0; L < kLists; L++) {
    rmax = max(rmax, rL[L]);
    if (!rL[L]) continue;
    uint32_t cnt = 0;
    for (uint32_t cc = 0; cc < kSampleCtas; cc++) cnt += pn[L * kSampleCtas + cc];
    if (cnt >= rL[L]) sel2 |= 1u << L;
  }
  uint32_t T2[kLists] = {0, 0, 0};
  auto merge = [&](auto qtag) {
    constexpr int QM = decltype(qtag)::value;
    uint32_t vq[kLists][QM];
    uint32_t hq = 0;
#pragma unroll
    for (int L = 0; L < kLists; L++) {
#pragma unroll
      for (int q = 0; q < QM; q++) {
        vq[L][q] = 0;
        // entry e of the concatenation: CTA e / r_L, slot e % r_L
        const uint32_t e = tid + kSampleThreads * q;
        if (!rL[L]) continue;
        const uint32_t cc = e / rL[L], slot = e % rL[L];
        if (cc < nct && slot < pn[L * kSampleCtas + cc]) {
          vq[L][q] = __ldcg(&S.part[((size_t)L * kSampleCtas + cc) * kMaxR + slot]);
          hq |= 1u << (L * QM + q);
        }
      }
    }
    joint_select32<QM>(vq, hq, sel2, rL, T2, hist, pick);
  };
  if (sel2) {
    if (nct * rmax <= kSampleThreads) merge(std::integral_constant<int, 1>());
    else merge(std::integral_constant<int, 4>());
  }
#pragma unroll
  for (int L = 0; L < kLists; L++) {
    // 0 (fewer than r_L eligible samples, or none taken): accept every eligible record
    const uint64_t thrv = ((sel2 >> L) & 1) ? summary_floor(T2[L]) : 0ull;
    if (tid == 0) {
      S.thr[L] = thrv;
      S.thr[kLists + L] = (act >> L) & 1;
    }
    if (tid < kLutN) {
      const uint64_t thr_ck = (L == 2) ? ~thrv : thrv;
      const uint64_t K = thr_ck >> 24;
      S.gthr[L * kLutN + tid] = make_uint2(g_at_least(K, S.sigma[tid], t2s[tid]), g_at_least(K + 1, S.sigma[tid], t2s[tid]));
    }
  }
}

// ------------------------------------------------------------- filter ----
__device__ __forceinline__ int set_of_tile(const RankSet *sets, int n_sets, uint32_t tile) {
  int lo = 0, hi = n_sets - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (sets[mid].tile0 <= tile) lo = mid; else hi = mid - 1;
  }
  return lo;
}

struct SetConst {
  uint32_t loV, loD, loP;      // index thresholds of the tie on the threshold key
  uint32_t dV, dD;             // completed records pass V / D iff lo >= dV / dD
  int32_t dP;                  // completed records pass P iff lo <= dP
  uint32_t act;                // active lists (bit L)
};

// ---- TMA 1-D bulk copies and mbarriers (inline PTX, sm_90+) ----
__device__ __forceinline__ uint32_t smem_addr(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}
__device__ __forceinline__ void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Bounded wait on an mbarrier phase; false when the bound ran out.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity) {
  for (uint32_t it = 0; it < (1u << 22); it++)
    if (mbar_try_wait(bar, parity)) return true;
  return false;
}

#ifndef UNISON_FILTER_STAGES
#define UNISON_FILTER_STAGES 2
#endif
#ifndef UNISON_FILTER_REC
#define UNISON_FILTER_REC 16
#endif
#ifndef UNISON_FILTER_CONSUMERS
#define UNISON_FILTER_CONSUMERS 256
#endif
#ifndef UNISON_FILTER_MINBLOCKS
#define UNISON_FILTER_MINBLOCKS 3
#endif
constexpr int kStages = UNISON_FILTER_STAGES;          // tiles in flight per CTA
constexpr uint32_t kRec = UNISON_FILTER_REC;           // records per consumer thread per tile
constexpr uint32_t kConsumers = UNISON_FILTER_CONSUMERS;  // consumer threads
constexpr uint32_t kBigTile = kConsumers * kRec;      // 4096 records per tile
constexpr uint32_t kGroups = kRec / 4;                 // groups of four records per thread
constexpr uint32_t kGroupStride = kConsumers * 4;      // records between a thread's groups
constexpr uint32_t kWarpBuf = 128;                     // flagged records a warp tests per pass
static_assert(kRec % 4 == 0 && kRec <= 32, "records per thread: a multiple of 4, at most 32");
static_assert(kConsumers >= kLutN * 5, "one consumer thread per bound-table entry");
constexpr uint32_t kFilterCtaThreads = kConsumers + 32;  // + one producer warp
struct __align__(128) FilterStage {
  uint32_t gap[kBigTile];
  uint16_t turn[kBigTile];
  uint8_t flags[kBigTile];
  uint8_t tier[kBigTile];
};
constexpr size_t kFilterSmem = sizeof(FilterStage) * kStages;

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
// Barrier 1 over the consumer warps only (the producer warp never joins it).
__device__ __forceinline__ void consumers_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kConsumers) : "memory"); }
// Barrier 1 with an OR reduction of p over the consumer threads.
__device__ __forceinline__ bool consumers_sync_or(bool p) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred pi, po;\n setp.ne.u32 pi, %1, 0;\n bar.red.or.pred po, 1, %2, pi;\n selp.u32 %0, 1, 0, po;\n}"
      : "=r"(r)
      : "r"((uint32_t)p), "n"(kConsumers)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ int set_of(const RankSet *sets, int si, uint32_t tile) {
  while (tile >= sets[si].tile0 + sets[si].ntiles) si++;
  return si;
}

// Thresholds of one set into shared memory (consumer threads call it).  Per
// turn index: vd = (gA_V, gB_V, gA_D, gB_D), pp = (gA_P, gB_P); an inactive
// list gets bounds no gap passes.
__device__ void load_set(const RankSet &S, uint4 *vd, uint2 *pp, uint64_t *t2s, uint64_t *mgs, SetConst &c) {
  consumers_sync();  // everyone is done with the previous set's tables
  const bool aV = S.thr[kLists + 0] != 0, aD = S.thr[kLists + 1] != 0, aP = S.thr[kLists + 2] != 0;
  if (threadIdx.x < kLutN) {
    const uint32_t t = threadIdx.x;
    const uint2 a0 = S.gthr[t], a1 = S.gthr[kLutN + t], a2 = S.gthr[2 * kLutN + t];
    vd[t] = make_uint4(aV ? a0.x : kFull, aV ? a0.y : kFull, aD ? a1.x : kFull, aD ? a1.y : kFull);
    pp[t] = aP ? a2 : make_uint2(0u, 0u);
    t2s[t] = S.t2v[t];
    mgs[t] = S.mgv[t];
  }
  if (threadIdx.x == 32) {
    uint32_t lo[kLists], dok[kLists];
#pragma unroll
    for (int L = 0; L < kLists; L++) {
      const uint64_t thrv = S.thr[L];
      const uint64_t thr_ck = (L == 2) ? ~thrv : thrv;
      const uint64_t K = thr_ck >> 24;
      lo[L] = (uint32_t)(thr_ck & kIdMask);
      // a completed record has the maximal key 2^40 - 1: 2 = always passes,
      // 1 = passes on the index part, 0 = never
      dok[L] = (L == 2) ? (kKeyMax40 == K ? 1u : 0u) : (kKeyMax40 > K ? 2u : (kKeyMax40 == K ? 1u : 0u));
    }
    c.loV = lo[0];
    c.loD = lo[1];
    c.loP = lo[2];
    c.dV = !aV ? 0x1000000u : (dok[0] == 2 ? 0u : (dok[0] == 1 ? lo[0] : 0x1000000u));
    c.dD = !aD ? 0x1000000u : (dok[1] == 2 ? 0u : (dok[1] == 1 ? lo[1] : 0x1000000u));
    c.dP = (aP && dok[2] == 1) ? (int32_t)lo[2] : -1;
    c.act = (aV ? 1u : 0u) | (aD ? 2u : 0u) | (aP ? 4u : 0u);
  }
  consumers_sync();
}

// Persistent streaming pass.  Each CTA takes every gridDim-th tile; its
// producer warp keeps kStages tiles in flight with TMA bulk copies into
// shared memory ("full" barriers), and its consumer warps copy each tile to
// registers, hand the stage back ("empty" barriers) and test every record
// against the set's thresholds.  Every wait is bounded; a CTA that gives up records
// UNISON_ERR_TIMEOUT, lets its own copies land (bounded) and returns.
__global__ void __launch_bounds__(kFilterCtaThreads, UNISON_FILTER_MINBLOCKS) rank_filter_kernel(const RankSet *sets, int n_sets,
                                                                        uint32_t total_tiles, int grouped) {
  pdl_launch_dependents();
  extern __shared__ __align__(128) unsigned char fsm[];
  FilterStage *stage = reinterpret_cast<FilterStage *>(fsm);
  __shared__ __align__(8) uint64_t full[kStages], empty[kStages];
  __shared__ uint4 vd[kLutN];
  __shared__ uint2 pp[kLutN];
  __shared__ uint64_t t2s[kLutN], mgs[kLutN];
  __shared__ uint2 ftab[kLutN * 5];
  __shared__ SetConst cset;
  __shared__ uint16_t wbuf[kConsumers / 32][kWarpBuf];  // per consumer warp: flagged records' offsets
  // Tiles are dealt round-robin, so the CTAs stream neighbouring tiles at any
  // moment, and the tiles whose records pass a threshold -- they cluster by
  // index, since ties on a key go to the smaller index -- spread over CTAs.
  // Grouped: set s owns CTAs [cta0, cta0 + nctas), which deal its tiles among
  // themselves (each CTA then loads one set's thresholds once).  Otherwise
  // (more sets than CTAs) the CTAs deal every set's tiles in one sequence.
  uint32_t t_begin, t_step, t_end;
  int si0;
  if (grouped) {
    int lo = 0, hi = n_sets - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (sets[mid].cta0 <= blockIdx.x) lo = mid; else hi = mid - 1;
    }
    si0 = lo;
    const RankSet &S = sets[si0];
    t_begin = S.tile0 + (blockIdx.x - S.cta0);
    t_step = S.nctas;
    t_end = S.tile0 + S.ntiles;
    if (blockIdx.x >= S.cta0 + S.nctas) return;
  } else {
    t_begin = blockIdx.x;
    t_step = gridDim.x;
    t_end = total_tiles;
    si0 = -1;
  }
  if (t_begin >= t_end) return;
  if (threadIdx.x == 0) {
    for (int q = 0; q < kStages; q++) {
      mbar_init(&full[q], 1);
      mbar_init(&empty[q], kConsumers / 32);
    }
    fence_mbar_init();
  }
  __syncthreads();
  if (si0 < 0) si0 = set_of_tile(sets, n_sets, t_begin);
  const int lane = threadIdx.x & 31;

  if (threadIdx.x >= kConsumers) {
    // ---------------- producer warp (one lane issues)
    if (lane != 0) return;
    int si = si0;
    uint32_t fills[kStages] = {};  // bulk copies issued into each stage (one full-barrier phase each)
    uint32_t issued = 0;           // bit q: the last copy into stage q may still be in flight
    bool failed = false;
    for (uint32_t i = 0, tile = t_begin; tile < t_end; i++, tile += t_step) {
      const int q = (int)(i % kStages);
      if (i >= (uint32_t)kStages) {
        // wait until the consumers released this stage's previous tile
        if (!mbar_wait_bounded(&empty[q], ((i / kStages) - 1) & 1)) {
          failed = true;
          break;
        }
        issued &= ~(1u << q);
      }
      si = set_of(sets, si, tile);
      const RankSet &T = sets[si];
      const uint32_t base = (tile - T.tile0) * kBigTile;
      if (base + kBigTile > T.n) continue;  // the partial last tile is read directly
      FilterStage &d = stage[q];
      fence_proxy_async();
      mbar_expect_tx(&full[q], kBigTile * 8);
      bulk_g2s(d.gap, T.gap + base, kBigTile * 4, &full[q]);
      bulk_g2s(d.turn, T.turn + base, kBigTile * 2, &full[q]);
      bulk_g2s(d.flags, T.flags + base, kBigTile, &full[q]);
      bulk_g2s(d.tier, T.tier + base, kBigTile, &full[q]);
      issued |= 1u << q;
      fills[q]++;
    }
    if (failed) {
      atomicExch(&sets[si0].work->status, (unsigned int)UNISON_ERR_TIMEOUT);
      // consumers that still wait will time out too; let this CTA's copies land
      // (phase fills-1 of each stage's full barrier) before the CTA exits
      for (int q = 0; q < kStages; q++)
        if ((issued >> q) & 1) mbar_wait_bounded(&full[q], (fills[q] - 1) & 1);
    }
    return;
  }

  // ---------------- consumer warps
  // The producer streams records (inputs) at once; the consumers first wait
  // for the sample's thresholds.
  pdl_wait();
  // Consumer thread ct owns, in each tile, kGroups groups of four consecutive
  // records, group gi starting at record gi * kGroupStride + 4 * ct: every
  // shared-memory read of the stage is lane-contiguous (no bank conflicts).
  const uint32_t ct = threadIdx.x;
  int si = si0;
  SetConst &c = cset;  // this set's constants, in shared memory
  uint32_t fph = 0;  // bit q: parity of the next full-barrier phase of stage q (flips per bulk tile)
  // this set's hot descriptor fields, cached when the set changes (pointers
  // used only on rare paths are read from the descriptor there)
  uint32_t s_n = 0, s_tile0 = 0, s_end = 0;
  bool s_keys = false;
  // Segment: a run of tiles over which every index condition of the set has
  // one class (all, none or mixed).  Within a set each condition changes class
  // at most twice (at the tile holding its boundary and the one after), so a
  // set has at most 13 segments.
  uint32_t seg_end = 0;  // first tile of the next segment
  bool seg_mixed = false, seg_none = false;
  for (uint32_t i = 0, tile = t_begin; tile < t_end; i++, tile += t_step) {
    const int q = (int)(i % kStages);
    if (i == 0 || tile >= s_end) {
      si = set_of(sets, si, tile);
      const RankSet &S = sets[si];
      load_set(S, vd, pp, t2s, mgs, c);
      s_n = S.n;
      s_tile0 = S.tile0;
      s_end = S.tile0 + S.ntiles;
      s_keys = S.keys != nullptr;
      seg_end = tile;  // force a new segment
    }
    const uint32_t tb = (tile - s_tile0) * kBigTile;
    if (tile >= seg_end) {
      // Index conditions over this tile: record indices rise through the
      // tile, so lo = ~index falls from lo_hi to lo_lo and each tie condition
      // on lo holds for all, none or a part of the tile.
      const uint32_t tcount = min(kBigTile, s_n - tb);
      const uint32_t lo_hi = (~tb) & kIdMask, lo_lo = (~(tb + tcount - 1)) & kIdMask;
      // 0 none, 1 all, 2 mixed
      auto ge_class = [&](uint32_t x) { return lo_lo >= x ? 1u : (lo_hi < x ? 0u : 2u); };                   // lo >= x
      auto le_class = [&](int64_t x) { return (int64_t)lo_hi <= x ? 1u : ((int64_t)lo_lo > x ? 0u : 2u); };  // lo <= x
      const uint32_t iV = ge_class(c.loV), iD = ge_class(c.loD), iP = le_class((int64_t)c.loP);
      const uint32_t dV = ge_class(c.dV), dD = ge_class(c.dD), dP = le_class((int64_t)c.dP);
      seg_mixed = ((c.act & 1) && (iV == 2 || dV == 2)) || ((c.act & 2) && (iD == 2 || dD == 2)) ||
                  ((c.act & 4) && (iP == 2 || dP == 2));
      // next tile where a condition can change class: lo >= x holds for
      // indices up to kIdMask - x, lo <= x from kIdMask - x on; the change
      // points are the tile holding that index and the tile after it
      const uint32_t r = tile - s_tile0;
      uint32_t nxt = s_end - s_tile0;
      auto upd = [&](int64_t lo_bound) {
        const int64_t b = (int64_t)kIdMask - lo_bound;
        if (b < 0 || b >= (int64_t)s_n) return;
        const uint32_t tbnd = (uint32_t)b / kBigTile;
        if (tbnd > r) nxt = min(nxt, tbnd);
        else if (tbnd + 1 > r) nxt = min(nxt, tbnd + 1);
      };
      upd(c.loV); upd(c.loD); upd(c.loP); upd(c.dV); upd(c.dD); upd(c.dP);
      seg_end = s_tile0 + nxt;
      // Per-segment bound table over (turn index, record class): a record of
      // class cls at turn index t may be a candidate of some list iff
      // g >= x or g < y.  Classes: 0 not eligible, 1 live fast tier, 2 live
      // HBM tier, 3 completed fast tier, 4 completed HBM tier.
      consumers_sync();  // everyone is done with the previous table
      bool live = false;
      if (!seg_mixed && ct < kLutN * 5) {
        const uint32_t t = ct / 5, cls = ct % 5;
        const uint4 a = vd[t];
        const uint2 bb = pp[t];
        const uint32_t bV = iV == 1 ? a.x : a.y, bD = iD == 1 ? a.z : a.w, bP = iP == 1 ? bb.y : bb.x;
        const bool pdV = (c.act & 1) && dV == 1, pdD = (c.act & 2) && dD == 1, pdP = (c.act & 4) && dP == 1;
        uint2 e = make_uint2(kFull, 0u);
        if (cls == 1) e = make_uint2(min(bV, bD), 0u);
        if (cls == 2) e = make_uint2(bV, bP);
        if (cls == 3) e = make_uint2(pdV || pdD ? 0u : kFull, 0u);
        if (cls == 4) e = make_uint2(pdV ? 0u : kFull, pdP ? kFull : 0u);
        ftab[ct] = e;
        // gaps are below 2^31: x >= 2^31 and y == 0 admit nothing
        live = e.x < 0x80000000u || e.y != 0u;
      }
      seg_none = !consumers_sync_or(live) && !seg_mixed;
    }
    const bool bulk = tb + kBigTile <= s_n;
    uint32_t g[kRec], tw[kRec / 2], fw[kGroups], rw[kGroups];
    if (bulk) {
      // a timed-out wait is reported, not collective: every wait here is
      // bounded, so the CTA still ends (with undefined results)
      if (!mbar_wait_bounded(&full[q], (fph >> q) & 1))
        atomicExch(&sets[si0].work->status, (unsigned int)UNISON_ERR_TIMEOUT);
      fph ^= 1u << q;
      const FilterStage &d = stage[q];
#pragma unroll
      for (int gi = 0; gi < (int)kGroups; gi++) {
        const uint32_t o = gi * kGroupStride + 4 * ct;
        const uint4 gq = *reinterpret_cast<const uint4 *>(d.gap + o);
        g[4 * gi] = gq.x; g[4 * gi + 1] = gq.y; g[4 * gi + 2] = gq.z; g[4 * gi + 3] = gq.w;
        const uint2 tq = *reinterpret_cast<const uint2 *>(d.turn + o);
        tw[2 * gi] = tq.x; tw[2 * gi + 1] = tq.y;
        fw[gi] = *reinterpret_cast<const uint32_t *>(d.flags + o);
        rw[gi] = *reinterpret_cast<const uint32_t *>(d.tier + o);
      }
    } else {
      const RankSet &S = sets[si];
      const uint32_t *s_gap = S.gap;
      const uint16_t *s_turn = S.turn;
      const uint8_t *s_flags = S.flags, *s_tier = S.tier;
#pragma unroll
      for (int gi = 0; gi < (int)kGroups; gi++) {
        tw[2 * gi] = tw[2 * gi + 1] = 0;
        fw[gi] = 0x01010101u;  // padding reads as pinned: never eligible
        rw[gi] = 0;
#pragma unroll
        for (uint32_t m = 0; m < 4; m++) {
          const uint32_t idx = tb + gi * kGroupStride + 4 * ct + m;
          g[4 * gi + m] = 0;
          if (idx < s_n) {
            g[4 * gi + m] = s_gap[idx];
            tw[2 * gi + (m >> 1)] |= (uint32_t)s_turn[idx] << (16 * (m & 1));
            const uint32_t sh = 8 * m;
            fw[gi] = (fw[gi] & ~(0xFFu << sh)) | ((uint32_t)s_flags[idx] << sh);
            rw[gi] = (rw[gi] & ~(0xFFu << sh)) | ((uint32_t)s_tier[idx] << sh);
          }
        }
      }
    }
    auto turn_of = [&](uint32_t k) { return min((tw[k >> 1] >> (16 * (k & 1))) & 0xFFFF, kTMax); };
    auto index_of = [&](uint32_t k) { return tb + (k >> 2) * kGroupStride + 4 * ct + (k & 3); };
    // 1. candidate bit per record (any list): one table lookup per record
    uint32_t cm = 0;
    if (seg_mixed) {
      // index conditions vary inside the tile: flag the records that pass
      // some list exactly
#pragma unroll
      for (uint32_t k = 0; k < kRec; k++) {
        const uint32_t sh = 8 * (k & 3);
        const uint32_t fl = (fw[k >> 2] >> sh) & 0xFF, tr = (rw[k >> 2] >> sh) & 0xFF;
        const uint32_t em = elig_mask((uint8_t)fl, (uint8_t)tr);
        const bool done = (fl & 2) != 0;
        const uint32_t gg = g[k], t = turn_of(k), lo = (~index_of(k)) & kIdMask;
        const uint4 a = vd[t];
        const uint2 b = pp[t];
        const bool pV = (em & 1) && (done ? lo >= c.dV : (gg >= a.y || (gg >= a.x && lo >= c.loV)));
        const bool pD = (em & 2) && (done ? lo >= c.dD : (gg >= a.w || (gg >= a.z && lo >= c.loD)));
        const bool pP = (em & 4) && (done ? (int32_t)lo <= c.dP : (gg < b.x || (gg < b.y && lo <= c.loP)));
        cm |= (uint32_t)(pV || pD || pP) << k;
      }
    } else if (!seg_none) {
      const unsigned char *tab = reinterpret_cast<const unsigned char *>(ftab);
#pragma unroll
      for (int gi = 0; gi < (int)kGroups; gi++) {
        // class * 8 per record, four records per word (SWAR)
        const uint32_t unp = __vcmpeq4(fw[gi] & 0x01010101u, 0u);
        const uint32_t isS = __vcmpeq4(rw[gi], 0x01010101u), isH = __vcmpeq4(rw[gi], 0x02020202u);
        const uint32_t dn = __vcmpne4(fw[gi] & 0x02020202u, 0u);
        const uint32_t c8 = (unp & ((isS & 0x08080808u) | (isH & 0x10101010u))) +
                            (unp & dn & (isS | isH) & 0x10101010u);
#pragma unroll
        for (uint32_t m = 0; m < 4; m++) {
          const uint32_t k = 4 * gi + m;
          const uint2 e = *reinterpret_cast<const uint2 *>(tab + turn_of(k) * 40 + ((c8 >> (8 * m)) & 0xFF));
          cm |= (uint32_t)(g[k] >= e.x || g[k] < e.y) << k;
        }
      }
    }
    // every record's key, when asked for (from registers)
    if (s_keys) {
      uint64_t *keys = sets[si].keys;
#pragma unroll
      for (uint32_t k = 0; k < kRec; k++) {
        const uint32_t idx = index_of(k);
        if (idx < s_n) {
          const bool dn = (fw[k >> 2] >> (8 * (k & 3) + 1)) & 1;
          keys[idx] = score_of(g[k], turn_of(k), dn, t2s, mgs);
        }
      }
    }
    // The stage is handed back to the producer as soon as this warp no longer
    // reads it: at once when none of its records is flagged, else after the
    // exact tests below, which read the flagged records back from the stage.
    const bool flagged = __any_sync(kFull, cm != 0);
    if (!flagged) {
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[q]);
      continue;
    }
    // 2. exact per-list tests of the flagged records: the warp lists their
    // offsets in the tile (kWarpBuf a pass), then each lane tests one and
    // appends its exact value to every list it passes (one atomic per warp
    // and list).
    uint16_t *wb = wbuf[ct >> 5];
    const FilterStage &d = stage[q];
    const RankSet &S = sets[si];
    uint32_t rem = cm;
    while (__any_sync(kFull, rem != 0)) {
      const uint32_t mine = __popc(rem);
      uint32_t incl = mine;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += y;
      }
      const uint32_t nb = min(__shfl_sync(kFull, incl, 31), kWarpBuf);
      uint32_t pos = incl - mine, wrote = 0;
#pragma unroll
      for (uint32_t k = 0; k < kRec; k++) {
        if ((rem >> k) & 1) {
          if (pos < kWarpBuf) {
            wb[pos] = (uint16_t)((k >> 2) * kGroupStride + 4 * ct + (k & 3));
            wrote |= 1u << k;
          }
          pos++;
        }
      }
      rem &= ~wrote;
      __syncwarp();
      for (uint32_t j0 = 0; j0 < nb; j0 += 32) {
        const uint32_t j = j0 + lane;
        bool pL[kLists] = {false, false, false};
        uint64_t ck = 0;
        if (j < nb) {
          const uint32_t o = wb[j], idx = tb + o;
          uint32_t gg, t, fl, tr;
          if (bulk) {
            gg = d.gap[o];
            t = d.turn[o];
            fl = d.flags[o];
            tr = d.tier[o];
          } else {  // the partial last tile: read from the set (padding is pinned)
            const bool in = idx < s_n;
            gg = in ? S.gap[idx] : 0u;
            t = in ? S.turn[idx] : 0u;
            fl = in ? S.flags[idx] : 1u;
            tr = in ? S.tier[idx] : 0u;
          }
          t = min(t, kTMax);
          const uint32_t em = elig_mask((uint8_t)fl, (uint8_t)tr);
          const bool done = (fl & 2) != 0;
          const uint32_t lo = (~idx) & kIdMask;
          const uint4 a = vd[t];
          const uint2 b = pp[t];
          pL[0] = (em & 1) && (done ? lo >= c.dV : (gg >= a.y || (gg >= a.x && lo >= c.loV)));
          pL[1] = (em & 2) && (done ? lo >= c.dD : (gg >= a.w || (gg >= a.z && lo >= c.loD)));
          pL[2] = (em & 4) && (done ? (int32_t)lo <= c.dP : (gg < b.x || (gg < b.y && lo <= c.loP)));
          if (pL[0] || pL[1] || pL[2]) ck = ck_of(score_of(gg, t, done, t2s, mgs), idx);
        }
#pragma unroll
        for (int L = 0; L < kLists; L++) {
          const unsigned bal = __ballot_sync(kFull, pL[L]);
          if (!bal) continue;
          unsigned base = 0;
          if (lane == 0) base = atomicAdd(&S.work->cand[L], (unsigned)__popc(bal));
          base = __shfl_sync(kFull, base, 0);
          const uint32_t at = base + __popc(bal & ((1u << lane) - 1));
          if (pL[L] && at < kCandCap) S.cand[(size_t)L * kCandCap + at] = list_val(ck, L);
        }
      }
      __syncwarp();  // the buffer is rewritten by the next pass
    }
    if (lane == 0) mbar_arrive(&empty[q]);
  }
}

// ------------------------------------------------------------- finish ----
constexpr uint32_t kIpt = kMaxSel / kFinishThreads;  // fill items per thread
static_assert(kMaxSel % kFinishThreads == 0 && kFinishThreads == 1024, "fill scan layout");

// Byte sums of up to 4096 moves reach 2^70: kept as lo + 2^64 hi.
struct Sum {
  uint64_t lo;
  uint32_t hi;
};
__device__ __forceinline__ Sum sum_add(Sum x, Sum y) {
  const uint64_t lo = x.lo + y.lo;
  return Sum{lo, x.hi + y.hi + (lo < x.lo ? 1u : 0u)};
}
__device__ __forceinline__ bool sum_le(Sum x, uint64_t cap) { return x.hi == 0 && x.lo <= cap; }
__device__ __forceinline__ Sum shfl_up_sum(Sum x, int o) {
  return Sum{__shfl_up_sync(kFull, x.lo, o), __shfl_up_sync(kFull, x.hi, o)};
}

// Block-wide inclusive prefix sums over items j = kIpt * tid + i of a and b.
__device__ void block_scan_pairs(Sum (&a)[kIpt], int64_t (&b)[kIpt], Sum *wa, int64_t *wb) {
  const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (uint32_t i = 1; i < kIpt; i++) {
    a[i] = sum_add(a[i], a[i - 1]);
    b[i] += b[i - 1];
  }
  Sum ia = a[kIpt - 1];
  int64_t ib = b[kIpt - 1];
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const Sum ya = shfl_up_sum(ia, o);
    const int64_t yb = __shfl_up_sync(kFull, ib, o);
    if ((int)lane >= o) {
      ia = sum_add(ia, ya);
      ib += yb;
    }
  }
  Sum ea = shfl_up_sum(ia, 1);
  int64_t eb = __shfl_up_sync(kFull, ib, 1);
  if (lane == 0) {
    ea = Sum{0, 0};
    eb = 0;
  }
  if (lane == 31) {
    wa[warp] = ia;
    wb[warp] = ib;
  }
  __syncthreads();
  if (warp == 0) {
    Sum xa = wa[lane];
    int64_t xb = wb[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const Sum ya = shfl_up_sum(xa, o);
      const int64_t yb = __shfl_up_sync(kFull, xb, o);
      if ((int)lane >= o) {
        xa = sum_add(xa, ya);
        xb += yb;
      }
    }
    const Sum pa = shfl_up_sum(xa, 1);
    const int64_t pb = __shfl_up_sync(kFull, xb, 1);
    __syncwarp();
    wa[lane] = lane ? pa : Sum{0, 0};
    wb[lane] = lane ? pb : 0ll;
  }
  __syncthreads();
  const Sum oa = sum_add(wa[warp], ea);
  const int64_t ob = wb[warp] + eb;
#pragma unroll
  for (uint32_t i = 0; i < kIpt; i++) {
    a[i] = sum_add(a[i], oa);
    b[i] += ob;
  }
  __syncthreads();  // wa, wb free again
}

// Exact top-M of list L over the whole set by one CTA, streaming records and
// keeping a pool of at most M + 4096 values (the fallback path).
__device__ uint32_t stream_topM(const RankSet &S, int L, uint32_t M, uint64_t *pool, const uint64_t *t2s,
                                const uint64_t *mgs, unsigned int (*hist)[256], unsigned int (*pick)[2],
                                unsigned long long *bcast, unsigned int *cnt) {
  if (threadIdx.x == 0) *cnt = 0;
  uint64_t floorv = 0;  // accept values strictly above (0 = accept all but 0)
  bool have_floor = false;
  __syncthreads();
  for (uint32_t b = 0; b < S.n; b += 4 * blockDim.x) {
    for (uint32_t q = 0; q < 4; q++) {
      const uint32_t r = b + q * blockDim.x + threadIdx.x;
      if (r < S.n) {
        const uint32_t m = elig_mask(S.flags[r], S.tier[r]);
        if ((m >> L) & 1) {
          const uint32_t t = min((uint32_t)S.turn[r], kTMax);
          const uint64_t v = list_val(ck_of(score_of(S.gap[r], t, (S.flags[r] & 2) != 0, t2s, mgs), r), L);
          if (!have_floor || v > floorv) {
            const uint32_t pos = atomicAdd(cnt, 1u);
            if (pos < kSmemCand) pool[pos] = v;
          }
        }
      }
    }
    __syncthreads();
    const uint32_t c = min(*cnt, kSmemCand);
    if (c > M) {
      const uint64_t th = block_select_rank([&](uint32_t i) { return pool[i]; }, c, M, hist, pick, bcast);
      // compact in place: values >= th (exactly M, values are unique)
      __syncthreads();
      if (threadIdx.x == 0) *cnt = 0;
      __syncthreads();
      // two-step compaction through registers to avoid overwriting unread values
      uint64_t keep[8];
      uint32_t nk = 0;
      for (uint32_t i = threadIdx.x; i < c; i += blockDim.x) {
        const uint64_t v = pool[i];
        if (v >= th && nk < 8) keep[nk++] = v;
      }
      __syncthreads();
      for (uint32_t i = 0; i < nk; i++) pool[atomicAdd(cnt, 1u)] = keep[i];
      __syncthreads();
      floorv = th;
      have_floor = true;
    }
    __syncthreads();
  }
  __syncthreads();
  return min(*cnt, M);
}

__global__ void __launch_bounds__(kFinishThreads) rank_finish_kernel(const RankSet *sets) {
  pdl_wait();  // candidates and counts come from the filter
  const RankSet &S = sets[blockIdx.y];
  const int L = blockIdx.x;  // this CTA's list
  extern __shared__ __align__(16) unsigned char smem[];
  uint64_t *buf = reinterpret_cast<uint64_t *>(smem);   // [kSmemCand]
  uint64_t *sel = buf + kSmemCand;                      // [kMaxSel]
  __shared__ uint64_t t2s[kLutN], mgs[kLutN];
  __shared__ unsigned int hist[2][256];
  __shared__ unsigned int pick[2][2];
  __shared__ unsigned long long bcast[2];
  __shared__ __align__(8) uint64_t cbar;
  __shared__ unsigned int cnt, is_last;
  if (threadIdx.x < kLutN) {
    t2s[threadIdx.x] = S.t2v[threadIdx.x];
    mgs[threadIdx.x] = S.mgv[threadIdx.x];
  }
  __syncthreads();
  {
    const bool active = S.thr[kLists + L] != 0;
    const uint32_t Mw = (L == 0) ? S.k : S.max_moves;
    const uint32_t emitted = S.work->cand[L];
    // Candidates are every eligible record at or beyond the threshold.  They
    // certify the top Mw when there are at least Mw of them, or when the
    // threshold admitted every eligible record; otherwise (or when the buffer
    // overflowed) the list is re-selected exactly from the whole set.
    const bool all_admitted = S.thr[L] == 0;
    const bool certified = emitted <= kCandCap && (emitted >= Mw || all_admitted);
    const uint32_t M = !active ? 0u : (certified ? min(Mw, emitted) : Mw);
    uint32_t got = 0;
    if (M > 0) {
      const uint64_t *cand = S.cand + (size_t)L * kCandCap;
      if (certified) {
        const uint32_t c = emitted;
        const uint64_t *src = cand;
        if (c <= kSmemCand) {
          // one bulk copy (an even count: 16-byte multiple; the buffer holds
          // kCandCap >= c + 1 entries)
          const uint32_t bytes = ((c + 1) & ~1u) * 8u;
          if (threadIdx.x == 0) {
            mbar_init(&cbar, 1);
            fence_mbar_init();
            mbar_expect_tx(&cbar, bytes);
            bulk_g2s(buf, cand, bytes, &cbar);
          }
          __syncthreads();
          if (!mbar_wait_bounded(&cbar, 0)) {
            atomicExch(&S.work->status, (unsigned int)UNISON_ERR_TIMEOUT);
            mbar_wait_bounded(&cbar, 0);  // let the copy land before the buffer is reused
          }
          src = buf;
        }
        uint64_t th = 0;
        if (c > M) th = block_select_rank([&](uint32_t i) { return src[i]; }, c, M, hist, pick, bcast);
        if (threadIdx.x == 0) cnt = 0;
        __syncthreads();
        // keep the values at or above the rank-M value (exactly M: values are
        // unique), warp-aggregated appends
        const uint32_t lane = threadIdx.x & 31;
        for (uint32_t base = 0; base < c; base += blockDim.x) {
          const uint32_t i = base + threadIdx.x;
          const uint64_t v = i < c ? src[i] : 0ull;
          const bool keep = i < c && (c <= M || v >= th);
          const unsigned bal = __ballot_sync(kFull, keep);
          unsigned wb = 0;
          if (lane == 0 && bal) wb = atomicAdd(&cnt, (unsigned)__popc(bal));
          wb = __shfl_sync(kFull, wb, 0);
          const uint32_t pos = wb + __popc(bal & ((1u << lane) - 1));
          if (keep && pos < kMaxSel) sel[pos] = v;
        }
        __syncthreads();
        got = min(cnt, M);
      } else {
        // candidates overflowed the buffer or fell short of M: exact re-selection
        got = stream_topM(S, L, M, buf, t2s, mgs, hist, pick, bcast, &cnt);
        for (uint32_t i = threadIdx.x; i < got; i += blockDim.x) sel[i] = buf[i];
        __syncthreads();
      }
      block_sort_desc(sel, got, buf);
      for (uint32_t i = threadIdx.x; i < got; i += blockDim.x) {
        const uint64_t v = sel[i];
        S.sorted[(size_t)L * kMaxSel + i] = v;
        // the fill reads the moved records' sizes: look them up here, in
        // parallel with the other lists
        if (L != 0) S.ssz[(size_t)L * kMaxSel + i] = S.kv[(~(uint32_t)(L == 2 ? ~v : v)) & kIdMask];
      }
    }
    if (threadIdx.x == 0) S.work->got[L] = got;
  }
  // the last of the set's list CTAs does the victims and the fill
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) is_last = (atomicAdd(&S.work->ticket, 1u) == (unsigned)kLists - 1);
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  const uint32_t nv = __ldcg(&S.work->got[0]), nd = __ldcg(&S.work->got[1]), np = __ldcg(&S.work->got[2]);
  const uint64_t *V = S.sorted, *D = S.sorted + kMaxSel, *P = S.sorted + 2 * kMaxSel;
  for (uint32_t i = threadIdx.x; i < nv; i += blockDim.x) S.victims[i] = (~(uint32_t)__ldcg(&V[i])) & kIdMask;

  // TIDE fill.  Stage P (ascending ck) and D (descending ck) with their sizes.
  // Layout inside the dynamic area (the selection buffers are free now):
  // pck, dck, dck2: kMaxSel u64 each; psz, dsz, dsz2: kMaxSel u32 each.
  uint64_t *pck = buf;
  uint64_t *dck = buf + kMaxSel;
  uint64_t *dck2 = buf + 2 * kMaxSel;
  uint32_t *psz = reinterpret_cast<uint32_t *>(buf + 3 * kMaxSel);
  uint32_t *dsz = psz + kMaxSel;
  uint32_t *dsz2 = dsz + kMaxSel;
  for (uint32_t i = threadIdx.x; i < np; i += blockDim.x) {
    pck[i] = ~__ldcg(&P[i]);
    psz[i] = __ldcg(&S.ssz[2 * kMaxSel + i]);
  }
  for (uint32_t i = threadIdx.x; i < nd; i += blockDim.x) {
    dck[i] = __ldcg(&D[i]);
    dsz[i] = __ldcg(&S.ssz[kMaxSel + i]);
  }
  __syncthreads();
  // Both fill phases take items in order and stop at the first that does not
  // fit; with the state after j items a function of prefix sums over items
  // 0..j, each phase is one block scan and a minimum over the failing items.
  __shared__ Sum wa[32];
  __shared__ int64_t wb[32];
  __shared__ unsigned int first_bad;
  __shared__ unsigned long long at_a;
  __shared__ long long at_b;
  const uint64_t kvb = S.kvb;
  const uint32_t tid = threadIdx.x;
  Sum a[kIpt];
  int64_t b[kIpt];
  // phase 1: promotions into free fast-tier space, least evictable first
  const uint32_t lim1 = (S.thr[kLists + 2] == 0) ? 0u : min(np, S.max_moves);
#pragma unroll
  for (uint32_t i = 0; i < kIpt; i++) {
    const uint32_t j = kIpt * tid + i;
    const uint64_t sz = j < lim1 ? psz[j] : 0;
    a[i] = Sum{sz * kvb, 0};  // bytes moved
    b[i] = (int64_t)sz;  // fast-tier tokens taken
  }
  if (tid == 0) first_bad = lim1;
  block_scan_pairs(a, b, wa, wb);
#pragma unroll
  for (uint32_t i = 0; i < kIpt; i++) {
    const uint32_t j = kIpt * tid + i;
    if (j < lim1 && !(sum_le(a[i], S.budget) && (uint64_t)b[i] <= S.free_s)) atomicMin(&first_bad, j);
  }
  __syncthreads();
  const uint32_t n1 = first_bad;
#pragma unroll
  for (uint32_t i = 0; i < kIpt; i++)
    if (n1 > 0 && kIpt * tid + i == n1 - 1) {
      at_a = a[i].lo;
      at_b = b[i];
    }
  __syncthreads();
  const uint64_t rem = S.budget - (n1 ? at_a : 0ull);
  const uint64_t fs = S.free_s - (n1 ? (uint64_t)at_b : 0ull), fh = S.free_h + (n1 ? (uint64_t)at_b : 0ull);
  __syncthreads();
  // phase 2 demotion order: fast-tier candidates merged with the promoted ones
  // (only the first lim2 positions can be paired)
  const uint32_t cap2 = S.max_moves > n1 ? S.max_moves - n1 : 0;
  const uint32_t nd2 = min(nd + n1, cap2);
  for (uint32_t i = threadIdx.x; i < nd; i += blockDim.x) {
    const uint64_t x = dck[i];
    uint32_t lo = 0, hi = n1;  // promoted (descending = P[n1-1..0]) greater than x
    while (lo < hi) {
      const uint32_t mid = (lo + hi) >> 1;
      if (pck[n1 - 1 - mid] > x) lo = mid + 1; else hi = mid;
    }
    if (i + lo < nd2) {
      dck2[i + lo] = x;
      dsz2[i + lo] = dsz[i];
    }
  }
  for (uint32_t q = threadIdx.x; q < n1; q += blockDim.x) {
    const uint64_t x = pck[n1 - 1 - q];
    uint32_t lo = 0, hi = nd;  // D entries greater than x
    while (lo < hi) {
      const uint32_t mid = (lo + hi) >> 1;
      if (dck[mid] > x) lo = mid + 1; else hi = mid;
    }
    if (q + lo < nd2) {
      dck2[q + lo] = x;
      dsz2[q + lo] = psz[n1 - 1 - q];
    }
  }
  __syncthreads();
  // phase 2: pair P[n1 + j] (next least evictable HBM record) with the j-th
  // most evictable fast-tier entry while the demoted one ranks above the
  // promoted one and the budget and both tiers' capacities hold
  const bool p2 = (S.thr[kLists + 2] != 0) && (S.thr[kLists + 1] != 0);
  const uint32_t lim2 = p2 ? min(np - min(np, n1), nd2) : 0u;
  bool order_ok[kIpt];
#pragma unroll
  for (uint32_t i = 0; i < kIpt; i++) {
    const uint32_t j = kIpt * tid + i;
    uint64_t sp = 0, sd = 0;
    order_ok[i] = false;
    if (j < lim2) {
      sp = psz[n1 + j];
      sd = dsz2[j];
      order_ok[i] = dck2[j] > pck[n1 + j];
    }
    a[i] = Sum{(sp + sd) * kvb, 0};         // bytes moved by the pair
    b[i] = (int64_t)sp - (int64_t)sd;      // fast tier gains sp, loses sd
  }
  if (tid == 0) first_bad = lim2;
  block_scan_pairs(a, b, wa, wb);
#pragma unroll
  for (uint32_t i = 0; i < kIpt; i++) {
    const uint32_t j = kIpt * tid + i;
    const bool ok = order_ok[i] && sum_le(a[i], rem) && (b[i] <= 0 || (uint64_t)b[i] <= fs) &&
                    (b[i] >= 0 || (uint64_t)(-b[i]) <= fh);
    if (j < lim2 && !ok) atomicMin(&first_bad, j);
  }
  __syncthreads();
  const uint32_t pairs = first_bad;
#pragma unroll
  for (uint32_t i = 0; i < kIpt; i++)
    if (pairs > 0 && kIpt * tid + i == pairs - 1) at_a = a[i].lo;
  __syncthreads();
  const uint64_t rem_end = rem - (pairs ? at_a : 0ull);
  for (uint32_t i = threadIdx.x; i < n1 + pairs; i += blockDim.x) S.promote[i] = (~(uint32_t)pck[i]) & kIdMask;
  for (uint32_t i = threadIdx.x; i < pairs; i += blockDim.x) S.demote[i] = (~(uint32_t)dck2[i]) & kIdMask;
  if (threadIdx.x == 0) {
    S.counts[0] = nv;
    S.counts[1] = n1 + pairs;
    S.counts[2] = pairs;
    S.counts[3] = S.work->status ? S.work->status : (unsigned int)UNISON_OK;
    S.moved[0] = S.budget - rem_end;
  }
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Device scratch of the ranking calls, kept per (device, stream) and grown
// when a call needs more: calls on one stream run in order, so each reuses
// the buffer after the previous one is done with it (stream order), and
// calls on different streams get different buffers.  Held for the life of
// the process.
std::mutex g_scratch_mu;
std::map<std::pair<int, cudaStream_t>, std::pair<char *, size_t>> g_scratch;

int scratch_acquire(cudaStream_t stream, size_t bytes, char **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return UNISON_ERR_CUDA;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  auto &e = g_scratch[std::make_pair(dev, stream)];
  if (e.second < bytes) {
    if (e.first) cudaFreeAsync(e.first, stream);  // ordered after the calls that used it
    e.first = nullptr;
    e.second = 0;
    char *p = nullptr;
    if (unison_fault_alloc() || cudaMallocAsync(reinterpret_cast<void **>(&p), bytes, stream) != cudaSuccess) {
      cudaGetLastError();
      return UNISON_ERR_OOM;
    }
    e.first = p;
    e.second = bytes;
  }
  *out = e.first;
  return UNISON_OK;
}

// Pinned host staging for the per-call upload, a ring of buffers per device.
// A buffer is handed out only after the copy that last read it has finished
// (its event); staging_release() ends the caller's hold.
struct Staging {
  unsigned char *host = nullptr;
  size_t cap = 0;
  cudaEvent_t done = nullptr;
};
constexpr int kStagingRing = 4;
std::mutex g_staging_mu;
Staging g_staging[64][kStagingRing];
int g_staging_next[64] = {};

int staging_acquire(size_t bytes, unsigned char **host, cudaEvent_t *done) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return UNISON_ERR_CUDA;
  }
  g_staging_mu.lock();
  Staging &b = g_staging[dev][g_staging_next[dev]];
  g_staging_next[dev] = (g_staging_next[dev] + 1) % kStagingRing;
  if (b.done && cudaEventSynchronize(b.done) != cudaSuccess) {
    cudaGetLastError();
    g_staging_mu.unlock();
    return UNISON_ERR_CUDA;
  }
  if (!b.done && cudaEventCreateWithFlags(&b.done, cudaEventDisableTiming) != cudaSuccess) {
    cudaGetLastError();
    b.done = nullptr;
    g_staging_mu.unlock();
    return UNISON_ERR_CUDA;
  }
  if (b.cap < bytes) {
    if (b.host) cudaFreeHost(b.host);
    b.host = nullptr;
    b.cap = 0;
    const size_t cap = std::max<size_t>(bytes, 64 << 10);
    if (cudaMallocHost(reinterpret_cast<void **>(&b.host), cap) != cudaSuccess) {
      cudaGetLastError();
      b.host = nullptr;
      g_staging_mu.unlock();
      return UNISON_ERR_OOM;
    }
    b.cap = cap;
  }
  *host = b.host;
  *done = b.done;
  return UNISON_OK;  // the lock is held until staging_release()
}
void staging_release() { g_staging_mu.unlock(); }

// Kernel attributes and the filter's resident-CTA count, set up once per
// device (the attributes belong to the device's context).
struct LaunchCfg {
  bool ok = false;
  uint32_t filter_ctas = 0, n_sm = 0;
};
const LaunchCfg &launch_cfg() {
  static std::mutex mu;
  static LaunchCfg cfgs[64];
  static bool done[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    static LaunchCfg bad;
    return bad;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!done[dev]) {
    LaunchCfg c;
    int n_sm = 0, per_sm = 0;
    const size_t smem_finish = sizeof(uint64_t) * (kSmemCand + kMaxSel);
    c.ok = cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess &&
           cudaFuncSetAttribute(rank_filter_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)kFilterSmem) == cudaSuccess &&
           cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, rank_filter_kernel, kFilterCtaThreads,
                                                         kFilterSmem) == cudaSuccess &&
           cudaFuncSetAttribute(rank_finish_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)smem_finish) == cudaSuccess;
    if (!c.ok) cudaGetLastError();
    c.filter_ctas = (uint32_t)std::max(1, n_sm * per_sm);
    c.n_sm = (uint32_t)std::max(1, n_sm);
    cfgs[dev] = c;
    done[dev] = c.ok;
  }
  return cfgs[dev];
}

}  // namespace

extern "C" int unison_rank_batch(const unison_records *sets, const unison_rank_params *params,
                                 const unison_rank_out *outs, int n_sets, void *cuda_stream) {
  if (n_sets < 0 || (n_sets > 0 && (!sets || !params || !outs))) return UNISON_ERR_ARG;
  if (n_sets == 0) return UNISON_OK;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  std::vector<RankSet> hs(n_sets);
  uint32_t tiles = 0;
  for (int i = 0; i < n_sets; i++) {
    const unison_records &r = sets[i];
    const unison_rank_params &p = params[i];
    const unison_rank_out &o = outs[i];
    if (r.n == 0 || r.n > (1ull << 24)) return UNISON_ERR_RANGE;
    if (!r.gap_q || !r.turn || !r.kv_tok || !r.tier || !r.flags) return UNISON_ERR_ARG;
    if (!aligned(r.gap_q, 16) || !aligned(r.turn, 16) || !aligned(r.tier, 16) || !aligned(r.flags, 16))
      return UNISON_ERR_ARG;
    if (p.k > kMaxSel || p.max_moves > kMaxSel) return UNISON_ERR_RANGE;
    if (p.penalty_q >= (1ull << 32) || p.kv_bytes_per_token == 0 || p.kv_bytes_per_token > (1u << 24))
      return UNISON_ERR_RANGE;
    if (!o.counts || !o.moved_bytes || (p.k && !o.victims) || (p.max_moves && (!o.promote || !o.demote)))
      return UNISON_ERR_ARG;
    for (int t = 0; t < (int)kLutN; t++)
      if (p.sigma_q[t] < kEpsQ || p.sigma_q[t] > kLambda) return UNISON_ERR_RANGE;
    RankSet &s = hs[i];
    s.gap = r.gap_q;
    s.turn = r.turn;
    s.kv = r.kv_tok;
    s.tier = r.tier;
    s.flags = r.flags;
    s.n = (uint32_t)r.n;
    s.k = p.k;
    s.max_moves = p.max_moves;
    s.kvb = p.kv_bytes_per_token;
    s.penalty = p.penalty_q;
    s.budget = p.budget_bytes;
    s.free_s = p.free_fast_tok;
    s.free_h = p.free_hbm_tok;
    s.victims = o.victims;
    s.promote = o.promote;
    s.demote = o.demote;
    s.counts = o.counts;
    s.moved = o.moved_bytes;
    s.keys = o.keys;
    s.tile0 = tiles;
    s.ntiles = (uint32_t)((r.n + kBigTile - 1) / kBigTile);
    tiles += s.ntiles;

    for (int t = 0; t < (int)kLutN; t++) {
      s.sigma[t] = p.sigma_q[t];
      s.t2v[t] = ((uint64_t)(kLambda - p.sigma_q[t]) * p.penalty_q) / kLambda;  // eq. (t2)
      s.mgv[t] = magic_for(p.sigma_q[t]);
    }
    s.act = 0;
    for (int L = 0; L < kLists; L++) s.act |= list_active(s, L) ? 1u << L : 0u;
  }
  const LaunchCfg &cfg = launch_cfg();
  if (!cfg.ok) return UNISON_ERR_CUDA;
  // samples per thread: 1 while every set's sample CTAs fit in one wave (two
  // 1,024-thread CTAs per SM), else 4
  uint32_t sq_per = 1;
  {
    uint64_t ctas1 = 0;
    for (int i = 0; i < n_sets; i++) ctas1 += sample_ctas(sample_size(hs[i], 1), 1);
    if (ctas1 > 2ull * cfg.n_sm) sq_per = 4;
  }
  for (int i = 0; i < n_sets; i++) {
    RankSet &s = hs[i];
    s.ns = sample_size(s, sq_per);
    s.sctas = sample_ctas(s.ns, sq_per);
    s.nruns = s.ns / 8;
    s.sq = s.nruns ? s.n / s.nruns : 0;
    s.srem = s.nruns ? s.n % s.nruns : 0;
    for (int L = 0; L < kLists; L++)
      s.rL[L] = (s.ns && list_active(s, L))
                    ? (uint32_t)umin64((list_target(s, L) * s.ns + s.n - 1) / s.n, kMaxR) : 0u;
  }
  // scratch: descriptors, every set's work words (one memset), then per set:
  // thresholds, tables, sorted lists and sizes, candidates, the sample's
  // partial lists
  const size_t per_set = align_up(sizeof(uint64_t) * 2 * kLists, 256) + align_up(sizeof(uint2) * kLists * kLutN, 256) +
                         align_up(sizeof(uint64_t) * kLists * kMaxSel, 256) +
                         align_up(sizeof(uint32_t) * kLists * kMaxSel, 256) +
                         align_up(sizeof(uint64_t) * kLists * kCandCap, 256) +
                         align_up(sizeof(uint32_t) * kLists * kSampleCtas * kMaxR, 256) +
                         align_up(sizeof(uint32_t) * kLists * kSampleCtas, 256);
  const size_t desc_b = align_up(sizeof(RankSet) * n_sets, 256);
  const size_t work_b = align_up(sizeof(RankWork) * n_sets, 256);
  char *scratch = nullptr;
  {
    const int ar = scratch_acquire(stream, desc_b + work_b + per_set * n_sets, &scratch);
    if (ar != UNISON_OK) return ar;
  }
  RankWork *works = reinterpret_cast<RankWork *>(scratch + desc_b);
  for (int i = 0; i < n_sets; i++) {
    char *p = scratch + desc_b + work_b + per_set * i;
    RankSet &s = hs[i];
    s.work = works + i;
    s.thr = reinterpret_cast<uint64_t *>(p);
    p += align_up(sizeof(uint64_t) * 2 * kLists, 256);
    s.gthr = reinterpret_cast<uint2 *>(p);
    p += align_up(sizeof(uint2) * kLists * kLutN, 256);
    s.sorted = reinterpret_cast<uint64_t *>(p);
    p += align_up(sizeof(uint64_t) * kLists * kMaxSel, 256);
    s.ssz = reinterpret_cast<uint32_t *>(p);
    p += align_up(sizeof(uint32_t) * kLists * kMaxSel, 256);
    s.cand = reinterpret_cast<uint64_t *>(p);
    p += align_up(sizeof(uint64_t) * kLists * kCandCap, 256);
    s.part = reinterpret_cast<uint32_t *>(p);
    p += align_up(sizeof(uint32_t) * kLists * kSampleCtas * kMaxR, 256);
    s.part_n = reinterpret_cast<uint32_t *>(p);
  }
  int rc = UNISON_OK;
  auto ck = [&](cudaError_t e) {
    if (e != cudaSuccess && rc == UNISON_OK) rc = UNISON_ERR_CUDA;
  };
  RankSet *d_sets = reinterpret_cast<RankSet *>(scratch);
  const size_t smem_finish = sizeof(uint64_t) * (kSmemCand + kMaxSel);
  // persistent filter: as many CTAs as fit at once (per device, set up once)
  uint32_t grid_filter = std::max(1u, std::min<uint32_t>(tiles, cfg.filter_ctas));
  // Filter schedule: each set gets a group of CTAs in proportion to its tiles
  // (at least 1, at most its tile count) when the groups fit in the resident
  // CTAs; otherwise every CTA deals from all sets' tiles.
  int grouped = 0;
  {
    uint64_t total = 0;
    for (int i = 0; i < n_sets; i++) {
      RankSet &s = hs[i];
      s.nctas = (uint32_t)std::max<uint64_t>(1, ((uint64_t)grid_filter * s.ntiles) / tiles);
      s.nctas = std::min(s.nctas, s.ntiles);
      s.cta0 = (uint32_t)total;
      total += s.nctas;
    }
    if (total <= grid_filter) {
      grouped = 1;
      grid_filter = (uint32_t)total;
    }
  }
  uint32_t max_sctas = 1;
  for (int i = 0; i < n_sets; i++) max_sctas = std::max(max_sctas, hs[i].sctas);
  // descriptors and zeroed work words: one copy from pinned staging
  {
    const size_t up = desc_b + sizeof(RankWork) * n_sets;
    unsigned char *h = nullptr;
    cudaEvent_t done = nullptr;
    const int sr = staging_acquire(up, &h, &done);
    if (sr != UNISON_OK) return sr;
    std::memcpy(h, hs.data(), sizeof(RankSet) * n_sets);
    std::memset(h + desc_b, 0, sizeof(RankWork) * n_sets);
    ck(cudaMemcpyAsync(d_sets, h, up, cudaMemcpyHostToDevice, stream));
    ck(cudaEventRecord(done, stream));  // the buffer is reused after this copy
    staging_release();
  }
  {
    ProfSpan span("rank_sample", stream);
    if (sq_per == 1)
      rank_sample_kernel<1><<<dim3(max_sctas, n_sets), kSampleThreads, 0, stream>>>(d_sets);
    else
      rank_sample_kernel<4><<<dim3(max_sctas, n_sets), kSampleThreads, 0, stream>>>(d_sets);
  }
  cudaLaunchAttribute pdl[1];
  pdl[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  pdl[0].val.programmaticStreamSerializationAllowed = 1;
  {
    ProfSpan span("rank_filter", stream);
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid_filter);
    lc.blockDim = dim3(kFilterCtaThreads);
    lc.dynamicSmemBytes = kFilterSmem;
    lc.stream = stream;
    lc.attrs = pdl;
    lc.numAttrs = 1;
    ck(cudaLaunchKernelEx(&lc, rank_filter_kernel, (const RankSet *)d_sets, n_sets, tiles, grouped));
  }
  {
    ProfSpan span("rank_finish", stream);
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(kLists, n_sets);
    lc.blockDim = dim3(kFinishThreads);
    lc.dynamicSmemBytes = smem_finish;
    lc.stream = stream;
    lc.attrs = pdl;
    lc.numAttrs = 1;
    ck(cudaLaunchKernelEx(&lc, rank_finish_kernel, (const RankSet *)d_sets));
  }
  count_launches(3);
  ck(cudaGetLastError());
  return rc;
}
