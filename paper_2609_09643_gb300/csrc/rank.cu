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
//
// One cooperative, persistent kernel does a whole call.  Each set owns a
// group of CTAs (in proportion to its records; with more sets than CTAs,
// each CTA takes whole sets in turn).  Per set, inside the group:
//   sample   up to 16 CTAs gather a jittered stratified sample, count it in
//            shared memory and add it to a 4,096-bin histogram per list (bins
//            monotone in the list value).  Once every sampling CTA's counts
//            are in, each CTA of the group cuts the histograms at the lists'
//            sample ranks itself: per-list thresholds and per-turn thresholds
//            on the gap average (the score is monotone in the gap for a fixed
//            turn, so the streaming test needs no division).  Meanwhile every
//            CTA's producer warp already streams its first tiles into shared
//            memory.
//   filter   the group's CTAs take the set's tiles from a shared counter;
//            every record is read once (8 B: gap average, turn, flags, tier)
//            by TMA bulk copies and tested against the thresholds, and the
//            exact values of the records that pass are appended per list to
//            the CTA's own region, which moves into the set's list when the
//            CTA is done.
//   finish   the last three CTAs of the group to finish streaming take one
//            list each: a 256-bucket cut below the candidates' common prefix
//            keeps the bucket holding the rank-M value and those above it,
//            which are bucket-sorted and the first M kept; a list whose cut
//            holds too many values falls back to a radix select, and one
//            whose candidates overflowed or fell short is re-selected exactly
//            by streaming the set.  The last list's CTA runs the fill, 256
//            items at a time, and writes the outputs.
// The work words and sample histograms of a call are held twice: calls on a
// stream alternate between the two, and each call zeroes the other.
// Every wait on another CTA or on a copy is bounded: a wait that gives up
// records UNISON_ERR_TIMEOUT in the set's status word and the CTA carries on
// to the end of the kernel.  A cooperative launch keeps every CTA of the grid
// resident, so the waits on other CTAs end.
#include <algorithm>
#include <cstring>
#include <map>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "profile.cuh"
#ifdef UNISON_DEBUG_HOOKS
#include "../../include/unison_debug.h"
#endif

using namespace unison;

namespace {

constexpr int kLists = 3;  // 0 = V, 1 = D, 2 = P
constexpr uint32_t kSample = 16384;      // largest sample of a set
constexpr uint32_t kCandCap = 65536;     // candidate slots per list and set
constexpr uint32_t kMaxGroup = 512;       // CTAs of one launch, at most (152 SMs x 3)
constexpr uint32_t kMaxSel = 4096;       // largest k and max_moves
constexpr uint32_t kFull = 0xFFFFFFFFu;
constexpr uint32_t kSampleCtas = 16;     // sampling CTAs per set, at most
constexpr uint32_t kSampleQ = 4;         // samples per consumer thread
constexpr uint32_t kSampleRank = 32;
constexpr uint32_t kBins = 4096;         // histogram bins per list
constexpr uint32_t kEndTile = 0xFFFFFFFFu;

// CTA layout: 8 consumer warps and one producer warp.  A tile is 4,096
// records; two tiles are in flight per CTA.
constexpr int kStages = 2;
constexpr uint32_t kRec = 16;                          // records per consumer thread per tile
constexpr uint32_t kConsumers = 256;                   // consumer threads
constexpr uint32_t kBigTile = kConsumers * kRec;       // 4096 records per tile
constexpr uint32_t kGroups = kRec / 4;                 // groups of four records per thread
constexpr uint32_t kGroupStride = kConsumers * 4;      // records between a thread's groups
constexpr uint32_t kWarpBuf = 128;                     // flagged records a warp tests per pass
constexpr uint32_t kCtaThreads = kConsumers + 32;
constexpr uint32_t kPerCtaSamples = kConsumers * kSampleQ;
constexpr uint32_t kIpt = kMaxSel / kConsumers;        // fill items per consumer thread
static_assert(kConsumers >= kLutN * 5, "one consumer thread per bound-table entry");
static_assert(kMaxSel % kConsumers == 0 && kIpt % 4 == 0, "fill layout");
static_assert(kBins == 16 * kConsumers, "histogram cut layout");

struct __align__(128) FilterStage {
  uint32_t gap[kBigTile];
  uint16_t turn[kBigTile];
  uint8_t flags[kBigTile];
  uint8_t tier[kBigTile];
};
constexpr size_t kDynSmem = sizeof(FilterStage) * kStages;  // 64 KB, reused by the finish
static_assert(sizeof(unsigned int) * kLists * kBins <= kDynSmem, "the sample's counts fit the stage area");
// the merge kernel's area: values and sizes, and the bucket sort's copies of both
constexpr size_t kMergeSmem = 3 * kMaxSel * sizeof(uint64_t);  // 96 KB
constexpr uint32_t kDynWords = kDynSmem / 8;                // 8192 u64
constexpr uint32_t kSmemCand = kDynWords - kMaxSel;          // candidates copied to shared memory
static_assert(kSmemCand >= kMaxSel && kDynWords >= 2 * kMaxSel, "finish layout");

// Every wait is bounded in time (%globaltimer, ns).  A wait on another CTA
// (thresholds, the group's last arrival) gives up after kWaitNs; a wait on
// this CTA's own pipeline (a tile's copies, a stage's release, the finish's
// copy) after kPipeNs, longer, so that a producer never gives up while its
// consumers still wait on another CTA.
// a suspended waiter re-checks its bound at least this often
constexpr uint32_t kWaitHintNs = 20000;
#ifdef UNISON_DEBUG_HOOKS
constexpr uint64_t kWaitNs = 2000000ull;     // 2 ms: the tests make one run out
constexpr uint64_t kPipeNs = 50000000ull;    // 50 ms: well above any ordinary copy
__device__ int g_hook_flag_set = -1;   // set whose threshold wait first waits on a flag nothing sets
__device__ int g_hook_mbar_set = -1;   // set whose first tile wait first waits on a barrier nothing arrives at
#else
constexpr uint64_t kWaitNs = 2000000000ull;  // 2 s
constexpr uint64_t kPipeNs = 4000000000ull;  // 4 s
#endif

// Each group of words that many CTAs poll or update at once has a 128-byte
// line of its own: a flag polled by every CTA of a group and counters taken
// by atomics in the same line would serialise at one L2 slice.
struct alignas(128) RankWork {
  // the streaming counters (atomics while the tiles stream)
  unsigned int cand[kLists];    // candidates emitted per list
  unsigned int next_tile;       // the group's tile counter
  unsigned int pad0[28];
  // the sample's reads done (polled by the producers)
  unsigned int gathered;        // sampling CTAs whose sample has arrived
  unsigned int pad1[31];
  // the sample's counts in the histogram (polled by every CTA of the group)
  unsigned int sample_ticket;   // sampling CTAs whose counts have landed
  unsigned int pad2[31];
  // the finish
  unsigned int done_ctas;       // CTAs of the group done streaming
  unsigned int list_ticket;     // lists finished
  unsigned int got[kLists];     // selected entries per list
  unsigned int status;          // UNISON_ERR_TIMEOUT if a bounded wait gave up
  unsigned int dummy;           // never written: the debug hook waits on it
  unsigned int pad3[25];
};
static_assert(sizeof(RankWork) == 512, "four lines");

// Per-turn tables of one (sigma, P_Z) pair, shared by the sets that use it.
struct RankTab {
  uint64_t t2v[kLutN];   // eq. (t2) per turn index
  uint64_t mgv[kLutN];   // division magic of sigma per turn index
  uint32_t sigma[kLutN];
};

struct RankSet {
  const uint32_t *gap;
  const uint16_t *turn;
  const uint32_t *kv;
  const uint8_t *tier;
  const uint8_t *flags;
  uint32_t n, k, max_moves, kvb;
  uint64_t budget, free_s, free_h;
  uint32_t *victims, *promote, *demote, *counts;
  uint64_t *moved, *keys;
  const RankTab *tab;
  uint32_t ntiles;
  uint32_t cta0, nctas;          // the group: CTAs [cta0, cta0 + nctas)
  uint32_t ns, nruns;            // sample size, its runs of 8
  uint64_t sstep;                // stratum width n / nruns in 16.16 fixed point
  uint32_t sctas;                // sampling CTAs (the group's first sctas)
  uint32_t act;                  // active lists (bit L)
  uint32_t rL[kLists];           // sample rank of each list's threshold
  uint32_t ccap;                 // candidate slots per list (kCandCap, or n rounded up for a set too small to sample)
  uint32_t off;                  // index of record 0 in the whole set (a shard's slice), else 0
  unsigned char *cands;          // a shard's candidate lists (unison_rank_shard), else null
  // scratch (per set)
  RankWork *work;
  uint64_t *cand;    // [3][ccap] the set's candidate lists (a global counter each)
  uint64_t *creg;    // [3][nctas][cr] each CTA's candidates while it streams
  uint32_t cr;       // region size
  uint64_t *sorted;  // [3][kMaxSel]
  uint32_t *ssz;     // [3][kMaxSel] KV tokens of the sorted entries (D and P)
  unsigned int *shist;  // [3][kBins] sample histogram (zero between calls)
};

// A shard's candidate lists (unison_rank_shard): a 64-byte header, then its
// V, D and P lists of (list value, KV tokens) in ranking order.
struct CandHeader {
  uint32_t count[kLists];
  uint32_t status;
  uint32_t n, off, k, max_moves;
  uint32_t pad[8];
};
static_assert(sizeof(CandHeader) == 64, "candidate header");
struct CandEntry {
  uint64_t v;
  uint32_t kv, pad;
};
constexpr uint32_t kMaxShards = 1024;
__host__ __device__ __forceinline__ size_t cand_bytes(uint32_t k, uint32_t m) {
  return sizeof(CandHeader) + sizeof(CandEntry) * ((size_t)k + 2ull * m);
}
__host__ __device__ __forceinline__ size_t cand_list_off(uint32_t k, uint32_t m, int L) {
  return sizeof(CandHeader) + sizeof(CandEntry) * (L == 0 ? 0ull : (L == 1 ? (size_t)k : (size_t)k + m));
}

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

__device__ __forceinline__ uint64_t list_val(uint64_t ck, int L) { return L == 2 ? ~ck : ck; }

// ------------------------------------------------- barriers and copies ----
__device__ __forceinline__ uint32_t smem_addr(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
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
// The same test, but a thread whose phase has not completed is suspended
// until it does or about hint_ns pass: a waiting thread then takes no issue
// slots from the warps that work.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t *bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity), "r"(hint_ns)
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

__device__ __forceinline__ uint64_t now_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Bounded wait on an mbarrier phase; false when the bound ran out.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity, uint64_t limit_ns = kPipeNs) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = now_ns();
  while (now_ns() - t0 < limit_ns)
    if (mbar_try_wait_sleep(bar, parity, kWaitHintNs)) return true;
  return false;
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

__device__ __forceinline__ void set_status(const RankSet &S, int code) { atomicExch(&S.work->status, (unsigned int)code); }

// Consumer thread 0 waits (bounded) until *word reaches target, then the
// consumers proceed with the other CTAs' writes visible.  False (for every
// consumer thread alike) on timeout.
__device__ bool wait_word(const RankSet &S, const unsigned int *word, unsigned int target) {
  __shared__ unsigned int ok;
  if (threadIdx.x == 0) {
    const uint64_t t0 = now_ns();
    uint32_t nap = 32;  // backoff: a word polled by many CTAs at once
    while (*(volatile const unsigned int *)word < target && now_ns() - t0 < kWaitNs) {
      __nanosleep(nap);
      nap = min(nap * 2, 256u);
    }
    ok = *(volatile const unsigned int *)word >= target;
    if (!ok) set_status(S, UNISON_ERR_TIMEOUT);
    __threadfence();
  }
  consumers_sync();
  return ok != 0;
}

// Consumer thread 0 waits (bounded) for an mbarrier phase; the others take
// its verdict, so every consumer thread takes the same path, then observe the
// completed phase themselves (one poll: it has completed) before they read
// what it guards.  False (for all) on timeout.
__device__ bool wait_phase_uniform(const RankSet &S, uint64_t *bar, uint32_t parity, uint64_t limit_ns = kPipeNs) {
  __shared__ unsigned int ok;
  if (threadIdx.x == 0) {
    ok = mbar_wait_bounded(bar, parity, limit_ns) ? 1u : 0u;
    if (!ok) set_status(S, UNISON_ERR_TIMEOUT);
  }
  consumers_sync();
  if (!ok) return false;
  mbar_try_wait(bar, parity);
  return true;
}

// ---------------------------------------------------- shared scratch ----
// The filter's bound table and flagged-record buffers, or the finish's
// radix-select scratch (never in use at the same time).
struct FilterScratch {
  uint2 ftab[kLutN * 5];
  uint16_t wbuf[kConsumers / 32][kWarpBuf];
};
struct SelectScratch {
  unsigned int hist[256];
  unsigned int off[256];  // the bucket sort's bucket starts
  unsigned int pick[2];
  unsigned long long bcast[2];
  unsigned int cnt;
  unsigned int wtot[kConsumers / 32];
  unsigned long long wsq[kConsumers / 32];
};
union CtaScratch {
  FilterScratch f;
  SelectScratch s;
};

// ---------------------------------------------------- histogram bins ----
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
// Bin of a summary, monotone: summaries below 2^31 by octave (the position
// e of the leading one) and the 6 bits after it (bins 0..1983, a 1/64-octave
// resolution; below 64 one bin per value); summaries at or above 2^31 (the
// maximal key) by index, 8,192 indices a bin (bins 2048..4095).
// bin_floor(b) is the smallest summary in bin b.
__device__ __forceinline__ uint32_t bin_of(uint32_t f) {
  if (f & 0x80000000u) return 2048u + ((f & kIdMask) >> 13);
  if (f < 64u) return (f ? (uint32_t)(31 - __clz(f)) : 0u) * 64u + f;
  const uint32_t e = 31 - __clz(f);
  return e * 64u + ((f >> (e - 6)) & 63u);
}
__device__ __forceinline__ uint32_t bin_floor(uint32_t b) {
  if (b >= 2048u) return 0x80000000u | ((b - 2048u) << 13);
  const uint32_t e = b / 64u, m = b % 64u;
  return e < 6u ? m : (64u + m) << (e - 6u);
}

// Value with the given rank (1 = largest) among get(0..n-1), 64-bit values,
// MSB-first over the bytes where the values differ.  Consumer threads only;
// hist must be zero on entry and is zero on return.
template <typename Get>
__device__ uint64_t block_select_rank(Get get, uint32_t n, uint32_t rank, SelectScratch &ss) {
  unsigned long long a = ~0ull, o = 0ull;
  for (uint32_t i = threadIdx.x; i < n; i += kConsumers) {
    const uint64_t v = get(i);
    a &= v;
    o |= v;
  }
  for (int s = 16; s; s >>= 1) {
    a &= __shfl_xor_sync(kFull, a, s);
    o |= __shfl_xor_sync(kFull, o, s);
  }
  if (threadIdx.x == 0) {
    ss.bcast[0] = ~0ull;
    ss.bcast[1] = 0ull;
  }
  consumers_sync();
  if ((threadIdx.x & 31) == 0) {
    atomicAnd(&ss.bcast[0], a);
    atomicOr(&ss.bcast[1], o);
  }
  consumers_sync();
  const uint64_t same = ~(ss.bcast[0] ^ ss.bcast[1]);  // bits equal in every value
  const uint64_t common = ss.bcast[0] & same;
  int top = 7;
  while (top > 0 && ((same >> (8 * top)) & 0xFF) == 0xFF) top--;
  uint64_t mask = top < 7 ? (~0ull << (8 * (top + 1))) : 0ull;
  uint64_t prefix = common & mask;
  uint32_t need = rank;
  unsigned int *hist = ss.hist;
  for (int b = top; b >= 0; b--) {
    for (uint32_t base = 0; base < n; base += kConsumers) {
      const uint32_t i = base + threadIdx.x;
      bool in = false;
      uint32_t d = 0;
      if (i < n) {
        const uint64_t v = get(i);
        in = (v & mask) == prefix;
        d = (uint32_t)(v >> (8 * b)) & 0xFF;
      }
      const unsigned act = __ballot_sync(kFull, in);
      if (in) {
        const unsigned grp = __match_any_sync(act, d);
        if ((__ffs(grp) - 1) == (int)(threadIdx.x & 31)) atomicAdd(&hist[d], (unsigned)__popc(grp));
      }
    }
    consumers_sync();
    if (threadIdx.x < 32) {
      const int l = threadIdx.x;
      uint32_t c[8], tot = 0;
#pragma unroll
      for (int q = 0; q < 8; q++) {
        c[q] = hist[255 - 8 * l - q];
        hist[255 - 8 * l - q] = 0;
        tot += c[q];
      }
      uint32_t incl = tot;
#pragma unroll
      for (int s = 1; s < 32; s <<= 1) {
        const uint32_t y = __shfl_up_sync(kFull, incl, s);
        if (l >= s) incl += y;
      }
      const uint32_t excl = incl - tot;
      const unsigned hit = __ballot_sync(kFull, excl < need && incl >= need);
      if (l == __ffs(hit) - 1) {
        uint32_t cum = excl;
#pragma unroll
        for (int q = 0; q < 8; q++) {
          if (cum + c[q] >= need) {
            ss.pick[0] = 255 - 8 * l - q;
            ss.pick[1] = need - cum;
            cum = 0xFFFFFFFFu;
            break;
          }
          cum += c[q];
        }
      }
    }
    consumers_sync();
    prefix |= (uint64_t)ss.pick[0] << (8 * b);
    mask |= 0xFFull << (8 * b);
    need = ss.pick[1];
  }
  consumers_sync();  // pick and bcast free for the caller
  return prefix;
}

// hist_cut over the kLists histograms hist[L * kBins ..] at once (their
// loads in flight together): cut[L] for need[L] > 0, -1 for need[L] == 0.
__device__ void hist_cut3(unsigned int *hist, const uint32_t (&need)[kLists], int (&cut)[kLists]) {
  __shared__ unsigned int wtot[kLists][kConsumers / 32];
  __shared__ int scut[kLists];
  const uint32_t tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t lo = kBins - 16 * (tid + 1);
  uint32_t c[kLists][16], tot[kLists], ex[kLists];
#pragma unroll
  for (int L = 0; L < kLists; L++) {
    uint4 *h4 = reinterpret_cast<uint4 *>(hist + L * kBins + lo);
#pragma unroll
    for (int q = 0; q < 4; q++) {
      const uint4 x = __ldcg(h4 + q);
      c[L][4 * q] = x.x; c[L][4 * q + 1] = x.y; c[L][4 * q + 2] = x.z; c[L][4 * q + 3] = x.w;
    }
  }
#pragma unroll
  for (int L = 0; L < kLists; L++) {
    tot[L] = 0;
#pragma unroll
    for (int q = 0; q < 16; q++) tot[L] += c[L][q];
    uint32_t incl = tot[L];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(kFull, incl, o);
      if ((int)lane >= o) incl += y;
    }
    if (lane == 31) wtot[L][warp] = incl;
    ex[L] = incl - tot[L];
  }
  if (tid < kLists) scut[tid] = -1;
  consumers_sync();
#pragma unroll
  for (int L = 0; L < kLists; L++) {
    for (uint32_t w = 0; w < warp; w++) ex[L] += wtot[L][w];
    if (need[L] && ex[L] < need[L] && ex[L] + tot[L] >= need[L]) {
      uint32_t acc = ex[L];
      for (int q = 15; q >= 0; q--) {
        if (acc + c[L][q] >= need[L]) {
          scut[L] = (int)(lo + q);
          break;
        }
        acc += c[L][q];
      }
    }
  }
  consumers_sync();
#pragma unroll
  for (int L = 0; L < kLists; L++) cut[L] = scut[L];
}

// Sort, descending, of a[0..n) padded with zeros to a power of two p >= 64
// (bitonic network in shared memory), carrying pay[] along when given.
// Stages whose partners lie less than 64 apart run warp by warp (each warp
// owns blocks of 64 entries), with a warp barrier; the wider stages pair
// entries across the array and take a block barrier.
__device__ void bitonic_sort_desc(uint64_t *a, uint32_t n, uint32_t *pay = nullptr) {
  if (n <= 1) return;
  uint32_t p = 64;
  while (p < n) p <<= 1;
  for (uint32_t i = n + threadIdx.x; i < p; i += kConsumers) {
    a[i] = 0;
    if (pay) pay[i] = 0;
  }
  consumers_sync();
  const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  auto cmpx = [&](uint32_t x, uint32_t y, bool desc) {
    const uint64_t u = a[x], v = a[y];
    if ((u < v) == desc) {
      a[x] = v;
      a[y] = u;
      if (pay) {
        const uint32_t t = pay[x];
        pay[x] = pay[y];
        pay[y] = t;
      }
    }
  };
  for (uint32_t k = 2; k <= p; k <<= 1) {
    for (uint32_t j = k >> 1; j > 0; j >>= 1) {
      if (j >= 64) {
        for (uint32_t i = threadIdx.x; i < p / 2; i += kConsumers) {
          const uint32_t x = ((i & ~(j - 1)) << 1) | (i & (j - 1));
          cmpx(x, x + j, (x & k) == 0);
        }
        consumers_sync();
      } else {
        // block b (64 entries) is warp b % 8's; lane l takes pair l of it
        for (uint32_t b = warp; b < p / 64; b += kConsumers / 32) {
          const uint32_t x = 64 * b + (((lane & ~(j - 1)) << 1) | (lane & (j - 1)));
          cmpx(x, x + j, (x & k) == 0);
        }
        __syncwarp();
      }
    }
    // the next level opens with a stride of k: across blocks once k >= 64
    if (k < p && k >= 64) consumers_sync();
  }
  consumers_sync();
}

// Sort, descending, of a[0..n) for n <= kRegSort: the same bitonic network
// over a fixed 2,048 entries (zeros pad the tail), held in registers, 8
// consecutive entries per consumer thread.  Partners less than 8 apart sit in
// one thread; less than 256 apart, in one warp (exchanged by shuffles); the
// three widest strides go through a[] with block barriers.  a[] must hold
// kRegSort entries.
constexpr uint32_t kRegSort = 8 * kConsumers;
template <uint32_t J>
__device__ __forceinline__ void reg_stage(uint64_t (&x)[8], uint32_t e0, uint32_t k) {
#pragma unroll
  for (uint32_t r = 0; r < 8; r++) {
    if (r & J) continue;
    const bool desc = ((e0 + r) & k) == 0;  // this k-block runs descending
    const uint64_t u = x[r], v = x[r + J];
    if ((u < v) == desc) {
      x[r] = v;
      x[r + J] = u;
    }
  }
}
__device__ void reg_bitonic_desc(uint64_t *a, uint32_t n) {
  const uint32_t tid = threadIdx.x, e0 = 8 * tid;
  uint64_t x[8];
#pragma unroll
  for (uint32_t r = 0; r < 8; r++) x[r] = e0 + r < n ? a[e0 + r] : 0ull;
  for (uint32_t k = 2; k <= kRegSort; k <<= 1) {
    for (uint32_t j = k >> 1; j > 0; j >>= 1) {
      if (j == 4) reg_stage<4>(x, e0, k);
      else if (j == 2) reg_stage<2>(x, e0, k);
      else if (j == 1) reg_stage<1>(x, e0, k);
      else if (j < 256) {
        const uint32_t pm = j >> 3;  // the partner thread is tid ^ pm
        const bool lower = (e0 & j) == 0, desc = (e0 & k) == 0;
#pragma unroll
        for (uint32_t r = 0; r < 8; r++) {
          const uint64_t y = __shfl_xor_sync(kFull, x[r], pm);
          x[r] = (lower == desc) ? (x[r] > y ? x[r] : y) : (x[r] < y ? x[r] : y);
        }
      } else {
#pragma unroll
        for (uint32_t r = 0; r < 8; r++) a[e0 + r] = x[r];
        consumers_sync();
        const bool lower = (e0 & j) == 0, desc = (e0 & k) == 0;
#pragma unroll
        for (uint32_t r = 0; r < 8; r++) {
          const uint64_t y = a[(e0 + r) ^ j];
          x[r] = (lower == desc) ? (x[r] > y ? x[r] : y) : (x[r] < y ? x[r] : y);
        }
        consumers_sync();
      }
    }
  }
#pragma unroll
  for (uint32_t r = 0; r < 8; r++)
    if (e0 + r < n) a[e0 + r] = x[r];
  consumers_sync();
}

// Sort, descending, of the distinct values a[0..n) by bucket: the 8 bits
// below the values' common prefix name 256 buckets, a counting pass places
// each value in its bucket's range (buckets in descending order, in tmp),
// and each value's place within its bucket is the count of the bucket's
// values above it.  pay[] (when given) moves along, through tmp_pay.  Costs
// the sum over buckets of size^2 comparisons; declines (false, a and pay
// unchanged) when that sum is large, i.e. the values crowd into few buckets.
static_assert(kConsumers == 256, "one bucket per consumer thread");

// The rank-M cut of the distinct values src[0..c), c > M: 256 buckets on
// the 8 bits below the values' common prefix (bucket of v: (v >> sh) & 255),
// and bcut the bucket holding the rank-M value.  Returns the count of values
// in bcut and the buckets above it: at least M.  each(fn) calls fn(v) once
// for every value, spread over the consumer threads in any order.
template <class Each>
__device__ uint32_t bucket_cut(Each each, uint32_t M, SelectScratch &ss, int &sh, uint32_t &bcut) {
  const uint32_t tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint64_t an = ~0ull, orv = 0ull;
  each([&](uint64_t v) {
    an &= v;
    orv |= v;
  });
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    an &= __shfl_xor_sync(kFull, an, o);
    orv |= __shfl_xor_sync(kFull, orv, o);
  }
  if (tid == 0) {
    ss.bcast[0] = ~0ull;
    ss.bcast[1] = 0ull;
  }
  ss.hist[tid] = 0;
  consumers_sync();
  if (lane == 0) {
    atomicAnd(&ss.bcast[0], an);
    atomicOr(&ss.bcast[1], orv);
  }
  consumers_sync();
  const uint64_t vary = ss.bcast[0] ^ ss.bcast[1];
  const int top = vary ? 64 - __clzll((long long)vary) : 0;
  sh = top > 8 ? top - 8 : 0;
  each([&](uint64_t v) { atomicAdd(&ss.hist[(uint32_t)(v >> sh) & 255u], 1u); });
  consumers_sync();
  // thread t owns bucket 255 - t: counts from the top
  const uint32_t own = ss.hist[255 - tid];
  uint32_t incl = own;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(kFull, incl, o);
    if ((int)lane >= o) incl += y;
  }
  if (lane == 31) ss.wtot[warp] = incl;
  consumers_sync();
  for (uint32_t w = 0; w < warp; w++) incl += ss.wtot[w];
  if (incl - own < M && incl >= M) {
    ss.pick[0] = 255 - tid;
    ss.pick[1] = incl;
  }
  consumers_sync();
  bcut = ss.pick[0];
  const uint32_t n = ss.pick[1];
  consumers_sync();  // pick, hist and bcast free for the caller
  return n;
}
__device__ bool bucket_sort_desc(uint64_t *a, uint32_t n, uint64_t *tmp, SelectScratch &ss, uint32_t *pay = nullptr,
                                 uint32_t *tmp_pay = nullptr) {
  if (n <= 1) return true;
  const uint32_t tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint64_t an = ~0ull, orv = 0ull;
  for (uint32_t i = tid; i < n; i += kConsumers) {
    const uint64_t v = a[i];
    an &= v;
    orv |= v;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    an &= __shfl_xor_sync(kFull, an, o);
    orv |= __shfl_xor_sync(kFull, orv, o);
  }
  if (tid == 0) {
    ss.bcast[0] = ~0ull;
    ss.bcast[1] = 0ull;
  }
  ss.hist[tid] = 0;
  consumers_sync();
  if (lane == 0) {
    atomicAnd(&ss.bcast[0], an);
    atomicOr(&ss.bcast[1], orv);
  }
  consumers_sync();
  const uint64_t vary = ss.bcast[0] ^ ss.bcast[1];  // non-zero: the values are distinct
  const int top = 64 - __clzll((long long)vary);
  const int sh = top > 8 ? top - 8 : 0;
  for (uint32_t i = tid; i < n; i += kConsumers) atomicAdd(&ss.hist[(uint32_t)(a[i] >> sh) & 255u], 1u);
  consumers_sync();
  // thread t owns bucket 255 - t: exclusive offsets in descending bucket order
  const uint32_t c = ss.hist[255 - tid];
  uint32_t incl = c;
  uint64_t sq = (uint64_t)c * c;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(kFull, incl, o);
    if ((int)lane >= o) incl += y;
    sq += __shfl_xor_sync(kFull, sq, o);
  }
  if (lane == 31) ss.wtot[warp] = incl;
  if (lane == 0) ss.wsq[warp] = sq;
  consumers_sync();
  uint32_t ex = incl - c;
  uint64_t sqt = 0;
  for (uint32_t w = 0; w < kConsumers / 32; w++) {
    if (w < warp) ex += ss.wtot[w];
    sqt += ss.wsq[w];
  }
  ss.off[255 - tid] = ex;
  consumers_sync();  // every count read before the cursors overwrite them
  if (sqt > 32ull * n + 8192ull) return false;  // the same verdict in every thread
  ss.hist[255 - tid] = ex;
  consumers_sync();
  for (uint32_t i = tid; i < n; i += kConsumers) {
    const uint64_t v = a[i];
    const uint32_t p = atomicAdd(&ss.hist[(uint32_t)(v >> sh) & 255u], 1u);
    tmp[p] = v;
    if (pay) tmp_pay[p] = pay[i];
  }
  consumers_sync();
  for (uint32_t p = tid; p < n; p += kConsumers) {
    const uint64_t v = tmp[p];
    const uint32_t b = (uint32_t)(v >> sh) & 255u, lo = ss.off[b], hi = ss.hist[b];
    uint32_t r = 0;
    for (uint32_t q = lo; q < hi; q++) r += tmp[q] > v ? 1u : 0u;
    a[lo + r] = v;
    if (pay) pay[lo + r] = tmp_pay[p];
  }
  consumers_sync();
  return true;
}

// The bucket sort, else a sorting network by size.  tmp: room for n values
// (and tmp_pay for n payloads when pay is given), apart from a and pay.
__device__ __forceinline__ void sort_desc(uint64_t *a, uint32_t n, uint64_t *tmp, SelectScratch &ss) {
  if (bucket_sort_desc(a, n, tmp, ss)) return;
  if (n <= kRegSort) reg_bitonic_desc(a, n);
  else bitonic_sort_desc(a, n);
}

// ------------------------------------------------------------- sample ----
// Sample size and per-list ranks: ns records (ns/8 runs of 8, one run per
// stratum) and rank r_L = ceil(target_L * ns / n), with ns about kSampleRank
// times n over the largest target, capped at kSample and at 1,024 per
// sampling CTA.  Candidates above the rank-r_L sample value number about
// target_L / r_L * Gamma(r_L), and fall short of M_L with probability
// P(Gamma(r_L) < r_L M_L / target_L).  Targets: 2 M + 1024 while the sample
// is not capped (r = 32 for the largest list: below 1e-6), else 6 M + 2048
// (r >= 8 at 2^24 records: about 1e-5).  The threshold is the floor of the
// histogram bin holding the rank-r_L sample, at or below that sample, so it
// admits a few more.  A shortfall costs time, never exactness (the finish
// re-selects the list).
__host__ __forceinline__ uint64_t umin64(uint64_t a, uint64_t b) { return a < b ? a : b; }
__host__ __forceinline__ bool list_active(const RankSet &S, int L) {
  const uint32_t M = (L == 0) ? S.k : S.max_moves;
  return M > 0 && (L == 0 || S.budget > 0);
}
__host__ __forceinline__ uint64_t list_target_of(const RankSet &S, int L, bool wide) {
  const uint32_t M = (L == 0) ? S.k : S.max_moves;
  return wide ? 6ull * M + 2048 : 2ull * M + 1024;
}
__host__ uint64_t sample_size_raw(const RankSet &S, bool wide) {
  if (S.n <= kSample) return 0;
  uint64_t tmax = 0;
  for (int L = 0; L < kLists; L++)
    if (list_active(S, L) && list_target_of(S, L, wide) > tmax) tmax = list_target_of(S, L, wide);
  if (tmax == 0) return 0;
  return ((uint64_t)kSampleRank * S.n) / tmax;
}

// The sample plan of a set whose group (cta0, nctas) is fixed.
void plan_sample(RankSet &s) {
  const uint32_t cap = (uint32_t)umin64(kSample, (uint64_t)kPerCtaSamples * std::min(s.nctas, kSampleCtas));
  const bool wide = sample_size_raw(s, false) > cap;
  uint64_t ns = umin64(sample_size_raw(s, wide), cap);
  s.sctas = ns ? (uint32_t)std::min<uint64_t>(std::min(s.nctas, kSampleCtas), (ns + kPerCtaSamples - 1) / kPerCtaSamples)
               : 1u;
  ns -= ns % (8ull * s.sctas);  // whole runs, evenly split over the sampling CTAs
  s.ns = (uint32_t)ns;
  s.nruns = s.ns / 8;
  s.sstep = s.nruns ? ((uint64_t)s.n << 16) / s.nruns : 0;
  for (int L = 0; L < kLists; L++)
    s.rL[L] = (s.ns && list_active(s, L)) ? (uint32_t)((list_target_of(s, L, wide) * s.ns + s.n - 1) / s.n) : 0u;
}

// Sampling CTA r of set S (consumer threads): samples j = r * per + jt of
// the CTA's share, run j / 8 covering stratum j / 8 (records from about
// run n / nruns to (run+1) n / nruns), 8 consecutive records at a hashed
// offset in it; each
// eligible sample is counted into its lists' histograms (first in shared
// memory, then the non-zero bins into the set's), and the CTA's ticket says
// its counts are in.
__device__ __noinline__ void sample_share(const RankSet &S, uint32_t r, const uint64_t *t2s, const uint64_t *mgs,
                                         unsigned int *lh, uint64_t *sfree) {
  const uint32_t tid = threadIdx.x;
  const uint32_t nct = S.sctas, act = S.act;
  const uint32_t per = S.ns / nct;  // samples of this CTA (<= 1024, a multiple of 8)
  // the CTA's counts first go to shared memory (lh: kLists * kBins words of
  // the idle stage area); only the non-zero bins then reach the global
  // histogram: samples of near keys share a few bins, and global atomics on
  // one address serialise
  uint4 *lh4 = reinterpret_cast<uint4 *>(lh);
  for (uint32_t i = tid; i < kLists * kBins / 4; i += kConsumers) lh4[i] = make_uint4(0u, 0u, 0u, 0u);
  consumers_sync();
  uint32_t rr[kSampleQ];
  bool ok[kSampleQ];
#pragma unroll
  for (int q = 0; q < (int)kSampleQ; q++) {
    const uint32_t jt = tid + kConsumers * q;
    ok[q] = jt < per;
    rr[q] = 0;
    if (ok[q]) {
      // stratum bounds about run n / nruns (16.16 fixed point: no division
      // on the sample's path; any stratification samples correctly)
      const uint32_t run = r * (per / 8) + jt / 8, o = jt % 8;
      const uint32_t lo = (uint32_t)((run * S.sstep) >> 16), hi = (uint32_t)(((run + 1) * S.sstep) >> 16);
      uint32_t h = run * 0x9E3779B1u;
      h ^= h >> 16;
      h *= 0x85EBCA6Bu;
      h ^= h >> 13;
      const uint32_t span = hi - lo >= 8 ? hi - lo - 8 : 0u;  // strata hold at least 8 records
      rr[q] = min(lo + __umulhi(h, span + 1) + o, S.n - 1);
    }
  }
  uint8_t fl[kSampleQ], tr[kSampleQ];
  uint16_t tu[kSampleQ];
  uint32_t gg[kSampleQ];
#pragma unroll
  for (int q = 0; q < (int)kSampleQ; q++) {  // index 0 for an unused slot: a valid record
    fl[q] = S.flags[rr[q]];
    tr[q] = S.tier[rr[q]];
    tu[q] = S.turn[rr[q]];
    gg[q] = S.gap[rr[q]];
  }
  // near keys share bins: the lanes of a warp that hit one bin add to it once
#pragma unroll
  for (int q = 0; q < (int)kSampleQ; q++) {
    const uint32_t t = min((uint32_t)tu[q], kTMax);
    const uint64_t ck = ck_of(score_of(gg[q], t, (fl[q] & 2) != 0, t2s, mgs), S.off + rr[q]);
    const uint32_t em = ok[q] ? elig_mask(fl[q], tr[q]) & act : 0u;
#pragma unroll
    for (int L = 0; L < kLists; L++) {
      const uint32_t b = ((em >> L) & 1) ? L * kBins + bin_of(summary_of(list_val(ck, L))) : 0xFFFFFFFFu;
      const unsigned grp = __match_any_sync(kFull, b);
      if (b != 0xFFFFFFFFu && (__ffs(grp) - 1) == (int)(tid & 31)) atomicAdd(&lh[b], (unsigned)__popc(grp));
    }
  }
  if (tid == 0) atomicAdd(&S.work->gathered, 1u);  // the group's copies may start now
  consumers_sync();
  for (uint32_t i = tid; i < kLists * kBins / 4; i += kConsumers) {
    const uint4 c = lh4[i];
    if (c.x) atomicAdd(&S.shist[4 * i], c.x);
    if (c.y) atomicAdd(&S.shist[4 * i + 1], c.y);
    if (c.z) atomicAdd(&S.shist[4 * i + 2], c.z);
    if (c.w) atomicAdd(&S.shist[4 * i + 3], c.w);
  }
  fence_proxy_async();  // these generic accesses before the producer's bulk copies into the area
  __threadfence();
  consumers_sync();
  if (tid == 0) {
    mbar_arrive(sfree);                      // the stage area is the producer's again
    atomicAdd(&S.work->sample_ticket, 1u);  // this CTA's counts are in the histogram
  }
}

// ------------------------------------------------------------- filter ----
struct SetConst {
  uint64_t thr[kLists];        // threshold per list, in list-value space (0: every eligible record)
  uint32_t loV, loD, loP;      // index thresholds of the tie on the threshold key
  uint32_t dV, dD;             // completed records pass V / D iff lo >= dV / dD
  int32_t dP;                  // completed records pass P iff lo <= dP
  uint32_t act;                // active lists (bit L)
};

// Thresholds of one set into shared memory (consumer threads), computed by
// every CTA of the group alike once the sample's counts are all in the
// histogram: each list's histogram is cut at its sample rank r_L, the
// threshold is the smallest list value of the cut's bin (0, every eligible
// record, when the sample holds fewer than r_L), and per turn index t the
// bounds are the smallest gap whose key reaches the threshold's key (gA) or
// exceeds it (gB): vd = (gA_V, gB_V, gA_D, gB_D), pp = (gA_P, gB_P).  An
// inactive list gets bounds no gap passes.
__device__ void thresholds(const RankSet &S, const uint64_t *t2s, const uint32_t *sgs, uint4 *vd, uint2 *pp,
                           SetConst &c) {
  __shared__ uint64_t sthr[kLists];
  int cut[kLists] = {-1, -1, -1};
  if (S.ns) {
    const uint32_t need[kLists] = {S.rL[0], S.rL[1], S.rL[2]};
    hist_cut3(S.shist, need, cut);
  }
  if (threadIdx.x < kLists) sthr[threadIdx.x] = cut[threadIdx.x] >= 0 ? summary_floor(bin_floor((uint32_t)cut[threadIdx.x])) : 0ull;
  consumers_sync();
  const bool aV = S.act & 1, aD = (S.act >> 1) & 1, aP = (S.act >> 2) & 1;
  if (threadIdx.x < kLutN) {
    const uint32_t t = threadIdx.x;
    uint2 g[kLists];
#pragma unroll
    for (int L = 0; L < kLists; L++) {
      const uint64_t thr_ck = (L == 2) ? ~sthr[L] : sthr[L];
      const uint64_t K = thr_ck >> 24;
      g[L] = make_uint2(g_at_least(K, sgs[t], t2s[t]), g_at_least(K + 1, sgs[t], t2s[t]));
    }
    vd[t] = make_uint4(aV ? g[0].x : kFull, aV ? g[0].y : kFull, aD ? g[1].x : kFull, aD ? g[1].y : kFull);
    pp[t] = aP ? g[2] : make_uint2(0u, 0u);
  }
  if (threadIdx.x == 32) {
    uint32_t lo[kLists], dok[kLists];
#pragma unroll
    for (int L = 0; L < kLists; L++) {
      const uint64_t thrv = sthr[L];
      c.thr[L] = thrv;
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
    c.act = S.act;
  }
  consumers_sync();
}

// ------------------------------------------------------------- finish ----
// Exact top-M of list L over the whole set by one CTA, streaming records and
// keeping a pool of at most M + 4 * kConsumers values in pool[] (the
// fallback path).  The result is in pool[0..return).
__device__ __noinline__ uint32_t stream_topM(const RankSet &S, int L, uint32_t M, uint64_t *pool, const uint64_t *t2s,
                                const uint64_t *mgs, SelectScratch &ss) {
  if (threadIdx.x == 0) ss.cnt = 0;
  uint64_t floorv = 0;  // accept values strictly above (once a floor exists)
  bool have_floor = false;
  consumers_sync();
  for (uint32_t b = 0; b < S.n; b += 4 * kConsumers) {
    for (uint32_t q = 0; q < 4; q++) {
      const uint32_t r = b + q * kConsumers + threadIdx.x;
      if (r < S.n) {
        const uint32_t m = elig_mask(S.flags[r], S.tier[r]);
        if ((m >> L) & 1) {
          const uint32_t t = min((uint32_t)S.turn[r], kTMax);
          const uint64_t v = list_val(ck_of(score_of(S.gap[r], t, (S.flags[r] & 2) != 0, t2s, mgs), S.off + r), L);
          if (!have_floor || v > floorv) pool[atomicAdd(&ss.cnt, 1u)] = v;
        }
      }
    }
    consumers_sync();
    const uint32_t c = ss.cnt;
    if (c > M) {
      const uint64_t th = block_select_rank([&](uint32_t i) { return pool[i]; }, c, M, ss);
      // compact in place to the values >= th (exactly M: values are unique),
      // through registers so that no unread value is overwritten
      constexpr uint32_t kKeep = (kMaxSel + 4 * kConsumers) / kConsumers;  // entries a thread scans, at most
      uint64_t keep[kKeep];
      uint32_t nk = 0;
      for (uint32_t i = threadIdx.x; i < c; i += kConsumers) {
        const uint64_t v = pool[i];
        if (v >= th && nk < kKeep) keep[nk++] = v;
      }
      if (threadIdx.x == 0) ss.cnt = 0;
      consumers_sync();
      for (uint32_t i = 0; i < nk; i++) pool[atomicAdd(&ss.cnt, 1u)] = keep[i];
      consumers_sync();
      floorv = th;
      have_floor = true;
    }
    consumers_sync();
  }
  const uint32_t got = min(ss.cnt, M);
  consumers_sync();
  return got;
}

// List L of set S: the exact top-M of its candidates, sorted, with the moved
// records' sizes; victims are written out directly.  fin: the 64 KB dynamic
// area (the stages are idle).  Returns true when this was the set's last list.
__device__ __noinline__ bool finish_list(const RankSet &S, int L, uint64_t *fin, const uint64_t *t2s, const uint64_t *mgs,
                                         SelectScratch &ss, const SetConst &cs) {
  __shared__ __align__(8) uint64_t cbar;
  __shared__ unsigned int last, sh_emitted, sh_flags, nsurv;
  uint64_t *buf = fin;               // [kSmemCand] candidates
  uint64_t *sel = fin + kSmemCand;   // [kMaxSel] the kept top-M
  const uint32_t tid = threadIdx.x, lane = tid & 31;
  // one thread reads the other CTAs' results, so that every consumer thread
  // takes the same path through the barriers below
  if (tid == 0) {
    sh_emitted = __ldcg(&S.work->cand[L]);
    sh_flags = ((cs.act >> L) & 1u) | (cs.thr[L] == 0 ? 2u : 0u);
  }
  consumers_sync();
  const bool active = sh_flags & 1;
  const uint32_t Mw = (L == 0) ? S.k : S.max_moves;
  const uint32_t emitted = sh_emitted;
  // Candidates are every eligible record at or beyond the threshold.  They
  // certify the top Mw when there are at least Mw of them, or when the
  // threshold admitted every eligible record; otherwise (or when the list
  // overflowed) the list is re-selected exactly from the whole set.
  const bool all_admitted = (sh_flags & 2) != 0;
  const bool certified = emitted <= S.ccap && (emitted >= Mw || all_admitted);
  const uint32_t M = !active ? 0u : (certified ? min(Mw, emitted) : Mw);
  uint32_t got = 0;
  uint64_t *out = sel;
  if (M > 0) {
    const uint64_t *cand = S.cand + (size_t)L * S.ccap;
    if (certified) {
      const uint32_t c = emitted;
      const bool in_smem = c <= kSmemCand;
      if (in_smem) {
        // one bulk copy (an even count: a 16-byte multiple; ccap is even, so
        // the list holds c + 1 entries when c is odd, and so does the area)
        const uint32_t bytes = ((c + 1) & ~1u) * 8u;
        fence_proxy_async();  // earlier generic accesses to the area before the async copy
        consumers_sync();
        if (tid == 0) {
          mbar_init(&cbar, 1);
          fence_mbar_init();
          mbar_expect_tx(&cbar, bytes);
          bulk_g2s(buf, cand, bytes, &cbar);
        }
        if (!wait_phase_uniform(S, &cbar, 0))
          wait_phase_uniform(S, &cbar, 0);  // let the copy land before the area is reused
      }
      const uint64_t *src = in_smem ? buf : cand;
      // every candidate, a block-wide pass (fn(v, ok): ok false past the end)
      auto each_w = [&](auto fn) {
        for (uint32_t base = 0; base < c; base += kConsumers) {
          const uint32_t i = base + tid;
          fn(i < c ? src[i] : 0ull, i < c);
        }
      };
      auto each = [&](auto fn) {
        each_w([&](uint64_t v, bool ok) {
          if (ok) fn(v);
        });
      };
      if (c <= M) {
        // every candidate is kept
        for (uint32_t i = tid; i < c; i += kConsumers) sel[i] = src[i];
        got = c;
      } else {
        // the values in the bucket holding the rank-M value and above it: at
        // least M of them, and the top M among them are the top M of all
        // candidates (every other value is in a lower bucket, hence smaller)
        int sh = 0;
        uint32_t bcut = 0;
        const uint32_t ns = bucket_cut(each, M, ss, sh, bcut);
        if (ns <= kMaxSel) {
          if (tid == 0) nsurv = 0;
          consumers_sync();
          each_w([&](uint64_t v, bool ok) {
            const bool keep = ok && ((uint32_t)(v >> sh) & 255u) >= bcut;
            const unsigned bal = __ballot_sync(kFull, keep);
            unsigned wb = 0;
            if (lane == 0 && bal) wb = atomicAdd(&nsurv, (unsigned)__popc(bal));
            wb = __shfl_sync(kFull, wb, 0);
            const uint32_t pos = wb + __popc(bal & ((1u << lane) - 1));
            if (keep) sel[pos] = v;
          });
          consumers_sync();
          got = ns;
        } else {
          // the cut's bucket holds too many values: radix select of the
          // rank-M value over every candidate
          ss.hist[tid] = 0;
          consumers_sync();
          const uint64_t th = block_select_rank([&](uint32_t i) { return src[i]; }, c, M, ss);
          if (tid == 0) ss.cnt = 0;
          consumers_sync();
          each_w([&](uint64_t v, bool ok) {
            const bool keep = ok && v >= th;
            const unsigned bal = __ballot_sync(kFull, keep);
            unsigned wb = 0;
            if (lane == 0 && bal) wb = atomicAdd(&ss.cnt, (unsigned)__popc(bal));
            wb = __shfl_sync(kFull, wb, 0);
            const uint32_t pos = wb + __popc(bal & ((1u << lane) - 1));
            if (keep && pos < kMaxSel) sel[pos] = v;
          });
          consumers_sync();
          got = min(ss.cnt, M);
        }
      }
      consumers_sync();
      sort_desc(sel, got, buf, ss);
      got = min(got, M);
    } else {
      // candidates overflowed the buffer or fell short of M: exact re-selection
      ss.hist[threadIdx.x] = 0;
      consumers_sync();
      got = stream_topM(S, L, M, fin, t2s, mgs, ss);
      out = fin;
      sort_desc(fin, got, fin + kMaxSel, ss);
    }
    // store the list; the fill reads the moved records' sizes, gathered here
    // eight at a time (independent random reads)
    for (uint32_t base = 0; base < got; base += 8 * kConsumers) {
      uint64_t v[8];
      uint32_t kv[8];
#pragma unroll
      for (int u = 0; u < 8; u++) {
        const uint32_t i = base + u * kConsumers + threadIdx.x;
        v[u] = i < got ? out[i] : 0ull;
        const uint32_t idx = (~(uint32_t)(L == 2 ? ~v[u] : v[u])) & kIdMask;
        kv[u] = (L != 0 && i < got) ? S.kv[idx - S.off] : 0u;
      }
#pragma unroll
      for (int u = 0; u < 8; u++) {
        const uint32_t i = base + u * kConsumers + threadIdx.x;
        if (i < got) {
          if (S.cands) {  // a shard: the list goes out, keyed by the whole set's index
            CandEntry *e = reinterpret_cast<CandEntry *>(S.cands + cand_list_off(S.k, S.max_moves, L));
            e[i] = CandEntry{v[u], kv[u], 0u};
          } else {
            S.sorted[(size_t)L * kMaxSel + i] = v[u];
            if (L == 0) S.victims[i] = (~(uint32_t)v[u]) & kIdMask;
            else S.ssz[(size_t)L * kMaxSel + i] = kv[u];
          }
        }
      }
    }
  }
  if (threadIdx.x == 0) {
    S.work->got[L] = got;
    if (S.cands) reinterpret_cast<CandHeader *>(S.cands)->count[L] = got;
  }
  __threadfence();
  consumers_sync();
  if (threadIdx.x == 0) last = (atomicAdd(&S.work->list_ticket, 1u) == (unsigned)kLists - 1);
  consumers_sync();
  return last != 0;
}

// ------------------------------------------------------------- fill ----
// Inclusive prefix over the consumer threads of (a, b); the block's totals
// come back in (ta, tb).  Two barriers.
__device__ void block_incl_scan2(uint64_t &a, int64_t &b, uint64_t &ta, int64_t &tb) {
  __shared__ uint64_t wa[kConsumers / 32];
  __shared__ int64_t wb[kConsumers / 32];
  const uint32_t lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint64_t ya = __shfl_up_sync(kFull, a, o);
    const int64_t yb = __shfl_up_sync(kFull, b, o);
    if ((int)lane >= o) {
      a += ya;
      b += yb;
    }
  }
  if (lane == 31) {
    wa[warp] = a;
    wb[warp] = b;
  }
  consumers_sync();
  uint64_t pa = 0, sa = 0;
  int64_t pb = 0, sb = 0;
#pragma unroll
  for (uint32_t w = 0; w < kConsumers / 32; w++) {
    if (w < warp) {
      pa += wa[w];
      pb += wb[w];
    }
    sa += wa[w];
    sb += wb[w];
  }
  a += pa;
  b += pb;
  ta = sa;
  tb = sb;
  consumers_sync();  // wa and wb free for the next call
}

// The TIDE fill of set S from its sorted lists (Sec. III-C): phase 1
// promotes the least evictable HBM records into free fast-tier space in order
// while the budget and the space last; phase 2 pairs the next HBM record with
// the j-th most evictable fast-tier record (demotions merged with the phase-1
// promotions) while the demoted one ranks above the promoted one and the
// budget and both tiers' capacities hold.  Each phase takes items in order
// and stops at the first that fails.  The state after j items is a prefix
// sum, so the consumer threads take a phase 256 items at a time, one item
// each: a block scan of the sizes, then the smallest failing item of the
// chunk; the fill stops at the first chunk that holds one (most fills end in
// the first).  Every size is in tokens and the budget test is on tokens: j
// items of s_1..s_j tokens cost (s_1 + ... + s_j) * kvb bytes, which is
// within the budget exactly when s_1 + ... + s_j <= floor(budget / kvb).
// The lists are staged in shared memory (P as ascending key, D descending,
// 12 bytes an entry) when they fit, else read in place.
__device__ __noinline__ void fill(const RankSet &S, uint64_t *fin) {
  __shared__ unsigned int sh_got[kLists], sh_act, sh_st, first_bad;
  __shared__ unsigned long long sh_tok;
  __threadfence();
  const uint32_t tid = threadIdx.x;
  if (tid == 0) {  // read once and shared: one path through the barriers
    for (int L = 0; L < kLists; L++) sh_got[L] = min(__ldcg(&S.work->got[L]), kMaxSel);
    sh_act = S.act & 6u;
    sh_st = *(volatile unsigned int *)&S.work->status;
  }
  consumers_sync();
  const uint32_t nv = sh_got[0], nd = sh_got[1], np = sh_got[2];
  const uint64_t *Pg = S.sorted + 2 * kMaxSel, *Dg = S.sorted + kMaxSel;
  const uint32_t *PSg = S.ssz + 2 * kMaxSel, *DSg = S.ssz + kMaxSel;
  const bool staged = 12ull * (np + nd) <= kDynSmem;
  uint64_t *pck = fin, *dck = fin + np;
  uint32_t *psz = reinterpret_cast<uint32_t *>(fin + np + nd), *dsz = psz + np;
  if (staged) {
    for (uint32_t i = tid; i < np; i += kConsumers) {
      const uint64_t x = ~__ldcg(Pg + i);
      const uint32_t z = __ldcg(PSg + i);
      pck[i] = x;
      psz[i] = z;
    }
    for (uint32_t i = tid; i < nd; i += kConsumers) {
      const uint64_t x = __ldcg(Dg + i);
      const uint32_t z = __ldcg(DSg + i);
      dck[i] = x;
      dsz[i] = z;
    }
  }
  auto p_ck = [&](uint32_t i) -> uint64_t { return staged ? pck[i] : ~__ldcg(Pg + i); };
  auto p_sz = [&](uint32_t i) -> uint32_t { return staged ? psz[i] : __ldcg(PSg + i); };
  auto d_ck = [&](uint32_t i) -> uint64_t { return staged ? dck[i] : __ldcg(Dg + i); };
  auto d_sz = [&](uint32_t i) -> uint32_t { return staged ? dsz[i] : __ldcg(DSg + i); };
  if (tid == 0) first_bad = kFull;
  consumers_sync();
  const uint64_t kvb = S.kvb, cap_b = S.budget / kvb;  // tokens the budget pays for
  // phase 1: promotions into free fast-tier space, least evictable first
  const uint32_t lim1 = (sh_act & 4) ? min(np, S.max_moves) : 0u;
  const uint64_t cap1 = min(cap_b, S.free_s);
  uint32_t n1 = lim1;
  uint64_t tok1 = 0;  // tokens promoted so far
  for (uint32_t base = 0; base < lim1; base += kConsumers) {
    const uint32_t j = base + tid;
    uint64_t a = j < lim1 ? p_sz(j) : 0u, ta;
    int64_t b = 0, tb;
    block_incl_scan2(a, b, ta, tb);
    if (j < lim1 && tok1 + a > cap1) atomicMin(&first_bad, j);
    consumers_sync();
    const uint32_t fb = first_bad;
    if (fb != kFull) {
      if (j + 1 == fb) sh_tok = tok1 + a;
      consumers_sync();
      n1 = fb;
      if (fb > base) tok1 = sh_tok;
      if (tid == 0) first_bad = kFull;
      consumers_sync();
      break;
    }
    tok1 += ta;
  }
  // phase 2: pair P[n1 + j] with the j-th entry of the demotion order
  const uint64_t cap2b = cap_b - tok1, fs = S.free_s - tok1, fh = S.free_h + tok1;
  const uint32_t cap2 = S.max_moves > n1 ? S.max_moves - n1 : 0;
  const uint32_t nd2 = min(nd + n1, cap2);
  const uint32_t lim2 = ((sh_act & 6) == 6) ? min(np - n1, nd2) : 0u;
  // the j-th entry (descending) of D merged with P[n1-1], ..., P[0]
  auto demote_at = [&](uint32_t j, uint64_t &val, uint32_t &sz) {
    uint32_t lo = j + 1 > n1 ? j + 1 - n1 : 0u, hi = min(j + 1, nd);
    while (lo < hi) {  // D entries among the top j + 1
      const uint32_t mid = (lo + hi) >> 1;
      if (d_ck(mid) > p_ck(n1 - 1 - (j - mid))) lo = mid + 1; else hi = mid;
    }
    const uint32_t i = lo;
    if (i == 0 || (j + 1 - i > 0 && p_ck(n1 - 1 - (j - i)) < d_ck(i - 1))) {
      const uint32_t pj = n1 - 1 - (j - i);  // the smaller of the two last taken is from P
      val = p_ck(pj);
      sz = p_sz(pj);
    } else {
      val = d_ck(i - 1);
      sz = d_sz(i - 1);
    }
  };
  uint32_t pairs = lim2;
  uint64_t tok2 = 0;  // tokens moved by the pairs so far (both directions)
  int64_t bal = 0;    // net tokens into the fast tier so far
  for (uint32_t base = 0; base < lim2; base += kConsumers) {
    const uint32_t j = base + tid;
    uint64_t a = 0, ta;
    int64_t b = 0, tb;
    bool order_ok = false;
    if (j < lim2) {
      uint64_t dv;
      uint32_t sd;
      demote_at(j, dv, sd);
      const uint32_t sp = p_sz(n1 + j);
      order_ok = dv > p_ck(n1 + j);
      a = (uint64_t)sp + sd;
      b = (int64_t)sp - (int64_t)sd;
    }
    block_incl_scan2(a, b, ta, tb);
    const uint64_t A = tok2 + a;
    const int64_t Bv = bal + b;
    const bool ok = order_ok && A <= cap2b && (Bv <= 0 || (uint64_t)Bv <= fs) && (Bv >= 0 || (uint64_t)(-Bv) <= fh);
    if (j < lim2 && !ok) atomicMin(&first_bad, j);
    consumers_sync();
    const uint32_t fb = first_bad;
    if (fb != kFull) {
      if (j + 1 == fb) sh_tok = A;
      consumers_sync();
      pairs = fb;
      if (fb > base) tok2 = sh_tok;
      break;
    }
    tok2 += ta;
    bal += tb;
  }
  for (uint32_t i = tid; i < n1 + pairs; i += kConsumers) S.promote[i] = (~(uint32_t)p_ck(i)) & kIdMask;
  for (uint32_t i = tid; i < pairs; i += kConsumers) {
    uint64_t dv;
    uint32_t sd;
    demote_at(i, dv, sd);
    S.demote[i] = (~(uint32_t)dv) & kIdMask;
  }
  if (tid == 0) {
    S.counts[0] = nv;
    S.counts[1] = n1 + pairs;
    S.counts[2] = pairs;
    S.counts[3] = sh_st ? sh_st : (unsigned int)UNISON_OK;
    S.moved[0] = (tok1 + tok2) * kvb;  // at most floor(budget / kvb) tokens
  }
  consumers_sync();
}

// ------------------------------------------------------------- kernel ----
// Grouped (sequential == 0): CTA c serves the set whose group holds it.
// Sequential: CTA c serves sets c, c + G, c + 2G, ... one after another, each
// as a group of one.  The producer warp takes the group's tiles from the
// set's counter and announces each stage's tile in stile[]; a partial last
// tile (read directly from global memory by the consumers) and the end of
// the set (kEndTile) are announced with a plain arrival.
// zero_a / zero_b (n_a, n_b 16-byte words): the other parity's work words
// and sample histograms, zeroed here for the next call on the stream.
// cmap (grouped launches): CTA b serves set cmap[b] & 0xFFFF, whose tables are
// tabs[cmap[b] >> 16]; null for a sequential launch.
__global__ void __launch_bounds__(kCtaThreads, 3)
    rank_kernel(const RankSet *sets, int n_sets, int sequential, const uint32_t *cmap, const RankTab *tabs,
                uint4 *zero_a, uint32_t n_a, uint4 *zero_b, uint32_t n_b) {
  extern __shared__ __align__(128) unsigned char dsm[];
  FilterStage *stage = reinterpret_cast<FilterStage *>(dsm);
  uint64_t *fin = reinterpret_cast<uint64_t *>(dsm);
  __shared__ __align__(8) uint64_t full[kStages], empty[kStages], sdone, sfree;
  __shared__ unsigned int stile[kStages];
  __shared__ uint4 vd[kLutN];
  __shared__ uint2 pp[kLutN];
  __shared__ uint64_t t2s[kLutN], mgs[kLutN];
  __shared__ SetConst cset;
  __shared__ RankSet rset;
  __shared__ unsigned int ccnt_s[kLists];  // candidates this CTA appended per list
  __shared__ unsigned int cbase_s[kLists];  // where its region goes in the set's list
  __shared__ uint32_t sgs[kLutN];
  __shared__ CtaScratch u;
  __shared__ unsigned int arrival;
#ifdef UNISON_DEBUG_HOOKS
  __shared__ __align__(8) uint64_t dummy_bar;
#endif

  {  // every CTA takes its share, before any returns
    const uint32_t g = blockIdx.x * blockDim.x + threadIdx.x, gs = gridDim.x * blockDim.x;
    for (uint32_t w = g; w < n_a; w += gs) zero_a[w] = make_uint4(0u, 0u, 0u, 0u);
    for (uint32_t w = g; w < n_b; w += gs) zero_b[w] = make_uint4(0u, 0u, 0u, 0u);
  }
  int s0, sstep;
  const RankTab *tab0 = nullptr;  // the first set's tables, when the map names them
  if (sequential) {
    s0 = blockIdx.x;
    sstep = gridDim.x;
  } else {
    const uint32_t e = __ldg(cmap + blockIdx.x);
    s0 = (int)(e & 0xFFFFu);
    tab0 = tabs + (e >> 16);
    sstep = n_sets;  // one set
  }
  if (s0 >= n_sets) return;
  if (threadIdx.x == 0) {
    for (int q = 0; q < kStages; q++) {
      mbar_init(&full[q], 1);
      mbar_init(&empty[q], kConsumers / 32);
    }
    mbar_init(&sdone, 1);
    mbar_init(&sfree, 1);
#ifdef UNISON_DEBUG_HOOKS
    mbar_init(&dummy_bar, 1);
#endif
    fence_mbar_init();
  }
  __syncthreads();
  const int lane = threadIdx.x & 31;

  if (threadIdx.x >= kConsumers) {
    // ---------------- producer warp (one lane issues)
    if (lane != 0) return;
    uint32_t lastph = 0;  // bit q: parity of the phase of stage q's last bulk copy
    uint32_t issued = 0;  // bit q: the last bulk copy into stage q may still be in flight
    uint32_t i = 0, nsets = 0, nsampled = 0;
    bool failed = false;
    int sfail = s0;
    for (int s = s0; s < n_sets && !failed; s += sstep) {
      const RankSet &T = sets[s];
      const uint32_t r = sequential ? 0u : blockIdx.x - T.cta0, nct = sequential ? 1u : T.nctas;
      // A sampling CTA counts its sample in the stage area: its copies wait
      // until the consumers are done with it.
      if (r < T.sctas) {
        if (!mbar_wait_bounded(&sfree, nsampled & 1)) {
          failed = true;
          sfail = s;
          break;
        }
        nsampled++;
      } else if (T.ns) {
        // The sample's random reads go first: the group's bulk copies would
        // otherwise queue ahead of them at the memory.  A short bounded wait;
        // if it runs out the copies simply start.
        const uint64_t t0 = now_ns();
        uint32_t nap = 64;
        while (*(volatile const unsigned int *)&T.work->gathered < T.sctas && now_ns() - t0 < 20000u) {
          __nanosleep(nap);
          nap = min(nap * 2, 512u);
        }
      }
      uint32_t claim = 0;  // the counter's answer for the next item, asked one item ahead
      for (uint32_t item = 0;; item++) {
        const int q = (int)(i % kStages);
        if (i >= (uint32_t)kStages) {
          // wait until the consumers released this stage's previous item
          if (!mbar_wait_bounded(&empty[q], ((i / kStages) - 1) & 1)) {
            failed = true;
            sfail = s;
            break;
          }
          issued &= ~(1u << q);
        }
        // the first kStages items of each CTA are dealt round-robin (every
        // CTA starts at once, and a set of few tiles spreads over the group);
        // the rest come from the group's counter, so that CTAs slowed by
        // candidate-heavy tiles take fewer
        const uint32_t t = item < (uint32_t)kStages ? r + item * nct : nct * kStages + claim;
        // ask for the next item's tile now: the answer's round trip overlaps
        // this item's copy and the wait for the next free stage
        if (item + 1 >= (uint32_t)kStages && t < T.ntiles) claim = atomicAdd(&T.work->next_tile, 1u);
        const uint32_t base = t < T.ntiles ? t * kBigTile : 0u;
        stile[q] = t < T.ntiles ? t : kEndTile;
        if (t >= T.ntiles || base + kBigTile > T.n) {
          mbar_arrive(&full[q]);  // the end of the set, or a partial tile read directly
          i++;
          if (t >= T.ntiles) break;
          continue;
        }
        FilterStage &d = stage[q];
        fence_proxy_async();
        mbar_expect_tx(&full[q], kBigTile * 8);
        bulk_g2s(d.gap, T.gap + base, kBigTile * 4, &full[q]);
        bulk_g2s(d.turn, T.turn + base, kBigTile * 2, &full[q]);
        bulk_g2s(d.flags, T.flags + base, kBigTile, &full[q]);
        bulk_g2s(d.tier, T.tier + base, kBigTile, &full[q]);
        issued |= 1u << q;
        lastph = (lastph & ~(1u << q)) | (((i / kStages) & 1) << q);
        i++;
      }
      // the consumers may use the stage memory for this set's finish: the next
      // set's copies wait until they are done with it
      if (!failed && s + sstep < n_sets) {
        if (!mbar_wait_bounded(&sdone, nsets & 1)) {
          failed = true;
          sfail = s;
        }
        nsets++;
      }
    }
    if (failed) {
      set_status(sets[sfail], UNISON_ERR_TIMEOUT);
      // consumers that still wait will time out too; let this CTA's copies land
      // before the CTA exits
      for (int q = 0; q < kStages; q++)
        if ((issued >> q) & 1) mbar_wait_bounded(&full[q], (lastph >> q) & 1);
    }
    return;
  }

  // ---------------- consumer warps
  const uint32_t ct = threadIdx.x;
  SetConst &c = cset;
  uint32_t i = 0;    // the CTA's running stage count (the producer's sequence)
  for (int s = s0; s < n_sets; s += sstep) {
    // the set's descriptor in shared memory: its fields are read throughout
    // the set's phases, each read from global memory a round trip.  The
    // tables come in the same round trip when the map names them.
    static_assert(sizeof(RankSet) % 8 == 0, "copied in 8-byte words");
    for (uint32_t w = ct; w < sizeof(RankSet) / 8; w += kConsumers)
      reinterpret_cast<uint64_t *>(&rset)[w] = reinterpret_cast<const uint64_t *>(sets + s)[w];
    if (tab0 && ct < kLutN) {
      t2s[ct] = tab0->t2v[ct];
      mgs[ct] = tab0->mgv[ct];
      sgs[ct] = tab0->sigma[ct];
    }
    consumers_sync();
    const RankSet &S = rset;
    const uint32_t r = sequential ? 0u : blockIdx.x - S.cta0;
    if (!tab0) {
      if (ct < kLutN) {
        t2s[ct] = S.tab->t2v[ct];
        mgs[ct] = S.tab->mgv[ct];
        sgs[ct] = S.tab->sigma[ct];
      }
      consumers_sync();
    }
    // 1. thresholds: the sampling CTAs sample; every CTA cuts the histograms
    if (r < S.sctas) sample_share(S, r, t2s, mgs, reinterpret_cast<unsigned int *>(dsm), &sfree);
#ifdef UNISON_DEBUG_HOOKS
    if (s == g_hook_flag_set) wait_word(S, &S.work->dummy, 1u);  // nothing sets it: runs out
#endif
    wait_word(S, &S.work->sample_ticket, S.sctas);
    if (ct < kLists) ccnt_s[ct] = 0;  // published by the barriers below
    thresholds(S, t2s, sgs, vd, pp, c);
    const uint32_t s_n = S.n;
    const bool s_keys = S.keys != nullptr;
    // Segment: a run of tiles over which every index condition of the set has
    // one class (all, none or mixed).  Within a set each condition changes
    // class at most twice (at the tile holding its boundary and the one
    // after), so a set has at most 13 segments.  A CTA's tiles come in
    // rising order.
    uint32_t seg_end = 0;  // first tile of the next segment
    bool seg_mixed = false, seg_none = false;
#ifdef UNISON_DEBUG_HOOKS
    bool first_tile = true;
#endif
    // 2. stream the tiles the group's counter hands this CTA: at most all of
    // the set's tiles and the end mark.  A wait that runs out ends the CTA's
    // streaming (its set's results are then undefined, and its status says so).
    for (uint32_t items = 0; items <= S.ntiles; items++, i++) {
      const int q = (int)(i % kStages);
#ifdef UNISON_DEBUG_HOOKS
      // a barrier nothing arrives at: the bounded wait runs out and reports
      if (first_tile && s == g_hook_mbar_set) wait_phase_uniform(S, &dummy_bar, 0, kWaitNs);
#endif
      if (!wait_phase_uniform(S, &full[q], (i / kStages) & 1)) {
        i++;
        break;
      }
      const uint32_t t = stile[q];
      if (t == kEndTile) {
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[q]);
        i++;
        break;
      }
      const uint32_t tb = t * kBigTile;
      if (t >= seg_end) {
        // Index conditions over this tile: record indices rise through the
        // tile, so lo = ~index falls from lo_hi to lo_lo and each tie condition
        // on lo holds for all, none or a part of the tile.
        const uint32_t tcount = min(kBigTile, s_n - tb);
        const uint32_t gtb = S.off + tb;  // the tile's first index in the whole set
        const uint32_t lo_hi = (~gtb) & kIdMask, lo_lo = (~(gtb + tcount - 1)) & kIdMask;
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
        uint32_t nxt = S.ntiles;
        auto upd = [&](int64_t lo_bound) {
          const int64_t b = (int64_t)kIdMask - lo_bound - S.off;  // a local index
          if (b < 0 || b >= (int64_t)s_n) return;
          const uint32_t tbnd = (uint32_t)b / kBigTile;
          if (tbnd > t) nxt = min(nxt, tbnd);
          else if (tbnd + 1 > t) nxt = min(nxt, tbnd + 1);
        };
        upd(c.loV); upd(c.loD); upd(c.loP); upd(c.dV); upd(c.dD); upd(c.dP);
        seg_end = nxt;
        // Per-segment bound table over (turn index, record class): a record of
        // class cls at turn index t may be a candidate of some list iff
        // g >= x or g < y.  Classes: 0 not eligible, 1 live fast tier, 2 live
        // HBM tier, 3 completed fast tier, 4 completed HBM tier.
        consumers_sync();  // everyone is done with the previous table
        bool live = false;
        if (!seg_mixed && ct < kLutN * 5) {
          const uint32_t tt = ct / 5, cls = ct % 5;
          const uint4 a = vd[tt];
          const uint2 bb = pp[tt];
          const uint32_t bV = iV == 1 ? a.x : a.y, bD = iD == 1 ? a.z : a.w, bP = iP == 1 ? bb.y : bb.x;
          const bool pdV = (c.act & 1) && dV == 1, pdD = (c.act & 2) && dD == 1, pdP = (c.act & 4) && dP == 1;
          uint2 e = make_uint2(kFull, 0u);
          if (cls == 1) e = make_uint2(min(bV, bD), 0u);
          if (cls == 2) e = make_uint2(bV, bP);
          if (cls == 3) e = make_uint2(pdV || pdD ? 0u : kFull, 0u);
          if (cls == 4) e = make_uint2(pdV ? 0u : kFull, pdP ? kFull : 0u);
          u.f.ftab[ct] = e;
          // gaps are below 2^31: x >= 2^31 and y == 0 admit nothing
          live = e.x < 0x80000000u || e.y != 0u;
        }
        seg_none = !consumers_sync_or(live) && !seg_mixed;
      }
      const bool bulk = tb + kBigTile <= s_n;
      uint32_t g[kRec], tw[kRec / 2], fw[kGroups], rw[kGroups];
      if (bulk) {
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
              g[4 * gi + m] = S.gap[idx];
              tw[2 * gi + (m >> 1)] |= (uint32_t)S.turn[idx] << (16 * (m & 1));
              const uint32_t sh = 8 * m;
              fw[gi] = (fw[gi] & ~(0xFFu << sh)) | ((uint32_t)S.flags[idx] << sh);
              rw[gi] = (rw[gi] & ~(0xFFu << sh)) | ((uint32_t)S.tier[idx] << sh);
            }
          }
        }
      }
#ifdef UNISON_DEBUG_HOOKS
      first_tile = false;
#endif
      auto turn_of = [&](uint32_t k) { return min((tw[k >> 1] >> (16 * (k & 1))) & 0xFFFF, kTMax); };
      auto index_of = [&](uint32_t k) { return tb + (k >> 2) * kGroupStride + 4 * ct + (k & 3); };
      // candidate bit per record (any list): one table lookup per record
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
          const uint32_t gg = g[k], tt = turn_of(k), lo = (~(S.off + index_of(k))) & kIdMask;
          const uint4 a = vd[tt];
          const uint2 b = pp[tt];
          const bool pV = (em & 1) && (done ? lo >= c.dV : (gg >= a.y || (gg >= a.x && lo >= c.loV)));
          const bool pD = (em & 2) && (done ? lo >= c.dD : (gg >= a.w || (gg >= a.z && lo >= c.loD)));
          const bool pP = (em & 4) && (done ? (int32_t)lo <= c.dP : (gg < b.x || (gg < b.y && lo <= c.loP)));
          cm |= (uint32_t)(pV || pD || pP) << k;
        }
      } else if (!seg_none) {
        const unsigned char *tab = reinterpret_cast<const unsigned char *>(u.f.ftab);
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
#pragma unroll
        for (uint32_t k = 0; k < kRec; k++) {
          const uint32_t idx = index_of(k);
          if (idx < s_n) {
            const bool dn = (fw[k >> 2] >> (8 * (k & 3) + 1)) & 1;
            S.keys[idx] = score_of(g[k], turn_of(k), dn, t2s, mgs);
          }
        }
      }
      // The stage is handed back as soon as this warp no longer reads it: at
      // once when none of its records is flagged, else after the exact tests
      // below, which read the flagged records back from the stage.
      const bool flagged = __any_sync(kFull, cm != 0);
      if (!flagged) {
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[q]);
        continue;
      }
      // exact per-list tests of the flagged records: the warp lists their
      // offsets in the tile (kWarpBuf a pass), then each lane tests one and
      // appends its exact value to every list it passes (one atomic per warp
      // and list, the lists' atomics in flight together).  When the last
      // records tested are in registers the stage is handed back before the
      // appends, whose atomics then overlap the stage's next copy.
      uint16_t *wb = u.f.wbuf[ct >> 5];
      const FilterStage &d = stage[q];
      uint32_t rem = cm;
      bool released = false;
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
        for (uint32_t m = rem; m != 0 && pos < kWarpBuf; m &= m - 1, pos++) {
          const uint32_t k = __ffs(m) - 1;
          wb[pos] = (uint16_t)((k >> 2) * kGroupStride + 4 * ct + (k & 3));
          wrote |= 1u << k;
        }
        rem &= ~wrote;
        const bool more = __any_sync(kFull, rem != 0);  // another pass follows
        __syncwarp();
        for (uint32_t j0 = 0; j0 < nb; j0 += 32) {
          const uint32_t j = j0 + lane;
          bool pL[kLists] = {false, false, false};
          uint64_t ck = 0;
          if (j < nb) {
            const uint32_t o = wb[j], idx = tb + o;
            uint32_t gg, tt, fl, tr;
            if (bulk) {
              gg = d.gap[o];
              tt = d.turn[o];
              fl = d.flags[o];
              tr = d.tier[o];
            } else {  // the partial last tile: read from the set (padding is pinned)
              const bool in = idx < s_n;
              gg = in ? S.gap[idx] : 0u;
              tt = in ? S.turn[idx] : 0u;
              fl = in ? S.flags[idx] : 1u;
              tr = in ? S.tier[idx] : 0u;
            }
            tt = min(tt, kTMax);
            const uint32_t em = elig_mask((uint8_t)fl, (uint8_t)tr);
            const bool done = (fl & 2) != 0;
            const uint32_t lo = (~(S.off + idx)) & kIdMask;
            const uint4 a = vd[tt];
            const uint2 b = pp[tt];
            pL[0] = (em & 1) && (done ? lo >= c.dV : (gg >= a.y || (gg >= a.x && lo >= c.loV)));
            pL[1] = (em & 2) && (done ? lo >= c.dD : (gg >= a.w || (gg >= a.z && lo >= c.loD)));
            pL[2] = (em & 4) && (done ? (int32_t)lo <= c.dP : (gg < b.x || (gg < b.y && lo <= c.loP)));
            if (pL[0] || pL[1] || pL[2]) ck = ck_of(score_of(gg, tt, done, t2s, mgs), S.off + idx);
          }
          if (!more && j0 + 32 >= nb) {  // the warp's last reads of the stage are done
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[q]);
            released = true;
          }
          unsigned bal[kLists], base[kLists];
#pragma unroll
          for (int L = 0; L < kLists; L++) {
            bal[L] = __ballot_sync(kFull, pL[L]);
            base[L] = 0;
          }
          if (lane == 0) {
#pragma unroll
            for (int L = 0; L < kLists; L++)
              if (bal[L]) base[L] = atomicAdd(&ccnt_s[L], (unsigned)__popc(bal[L]));
          }
#pragma unroll
          for (int L = 0; L < kLists; L++) {
            if (!bal[L]) continue;
            const uint32_t lt = (1u << lane) - 1;
            const uint32_t at = __shfl_sync(kFull, base[L], 0) + __popc(bal[L] & lt);
            const uint64_t v = list_val(ck, L);
            if (pL[L] && at < S.cr) S.creg[((size_t)L * S.nctas + r) * S.cr + at] = v;
            // past the end of the CTA's region: straight into the set's list
            const unsigned ovf = __ballot_sync(kFull, pL[L] && at >= S.cr);
            if (ovf) {
              unsigned ob = 0;
              if (lane == 0) ob = atomicAdd(&S.work->cand[L], (unsigned)__popc(ovf));
              ob = __shfl_sync(kFull, ob, 0) + __popc(ovf & lt);
              if (pL[L] && at >= S.cr && ob < S.ccap) S.cand[(size_t)L * S.ccap + ob] = v;
            }
          }
        }
        __syncwarp();  // the buffer is rewritten by the next pass
      }
      if (!released && lane == 0) mbar_arrive(&empty[q]);
    }
    // 3. done streaming: the last three CTAs of the group take one list each
    // (a group of fewer CTAs: the last one takes the rest), once every CTA of
    // the group has emitted its candidates; the last list's CTA runs the fill
    // the CTA's region moves to the set's list: one range taken per list
    // (the three atomics in flight together), then copied
    consumers_sync();  // every warp's appends counted
    if (ct < kLists) {
      const uint32_t nr = min(ccnt_s[ct], S.cr);
      cbase_s[ct] = nr ? atomicAdd(&S.work->cand[ct], nr) : 0u;
    }
    consumers_sync();
#pragma unroll 1
    for (int L = 0; L < kLists; L++) {
      const uint32_t nr = min(ccnt_s[L], S.cr), b0 = cbase_s[L];
      const uint64_t *rg = S.creg + ((size_t)L * S.nctas + r) * S.cr;
      for (uint32_t j = ct; j < nr; j += kConsumers)
        if (b0 + j < S.ccap) S.cand[(size_t)L * S.ccap + b0 + j] = __ldcg(rg + j);
    }
    __threadfence();
    consumers_sync();
    if (ct == 0) {
      arrival = atomicAdd(&S.work->done_ctas, 1u);
      __threadfence();  // the earlier arrivals' candidates are visible after this
    }
    consumers_sync();
    const uint32_t nct = sequential ? 1u : S.nctas;
    const uint32_t qr = nct - 1 - arrival;
    uint32_t mine = 0;
#pragma unroll
    for (int L = 0; L < kLists; L++)
      if ((uint32_t)L == qr || (qr == 0 && (uint32_t)L >= nct)) mine |= 1u << L;
    if (mine) {
      if (qr > 0) wait_word(S, &S.work->done_ctas, nct);
      bool last = false;
#pragma unroll 1
      for (int L = 0; L < kLists; L++)
        if ((mine >> L) & 1) last = finish_list(S, L, fin, t2s, mgs, u.s, c);
      if (last && !S.cands) fill(S, fin);
      if (last && S.cands && ct == 0) {  // a shard: the header closes its lists
        CandHeader *h = reinterpret_cast<CandHeader *>(S.cands);
        h->n = S.n;
        h->off = S.off;
        h->k = S.k;
        h->max_moves = S.max_moves;
        h->status = *(volatile unsigned int *)&S.work->status;
      }
    }
    // 4. the stage memory is free for the next set's copies
    consumers_sync();
    if (ct == 0) mbar_arrive(&sdone);
  }
}

// ------------------------------------------------------------- merge ----
// The shards' candidate lists, gathered (n_shards buffers of `stride` bytes
// each): CTA L selects list L's global top M (a radix select when the
// shards hold more than 4,096 entries, then a bitonic sort carrying the
// sizes), writes it as the finish does, and the last list's CTA runs the
// fill.  One CTA per list, consumer-sized (256 threads).
__global__ void __launch_bounds__(kConsumers) rank_merge_kernel(const RankSet *Sp, const unsigned char *gathered,
                                                                int n_shards, uint64_t stride) {
  extern __shared__ __align__(128) unsigned char dsm[];
  uint64_t *fin = reinterpret_cast<uint64_t *>(dsm);
  __shared__ SelectScratch ss;
  __shared__ unsigned int pre[kMaxShards + 1];
  __shared__ unsigned int last;
  const RankSet &S = *Sp;
  const int L = blockIdx.x;
  const uint32_t Mw = L == 0 ? S.k : S.max_moves;
  const bool active = (S.act >> L) & 1;
  const size_t loff = cand_list_off(S.k, S.max_moves, L);
  if (threadIdx.x == 0) {
    pre[0] = 0;
    for (int sh = 0; sh < n_shards; sh++) {
      const CandHeader *h = reinterpret_cast<const CandHeader *>(gathered + stride * sh);
      pre[sh + 1] = pre[sh] + min(h->count[L], Mw);
      if (h->status) set_status(S, (int)h->status);
    }
  }
  ss.hist[threadIdx.x] = 0;
  consumers_sync();
  const uint32_t c = pre[n_shards];
  const uint32_t M = active ? min(Mw, c) : 0u;
  auto entry = [&](uint32_t i) -> const CandEntry & {
    uint32_t lo = 0, hi = (uint32_t)n_shards - 1;  // the shard holding entry i: pre[sh] <= i < pre[sh + 1]
    while (lo < hi) {
      const uint32_t mid = (lo + hi + 1) >> 1;
      if (pre[mid] <= i) lo = mid; else hi = mid - 1;
    }
    return reinterpret_cast<const CandEntry *>(gathered + stride * lo + loff)[i - pre[lo]];
  };
  uint64_t *val = fin;                                       // [kMaxSel]
  uint32_t *szs = reinterpret_cast<uint32_t *>(fin + kMaxSel);  // [kMaxSel]
  uint32_t got = 0;
  if (M > 0) {
    uint32_t keepn;
    if (c <= kMaxSel) {
      for (uint32_t i = threadIdx.x; i < c; i += kConsumers) {
        const CandEntry &e = entry(i);
        val[i] = e.v;
        szs[i] = e.kv;
      }
      keepn = c;
    } else {
      const uint64_t th = block_select_rank([&](uint32_t i) { return entry(i).v; }, c, M, ss);
      if (threadIdx.x == 0) ss.cnt = 0;
      consumers_sync();
      for (uint32_t i = threadIdx.x; i < c; i += kConsumers) {
        const CandEntry &e = entry(i);
        if (e.v >= th) {
          const uint32_t pos = atomicAdd(&ss.cnt, 1u);
          if (pos < kMaxSel) {
            val[pos] = e.v;
            szs[pos] = e.kv;
          }
        }
      }
      consumers_sync();
      keepn = min(ss.cnt, kMaxSel);
    }
    consumers_sync();
    if (!bucket_sort_desc(val, keepn, fin + 3 * kMaxSel / 2, ss, szs, reinterpret_cast<uint32_t *>(fin + 5 * kMaxSel / 2)))
      bitonic_sort_desc(val, keepn, szs);
    got = min(keepn, M);
    for (uint32_t i = threadIdx.x; i < got; i += kConsumers) {
      S.sorted[(size_t)L * kMaxSel + i] = val[i];
      if (L == 0) S.victims[i] = (~(uint32_t)val[i]) & kIdMask;
      else S.ssz[(size_t)L * kMaxSel + i] = szs[i];
    }
  }
  if (threadIdx.x == 0) S.work->got[L] = got;
  __threadfence();
  consumers_sync();
  if (threadIdx.x == 0) last = (atomicAdd(&S.work->list_ticket, 1u) == (unsigned)kLists - 1);
  consumers_sync();
  if (last) fill(S, fin);
}

// ------------------------------------------------------------ host side ----
size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Device scratch of the ranking calls, kept per (device, stream) and grown
// when a call needs more: calls on one stream run in order, so each reuses
// the buffer after the previous one is done with it (stream order), and
// calls on different streams get different buffers.  Held for the life of
// the process.  The stream handle is the key: a stream must outlive the
// ranking calls queued on it (a new stream that reuses a destroyed one's
// handle would otherwise share its scratch without being ordered after it).
// Two blocks per key: the call's working scratch, and the per-set
// histograms, which are zeroed when allocated and left zero by every call
// (each is zeroed by the thread that reads it).
struct Scratch {
  char *p = nullptr;
  size_t bytes = 0;
};
std::mutex g_scratch_mu;
std::map<std::pair<int, cudaStream_t>, std::pair<Scratch, Scratch>> g_scratch;

int grow(Scratch &e, size_t bytes, bool zero, cudaStream_t stream) {
  if (e.bytes >= bytes) return UNISON_OK;
  if (e.p) cudaFreeAsync(e.p, stream);  // ordered after the calls that used it
  e.p = nullptr;
  e.bytes = 0;
  char *p = nullptr;
  if (unison_fault_alloc() || cudaMallocAsync(reinterpret_cast<void **>(&p), bytes, stream) != cudaSuccess) {
    cudaGetLastError();
    return UNISON_ERR_OOM;
  }
  if (zero && cudaMemsetAsync(p, 0, bytes, stream) != cudaSuccess) {
    cudaGetLastError();
    cudaFreeAsync(p, stream);
    return UNISON_ERR_CUDA;
  }
  e.p = p;
  e.bytes = bytes;
  return UNISON_OK;
}

int scratch_acquire(cudaStream_t stream, size_t bytes, size_t hist_bytes, char **out, char **hist) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return UNISON_ERR_CUDA;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  auto &e = g_scratch[std::make_pair(dev, stream)];
  int rc = grow(e.first, bytes, false, stream);
  if (rc == UNISON_OK) rc = grow(e.second, hist_bytes, true, stream);
  if (rc != UNISON_OK) return rc;
  *out = e.first.p;
  *hist = e.second.p;
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
constexpr int kStagingRing = 8;
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

// Kernel attributes and the grid (every CTA resident at once), set up once
// per device (the attributes belong to the device's context).
struct LaunchCfg {
  bool ok = false;
  uint32_t ctas = 0;
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
    int n_sm = 0, per_sm = 0, coop = 0;
    c.ok = cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess &&
           cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev) == cudaSuccess && coop &&
           cudaFuncSetAttribute(rank_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kDynSmem) ==
               cudaSuccess &&
           cudaFuncSetAttribute(rank_merge_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kMergeSmem) ==
               cudaSuccess &&
           cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, rank_kernel, kCtaThreads, kDynSmem) ==
               cudaSuccess &&
           per_sm > 0;
    if (!c.ok) cudaGetLastError();
    c.ctas = (uint32_t)std::min(std::max(1, n_sm * per_sm), (int)kMaxGroup);
    cfgs[dev] = c;
    done[dev] = c.ok;
  }
  return cfgs[dev];
}

}  // namespace

#ifdef UNISON_DEBUG_HOOKS
// Test hooks of the debug build (absent from the default build): the next
// ranking calls' threshold wait of set flag_set first waits on a flag that
// nothing sets, and the first tile wait of set mbar_set first waits on a
// barrier nothing arrives at; both bounded waits run out and report
// UNISON_ERR_TIMEOUT in that set's counts[3].  -1 turns a hook off.
extern "C" int unison_debug_rank_wait_hooks(int flag_set, int mbar_set) {
  if (cudaMemcpyToSymbol(g_hook_flag_set, &flag_set, sizeof(int)) != cudaSuccess ||
      cudaMemcpyToSymbol(g_hook_mbar_set, &mbar_set, sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    return UNISON_ERR_CUDA;
  }
  return UNISON_OK;
}
#endif

namespace {

// The ranking call: n_sets sets with their outputs, or (cands != null) one
// shard of a set whose record 0 has index `off` in the whole set, with its
// candidate lists going to cands instead of outputs.
// The last ranking call's plan per (device, stream): a call whose arguments
// are byte for byte those of the previous call on its stream finds its
// descriptors, tables and scratch layout already on the device and only
// launches.  The per-call state (work words, sample histograms) is held
// twice; calls alternate between the two, and each launch zeroes the
// other's for the next call.  Any other use of the stream's scratch (a
// merge, a different call, a reallocation) replaces or drops the plan.
struct RankPlan {
  std::vector<unsigned char> key;
  size_t bytes = 0, hist_bytes = 0;
  size_t desc_b = 0, work_off = 0, work_b = 0, hist_b = 0;  // per parity: descriptors, work words, histograms
  size_t cmap_off = 0, tabs_off = 0;
  char *scratch = nullptr, *hists = nullptr;
  uint32_t grid = 0;
  int sequential = 0;
  int parity = 0;  // the parity the next call uses (its state is zero)
};
std::mutex g_plan_mu;
std::map<std::pair<int, cudaStream_t>, RankPlan> g_plan;

void plan_key(std::vector<unsigned char> &k, const unison_records *sets, const unison_rank_params *params,
              const unison_rank_out *outs, int n_sets, uint32_t off, const unsigned char *cands) {
  k.clear();
  auto put = [&](const void *q, size_t b) {
    const unsigned char *c = static_cast<const unsigned char *>(q);
    k.insert(k.end(), c, c + b);
  };
  put(&n_sets, sizeof n_sets);
  put(&off, sizeof off);
  put(&cands, sizeof cands);
  put(sets, sizeof(unison_records) * n_sets);
  put(params, sizeof(unison_rank_params) * n_sets);
  if (!cands) put(outs, sizeof(unison_rank_out) * n_sets);
}

void plan_drop(cudaStream_t stream) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return;
  }
  std::lock_guard<std::mutex> lock(g_plan_mu);
  g_plan.erase(std::make_pair(dev, stream));
}

cudaError_t launch_rank_kernel(uint32_t grid, const RankSet *d_sets, int n_sets, int sequential, const uint32_t *cmap,
                               const RankTab *tabs, char *zero_a, size_t bytes_a, char *zero_b, size_t bytes_b,
                               cudaStream_t stream) {
  ProfSpan span("rank", stream);
  cudaLaunchAttribute coop[1];
  coop[0].id = cudaLaunchAttributeCooperative;
  coop[0].val.cooperative = 1;
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(grid);
  lc.blockDim = dim3(kCtaThreads);
  lc.dynamicSmemBytes = kDynSmem;
  lc.stream = stream;
  lc.attrs = coop;
  lc.numAttrs = 1;
  return cudaLaunchKernelEx(&lc, rank_kernel, d_sets, n_sets, sequential, cmap, tabs, reinterpret_cast<uint4 *>(zero_a),
                            (uint32_t)(bytes_a / 16), reinterpret_cast<uint4 *>(zero_b), (uint32_t)(bytes_b / 16));
}

int rank_launch(const unison_records *sets, const unison_rank_params *params, const unison_rank_out *outs,
                int n_sets, uint32_t off, unsigned char *cands, cudaStream_t stream) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return UNISON_ERR_CUDA;
  }
  thread_local std::vector<unsigned char> key;
  plan_key(key, sets, params, outs, n_sets, off, cands);
  {
    std::lock_guard<std::mutex> lock(g_plan_mu);
    auto it = g_plan.find(std::make_pair(dev, stream));
    if (it != g_plan.end() && it->second.key == key) {
      RankPlan &pl = it->second;
      char *scratch = nullptr, *hists = nullptr;
      if (scratch_acquire(stream, pl.bytes, pl.hist_bytes, &scratch, &hists) == UNISON_OK && scratch == pl.scratch &&
          hists == pl.hists) {
        const int pa = pl.parity, pb = 1 - pa;
        int rc = UNISON_OK;
        if (launch_rank_kernel(pl.grid, reinterpret_cast<const RankSet *>(scratch + pa * pl.desc_b), n_sets,
                               pl.sequential,
                               pl.sequential ? nullptr : reinterpret_cast<const uint32_t *>(scratch + pl.cmap_off),
                               reinterpret_cast<const RankTab *>(scratch + pl.tabs_off),
                               scratch + pl.work_off + pb * pl.work_b, pl.work_b, hists + pb * pl.hist_b, pl.hist_b,
                               stream) != cudaSuccess)
          rc = UNISON_ERR_CUDA;
        count_launches(1);
        if (cudaGetLastError() != cudaSuccess) rc = UNISON_ERR_CUDA;
        if (rc == UNISON_OK) pl.parity = pb;
        else g_plan.erase(it);
        return rc;
      }
      g_plan.erase(it);
    }
  }
  std::vector<RankSet> hs(n_sets);
  std::vector<RankTab> tabs;
  std::vector<int> tab_of(n_sets);
  std::vector<std::pair<const unison_rank_params *, int>> tab_keys;  // params whose tables are built
  uint64_t tiles = 0;
  for (int i = 0; i < n_sets; i++) {
    const unison_records &r = sets[i];
    const unison_rank_params &p = params[i];
    const unison_rank_out o = cands ? unison_rank_out{} : outs[i];
    if (r.n == 0 || r.n + off > (1ull << 24)) return UNISON_ERR_RANGE;
    if (!r.gap_q || !r.turn || !r.kv_tok || !r.tier || !r.flags) return UNISON_ERR_ARG;
    if (!aligned(r.gap_q, 16) || !aligned(r.turn, 16) || !aligned(r.tier, 16) || !aligned(r.flags, 16))
      return UNISON_ERR_ARG;
    if (p.k > kMaxSel || p.max_moves > kMaxSel) return UNISON_ERR_RANGE;
    if (p.penalty_q >= (1ull << 32) || p.kv_bytes_per_token == 0 || p.kv_bytes_per_token > (1u << 24))
      return UNISON_ERR_RANGE;
    if (!cands && (!o.counts || !o.moved_bytes || (p.k && !o.victims) || (p.max_moves && (!o.promote || !o.demote))))
      return UNISON_ERR_ARG;
    for (int t = 0; t < (int)kLutN; t++)
      if (p.sigma_q[t] < kEpsQ || p.sigma_q[t] > kLambda) return UNISON_ERR_RANGE;
    // per-turn tables, one per distinct (sigma, P_Z)
    int ti = -1;
    for (size_t j = 0; j < tab_keys.size() && ti < 0; j++) {
      const unison_rank_params &q = *tab_keys[j].first;
      if (q.penalty_q == p.penalty_q && std::memcmp(q.sigma_q, p.sigma_q, sizeof(p.sigma_q)) == 0)
        ti = tab_keys[j].second;
    }
    if (ti < 0) {
      RankTab tb;
      for (int t = 0; t < (int)kLutN; t++) {
        tb.sigma[t] = p.sigma_q[t];
        tb.t2v[t] = ((uint64_t)(kLambda - p.sigma_q[t]) * p.penalty_q) / kLambda;  // eq. (t2)
        tb.mgv[t] = magic_for(p.sigma_q[t]);
      }
      ti = (int)tabs.size();
      tabs.push_back(tb);
      tab_keys.emplace_back(&p, ti);
    }
    tab_of[i] = ti;
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
    s.budget = p.budget_bytes;
    s.free_s = p.free_fast_tok;
    s.free_h = p.free_hbm_tok;
    s.victims = o.victims;
    s.promote = o.promote;
    s.demote = o.demote;
    s.counts = o.counts;
    s.moved = o.moved_bytes;
    s.keys = o.keys;
    s.off = off;
    s.cands = cands;
    s.ntiles = (uint32_t)((r.n + kBigTile - 1) / kBigTile);
    tiles += s.ntiles;
    s.act = 0;
    for (int L = 0; L < kLists; L++) s.act |= list_active(s, L) ? 1u << L : 0u;
  }
  const LaunchCfg &cfg = launch_cfg();
  if (!cfg.ok) return UNISON_ERR_CUDA;
  // Groups: each set gets CTAs in proportion to its tiles (at least 1, at
  // most its tile count); CTAs left over go to the sets with the most tiles
  // per CTA.  With more sets than CTAs, CTA c takes sets c, c + G, ...
  const int sequential = (uint64_t)n_sets > cfg.ctas ? 1 : 0;
  uint32_t grid = cfg.ctas;
  if (!sequential) {
    uint64_t used = 0;
    for (int i = 0; i < n_sets; i++) {
      RankSet &s = hs[i];
      s.nctas = (uint32_t)std::max<uint64_t>(1, (uint64_t)cfg.ctas * s.ntiles / tiles);
      s.nctas = std::min(s.nctas, s.ntiles);
      used += s.nctas;
    }
    while (used < cfg.ctas) {
      int best = -1;
      for (int i = 0; i < n_sets; i++)
        if (hs[i].nctas < hs[i].ntiles &&
            (best < 0 || (uint64_t)hs[i].ntiles * hs[best].nctas > (uint64_t)hs[best].ntiles * hs[i].nctas))
          best = i;
      if (best < 0) break;
      hs[best].nctas++;
      used++;
    }
    uint32_t cta = 0;
    for (int i = 0; i < n_sets; i++) {
      hs[i].cta0 = cta;
      cta += hs[i].nctas;
    }
    grid = cta;
  } else {
    for (int i = 0; i < n_sets; i++) {
      hs[i].cta0 = (uint32_t)(i % cfg.ctas);
      hs[i].nctas = 1;
    }
  }
  for (int i = 0; i < n_sets; i++) plan_sample(hs[i]);
  // scratch: descriptors, tables, every set's work words (zeroed by the
  // upload), then per set: thresholds, tables, sorted lists and sizes,
  // candidates; and the per-set histograms in their own block
  const size_t fixed_set = align_up(sizeof(uint64_t) * kLists * kMaxSel, 256) +
                           align_up(sizeof(uint32_t) * kLists * kMaxSel, 256);
  const size_t hist_set = sizeof(unsigned int) * kLists * kBins;
  size_t sets_b = 0, hist_b = 0;  // hist_b: one parity's histograms (sampled sets only)
  for (int i = 0; i < n_sets; i++) {
    RankSet &s = hs[i];
    // without a sample every eligible record is a candidate: at most n
    s.ccap = s.n > kSample ? kCandCap : (s.n + 31) & ~31u;
    // each CTA's region holds its share of ccap (at least 1,024 entries);
    // a CTA whose region fills appends the rest to the list directly
    s.cr = std::max<uint32_t>(s.ccap / s.nctas, std::min<uint32_t>(s.ccap, 1024u));
    sets_b += fixed_set + align_up(sizeof(uint64_t) * kLists * s.ccap, 256) +
              align_up(sizeof(uint64_t) * kLists * s.nctas * s.cr, 256);
    if (s.ns) hist_b += hist_set;
  }
  const size_t desc_b = align_up(sizeof(RankSet) * n_sets, 256);
  const size_t cmap_b = sequential ? 0 : align_up(sizeof(uint32_t) * grid, 256);
  const size_t tab_b = align_up(sizeof(RankTab) * tabs.size(), 256);
  const size_t work_b = align_up(sizeof(RankWork) * n_sets, 256);
  char *scratch = nullptr, *hists = nullptr;
  {
    plan_drop(stream);  // the scratch is rewritten below; the plan returns only if the launch succeeds
    const int ar = scratch_acquire(stream, 2 * desc_b + cmap_b + tab_b + 2 * work_b + sets_b,
                                   std::max<size_t>(2 * hist_b, 256), &scratch, &hists);
    if (ar != UNISON_OK) return ar;
  }
  // image: descriptors of parity 0 and 1, the CTA map, tables, work words of
  // parity 0 and 1, then the per-set areas; histograms of parity 0 then 1
  const size_t cmap_off = 2 * desc_b, tabs_off = cmap_off + cmap_b;
  RankTab *d_tabs = reinterpret_cast<RankTab *>(scratch + tabs_off);
  const size_t work_off = tabs_off + tab_b;
  RankWork *works = reinterpret_cast<RankWork *>(scratch + work_off);
  char *p = scratch + work_off + 2 * work_b;
  size_t hoff = 0;
  for (int i = 0; i < n_sets; i++) {
    RankSet &s = hs[i];
    s.tab = d_tabs + tab_of[i];
    s.work = works + i;
    s.shist = s.ns ? reinterpret_cast<unsigned int *>(hists + hoff) : nullptr;
    if (s.ns) hoff += hist_set;
    s.sorted = reinterpret_cast<uint64_t *>(p);
    p += align_up(sizeof(uint64_t) * kLists * kMaxSel, 256);
    s.ssz = reinterpret_cast<uint32_t *>(p);
    p += align_up(sizeof(uint32_t) * kLists * kMaxSel, 256);
    s.cand = reinterpret_cast<uint64_t *>(p);
    p += align_up(sizeof(uint64_t) * kLists * s.ccap, 256);
    s.creg = reinterpret_cast<uint64_t *>(p);
    p += align_up(sizeof(uint64_t) * kLists * s.nctas * s.cr, 256);
  }
  int rc = UNISON_OK;
  auto ck = [&](cudaError_t e) {
    if (e != cudaSuccess && rc == UNISON_OK) rc = UNISON_ERR_CUDA;
  };
  RankSet *d_sets = reinterpret_cast<RankSet *>(scratch);
  // descriptors of both parities, tables and both parities' zeroed work
  // words: one copy from pinned staging; both parities' histograms zeroed
  {
    const size_t up = work_off + 2 * work_b;
    unsigned char *h = nullptr;
    cudaEvent_t done = nullptr;
    const int sr = staging_acquire(up, &h, &done);
    if (sr != UNISON_OK) return sr;
    std::memcpy(h, hs.data(), sizeof(RankSet) * n_sets);
    for (int i = 0; i < n_sets; i++) {  // parity 1: the other work words and histograms
      RankSet s1 = hs[i];
      s1.work = reinterpret_cast<RankWork *>(reinterpret_cast<char *>(s1.work) + work_b);
      if (s1.shist) s1.shist = reinterpret_cast<unsigned int *>(reinterpret_cast<char *>(s1.shist) + hist_b);
      std::memcpy(h + desc_b + sizeof(RankSet) * i, &s1, sizeof(RankSet));
    }
    if (!sequential) {
      uint32_t *cm = reinterpret_cast<uint32_t *>(h + cmap_off);
      for (int i = 0; i < n_sets; i++)
        for (uint32_t b = hs[i].cta0; b < hs[i].cta0 + hs[i].nctas; b++) cm[b] = (uint32_t)i | ((uint32_t)tab_of[i] << 16);
    }
    std::memcpy(h + tabs_off, tabs.data(), sizeof(RankTab) * tabs.size());
    std::memset(h + work_off, 0, 2 * work_b);
    ck(cudaMemcpyAsync(d_sets, h, up, cudaMemcpyHostToDevice, stream));
    ck(cudaEventRecord(done, stream));  // the buffer is reused after this copy
    staging_release();
    if (hist_b) ck(cudaMemsetAsync(hists, 0, 2 * hist_b, stream));
  }
  ck(launch_rank_kernel(grid, d_sets, n_sets, sequential,
                        sequential ? nullptr : reinterpret_cast<const uint32_t *>(scratch + cmap_off), d_tabs,
                        scratch + work_off + work_b, work_b, hists + hist_b, hist_b, stream));
  count_launches(1);
  ck(cudaGetLastError());
  if (rc == UNISON_OK) {
    std::lock_guard<std::mutex> lock(g_plan_mu);
    RankPlan &pl = g_plan[std::make_pair(dev, stream)];
    pl.key = key;
    pl.bytes = 2 * desc_b + cmap_b + tab_b + 2 * work_b + sets_b;
    pl.cmap_off = cmap_off;
    pl.tabs_off = tabs_off;
    pl.hist_bytes = std::max<size_t>(2 * hist_b, 256);
    pl.desc_b = desc_b;
    pl.work_off = work_off;
    pl.work_b = work_b;
    pl.hist_b = hist_b;
    pl.parity = 1;
    pl.scratch = scratch;
    pl.hists = hists;
    pl.grid = grid;
    pl.sequential = sequential;
  }
  return rc;
}

}  // namespace

extern "C" int unison_rank_batch(const unison_records *sets, const unison_rank_params *params,
                                 const unison_rank_out *outs, int n_sets, void *cuda_stream) {
  if (n_sets < 0 || (n_sets > 0 && (!sets || !params || !outs))) return UNISON_ERR_ARG;
  if (n_sets == 0) return UNISON_OK;
  return rank_launch(sets, params, outs, n_sets, 0u, nullptr, static_cast<cudaStream_t>(cuda_stream));
}

extern "C" int unison_rank(const unison_records *records, const unison_rank_params *params,
                           const unison_rank_out *out, void *cuda_stream) {
  if (!records || !params || !out) return UNISON_ERR_ARG;
  return unison_rank_batch(records, params, out, 1, cuda_stream);
}

extern "C" uint64_t unison_rank_cands_bytes(uint32_t k, uint32_t max_moves) { return cand_bytes(k, max_moves); }

extern "C" int unison_rank_shard(const unison_records *slice, uint64_t index_offset, const unison_rank_params *params,
                                 void *cands_dev, void *cuda_stream) {
  if (!slice || !params || !cands_dev || !aligned(cands_dev, 256)) return UNISON_ERR_ARG;
  if (index_offset >= (1ull << 24)) return UNISON_ERR_RANGE;
  return rank_launch(slice, params, nullptr, 1, (uint32_t)index_offset, static_cast<unsigned char *>(cands_dev),
                     static_cast<cudaStream_t>(cuda_stream));
}

extern "C" int unison_rank_merge(const void *gathered_dev, int n_shards, const unison_rank_params *params,
                                 const unison_rank_out *out, void *cuda_stream) {
  if (!gathered_dev || !params || !out || n_shards < 1) return UNISON_ERR_ARG;
  if (n_shards > (int)kMaxShards) return UNISON_ERR_RANGE;
  const unison_rank_params &p = *params;
  const unison_rank_out &o = *out;
  if (p.k > kMaxSel || p.max_moves > kMaxSel) return UNISON_ERR_RANGE;
  if (p.kv_bytes_per_token == 0 || p.kv_bytes_per_token > (1u << 24)) return UNISON_ERR_RANGE;
  if (!o.counts || !o.moved_bytes || (p.k && !o.victims) || (p.max_moves && (!o.promote || !o.demote)))
    return UNISON_ERR_ARG;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  RankSet s{};
  s.k = p.k;
  s.max_moves = p.max_moves;
  s.kvb = p.kv_bytes_per_token;
  s.budget = p.budget_bytes;
  s.free_s = p.free_fast_tok;
  s.free_h = p.free_hbm_tok;
  s.victims = o.victims;
  s.promote = o.promote;
  s.demote = o.demote;
  s.counts = o.counts;
  s.moved = o.moved_bytes;
  for (int L = 0; L < kLists; L++) s.act |= list_active(s, L) ? 1u << L : 0u;
  // scratch: descriptor and work words (one upload), sorted lists
  const size_t desc_b = align_up(sizeof(RankSet), 256), work_b = align_up(sizeof(RankWork), 256);
  const size_t lists_b = align_up(sizeof(uint64_t) * kLists * kMaxSel, 256) + align_up(sizeof(uint32_t) * kLists * kMaxSel, 256);
  char *scratch = nullptr, *hists = nullptr;
  {
    plan_drop(stream);  // the descriptor area is rewritten below
    const int ar = scratch_acquire(stream, desc_b + work_b + lists_b, 0, &scratch, &hists);
    if (ar != UNISON_OK) return ar;
  }
  s.work = reinterpret_cast<RankWork *>(scratch + desc_b);
  s.sorted = reinterpret_cast<uint64_t *>(scratch + desc_b + work_b);
  s.ssz = reinterpret_cast<uint32_t *>(scratch + desc_b + work_b + align_up(sizeof(uint64_t) * kLists * kMaxSel, 256));
  const LaunchCfg &cfg = launch_cfg();
  if (!cfg.ok) return UNISON_ERR_CUDA;
  int rc = UNISON_OK;
  auto ck = [&](cudaError_t e) {
    if (e != cudaSuccess && rc == UNISON_OK) rc = UNISON_ERR_CUDA;
  };
  {
    const size_t up = desc_b + work_b;
    unsigned char *h = nullptr;
    cudaEvent_t done = nullptr;
    const int sr = staging_acquire(up, &h, &done);
    if (sr != UNISON_OK) return sr;
    std::memset(h, 0, up);
    std::memcpy(h, &s, sizeof(RankSet));
    ck(cudaMemcpyAsync(scratch, h, up, cudaMemcpyHostToDevice, stream));
    ck(cudaEventRecord(done, stream));
    staging_release();
  }
  rank_merge_kernel<<<kLists, kConsumers, kMergeSmem, stream>>>(reinterpret_cast<const RankSet *>(scratch),
                                                             static_cast<const unsigned char *>(gathered_dev), n_shards,
                                                             (uint64_t)cand_bytes(p.k, p.max_moves));
  count_launches(1);
  ck(cudaGetLastError());
  return rc;
}
