// Batched trace replay of UNISON's joint event loop (Algorithm 1) on GB300.
//
// Kernels, in launch order:
//   hazard_lut_kernel   eqs. (hazard), (surv), (uq), (hq), (survq), (t2): one
//                       block per (trace, bucket width, P_Z) builds sigma_q[t]
//                       and T2[t] from the trace's turns-per-session counts.
//   key_stream_kernel   eqs. (gap), (ema-int), (t1), (scoreq): one thread per
//                       session walks its turns and writes, for each of its
//                       events, the session's packed SPEAR key and gap average
//                       after that event.  With the offline table of Sec. V-E
//                       a session's score changes only at its own events, so
//                       the event loop re-ranks from these values instead of
//                       re-dividing every live score at every event; the
//                       decisions are identical.
//   replay_kernel       Algorithm 1: one warp per replay; the unpinned
//                       residents of each tier kept sorted by packed 64-bit
//                       key in shared memory (the most evictable last), so
//                       the argmax of a decision is a pop and an update is a
//                       warp-parallel lower bound plus a block shift.
//   ttft_median_kernel  Sec. V-A TTFT p50: radix select of the lower median
//                       over each replay's per-request TTFT values.
#include <algorithm>
#include <cmath>
#include <map>
#include <mutex>
#include <tuple>
#include <vector>

#include "common.cuh"
#include "profile.cuh"

using namespace unison;

namespace {

constexpr uint32_t kFull = 0xFFFFFFFFu;
constexpr uint32_t kTierNone = 0, kTierS = 1, kTierH = 2;
// Per-session maps in shared memory beside the resident lists: none, the tier
// byte and the pin slot, or the tier byte alone.
constexpr uint32_t kMapNone = 0, kMapSlots = 1, kMapTier = 2;

struct ComboDesc {
  const uint32_t *turn_ev;   // [2T]
  const uint32_t *turn_t;    // [2T]
  const uint32_t *turn_off;  // [S+1]
  const uint32_t *tps;       // [S]
  uint32_t n_sessions, n_events;
  uint32_t ema_num, ema_den, bucket, signals;  // signals: UNISON_SIGNAL_* bits of the flags
  uint64_t penalty_q;
  uint16_t *sigma;  // [51]
  uint64_t *t2;     // [51]
  uint64_t *pkey;   // [E] key after the event
  uint32_t *gq;     // [E] gap average after the event
  uint64_t *pkb;    // [E] key before the event (arrivals of turn >= 1)
};

struct ReplayDesc {
  const uint4 *ev;
  const uint32_t *prev_out;
  const uint32_t *nref;
  const uint32_t *prev_ev;  // previous completion event of each arrival's session
  const uint64_t *pkey;  // key stream (SPEAR policies) or null
  const uint64_t *pkb;   // key before each arrival (SPEAR policies) or null
  const uint32_t *gq;    // gap-average stream (TIDE policies) or null
  uint64_t *ttft;        // [n_turns]
  uint32_t *glist;       // resident lists in global memory, or null (shared)
  unison_decision *log;
  uint64_t log_cap;
  unison_replay_result *result;
  uint64_t cap_s, cap_h;  // tokens
  uint64_t dma;           // bytes per us
  uint64_t prefill_ns;    // ns per prefill token
  uint32_t n_events, n_turns, n_sessions, policy;
  uint32_t max_sessions, kvb, ttl, load;
  uint32_t rcap_s, rcap_h;
  uint32_t tmap;    // kMapNone, kMapSlots (tier byte and pin slot per session) or kMapTier (tier byte)
  uint32_t bucket;  // hazard bucket width (online hazard replays)
  uint64_t penalty;  // P_Z in quantised units (online hazard replays)
  const uint64_t *t2;  // eq. (t2) per turn index of the offline table (stale-snapshot replays)
  uint32_t stale_sync, stale_m;  // UNISON_SYNC_* and arrivals per sync
};

// --------------------------------------------------------------------------
// Hazard table: n(t) = #{T_s >= t+1}, d(t) = #{T_s = t+1}, pooled over
// buckets of consecutive turns, h_q = round-half-up(Lambda * d / n),
// sigma_q = max(eps_q, Lambda - h_q), T2 = floor((Lambda - sigma_q) P_Z / Lambda).
// --------------------------------------------------------------------------
__device__ void build_lut(const uint32_t *tps, uint32_t n_sessions, uint32_t bucket, uint64_t penalty,
                          uint16_t *sigma_out, uint16_t *hq_out, uint64_t *t2_out) {
  __shared__ unsigned long long cnt[kLutN + 2];  // cnt[j] = #{T_s = j}, j = 1..51; cnt[52] = #{T_s >= 52}
  __shared__ unsigned long long nn[kLutN], dd[kLutN];
  for (uint32_t i = threadIdx.x; i < kLutN + 2; i += blockDim.x) cnt[i] = 0;
  __syncthreads();
  for (uint32_t s = threadIdx.x; s < n_sessions; s += blockDim.x) {
    uint32_t t = tps[s];
    atomicAdd(&cnt[t < kLutN + 1 ? t : kLutN + 1], 1ull);
  }
  __syncthreads();
  if (threadIdx.x < kLutN) {
    const uint32_t t = threadIdx.x;
    unsigned long long n = 0;
    for (uint32_t j = t + 1; j <= kLutN + 1; j++) n += cnt[j];  // live at turn t
    nn[t] = n;
    dd[t] = cnt[t + 1];                                         // complete at turn t
  }
  __syncthreads();
  if (threadIdx.x < kLutN) {
    const uint32_t t = threadIdx.x, b = t / bucket;
    unsigned long long n = 0, d = 0;
    for (uint32_t u = b * bucket; u < kLutN && u < (b + 1) * bucket; u++) {
      n += nn[u];
      d += dd[u];
    }
    uint64_t hq = 0;
    if (n) {
      hq = (2ull * d * kLambda + n) / (2ull * n);
      if (hq > kLambda) hq = kLambda;
    }
    uint64_t sq = kLambda - hq;
    if (sq < kEpsQ) sq = kEpsQ;
    sigma_out[t] = (uint16_t)sq;
    if (hq_out) hq_out[t] = (uint16_t)hq;
    if (t2_out) t2_out[t] = ((kLambda - sq) * penalty) / kLambda;
  }
}

__global__ void hazard_lut_kernel(const ComboDesc *combos) {
  const ComboDesc &c = combos[blockIdx.x];
  build_lut(c.tps, c.n_sessions, c.bucket, c.penalty_q, c.sigma, nullptr, c.t2);
  // without the hazard signal (Sec. V-D) the score sees zero hazard: sigma =
  // Lambda and T2 = 0 (each entry is rewritten by the thread that wrote it)
  if ((c.signals & UNISON_SIGNAL_NO_HAZARD) && threadIdx.x < kLutN) {
    c.sigma[threadIdx.x] = (uint16_t)kLambda;
    c.t2[threadIdx.x] = 0;
  }
}

__global__ void hazard_lut_single_kernel(const uint32_t *tps, uint32_t n, uint32_t bucket, uint16_t *sigma,
                                         uint16_t *hq) {
  build_lut(tps, n, bucket, 0, sigma, hq, nullptr);
}

// --------------------------------------------------------------------------
// Key stream: per session, gap average (eq. ema-int) and score (eqs. t1, t2,
// scoreq) after each of its events, packed with the session id.
// --------------------------------------------------------------------------
// Every thread loads the table before any may leave, so the barrier is uniform.
__global__ void key_stream_kernel(const ComboDesc *combos) {
  const ComboDesc &c = combos[blockIdx.y];
  __shared__ unsigned long long mg[kLutN], t2[kLutN];
  for (uint32_t i = threadIdx.x; i < kLutN; i += blockDim.x) {
    mg[i] = magic_for(c.sigma[i]);  // eq. (t1)'s division by sigma as a multiply-high
    t2[i] = c.t2[i];
  }
  __syncthreads();
  const uint32_t s = blockIdx.x * blockDim.x + threadIdx.x;
  if (s >= c.n_sessions) return;
  const uint32_t b = c.turn_off[s], ts = c.tps[s];
  const uint64_t a_num = c.ema_num, a_rest = c.ema_den - c.ema_num, a_den = c.ema_den;
  // eq. (ema-int)'s division by a_den: its numerator stays below a_den * 2^31,
  // so below 2^43 when a_den < 2^12 -- then a multiply-high (a_den >= 2)
  const bool den_magic = a_den >= 2 && a_den < 4096;
  const uint64_t den_mg = den_magic ? magic_for((uint32_t)a_den) : 0;
  const bool no_gap = (c.signals & UNISON_SIGNAL_NO_GAP) != 0;
  uint64_t g = 0, prev_pk = 0;
  uint32_t prev_c = 0;
  for (uint32_t k = 0; k < ts; k++) {
    const uint32_t ti = b + k;
    const uint32_t ta = c.turn_t[2 * ti], tc = c.turn_t[2 * ti + 1];
    if (k) {
      const uint64_t gap = (uint32_t)(ta - prev_c);
      const uint64_t num = a_num * gap + a_rest * g;
      g = den_magic ? __umul64hi(num, den_mg) : num / a_den;
    }
    prev_c = tc;
    const uint32_t t = k < kTMax ? k : kTMax;
    // without the gap signal (Sec. V-D) the score sees a zero gap average;
    // g < 2^31 (gaps are clamped below 2^31 us), so g * Lambda < 2^43
    const uint64_t key = __umul64hi((no_gap ? 0 : g) * kLambda, mg[t]) + t2[t];
    const uint64_t pk = pack_key(key, s);
    const uint32_t ea = c.turn_ev[2 * ti], ec = c.turn_ev[2 * ti + 1];
    c.pkey[ea] = pk;
    c.gq[ea] = (uint32_t)g;
    c.pkb[ea] = prev_pk;  // the key the session carried into this arrival
    prev_pk = (k + 1 == ts) ? pack_key(kKeyMax40, s) : pk;
    c.pkey[ec] = prev_pk;
    c.gq[ec] = (uint32_t)g;
  }
}

// --------------------------------------------------------------------------
// Resident sessions.  The unpinned residents of each tier sit in an array
// sorted by packed key, ascending: the most evictable is the last entry and
// the least evictable the first, so every argmax / argmin of Algorithm 1 and
// of TIDE is an array end.  Pinned (mid-turn) residents, which no decision
// may touch, sit in a small unordered list.  Keys change only at a session's
// own events, so an arriving session is found by binary search on the key it
// was given at its previous event.  Entries (16 B):
//   sorted: {key lo, key hi, size | promoted << 31, last return time}
//   pinned: {key lo, key hi, size, session | tier << 30}
// All list state is warp-uniform; lane 0 writes single entries, all lanes
// move blocks (warp-parallel shifts, top or bottom chunk first).
// --------------------------------------------------------------------------
constexpr uint32_t kPromotedBit = 0x80000000u;
constexpr uint32_t kSizeMask = 0x7FFFFFFFu;

struct Sorted {
  uint4 *e;
  uint32_t n, cap;
};

// Smallest power of two >= x (x >= 1).
__host__ __device__ __forceinline__ uint32_t ring_size(uint32_t x) {
  uint32_t r = 1;
  while (r < x) r <<= 1;
  return r;
}

__device__ __forceinline__ uint64_t ekey(uint4 v) { return ((uint64_t)v.y << 32) | v.x; }

// Number of entries with key < k (warp-uniform result).
__device__ __forceinline__ uint32_t lower_bound(const Sorted &T, uint64_t k, int lane) {
  uint32_t lo = 0, hi = T.n;  // the answer lies in [lo, hi]
  while (hi - lo > 32) {
    const uint32_t step = (hi - lo + 31) / 32;
    const uint32_t i = lo + lane * step;
    const bool less = i < hi && ekey(T.e[i]) < k;
    const uint32_t cnt = __popc(__ballot_sync(kFull, less));  // 'less' holds for a prefix of lanes
    const uint32_t nlo = cnt ? lo + (cnt - 1) * step + 1 : lo;
    const uint32_t nhi = min(hi, lo + cnt * step);
    lo = nlo;
    hi = nhi;
  }
  const uint32_t i = lo + lane;
  return lo + __popc(__ballot_sync(kFull, i < hi && ekey(T.e[i]) < k));
}

// Move e[lo, hi) by delta places (delta > 0 toward the end), warp-parallel.
// Out of line on purpose: inlined at every call site, the shifts' register
// demand crowds the event loop (measured: the sweep runs about 8% faster).
__device__ __noinline__ void shift_block(uint4 *e, uint32_t lo, uint32_t hi, int32_t delta, int lane) {
  if (lo >= hi || delta == 0) return;
  if (delta > 0) {  // top chunk first
    uint32_t top = hi;
    while (top > lo) {
      const uint32_t bot = top - lo > 128 ? top - 128 : lo;
      uint4 v[4];
#pragma unroll
      for (int j = 0; j < 4; j++) {
        const uint32_t i = bot + lane + 32 * j;
        if (i < top) v[j] = e[i];
      }
      __syncwarp();
#pragma unroll
      for (int j = 0; j < 4; j++) {
        const uint32_t i = bot + lane + 32 * j;
        if (i < top) e[i + delta] = v[j];
      }
      __syncwarp();
      top = bot;
    }
  } else {  // bottom chunk first
    uint32_t bot = lo;
    while (bot < hi) {
      const uint32_t top = hi - bot > 128 ? bot + 128 : hi;
      uint4 v[4];
#pragma unroll
      for (int j = 0; j < 4; j++) {
        const uint32_t i = bot + lane + 32 * j;
        if (i < top) v[j] = e[i];
      }
      __syncwarp();
#pragma unroll
      for (int j = 0; j < 4; j++) {
        const uint32_t i = bot + lane + 32 * j;
        if (i < top) e[(int32_t)i + delta] = v[j];
      }
      __syncwarp();
      bot = top;
    }
  }
}

// The fast tier in registers (kRegS launches, every replay's fast tier at
// most 32 entries): lane i holds entry i of the sorted array, so a search is
// one ballot and an insert, an erase or a pop is a few shuffles, with no
// shared-memory round trip.
struct RegTier {
  uint4 v;  // this lane's entry
  uint32_t n;
};
__device__ __forceinline__ uint32_t reg_lower_bound(const RegTier &R, uint64_t k, int lane) {
  return __popc(__ballot_sync(kFull, (uint32_t)lane < R.n && ekey(R.v) < k));
}
__device__ __forceinline__ uint4 reg_at(const RegTier &R, uint32_t i) {
  return make_uint4(__shfl_sync(kFull, R.v.x, i), __shfl_sync(kFull, R.v.y, i), __shfl_sync(kFull, R.v.z, i),
                    __shfl_sync(kFull, R.v.w, i));
}
__device__ __forceinline__ void reg_insert_at(RegTier &R, uint32_t p, uint4 e, int lane) {
  const uint4 u = make_uint4(__shfl_up_sync(kFull, R.v.x, 1), __shfl_up_sync(kFull, R.v.y, 1),
                             __shfl_up_sync(kFull, R.v.z, 1), __shfl_up_sync(kFull, R.v.w, 1));
  if ((uint32_t)lane > p) R.v = u;
  if ((uint32_t)lane == p) R.v = e;
  R.n++;
}
__device__ __forceinline__ void reg_erase_at(RegTier &R, uint32_t p, int lane) {
  const uint4 u = make_uint4(__shfl_down_sync(kFull, R.v.x, 1), __shfl_down_sync(kFull, R.v.y, 1),
                             __shfl_down_sync(kFull, R.v.z, 1), __shfl_down_sync(kFull, R.v.w, 1));
  if ((uint32_t)lane >= p) R.v = u;
  R.n--;
}

// The HBM tier in registers (kHK > 0 slots a lane): lane l holds entries l,
// 32 + l, 64 + l, ... of the sorted array, three words each (key and size; an
// entry's fourth word, its completion time, is read only by the timeout
// policy, which these launches never run).  A search is kHK ballots; an
// insert, an erase or a drop of the first entries one shuffle per word and
// slot.  A replay whose HBM tier would pass 32 kHK entries stops (kRegFull)
// and is replayed from its start with the tier in shared memory: a replay is
// deterministic, so its results are the same, and the register body needs no
// test of where the tier is (measured: the sweep runs 6% faster than with a
// one-way move of the tier to shared memory tested at every operation).
// The restart is kept for the rare replay: while warps of one SM run
// different bodies the launch slows down far beyond the repeated work
// (measured: independent-gap sweep, 128 GiB replays restarting with 6
// slots: 121 ms, against 70 ms with 6 slots from the start).  Five slots hold
// both sweeps' HBM tiers (at most about 125 entries with per-session gap
// recurrence, about 140 with independent gaps); four run the recurrent-gap
// sweep 7% faster but send the other's 128 GiB replays to shared memory.
constexpr int kHSlots = 5;
constexpr int kRegFull = -1000;  // internal status: never reported
struct RegTierH {
  // key low, key high, size (and the promoted bit)
  uint32_t x[kHSlots], y[kHSlots], z[kHSlots];
};
__device__ __forceinline__ uint64_t hkey(const RegTierH &G, int j) { return ((uint64_t)G.y[j] << 32) | G.x[j]; }
// Entry i (warp-uniform, below 32 K; a larger i reads a slot-0 entry).
template <int K>
__device__ __forceinline__ uint4 hreg_at(const RegTierH &G, uint32_t i) {
  const uint32_t sl = i >> 5, ln = i & 31;
  uint32_t a = G.x[0], b = G.y[0], c = G.z[0];
#pragma unroll
  for (int j = 1; j < K; j++)
    if (sl == (uint32_t)j) {
      a = G.x[j];
      b = G.y[j];
      c = G.z[j];
    }
  return make_uint4(__shfl_sync(kFull, a, ln), __shfl_sync(kFull, b, ln), __shfl_sync(kFull, c, ln), 0u);
}
// Entries with key < k among the first n.
template <int K>
__device__ __forceinline__ uint32_t hreg_lower_bound(const RegTierH &G, uint32_t n, uint64_t k, int lane) {
  uint32_t cnt = 0;
#pragma unroll
  for (int j = 0; j < K; j++) cnt += __popc(__ballot_sync(kFull, 32u * j + lane < n && hkey(G, j) < k));
  return cnt;
}
// Insert e at position p (fewer than 32 K entries): entries p.. move up one
// place.  Lane l of a slot takes lane l - 1's entry, lane 0 the slot below's
// lane 31: the providing lane picks the slot, so a word moves in one shuffle
// (slots from the top down, each reading the slot below before it changes).
// Here and below every slot moves whatever the count and position: entries
// past the count may hold anything, and the shuffles cost less than branches
// that would skip the unchanged slots (measured: the sweep runs 8% faster).
template <int K>
__device__ __forceinline__ void hreg_insert_at(RegTierH &G, uint32_t p, uint4 e, int lane) {
  const uint32_t from = (lane - 1) & 31;
#pragma unroll
  for (int j = K - 1; j >= 0; j--) {
    const bool low = j > 0 && lane == 31;  // lane 31 provides the slot below's entry
    const uint32_t ux = __shfl_sync(kFull, low ? G.x[j > 0 ? j - 1 : 0] : G.x[j], from),
                   uy = __shfl_sync(kFull, low ? G.y[j > 0 ? j - 1 : 0] : G.y[j], from),
                   uz = __shfl_sync(kFull, low ? G.z[j > 0 ? j - 1 : 0] : G.z[j], from);
    const uint32_t idx = 32u * j + lane;
    if (idx > p) {
      G.x[j] = ux;
      G.y[j] = uy;
      G.z[j] = uz;
    } else if (idx == p) {
      G.x[j] = e.x;
      G.y[j] = e.y;
      G.z[j] = e.z;
    }
  }
}
// Erase position p: entries p + 1.. move down one place.  Lane l
// takes lane l + 1's entry, lane 31 the slot above's lane 0 (slots from the
// bottom up, each reading the slot above before it changes).
template <int K>
__device__ __forceinline__ void hreg_erase_at(RegTierH &G, uint32_t p, int lane) {
  const uint32_t from = (lane + 1) & 31;
#pragma unroll
  for (int j = 0; j < K; j++) {
    constexpr int kTop = K - 1;
    const bool high = j < kTop && lane == 0;  // lane 0 provides the slot above's entry
    const uint32_t dx = __shfl_sync(kFull, high ? G.x[j < kTop ? j + 1 : kTop] : G.x[j], from),
                   dy = __shfl_sync(kFull, high ? G.y[j < kTop ? j + 1 : kTop] : G.y[j], from),
                   dz = __shfl_sync(kFull, high ? G.z[j < kTop ? j + 1 : kTop] : G.z[j], from);
    if (32u * j + lane >= p) {
      G.x[j] = dx;
      G.y[j] = dy;
      G.z[j] = dz;
    }
  }
}
// Drop the first m (1..32) entries: entry i takes entry i + m, from
// lane (l + m) mod 32 of the same slot, or of the next one where l + m >= 32;
// the providing lanes below m give the next slot's entry.
template <int K>
__device__ __forceinline__ void hreg_drop_front(RegTierH &G, uint32_t m, int lane) {
  const uint32_t from = (lane + m) & 31;
  const bool next = (uint32_t)lane < m;
#pragma unroll
  for (int j = 0; j < K; j++) {
    constexpr int kTop = K - 1;
    const bool up = j < kTop && next;
    G.x[j] = __shfl_sync(kFull, up ? G.x[j < kTop ? j + 1 : kTop] : G.x[j], from);
    G.y[j] = __shfl_sync(kFull, up ? G.y[j < kTop ? j + 1 : kTop] : G.y[j], from);
    G.z[j] = __shfl_sync(kFull, up ? G.z[j < kTop ? j + 1 : kTop] : G.z[j], from);
  }
}

// Descriptor fields the placement and fill read on every event, held in
// registers (the descriptor itself sits in shared memory).
struct Hot {
  uint64_t cap_s, cap_h;  // tokens
  uint64_t kvb, dma;      // bytes per token, bytes per us
  uint32_t max_sessions;
};

struct ReplayState {
  Sorted S, H;      // unpinned residents per tier
  RegTier R;        // the fast tier's residents instead of S, in kRegS launches
  RegTierH G;       // the HBM tier's residents instead of H.e, in kHK > 0 bodies; the count is H.n
  uint4 *pin;       // pinned residents
  uint32_t npin, pin_cap;
  uint4 *tmp;       // TIDE staging: [0, cap_s) promoted, [cap_s, 2 cap_s) demoted
  uint8_t *tmap;    // tier of each unpinned resident session (kTierNone otherwise), or null
  uint16_t *pslot;  // slot of each pinned session in `pin` (kNoSlot otherwise), or null
  uint64_t used_s, used_h, pinned_s, pinned_h;  // tokens
  unison_decision *log;
  uint64_t log_cap;
  uint32_t e;  // current event index
  int status;
  uint64_t hash, log_len;  // decision stream state
  // counters (warp-uniform registers: every lane keeps the same copy)
  uint32_t n_warm, n_cold, n_hit_s, n_hit_h, n_miss, n_bypass, n_place_s, n_place_h;
  uint32_t n_evict, n_demote, n_promote, n_tide_demote, n_expire, n_tide_calls, n_pth;
  uint64_t tok_hit_s, tok_hit_h, tok_miss, tok_computed, tok_needed, dma_bytes;
  // stale-snapshot replays: every session's live key, and the choices made
  // against it
  const uint64_t *live;
  uint32_t vict_n, vict_diff, prom_n, prom_diff;
};

#define CNT(st, field, v) ((st).field += (v))

constexpr uint16_t kNoSlot = 0xFFFF;

// kLean (here and below): the replay keeps no decision log, has the tier map
// and pin slots, and no slot limit -- known at compile time.
template <bool kLean>
__device__ __forceinline__ void log_dec(ReplayState &st, uint32_t kind, uint32_t s, int lane) {
  const uint64_t w = ((uint64_t)st.e << 32) | ((uint64_t)kind << 24) | s;
  st.hash = (st.hash ^ w) * kFnvPrime;
  if (!kLean && st.log) {
    if (st.log_len < st.log_cap) {
      if (lane == 0) {
        unison_decision d;
        d.event = st.e;
        d.kind_session = (kind << 24) | s;
        st.log[st.log_len] = d;
      }
    } else if (st.status == UNISON_OK) {
      st.status = UNISON_ERR_LOG_FULL;
    }
  }
  st.log_len++;
}

// Tier-map update: every lane stores the same byte, so each lane's later
// reads see it without a warp barrier.
template <bool kLean>
__device__ __forceinline__ void set_tier(ReplayState &st, uint32_t id, uint32_t tier) {
  if (kLean || st.tmap) st.tmap[id] = (uint8_t)tier;
}

template <bool kLean>
__device__ __forceinline__ bool sorted_insert(ReplayState &st, Sorted &T, uint4 v, int lane, uint32_t tier) {
  if (T.n >= T.cap) {
    st.status = UNISON_ERR_CAPACITY;
    return false;
  }
  uint32_t p = T.n;  // past the last key: an append, no search or shift
  if (T.n > 0 && ekey(v) < ekey(T.e[T.n - 1])) {
    p = lower_bound(T, ekey(v), lane);
    shift_block(T.e, p, T.n, 1, lane);
  }
  if (lane == 0) T.e[p] = v;
  __syncwarp();
  T.n++;
  set_tier<kLean>(st, packed_id(ekey(v)), tier);
  return true;
}

__device__ __forceinline__ void sorted_erase(Sorted &T, uint32_t p, int lane) {
  shift_block(T.e, p + 1, T.n, -1, lane);
  T.n--;
}

template <bool kLean>
__device__ __forceinline__ uint4 sorted_pop_back(ReplayState &st, Sorted &T) {
  const uint4 v = T.e[T.n - 1];
  __syncwarp();
  T.n--;
  set_tier<kLean>(st, packed_id(ekey(v)), kTierNone);
  return v;
}

template <bool kLean>
__device__ __forceinline__ bool reg_sorted_insert(ReplayState &st, uint4 v, int lane) {
  if (st.R.n >= st.S.cap) {
    st.status = UNISON_ERR_CAPACITY;
    return false;
  }
  reg_insert_at(st.R, reg_lower_bound(st.R, ekey(v), lane), v, lane);
  set_tier<kLean>(st, packed_id(ekey(v)), kTierS);
  return true;
}
template <bool kLean>
__device__ __forceinline__ uint4 reg_pop_back(ReplayState &st) {
  const uint4 v = reg_at(st.R, st.R.n - 1);
  st.R.n--;
  set_tier<kLean>(st, packed_id(ekey(v)), kTierNone);
  return v;
}

// HBM-tier operations on kHK register slots a lane, or on the array (kHK 0).
template <int kHK>
__device__ __forceinline__ uint4 h_at(const ReplayState &st, uint32_t i) {
  if constexpr (kHK > 0) return hreg_at<kHK>(st.G, i);
  return st.H.e[i];
}
template <int kHK>
__device__ __forceinline__ void h_erase_at(ReplayState &st, uint32_t p, int lane) {
  if constexpr (kHK > 0) {
    hreg_erase_at<kHK>(st.G, p, lane);
    st.H.n--;
  } else {
    sorted_erase(st.H, p, lane);
  }
}
template <bool kLean, int kHK>
__device__ __forceinline__ uint4 h_pop_back(ReplayState &st) {
  if constexpr (kHK > 0) {
    const uint4 v = hreg_at<kHK>(st.G, st.H.n - 1);
    st.H.n--;
    set_tier<kLean>(st, packed_id(ekey(v)), kTierNone);
    return v;
  }
  return sorted_pop_back<kLean>(st, st.H);
}
// Drop the first m entries (m <= 32 in register bodies).
template <int kHK>
__device__ __forceinline__ void h_drop_front(ReplayState &st, uint32_t m, int lane) {
  if constexpr (kHK > 0) hreg_drop_front<kHK>(st.G, m, lane);
  else shift_block(st.H.e, m, st.H.n, -(int32_t)m, lane);
  st.H.n -= m;
}
template <bool kLean, int kHK>
__device__ __forceinline__ bool h_insert(ReplayState &st, uint4 v, int lane) {
  if constexpr (kHK > 0) {
    if (st.H.n >= st.H.cap || st.H.n >= 32u * kHK) {
      // the list bound, or the registers' 32 kHK entries (the replay starts over)
      st.status = st.H.n >= st.H.cap ? UNISON_ERR_CAPACITY : kRegFull;
      return false;
    }
    hreg_insert_at<kHK>(st.G, hreg_lower_bound<kHK>(st.G, st.H.n, ekey(v), lane), v, lane);
    st.H.n++;
    set_tier<kLean>(st, packed_id(ekey(v)), kTierH);
    return true;
  }
  return sorted_insert<kLean>(st, st.H, v, lane, kTierH);
}

__device__ __forceinline__ uint32_t esize(uint4 v) { return v.z & kSizeMask; }

// Stale-snapshot replays (eq. stale): the arrays are ordered by snapshot
// keys; a choice made on them is compared with the most (least) evictable
// candidate by live keys.  Live keys are packed with the session id, so the
// extreme key names one session.
__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = max(v, (uint64_t)__shfl_xor_sync(kFull, (unsigned long long)v, o));
  return v;
}
__device__ __forceinline__ uint64_t warp_min_u64(uint64_t v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, (uint64_t)__shfl_xor_sync(kFull, (unsigned long long)v, o));
  return v;
}
__device__ __forceinline__ uint64_t live_max(const ReplayState &st, const Sorted &T, uint32_t lo, uint32_t hi,
                                             int lane) {
  uint64_t m = 0;
  for (uint32_t i = lo + lane; i < hi; i += 32) m = max(m, st.live[packed_id(ekey(T.e[i]))]);
  return warp_max_u64(m);
}
__device__ __forceinline__ uint64_t live_min(const ReplayState &st, const Sorted &T, uint32_t lo, uint32_t hi,
                                             int lane) {
  uint64_t m = ~0ull;
  for (uint32_t i = lo + lane; i < hi; i += 32) m = min(m, st.live[packed_id(ekey(T.e[i]))]);
  return warp_min_u64(m);
}
__device__ __forceinline__ void count_victim(ReplayState &st, uint32_t chosen, uint64_t live_best) {
  st.vict_n++;
  st.vict_diff += packed_id(live_best) != chosen;
}
__device__ __forceinline__ void count_promotion(ReplayState &st, uint32_t chosen, uint64_t live_best) {
  st.prom_n++;
  st.prom_diff += packed_id(live_best) != chosen;
}

// A session demoted out of the fast tier enters HBM, displacing the most
// evictable unpinned HBM sessions, or is dropped when it is itself the most
// evictable of (unpinned HBM) + {itself}.
template <bool kStale, bool kLean, int kHK = 0>
__device__ __forceinline__ bool admit_demoted(ReplayState &st, const Hot &D, uint4 d, int lane) {
  static_assert(!(kHK > 0 && kStale), "the register HBM tier serves live-key replays only");
  const uint32_t id = packed_id(ekey(d));
  const uint32_t size = esize(d);
  if (st.pinned_h > D.cap_h || size > D.cap_h - st.pinned_h) {
    log_dec<kLean>(st, UNISON_KIND_EVICT, id, lane);
    CNT(st, n_evict, 1);
    return true;
  }
  while (st.used_h + size > D.cap_h) {
    if (kStale) {
      const bool drop = st.H.n == 0 || ekey(d) > ekey(st.H.e[st.H.n - 1]);
      count_victim(st, drop ? id : packed_id(ekey(st.H.e[st.H.n - 1])),
                   max(live_max(st, st.H, 0, st.H.n, lane), st.live[id]));
    }
    if (st.H.n == 0 || ekey(d) > ekey(h_at<kHK>(st, st.H.n - 1))) {
      log_dec<kLean>(st, UNISON_KIND_EVICT, id, lane);
      CNT(st, n_evict, 1);
      return true;
    }
    const uint4 v = h_pop_back<kLean, kHK>(st);
    st.used_h -= esize(v);
    log_dec<kLean>(st, UNISON_KIND_EVICT, packed_id(ekey(v)), lane);
    CNT(st, n_evict, 1);
  }
  if (!h_insert<kLean, kHK>(st, d, lane)) return false;
  st.used_h += size;
  log_dec<kLean>(st, UNISON_KIND_DEMOTE, id, lane);
  CNT(st, n_demote, 1);
  return true;
}

__device__ __forceinline__ bool pin_append(ReplayState &st, uint64_t pk, uint32_t size, uint32_t s, uint32_t tier,
                                           int lane) {
  if (st.npin >= st.pin_cap) {
    st.status = UNISON_ERR_CAPACITY;
    return false;
  }
  if (lane == 0) st.pin[st.npin] = make_uint4((uint32_t)pk, (uint32_t)(pk >> 32), size, s | (tier << 30));
  if (st.pslot) st.pslot[s] = (uint16_t)st.npin;  // every lane stores the same slot
  __syncwarp();
  st.npin++;
  return true;
}

// Placement of the arriving (pinned) session s with n tokens.
template <bool kStale, bool kLean, bool kRegS = false, int kHK = 0>
__device__ __forceinline__ bool place(ReplayState &st, const Hot &D, uint32_t s, uint64_t pk, uint32_t n,
                                      int lane) {
  if (!kLean && D.max_sessions && st.npin >= D.max_sessions) {
    log_dec<kLean>(st, UNISON_KIND_BYPASS, s, lane);
    CNT(st, n_bypass, 1);
    return true;
  }
  if (st.pinned_s <= D.cap_s && n <= D.cap_s - st.pinned_s) {
    while (st.used_s + n > D.cap_s) {
      if ((kRegS ? st.R.n : st.S.n) == 0) {
        st.status = UNISON_ERR_CAPACITY;
        return false;
      }
      if (kStale) count_victim(st, packed_id(ekey(st.S.e[st.S.n - 1])), live_max(st, st.S, 0, st.S.n, lane));
      // most evictable unpinned fast-tier session
      const uint4 d = kRegS ? reg_pop_back<kLean>(st) : sorted_pop_back<kLean>(st, st.S);
      st.used_s -= esize(d);
      if (!admit_demoted<kStale, kLean, kHK>(st, D, d, lane)) return false;
    }
    if (!pin_append(st, pk, n, s, kTierS, lane)) return false;
    st.used_s += n;
    st.pinned_s += n;
    log_dec<kLean>(st, UNISON_KIND_PLACE_S, s, lane);
    CNT(st, n_place_s, 1);
  } else if (st.pinned_h <= D.cap_h && n <= D.cap_h - st.pinned_h) {
    while (st.used_h + n > D.cap_h) {
      if (st.H.n == 0) {
        st.status = UNISON_ERR_CAPACITY;
        return false;
      }
      if (kStale) count_victim(st, packed_id(ekey(st.H.e[st.H.n - 1])), live_max(st, st.H, 0, st.H.n, lane));
      const uint4 v = h_pop_back<kLean, kHK>(st);
      st.used_h -= esize(v);
      log_dec<kLean>(st, UNISON_KIND_EVICT, packed_id(ekey(v)), lane);
      CNT(st, n_evict, 1);
    }
    if (!pin_append(st, pk, n, s, kTierH, lane)) return false;
    st.used_h += n;
    st.pinned_h += n;
    log_dec<kLean>(st, UNISON_KIND_PLACE_H, s, lane);
    CNT(st, n_place_h, 1);
  } else {
    log_dec<kLean>(st, UNISON_KIND_BYPASS, s, lane);
    CNT(st, n_bypass, 1);
    return true;
  }
  if (!kLean && D.max_sessions) {
    while (st.S.n + st.H.n + st.npin > D.max_sessions) {
      if (st.S.n == 0 && st.H.n == 0) {
        st.status = UNISON_ERR_CAPACITY;
        return false;
      }
      const bool from_s =
          st.H.n == 0 || (st.S.n > 0 && ekey(st.S.e[st.S.n - 1]) > ekey(st.H.e[st.H.n - 1]));
      if (kStale)
        count_victim(st, packed_id(ekey(from_s ? st.S.e[st.S.n - 1] : st.H.e[st.H.n - 1])),
                     max(live_max(st, st.S, 0, st.S.n, lane), live_max(st, st.H, 0, st.H.n, lane)));
      const uint4 v = sorted_pop_back<kLean>(st, from_s ? st.S : st.H);
      if (from_s)
        st.used_s -= esize(v);
      else
        st.used_h -= esize(v);
      log_dec<kLean>(st, UNISON_KIND_EVICT, packed_id(ekey(v)), lane);
      CNT(st, n_evict, 1);
    }
  }
  return true;
}

// TIDE at a gap_start with `budget` bytes.  The moves are decided on the
// sorted arrays in the list form (phase 1: least evictable HBM sessions into
// free fast-tier space; phase 2: pair the next least evictable HBM session
// with the most evictable fast-tier one), which makes the same moves as the
// pair loop of Algorithm 1, and are then applied in bulk.
template <bool kStale, bool kLean, bool kRegS = false, int kHK = 0>
__device__ __forceinline__ uint64_t tide(ReplayState &st, const Hot &D, uint64_t budget, uint32_t rcap_s,
                                         int lane) {
  const uint32_t sn = kRegS ? st.R.n : st.S.n;  // fast-tier entries; the fast tier changes only at the end
  uint64_t rem = budget;
  const uint64_t kvb = D.kvb;
  uint32_t n1 = 0;
  while (n1 < st.H.n) {
    const uint4 p = h_at<kHK>(st, n1);
    const uint64_t sz = esize(p), by = sz * kvb;
    if (by > rem || st.used_s + sz > D.cap_s) break;
    // (the loop form's candidates: HBM less the sessions promoted so far)
    if (kStale) count_promotion(st, packed_id(ekey(p)), live_min(st, st.H, n1, st.H.n, lane));
    rem -= by;
    st.used_s += sz;
    st.used_h -= sz;
    log_dec<kLean>(st, UNISON_KIND_PROMOTE, packed_id(ekey(p)), lane);
    n1++;
  }
  uint32_t pairs = 0;
  for (;;) {
    if (n1 + pairs >= st.H.n || pairs >= sn) break;
    const uint4 p = h_at<kHK>(st, n1 + pairs);
    const uint4 d = kRegS ? reg_at(st.R, sn - 1 - pairs) : st.S.e[st.S.n - 1 - pairs];
    // the next most evictable of (fast tier + promoted) is a promoted session
    // when the largest promoted key beats d: then it cannot beat p, stop
    if (n1 > 0 && ekey(h_at<kHK>(st, n1 - 1)) > ekey(d)) break;
    if (!(ekey(d) > ekey(p))) break;
    const uint64_t sp = esize(p), sd = esize(d), by = (sp + sd) * kvb;
    if (by > rem) break;
    if (st.used_s - sd + sp > D.cap_s) break;
    if (st.used_h - sp + sd > D.cap_h) break;
    if (kStale) {
      // at this step HBM holds its entries from n1 + pairs on plus the pairs
      // demoted so far (the top `pairs` fast-tier entries); the fast tier
      // its first S.n - pairs entries plus the n1 + pairs promoted so far
      count_promotion(st, packed_id(ekey(p)),
                      min(live_min(st, st.H, n1 + pairs, st.H.n, lane), live_min(st, st.S, st.S.n - pairs, st.S.n, lane)));
      count_victim(st, packed_id(ekey(d)),
                   max(live_max(st, st.S, 0, st.S.n - pairs, lane), live_max(st, st.H, 0, n1 + pairs, lane)));
    }
    rem -= by;
    st.used_s = st.used_s - sd + sp;
    st.used_h = st.used_h - sp + sd;
    log_dec<kLean>(st, UNISON_KIND_PROMOTE, packed_id(ekey(p)), lane);
    log_dec<kLean>(st, UNISON_KIND_TIDE_DEMOTE, packed_id(ekey(d)), lane);
    pairs++;
  }
  const uint32_t m = n1 + pairs;
  CNT(st, n_promote, m);
  CNT(st, n_tide_demote, pairs);
  if (m == 0) return 0;
  if (m > rcap_s || pairs > rcap_s) {
    st.status = UNISON_ERR_CAPACITY;
    return budget - rem;
  }
  if (m == 1 && pairs == 0) {  // one promotion (the common case): move it directly
    uint4 v = h_at<kHK>(st, 0);
    v.z |= kPromotedBit;
    __syncwarp();
    h_drop_front<kHK>(st, 1, lane);
    if (kRegS) reg_sorted_insert<kLean>(st, v, lane);
    else sorted_insert<kLean>(st, st.S, v, lane, kTierS);
    return budget - rem;
  }
  if (m == 1 && pairs == 1) {  // one pair (the next most common): swap it directly
    uint4 v = h_at<kHK>(st, 0);
    v.z |= kPromotedBit;
    const uint4 d = kRegS ? reg_at(st.R, sn - 1) : st.S.e[st.S.n - 1];
    __syncwarp();
    h_drop_front<kHK>(st, 1, lane);
    if (kRegS) {
      st.R.n -= 1;
      if (!reg_sorted_insert<kLean>(st, v, lane)) return budget - rem;
    } else {
      st.S.n -= 1;
      if (!sorted_insert<kLean>(st, st.S, v, lane, kTierS)) return budget - rem;
    }
    h_insert<kLean, kHK>(st, d, lane);
    return budget - rem;
  }
  // stage the moved entries, then fix both arrays
  uint4 *pro = st.tmp, *dem = st.tmp + rcap_s;
  if constexpr (kHK > 0) {  // m <= 32: the first m entries are slot 0's
    if ((uint32_t)lane < m) pro[lane] = make_uint4(st.G.x[0], st.G.y[0], st.G.z[0] | kPromotedBit, 0u);
  } else {
    for (uint32_t i = lane; i < m; i += 32) {
      uint4 v = st.H.e[i];
      v.z |= kPromotedBit;
      pro[i] = v;
    }
  }
  if (kRegS) {  // pairs <= fast-tier entries <= 32: one entry a lane
    const uint4 dv = reg_at(st.R, min(sn - pairs + (uint32_t)lane, 31u));
    if ((uint32_t)lane < pairs) dem[lane] = dv;
  } else {
    for (uint32_t i = lane; i < pairs; i += 32) dem[i] = st.S.e[st.S.n - pairs + i];
  }
  __syncwarp();
  h_drop_front<kHK>(st, m, lane);
  if (kRegS) st.R.n -= pairs;
  else st.S.n -= pairs;
  for (uint32_t i = 0; i < m; i++)
    if (kRegS ? !reg_sorted_insert<kLean>(st, pro[i], lane) : !sorted_insert<kLean>(st, st.S, pro[i], lane, kTierS))
      return budget - rem;
  for (uint32_t i = 0; i < pairs; i++)
    if (!h_insert<kLean, kHK>(st, dem[i], lane)) return budget - rem;
  return budget - rem;
}

// Timeout: expire unpinned residents idle >= ttl, smallest session id first.
// Under recency keys the last return time falls as the key grows, so the
// expired sessions of a tier are a top suffix of its array.
template <bool kLean>
__device__ __forceinline__ void expire_idle(ReplayState &st, uint32_t now, uint32_t ttl, int lane) {
  for (;;) {
    // expired suffix lengths
    uint32_t cs = 0, ch = 0;
    while (cs < st.S.n && now - st.S.e[st.S.n - 1 - cs].w >= ttl) cs++;
    while (ch < st.H.n && now - st.H.e[st.H.n - 1 - ch].w >= ttl) ch++;
    if (cs + ch == 0) return;
    // smallest session id among them
    uint32_t bid = kFull, bpos = 0, btier = 0;
    for (uint32_t i = lane; i < cs + ch; i += 32) {
      const bool inS = i < cs;
      const uint32_t pos = inS ? st.S.n - 1 - i : st.H.n - 1 - (i - cs);
      const uint32_t id = packed_id(ekey(inS ? st.S.e[pos] : st.H.e[pos]));
      if (id < bid) {
        bid = id;
        bpos = pos;
        btier = inS ? kTierS : kTierH;
      }
    }
    const uint32_t mid = __reduce_min_sync(kFull, bid);
    const int src = __ffs(__ballot_sync(kFull, bid == mid)) - 1;
    const uint32_t pos = __shfl_sync(kFull, bpos, src), tier = __shfl_sync(kFull, btier, src);
    Sorted &T = tier == kTierS ? st.S : st.H;
    const uint32_t sz = esize(T.e[pos]);
    __syncwarp();
    if (tier == kTierS)
      st.used_s -= sz;
    else
      st.used_h -= sz;
    sorted_erase(T, pos, lane);
    set_tier<kLean>(st, mid, kTierNone);
    log_dec<kLean>(st, UNISON_KIND_EXPIRE, mid, lane);
    CNT(st, n_expire, 1);
  }
}

__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async8(void *dst, const void *src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async4(void *dst, const void *src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"((uint32_t)__cvta_generic_to_shared(dst)), "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_one() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ bool has_tide(uint32_t policy) {
  return policy == UNISON_SPEAR_TIDE || policy == UNISON_LRU_TIDE;
}

// --------------------------------------------------------------------------
// Online hazard table (Sec. V-F): counts n(t), d(t) of the sessions completed
// so far, and the table built from them exactly as the offline one (eqs.
// (hazard), (hq), (survq), (t2); bucket pooling).  Lives in shared memory
// after the per-session state of an online replay.
// --------------------------------------------------------------------------
struct OnlineTable {
  uint32_t n[kLutN], d[kLutN], sig[kLutN];
  unsigned long long t2[kLutN];
  unsigned long long mg[kLutN];  // magic_for(sig): eq. (t1)'s division by a multiply-high
};

// g < 2^31 (gaps are clamped below 2^31 us), so g * Lambda < 2^43.
__device__ __forceinline__ uint64_t online_key(const OnlineTable &ot, uint32_t g, uint32_t t, uint32_t s) {
  const uint32_t tt = t < kTMax ? t : kTMax;
  return pack_key(__umul64hi((uint64_t)g * kLambda, ot.mg[tt]) + ot.t2[tt], s);
}

// A session of `turns` turns has completed: add it to the counts and rebuild
// sigma and T2 for every turn index.
__device__ bool online_add(OnlineTable &ot, uint32_t turns, uint32_t bucket, uint64_t penalty, int lane) {
  for (uint32_t t = lane; t < kLutN; t += 32) {
    ot.n[t] += turns >= t + 1 ? 1u : 0u;
    ot.d[t] += turns == t + 1 ? 1u : 0u;
  }
  __syncwarp();
  uint32_t sg[2];
  unsigned long long t2[2];
#pragma unroll
  for (int q = 0; q < 2; q++) {
    const uint32_t t = lane + 32 * q;
    sg[q] = kLambda;
    t2[q] = 0;
    if (t < kLutN) {
      uint64_t nn = 0, dd = 0;
      for (uint32_t u = (t / bucket) * bucket; u < kLutN && u / bucket == t / bucket; u++) {
        nn += ot.n[u];
        dd += ot.d[u];
      }
      uint64_t hq = nn ? (2 * dd * kLambda + nn) / (2 * nn) : 0;
      if (hq > kLambda) hq = kLambda;
      const uint32_t sq = (uint32_t)(kLambda - hq) < kEpsQ ? kEpsQ : (uint32_t)(kLambda - hq);
      sg[q] = sq;
      t2[q] = ((unsigned long long)(kLambda - sq) * penalty) / kLambda;
    }
  }
  bool changed = false;
#pragma unroll
  for (int q = 0; q < 2; q++) changed |= (lane + 32 * q < kLutN) && ot.sig[lane + 32 * q] != sg[q];
  __syncwarp();
#pragma unroll
  for (int q = 0; q < 2; q++) {
    const uint32_t t = lane + 32 * q;
    if (t < kLutN) {
      if (ot.sig[t] != sg[q]) ot.mg[t] = magic_for(sg[q]);
      ot.sig[t] = sg[q];
      ot.t2[t] = t2[q];
    }
  }
  __syncwarp();
  return __any_sync(kFull, changed);  // T2 is a function of sigma
}

// Every resident takes a new key (new_key maps an entry's key to it), then the
// tier is re-sorted if that broke its order: bitonic network (descending,
// padded to a power of two with key 0, which no packed key equals since
// session ids stay below 2^24 - 1), then reversed.  The tier's array holds a
// power of two >= its capacity.
template <class KeyFn>
__device__ void rerank(Sorted &T, KeyFn new_key, int lane) {
  for (uint32_t i = lane; i < T.n; i += 32) {
    uint4 v = T.e[i];
    const uint64_t nk = new_key(ekey(v));
    v.x = (uint32_t)nk;
    v.y = (uint32_t)(nk >> 32);
    T.e[i] = v;
  }
  __syncwarp();
  // a small change of the keys often keeps the order: then nothing moves
  bool out_of_order = false;
  for (uint32_t i = lane + 1; i < T.n; i += 32) out_of_order |= ekey(T.e[i - 1]) > ekey(T.e[i]);
  if (!__any_sync(kFull, out_of_order)) return;
  const uint32_t ring = ring_size(T.n);
  for (uint32_t i = T.n + lane; i < ring; i += 32) T.e[i] = make_uint4(0u, 0u, 0u, 0u);
  __syncwarp();
  for (uint32_t k = 2; k <= ring; k <<= 1) {
    for (uint32_t j = k >> 1; j > 0; j >>= 1) {
      for (uint32_t q = lane; q < ring / 2; q += 32) {
        // q-th pair (i, i + j): i has a zero at bit j
        const uint32_t i = ((q & ~(j - 1)) << 1) | (q & (j - 1)), ij = i | j;
        const uint4 a = T.e[i], b = T.e[ij];
        const bool desc = (i & k) == 0;
        if (desc ? ekey(a) < ekey(b) : ekey(a) > ekey(b)) {
          T.e[i] = b;
          T.e[ij] = a;
        }
      }
      __syncwarp();
    }
  }
  for (uint32_t i = lane; i < T.n / 2; i += 32) {
    const uint4 a = T.e[i], b = T.e[T.n - 1 - i];
    T.e[i] = b;
    T.e[T.n - 1 - i] = a;
  }
  __syncwarp();
}

// Keys of every resident under a rebuilt online table; completed sessions
// keep the maximal key.
__device__ void online_rerank(Sorted &T, const OnlineTable &ot, const uint32_t *gs, const uint16_t *ks, int lane) {
  rerank(T, [&](uint64_t k) {
    if ((k >> 24) == kKeyMax40) return k;
    const uint32_t id = packed_id(k);
    return online_key(ot, gs[id], (uint32_t)ks[id] - 1, id);
  }, lane);
}

constexpr uint32_t kDirtyCap = 32;  // sessions a stale-snapshot sync updates one by one
constexpr int kKeyStream = 0;  // keys from the per-session key stream
constexpr int kKeyOnline = 1;  // keys under the online hazard table
constexpr int kKeyStale = 2;   // snapshot keys of a dual design

// Event prefetch: the next batch of 32 events and their side streams are
// copied into this shared-memory double buffer with cp.async while the
// current batch is processed.
struct EventBufs {
  uint4 sev[2][32];
  uint32_t sprev[2][32], spev[2][32], snref[2][32], sgq[2][32];
  unsigned long long spk[2][32], spkb[2][32];
};

// One replay: Algorithm 1 over the trace's events.  kPol is the replay's
// policy when the body is specialised for it (its policy tests then fold
// away), or -1 for the body that reads the policy from the descriptor.
// False when a register body (kHK > 0) stopped at its HBM tier's register
// bound (no result written): the caller replays it again with more slots or
// none.
template <bool kGlobalLists, int kKeys, int kPol, bool kLean, bool kRegS = false, int kHK = 0>
__device__ __forceinline__ bool replay_body(const ReplayDesc &D, EventBufs &bufs, unsigned char *smem, int lane) {
  constexpr bool kOnline = kKeys == kKeyOnline, kStale = kKeys == kKeyStale;
  // the register HBM tier drops the entries' completion times (timeout only)
  // and drop_front's m <= 32 rests on the fast tier's 32-entry bound
  static_assert(kHK == 0 || (kHK <= kHSlots && kRegS && kLean && kPol == UNISON_SPEAR_TIDE && !kOnline && !kStale),
                "register HBM tier: lean SPEAR+TIDE launches with the register fast tier");
  const Hot hot{D.cap_s, D.cap_h, D.kvb, D.dma, D.max_sessions};

  ReplayState st;
  uint32_t *online_gs = nullptr;
  uint16_t *online_ks = nullptr;
  OnlineTable *online_tab = nullptr;
  uint64_t *stale_live = nullptr, *stale_snap = nullptr;
  uint8_t *stale_dflag = nullptr;
  uint32_t *stale_dlist = nullptr, stale_ndirty = 0;
  // a session's live key changed: note it for the next sync (every lane
  // stores the same values)
  auto mark_dirty = [&](uint32_t s) {
    if (!stale_dflag[s]) {
      stale_dflag[s] = 1;
      if (stale_ndirty < kDirtyCap) stale_dlist[stale_ndirty] = s;
      stale_ndirty++;
    }
  };
  {
    uint4 *p = reinterpret_cast<uint4 *>(kGlobalLists ? reinterpret_cast<unsigned char *>(D.glist) : smem);
    // online and stale-snapshot replays keep power-of-two tiers (for re-sorts)
    st.S.e = p;
    p += (kOnline || kStale) ? ring_size(D.rcap_s) : D.rcap_s;
    st.H.e = p;
    p += (kOnline || kStale) ? ring_size(D.rcap_h) : D.rcap_h;
    st.pin = p;
    p += D.rcap_s + D.rcap_h;
    st.tmp = p;
    p += 2 * D.rcap_s;
    st.tmap = nullptr;
    st.pslot = nullptr;
    if (!kGlobalLists && D.tmap != kMapNone) {
      // tier map (1 B per session), then pin slots (2 B per session)
      st.tmap = reinterpret_cast<uint8_t *>(p);
      uint32_t *m32 = reinterpret_cast<uint32_t *>(p);
      for (uint32_t i = lane; i < (D.n_sessions + 3) / 4; i += 32) m32[i] = 0u;
      if (kLean || D.tmap == kMapSlots) {
        st.pslot = reinterpret_cast<uint16_t *>(reinterpret_cast<unsigned char *>(p) + ((D.n_sessions + 15) & ~15u));
        uint32_t *s32 = reinterpret_cast<uint32_t *>(st.pslot);
        for (uint32_t i = lane; i < (D.n_sessions + 1) / 2; i += 32) s32[i] = 0xFFFFFFFFu;
      }
      __syncwarp();
    }
    if (kOnline) {
      // after the tier map: gap average (u32) and arrivals so far (u16) per
      // session, then the table
      unsigned char *q = reinterpret_cast<unsigned char *>(p) + ((D.n_sessions + 15) & ~15u) +
                         2 * ((D.n_sessions + 7) & ~7u);
      online_gs = reinterpret_cast<uint32_t *>(q);
      q += 4 * ((D.n_sessions + 3) & ~3u);
      online_ks = reinterpret_cast<uint16_t *>(q);
      q += 2 * ((D.n_sessions + 7) & ~7u);
      online_tab = reinterpret_cast<OnlineTable *>(q);
      for (uint32_t i = lane; i < D.n_sessions; i += 32) {
        online_gs[i] = 0u;
        online_ks[i] = 0;
      }
      for (uint32_t t = lane; t < kLutN; t += 32) {
        online_tab->n[t] = online_tab->d[t] = 0u;
        online_tab->sig[t] = kLambda;  // no session completed: zero hazard
        online_tab->t2[t] = 0ull;
        online_tab->mg[t] = magic_for(kLambda);
      }
      __syncwarp();
    }
    if (kStale) {
      // after the tier map: each session's live key and snapshot key; a zero
      // register row (gap average 0, turn 0, not done) scores T2 of turn 0
      unsigned char *q = reinterpret_cast<unsigned char *>(p) + ((D.n_sessions + 15) & ~15u) +
                         2 * ((D.n_sessions + 7) & ~7u);
      stale_live = reinterpret_cast<uint64_t *>(q);
      stale_snap = stale_live + ((D.n_sessions + 1) & ~1u);
      // then a flag per session changed since the last sync, and the list of
      // the first kDirtyCap of them
      stale_dflag = reinterpret_cast<uint8_t *>(stale_snap + ((D.n_sessions + 1) & ~1u));
      stale_dlist = reinterpret_cast<uint32_t *>(stale_dflag + ((D.n_sessions + 15) & ~15u));
      const uint64_t k0 = D.t2[0];
      for (uint32_t i = lane; i < D.n_sessions; i += 32) {
        stale_live[i] = stale_snap[i] = pack_key(k0, i);
        stale_dflag[i] = 0;
      }
      __syncwarp();
    }
    st.live = stale_live;
    st.vict_n = st.vict_diff = st.prom_n = st.prom_diff = 0;
    st.S.n = st.H.n = 0;
    st.R.n = 0;
    st.R.v = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
    for (int j = 0; j < kHK; j++) st.G.x[j] = st.G.y[j] = st.G.z[j] = 0u;
    st.S.cap = D.rcap_s;
    st.H.cap = D.rcap_h;
    st.npin = 0;
    st.pin_cap = D.rcap_s + D.rcap_h;
    st.used_s = st.used_h = st.pinned_s = st.pinned_h = 0;
  }
  st.log = D.log;
  st.log_cap = D.log_cap;
  st.status = UNISON_OK;
  st.hash = kFnvOffset;
  st.log_len = 0;
  st.n_warm = st.n_cold = st.n_hit_s = st.n_hit_h = st.n_miss = st.n_bypass = st.n_place_s = st.n_place_h = 0;
  st.n_evict = st.n_demote = st.n_promote = st.n_tide_demote = st.n_expire = st.n_tide_calls = st.n_pth = 0;
  st.tok_hit_s = st.tok_hit_h = st.tok_miss = st.tok_computed = st.tok_needed = st.dma_bytes = 0;

  const uint32_t policy = kPol >= 0 ? (uint32_t)kPol : D.policy;
  const bool spear_keys = policy == UNISON_SPEAR || policy == UNISON_SPEAR_TIDE;
  const bool tide_on = has_tide(policy);
  const bool belady = policy == UNISON_BELADY;
  const bool timeout = policy == UNISON_TIMEOUT && D.ttl != 0xFFFFFFFFu;

  // TTFT queue (Sec. V-A): arrivals compressed by the load factor.
  uint64_t rel_us = 0, q_free = 0;
  uint32_t prev_now = 0, n_arr = 0, n_ev = 0;
  const uint32_t load = D.load;
  const uint64_t prefill_ns = D.prefill_ns;
  const uint32_t n_turns = D.n_turns;
  uint64_t *const ttft_out = D.ttft;
  const uint64_t ns_per_us = (1000u % load == 0) ? 1000u / load : 0u;  // 0: divide exactly
  unsigned long long s_lo = 0, s_hi = 0;
  uint32_t stale_arrivals = 0;
  bool dma_busy = false;
  uint64_t busy_from = 0, busy_bytes = 0;  // the DMA's last batch: start (rel_us) and bytes

  auto &sev = bufs.sev;
  auto &sprev = bufs.sprev, &spev = bufs.spev, &snref = bufs.snref, &sgq = bufs.sgq;
  auto &spk = bufs.spk, &spkb = bufs.spkb;
  const uint32_t E = D.n_events;
  auto fetch = [&](uint32_t b, int bi) {
    const uint32_t i = b + lane;
    if (i < E) {
      cp_async16(&sev[bi][lane], &D.ev[i]);
      cp_async4(&sprev[bi][lane], &D.prev_out[i]);
      if (!spear_keys) cp_async4(&spev[bi][lane], &D.prev_ev[i]);  // recency keys only
      if (belady) cp_async4(&snref[bi][lane], &D.nref[i]);
      if (spear_keys && !kOnline) {
        cp_async8(&spk[bi][lane], &D.pkey[i]);
        cp_async8(&spkb[bi][lane], &D.pkb[i]);
      }
      if (tide_on || kOnline) cp_async4(&sgq[bi][lane], &D.gq[i]);
    }
    cp_async_commit();
  };
  fetch(0, 0);
  cp_async_wait_all();
  __syncwarp();
  if (E) prev_now = sev[0][0].x;

  int bi = 0;
  for (uint32_t b = 0; b < E && st.status != UNISON_ERR_CAPACITY && st.status != kRegFull; b += 32, bi ^= 1) {
    if (b + 32 < E) {
      fetch(b + 32, bi ^ 1);
      cp_async_wait_one();  // this batch's copies have landed
    } else {
      cp_async_wait_all();
    }
    __syncwarp();
    const uint32_t cnt = min(32u, E - b);
    for (uint32_t j = 0; j < cnt; j++) {
      const uint32_t e = b + j;
      const uint4 ev = sev[bi][j];
      const uint32_t now = ev.x;
      const uint32_t w1 = ev.y;
      const uint32_t s = w1 & kIdMask;
      const bool arrival = (w1 & kEvArrival) != 0;
      const bool edge = (w1 & kEvEdge) != 0;
      st.e = e;
      n_ev++;
      rel_us += (uint32_t)(now - prev_now);
      prev_now = now;
      if (timeout) expire_idle<kLean>(st, now, D.ttl, lane);
      // the DMA is free again from start + ceil(bytes / rate) us on, i.e. once
      // the elapsed us times the rate cover the bytes (no division; the high
      // word of the product catches a product past 2^64)
      if (dma_busy) {
        const uint64_t el = rel_us - busy_from;
        if (__umul64hi(el, hot.dma) != 0 || el * hot.dma >= busy_bytes) dma_busy = false;
      }

      if (arrival) {
        const uint32_t in = ev.z;
        const uint32_t out = ev.w;
        const uint32_t prev = sprev[bi][j];
        // where is s?  search both tiers for the key of its previous event
        uint32_t tier = kTierNone;
        uint4 ent = make_uint4(0, 0, 0, 0);
        uint32_t pos = 0;
        if (!edge) {
          uint64_t pkb;
          if (kOnline)
            pkb = online_key(*online_tab, online_gs[s], (uint32_t)online_ks[s] - 1, s);
          else if (kStale)
            pkb = stale_snap[s];  // residents carry their snapshot keys
          else if (spear_keys)
            pkb = spkb[bi][j];
          else if (belady)
            pkb = pack_key(e, s);  // the previous arrival's next reference is this event
          else
            pkb = pack_key(0xFFFFFFFFull - spev[bi][j], s);
          // with the tier map only the session's own tier is searched (and
          // nothing for a session that is not resident)
          if constexpr (kHK > 0) {
            // both tiers in registers: one equality ballot per slot finds the
            // key (unique: it carries the session id) without the tier map
            const unsigned fs = __ballot_sync(kFull, (uint32_t)lane < st.R.n && ekey(st.R.v) == pkb);
            unsigned fh[kHK];
#pragma unroll
            for (int j = 0; j < kHK; j++)
              fh[j] = __ballot_sync(kFull, 32u * j + lane < st.H.n && hkey(st.G, j) == pkb);
            uint32_t ph = 0;
            unsigned inh = 0;
#pragma unroll
            for (int j = kHK - 1; j >= 0; j--) {
              if (fh[j]) ph = 32u * j + __ffs(fh[j]) - 1;
              inh |= fh[j];
            }
            const uint32_t ps = fs ? __ffs(fs) - 1 : 0u;
            const uint4 es = reg_at(st.R, ps), eh = hreg_at<kHK>(st.G, ph);
            tier = fs ? kTierS : (inh ? kTierH : kTierNone);
            pos = fs ? ps : ph;
            ent = fs ? es : eh;
          }
          const uint32_t mt = kHK > 0 ? 0u : ((kLean || st.tmap) ? st.tmap[s] : (kTierS | kTierH));
          if (mt & kTierS) {
            if (kRegS) {
              pos = reg_lower_bound(st.R, pkb, lane);
              const uint4 cand = reg_at(st.R, min(pos, 31u));
              if (pos < st.R.n && ekey(cand) == pkb) {
                tier = kTierS;
                ent = cand;
              }
            } else {
              pos = lower_bound(st.S, pkb, lane);
              if (pos < st.S.n && ekey(st.S.e[pos]) == pkb) {
                tier = kTierS;
                ent = st.S.e[pos];
              }
            }
          }
          if (tier == kTierNone && (mt & kTierH)) {
            pos = lower_bound(st.H, pkb, lane);
            if (pos < st.H.n && ekey(st.H.e[pos]) == pkb) {
              tier = kTierH;
              ent = st.H.e[pos];
            }
          }
          __syncwarp();
        }
        uint64_t prefill;
        if (edge) {
          log_dec<kLean>(st, UNISON_KIND_COLD, s, lane);
          CNT(st, n_cold, 1);
          prefill = in;
        } else {
          CNT(st, n_warm, 1);
          CNT(st, tok_needed, in);
          if (tier == kTierS) {
            log_dec<kLean>(st, UNISON_KIND_HIT_S, s, lane);
            CNT(st, n_hit_s, 1);
            CNT(st, tok_hit_s, prev);
            prefill = in - prev;
            if (ent.z & kPromotedBit) CNT(st, n_pth, 1);
          } else if (tier == kTierH) {
            log_dec<kLean>(st, UNISON_KIND_HIT_H, s, lane);
            CNT(st, n_hit_h, 1);
            CNT(st, tok_hit_h, prev);
            prefill = in - prev;
          } else {
            log_dec<kLean>(st, UNISON_KIND_MISS, s, lane);
            CNT(st, n_miss, 1);
            CNT(st, tok_miss, prev);
            prefill = in;
          }
          CNT(st, tok_computed, prefill);
        }
        {
          const uint64_t arr = ns_per_us ? rel_us * ns_per_us : rel_us * 1000ull / load;
          if (q_free < arr) q_free = arr;
          q_free += prefill * prefill_ns;
          const uint64_t v = q_free - arr;
          if (lane == 0 && n_arr < n_turns) ttft_out[n_arr] = v;
          n_arr++;
          const unsigned long long lo2 = s_lo + v;
          s_hi += (lo2 < s_lo);
          s_lo = lo2;
        }
        if (tier == kTierS) {
          st.used_s -= esize(ent);
          if (kRegS) reg_erase_at(st.R, pos, lane);
          else sorted_erase(st.S, pos, lane);
          set_tier<kLean>(st, s, kTierNone);
        } else if (tier == kTierH) {
          st.used_h -= esize(ent);
          h_erase_at<kHK>(st, pos, lane);
          set_tier<kLean>(st, s, kTierNone);
        }
        uint64_t pk;
        if (kOnline) {
          // turn k = arrivals so far; the session's gap average and turn
          // index advance (the count saturates far above the last table row)
          const uint32_t k = online_ks[s];
          pk = online_key(*online_tab, sgq[bi][j], k, s);
          __syncwarp();
          if (lane == 0) {
            online_gs[s] = sgq[bi][j];
            online_ks[s] = (uint16_t)(k < 0xFFFFu ? k + 1 : k);
          }
          __syncwarp();
        } else if (kStale) {
          pk = stale_snap[s];
          stale_live[s] = spk[bi][j];  // every lane stores the same key
          mark_dirty(s);
        } else if (spear_keys)
          pk = spk[bi][j];
        else if (belady) {
          const uint32_t nr = snref[bi][j];
          pk = pack_key(nr == kNoRef ? kKeyMax40 : (uint64_t)nr, s);
        } else
          pk = pack_key(0xFFFFFFFFull - e, s);
        if (!place<kStale, kLean, kRegS, kHK>(st, hot, s, pk, out, lane)) break;
      } else {
        // completion: unpin (if resident) and rank the session with its new key
        if (kStale) {
          stale_live[s] = spk[bi][j];
          mark_dirty(s);
        }
        uint32_t pi = kNoSlot;
        if (kLean || st.pslot) {
          pi = st.pslot[s];
        } else {
          int mine = -1;
          for (uint32_t i = lane; i < st.npin; i += 32)
            if ((st.pin[i].w & kIdMask) == s) mine = (int)i;
          const uint32_t who = __ballot_sync(kFull, mine >= 0);
          if (who) pi = (uint32_t)__shfl_sync(kFull, mine, __ffs(who) - 1);
        }
        if (pi != kNoSlot) {
          const uint4 pe = st.pin[pi];
          const uint4 last = st.pin[st.npin - 1];
          __syncwarp();
          if (lane == 0) st.pin[pi] = last;
          if (kLean || st.pslot) {  // the last entry moves into the freed slot
            st.pslot[last.w & kIdMask] = (uint16_t)pi;
            st.pslot[s] = kNoSlot;
          }
          __syncwarp();
          st.npin--;
          const uint32_t tier = pe.w >> 30, sz = pe.z;
          uint64_t pk = ((uint64_t)pe.y << 32) | pe.x;
          if (kOnline)
            pk = edge ? pack_key(kKeyMax40, s)
                      : online_key(*online_tab, online_gs[s], (uint32_t)online_ks[s] - 1, s);
          else if (kStale)
            pk = stale_snap[s];
          else if (spear_keys)
            pk = spk[bi][j];
          else if (!belady)
            pk = pack_key(0xFFFFFFFFull - e, s);
          const uint4 v = make_uint4((uint32_t)pk, (uint32_t)(pk >> 32), sz, now);
          if (tier == kTierS) {
            st.pinned_s -= sz;
            if (kRegS ? !reg_sorted_insert<kLean>(st, v, lane) : !sorted_insert<kLean>(st, st.S, v, lane, kTierS)) break;
          } else {
            st.pinned_h -= sz;
            if (!h_insert<kLean, kHK>(st, v, lane)) break;
          }
        }
        if (kOnline && edge) {
          // Sec. V-F: the finished session's turn count joins the table and
          // every resident is ranked under the rebuilt one
          if (online_add(*online_tab, online_ks[s], D.bucket, D.penalty, lane)) {
            online_rerank(st.S, *online_tab, online_gs, online_ks, lane);
            online_rerank(st.H, *online_tab, online_gs, online_ks, lane);
          }
        }
        if (!edge && tide_on && !dma_busy) {
          const uint64_t g = sgq[bi][j];
          const uint64_t budget = g * D.dma;
          CNT(st, n_tide_calls, 1);
          const uint64_t moved = tide<kStale, kLean, kRegS, kHK>(st, hot, budget, D.rcap_s, lane);
          CNT(st, dma_bytes, moved);
          if (moved > 0 && D.dma > 0) {
            dma_busy = true;
            busy_from = rel_us;
            busy_bytes = moved;
          }
          if (st.status == UNISON_ERR_CAPACITY || st.status == kRegFull) break;
        }
      }
      if (kStale) {
        // a sync point copies every live row into the snapshot, after the
        // event's own decisions; residents then carry their live keys
        bool sync = D.stale_sync == UNISON_SYNC_EVENT;
        if (arrival && D.stale_sync == UNISON_SYNC_ARRIVALS) sync = ++stale_arrivals % D.stale_m == 0;
        if (!arrival && D.stale_sync == UNISON_SYNC_GAP_START) sync = !edge;
        if (sync && stale_ndirty <= kDirtyCap) {
          // few sessions changed: move just their resident entries
          for (uint32_t k = 0; k < stale_ndirty; k++) {
            const uint32_t d = stale_dlist[k];
            const uint64_t nk = stale_live[d], ok = stale_snap[d];
            stale_snap[d] = nk;
            stale_dflag[d] = 0;
            const uint32_t t = st.tmap[d];
            if (t != kTierNone && nk != ok) {
              Sorted &T = t == kTierS ? st.S : st.H;
              const uint32_t pos = lower_bound(T, ok, lane);
              uint4 v = T.e[pos];
              __syncwarp();
              v.x = (uint32_t)nk;
              v.y = (uint32_t)(nk >> 32);
              sorted_erase(T, pos, lane);
              sorted_insert<kLean>(st, T, v, lane, t);
            }
          }
          __syncwarp();
          stale_ndirty = 0;
        } else if (sync) {
          for (uint32_t i = lane; i < D.n_sessions; i += 32) {
            stale_snap[i] = stale_live[i];
            stale_dflag[i] = 0;
          }
          __syncwarp();
          const auto snap_key = [&](uint64_t k) { return stale_snap[packed_id(k)]; };
          rerank(st.S, snap_key, lane);
          rerank(st.H, snap_key, lane);
          stale_ndirty = 0;
        }
      }
    }
  }
  if (kHK > 0 && st.status == kRegFull) {
    cp_async_wait_all();  // the next batch's copies land before the replay starts over
    __syncwarp();
    return false;
  }
  if (lane == 0) {
    unison_replay_result r = {};
    r.events = n_ev;
    r.req_warm = st.n_warm;
    r.cold = st.n_cold;
    r.hit_s = st.n_hit_s;
    r.hit_h = st.n_hit_h;
    r.miss = st.n_miss;
    r.bypass = st.n_bypass;
    r.place_s = st.n_place_s;
    r.place_h = st.n_place_h;
    r.evict = st.n_evict;
    r.demote = st.n_demote;
    r.promote = st.n_promote;
    r.tide_demote = st.n_tide_demote;
    r.expire = st.n_expire;
    r.tok_hit_s = st.tok_hit_s;
    r.tok_hit_h = st.tok_hit_h;
    r.tok_miss = st.tok_miss;
    r.tok_computed = st.tok_computed;
    r.tok_needed = st.tok_needed;
    r.dma_bytes = st.dma_bytes;
    r.tide_calls = st.n_tide_calls;
    r.promoted_then_hit_s = st.n_pth;
    r.ttft_sum_lo = s_lo;
    r.ttft_sum_hi = s_hi;
    r.ttft_p50_ns = 0;
    r.ttft_n = n_arr;
    r.decision_hash = st.hash;
    r.log_len = st.log_len;
    r.vict_n = st.vict_n;
    r.vict_diff = st.vict_diff;
    r.prom_n = st.prom_n;
    r.prom_diff = st.prom_diff;
    r.status = st.status;
    *D.result = r;
  }
  return true;
}

// One warp per replay.  SPEAR+TIDE replays (the sweep's policy) run a body
// specialised for it: a smaller, branch-free event loop.  kOnly >= 0: every
// replay of the launch has that policy, and the kernel holds only its body
// (and is sized for it alone); kLean: every replay of the launch is lean
// (see log_dec).
template <bool kGlobalLists, int kKeys, int kOnly, bool kLean, bool kRegS = false, int kHK = 0>
__global__ void __launch_bounds__(32) replay_kernel(const ReplayDesc *descs, const uint32_t *order) {
  extern __shared__ __align__(16) unsigned char smem[];
  __shared__ ReplayDesc Dsh;
  __shared__ __align__(16) EventBufs bufs;
  const int lane = threadIdx.x & 31;
  if (lane == 0) Dsh = descs[order[blockIdx.x]];
  __syncwarp();
  if (kOnly >= 0) {
    if constexpr (kHK > 0) {
      // a replay whose HBM tier outgrows kHK slots starts over with the tier
      // in shared memory
      if (!replay_body<kGlobalLists, kKeys, kOnly, kLean, kRegS, kHK>(Dsh, bufs, smem, lane))
        replay_body<kGlobalLists, kKeys, kOnly, kLean, kRegS, 0>(Dsh, bufs, smem, lane);
    } else {
      replay_body<kGlobalLists, kKeys, kOnly, kLean, kRegS, 0>(Dsh, bufs, smem, lane);
    }
  } else if (kKeys == kKeyStream && Dsh.policy == UNISON_SPEAR_TIDE)
    replay_body<kGlobalLists, kKeys, UNISON_SPEAR_TIDE, false>(Dsh, bufs, smem, lane);
  else
    replay_body<kGlobalLists, kKeys, -1, false>(Dsh, bufs, smem, lane);
}

// Lower median (element floor((n-1)/2) in sorted order) by MSB-first radix select.
__global__ void __launch_bounds__(256) ttft_median_kernel(const ReplayDesc *descs, uint32_t n_replays) {
  const ReplayDesc &D = descs[blockIdx.x];
  __shared__ unsigned int hist[256];
  __shared__ unsigned long long red[8];
  __shared__ unsigned int sel_digit, sel_count;
  __shared__ unsigned long long sel_target;
  const uint64_t n = min((uint64_t)D.result->ttft_n, (uint64_t)D.n_turns);
  if (n == 0) {
    if (threadIdx.x == 0) D.result->ttft_p50_ns = 0;
    return;
  }
  const uint64_t *v = D.ttft;
  unsigned long long orv = 0;
  for (uint64_t i = threadIdx.x; i < n; i += blockDim.x) orv |= v[i];
  for (int o = 16; o; o >>= 1) orv |= __shfl_xor_sync(kFull, orv, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = orv;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long a = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); w++) a |= red[w];
    red[0] = a;
  }
  __syncthreads();
  const unsigned long long all = red[0];
  int top = 0;
  for (int b = 7; b >= 0; b--)
    if ((all >> (8 * b)) & 0xFF) {
      top = b;
      break;
    }
  // Once the values that share the selected prefix fit in shared memory, a
  // global pass copies them there and the remaining passes read only those.
  constexpr uint32_t kMedCap = 4096;
  __shared__ unsigned long long cand[kMedCap];
  __shared__ unsigned int ncand;
  uint64_t target = (n - 1) / 2, prefix = 0, mask = 0, cnt = n;  // cnt: values matching the prefix
  bool in_smem = false;
  uint32_t m = 0;
  for (int b = top; b >= 0; b--) {
    for (uint32_t i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    const bool copy = !in_smem && cnt <= kMedCap;
    if (threadIdx.x == 0) ncand = 0;
    __syncthreads();
    if (in_smem) {
      for (uint32_t i = threadIdx.x; i < m; i += blockDim.x) {
        const uint64_t x = cand[i];
        if ((x & mask) == prefix) atomicAdd(&hist[(x >> (8 * b)) & 0xFF], 1u);
      }
    } else {
      for (uint64_t i = threadIdx.x; i < n; i += blockDim.x) {
        const uint64_t x = v[i];
        if ((x & mask) == prefix) {
          atomicAdd(&hist[(x >> (8 * b)) & 0xFF], 1u);
          if (copy) cand[atomicAdd(&ncand, 1u)] = x;
        }
      }
    }
    __syncthreads();
    if (copy) {
      in_smem = true;
      m = ncand;
    }
    if (threadIdx.x == 0) {
      uint64_t cum = 0;
      uint32_t d = 0;
      for (; d < 256; d++) {
        if (cum + hist[d] > target) break;
        cum += hist[d];
      }
      sel_digit = d < 256 ? d : 255;
      sel_target = target - cum;
      sel_count = d < 256 ? hist[d] : 0;
    }
    __syncthreads();
    prefix |= (uint64_t)sel_digit << (8 * b);
    mask |= 0xFFull << (8 * b);
    target = sel_target;
    cnt = sel_count;
    __syncthreads();
  }
  if (threadIdx.x == 0) D.result->ttft_p50_ns = prefix;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool needs_stream(uint32_t p) { return p == UNISON_SPEAR || p == UNISON_SPEAR_TIDE || p == UNISON_LRU_TIDE; }

int check_params(const unison_replay_params &p, int n_traces) {
  if (p.policy > UNISON_LRU_TIDE) return UNISON_ERR_ARG;
  if ((int)p.trace_idx >= n_traces) return UNISON_ERR_ARG;
  if (p.kv_bytes_per_token == 0 || p.kv_bytes_per_token > (1u << 24)) return UNISON_ERR_RANGE;
  if (p.ema_den == 0 || p.ema_num > p.ema_den || p.ema_den > (1u << 20)) return UNISON_ERR_RANGE;
  if (p.hazard_bucket == 0) return UNISON_ERR_ARG;
  if (p.penalty_q >= (1ull << 32)) return UNISON_ERR_RANGE;
  if (p.dma_bytes_per_us >= (1ull << 32)) return UNISON_ERR_RANGE;
  if (p.ttl_us != 0xFFFFFFFFu && p.ttl_us >= (1u << 31)) return UNISON_ERR_RANGE;
  if (p.ttft_load == 0) return UNISON_ERR_ARG;
  constexpr uint32_t kSignals = UNISON_SIGNAL_NO_GAP | UNISON_SIGNAL_NO_HAZARD;
  if (p.flags & ~(UNISON_HAZARD_ONLINE | kSignals)) return UNISON_ERR_ARG;
  if ((p.flags & kSignals) &&
      ((p.flags & UNISON_HAZARD_ONLINE) || (p.policy != UNISON_SPEAR && p.policy != UNISON_SPEAR_TIDE)))
    return UNISON_ERR_ARG;
  if ((p.flags & UNISON_HAZARD_ONLINE) && p.policy != UNISON_SPEAR && p.policy != UNISON_SPEAR_TIDE)
    return UNISON_ERR_ARG;
  if (p.stale_sync > UNISON_SYNC_GAP_START || (p.stale_sync == UNISON_SYNC_ARRIVALS && p.stale_m == 0))
    return UNISON_ERR_ARG;
  if (p.stale_sync != UNISON_SYNC_LIVE &&
      ((p.flags & UNISON_HAZARD_ONLINE) || (p.policy != UNISON_SPEAR && p.policy != UNISON_SPEAR_TIDE)))
    return UNISON_ERR_ARG;
  return UNISON_OK;
}

}  // namespace

extern "C" int unison_hazard_lut(const uint32_t *turns_dev, uint64_t n_sessions, uint32_t bucket,
                                 uint16_t *sigma_q_dev, uint16_t *h_q_dev, void *cuda_stream) {
  if (!turns_dev || !sigma_q_dev || bucket == 0 || n_sessions >= (1ull << 32)) return UNISON_ERR_ARG;
  hazard_lut_single_kernel<<<1, 256, 0, static_cast<cudaStream_t>(cuda_stream)>>>(
      turns_dev, (uint32_t)n_sessions, bucket, sigma_q_dev, h_q_dev);
  count_launches(1);
  return cudaGetLastError() == cudaSuccess ? UNISON_OK : UNISON_ERR_CUDA;
}

namespace {

// Scratch layout and launch plan of one batch (shared by both entry points).
struct ReplayPlan {
  std::vector<std::tuple<uint32_t, uint32_t, uint32_t, uint32_t, uint64_t, uint32_t>> combos;
  std::vector<int> replay_combo;
  size_t off_desc = 0, off_order = 0, off_combo = 0, bytes = 0;
  std::vector<size_t> off_lut, off_stream, off_ttft, off_glist;
  // Replay groups, one kernel launch each: lists in shared memory (SPEAR+TIDE,
  // other policies), in global memory (the same split), online hazard table,
  // stale snapshot.  The launches are independent and run concurrently.
  std::vector<uint32_t> in_st, in_mix, in_gst, in_gmix, in_online, in_stale;
  std::vector<uint32_t> rcap_s, rcap_h, tmap;
  size_t max_smem_st = 0, max_smem_mix = 0, max_smem_online = 0, max_smem_stale = 0;
  bool st_lean = true;  // every shared-memory SPEAR+TIDE replay has the map with pin slots and no slot limit
  bool st_reg = true;   // and a fast tier of at most 32 entries (held in the warp's registers)
};

// Resident-list capacity of a tier: at most one entry per session and no more
// than the tier's token capacity over the smallest l^out of the trace (+1
// for the transient extra entry while a pair is swapped).
uint32_t list_cap(uint64_t cap_tok, const unison_trace *tr) {
  const uint64_t mo = std::max<uint32_t>(tr->min_out_tok, 1);
  return (uint32_t)std::min<uint64_t>(tr->n_sessions, cap_tok / mo) + 1;
}

// 16-byte entries: fast and HBM arrays, the pinned list (both tiers) and the
// TIDE staging area (two fast-tier capacities).  The tier map and pin slots
// (3 B per session) follow when the trace has at most kTierMapMax sessions
// and they fit; else the tier map alone (1 B per session) when the launch's
// replays still run in as few waves of CTAs.
constexpr uint32_t kTierMapMax = 32768;
size_t list_bytes(uint32_t cs, uint32_t ch) { return 16ull * (4ull * cs + 2ull * ch); }

// An online hazard replay: both tiers rounded up to powers of two, the tier
// map, the per-session gap average (4 B) and arrival count (2 B), the table.
// A stale-snapshot replay: power-of-two tiers, the tier map, then the live
// and snapshot key of every session.
size_t stale_bytes(uint32_t cs, uint32_t ch, uint32_t n_sessions) {
  const size_t n = n_sessions;
  return 16ull * (ring_size(cs) + ring_size(ch) + 3ull * cs + ch) + align_up(n, 16) + 2 * align_up(n, 8) +
         16 * align_up(n, 2) + align_up(n, 16) + 4 * kDirtyCap;
}

size_t online_bytes(uint32_t cs, uint32_t ch, uint32_t n_sessions) {
  const size_t n = n_sessions;
  return 16ull * (ring_size(cs) + ring_size(ch) + 3ull * cs + ch) + align_up(n, 16) + 2 * align_up(n, 8) +
         4 * align_up(n, 4) +
         2 * align_up(n, 8) + align_up(sizeof(OnlineTable), 16);
}

using ReplayKernel = void (*)(const ReplayDesc *, const uint32_t *);

// The kernel of the shared-memory SPEAR+TIDE group, for a log or not.
ReplayKernel st_kernel(const ReplayPlan &P, bool logged) {
  if (P.st_lean && !logged)
    return P.st_reg ? replay_kernel<false, kKeyStream, UNISON_SPEAR_TIDE, true, true, kHSlots>
                    : replay_kernel<false, kKeyStream, UNISON_SPEAR_TIDE, true>;
  return replay_kernel<false, kKeyStream, UNISON_SPEAR_TIDE, false>;
}

// Waves of CTAs a group of n replays needs with `dyn` bytes per CTA.
uint64_t smem_waves(ReplayKernel k, size_t n, size_t dyn) {
  int dev = 0, sms = 0, nb = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, k, 32, dyn) != cudaSuccess || nb <= 0 || sms <= 0) {
    cudaGetLastError();
    return ~0ull;
  }
  const uint64_t slots = (uint64_t)nb * (uint64_t)sms;
  return (n + slots - 1) / slots;
}

// Replays of a shared-memory group without a map take the tier map alone (an
// arrival then searches only its own tier, and nothing on a miss) when it
// fits and the group needs no more waves with it.
void add_tier_maps(const unison_trace *const *traces, const unison_replay_params *params, size_t smem_limit,
                   const std::vector<uint32_t> &group, ReplayKernel k, size_t &max_smem, ReplayPlan &P) {
  size_t with = max_smem;
  std::vector<uint32_t> add;
  for (uint32_t r : group) {
    if (P.tmap[r] != kMapNone) continue;
    const unison_trace *tr = traces[params[r].trace_idx];
    const size_t b = list_bytes(P.rcap_s[r], P.rcap_h[r]) + align_up(tr->n_sessions, 16);
    if (b > smem_limit) continue;
    add.push_back(r);
    with = std::max(with, b);
  }
  if (add.empty()) return;
  if (with > max_smem && smem_waves(k, group.size(), with) > smem_waves(k, group.size(), max_smem)) return;
  for (uint32_t r : add) P.tmap[r] = kMapTier;
  max_smem = with;
}

int plan_replays(const unison_trace *const *traces, const unison_replay_params *params, int n_replays,
                 size_t smem_limit, bool results_in_scratch, ReplayPlan &P, size_t &off_res) {
  std::map<std::tuple<uint32_t, uint32_t, uint32_t, uint32_t, uint64_t, uint32_t>, int> combo_of;
  P.replay_combo.assign(n_replays, -1);
  for (int r = 0; r < n_replays; r++) {
    const unison_replay_params &p = params[r];
    if (!needs_stream(p.policy)) continue;
    auto key = std::make_tuple(p.trace_idx, p.ema_num, p.ema_den, p.hazard_bucket, p.penalty_q,
                               p.flags & (UNISON_SIGNAL_NO_GAP | UNISON_SIGNAL_NO_HAZARD));
    auto it = combo_of.find(key);
    if (it == combo_of.end()) {
      it = combo_of.emplace(key, (int)P.combos.size()).first;
      P.combos.push_back(key);
    }
    P.replay_combo[r] = it->second;
  }
  size_t off = 0;
  P.off_desc = off;
  off = align_up(off + sizeof(ReplayDesc) * n_replays, 256);
  P.off_order = off;
  off = align_up(off + sizeof(uint32_t) * 2 * n_replays, 256);
  P.off_combo = off;
  off = align_up(off + sizeof(ComboDesc) * P.combos.size() + 1, 256);
  P.off_lut.resize(P.combos.size());
  P.off_stream.resize(P.combos.size());
  for (size_t c = 0; c < P.combos.size(); c++) {
    P.off_lut[c] = off;
    off = align_up(off + 128 + 51 * 8, 256);
    const uint64_t E = traces[std::get<0>(P.combos[c])]->n_events;
    P.off_stream[c] = off;
    off = align_up(off + align_up(12 * E, 8) + 8 * E, 256);
  }
  P.off_ttft.assign(n_replays, 0);
  P.off_glist.assign(n_replays, 0);
  P.rcap_s.resize(n_replays);
  P.rcap_h.resize(n_replays);
  P.tmap.assign(n_replays, 0);
  for (int r = 0; r < n_replays; r++) {
    const unison_replay_params &p = params[r];
    const unison_trace *tr = traces[p.trace_idx];
    P.rcap_s[r] = list_cap(p.cap_fast_bytes / p.kv_bytes_per_token, tr);
    P.rcap_h[r] = list_cap(p.cap_hbm_bytes / p.kv_bytes_per_token, tr);
    const size_t lists = list_bytes(P.rcap_s[r], P.rcap_h[r]);
    // the tier map and pin slots (3 bytes per session) when they fit beside the lists
    const size_t map = align_up(tr->n_sessions, 16) + 2 * align_up(tr->n_sessions, 8);
    P.tmap[r] = tr->n_sessions <= kTierMapMax && lists + map <= smem_limit ? kMapSlots : kMapNone;
    if (p.flags & UNISON_HAZARD_ONLINE) {
      // online hazard replays run from shared memory only
      const size_t ob = online_bytes(P.rcap_s[r], P.rcap_h[r], tr->n_sessions);
      if (tr->n_sessions > kTierMapMax || ob > smem_limit) return UNISON_ERR_RANGE;
      P.tmap[r] = kMapSlots;
      P.in_online.push_back((uint32_t)r);
      P.max_smem_online = std::max(P.max_smem_online, ob);
    } else if (p.stale_sync != UNISON_SYNC_LIVE) {
      // stale-snapshot replays too
      const size_t sb = stale_bytes(P.rcap_s[r], P.rcap_h[r], tr->n_sessions);
      if (tr->n_sessions > kTierMapMax || sb > smem_limit) return UNISON_ERR_RANGE;
      P.tmap[r] = kMapSlots;
      P.in_stale.push_back((uint32_t)r);
      P.max_smem_stale = std::max(P.max_smem_stale, sb);
    } else if (lists <= smem_limit) {
      const bool st = p.policy == UNISON_SPEAR_TIDE;
      (st ? P.in_st : P.in_mix).push_back((uint32_t)r);
      size_t &m = st ? P.max_smem_st : P.max_smem_mix;
      m = std::max<size_t>(m, lists + (P.tmap[r] == kMapSlots ? map : 0));
    } else {
      P.tmap[r] = kMapNone;
      (p.policy == UNISON_SPEAR_TIDE ? P.in_gst : P.in_gmix).push_back((uint32_t)r);
      P.off_glist[r] = off;
      off = align_up(off + lists, 256);
    }
    P.off_ttft[r] = off;
    off = align_up(off + 8 * (tr->n_turns + 1), 256);
  }
  add_tier_maps(traces, params, smem_limit, P.in_st, st_kernel(P, true), P.max_smem_st, P);
  add_tier_maps(traces, params, smem_limit, P.in_mix, replay_kernel<false, kKeyStream, -1, false>, P.max_smem_mix,
                P);
  for (uint32_t r : P.in_st) P.st_lean &= P.tmap[r] == kMapSlots && params[r].max_sessions == 0;
  for (uint32_t r : P.in_st) P.st_reg &= P.rcap_s[r] <= 32;
  off_res = 0;
  if (results_in_scratch) {
    off_res = off;
    off = align_up(off + sizeof(unison_replay_result) * n_replays, 256);
  }
  P.bytes = off;
  return UNISON_OK;
}

// Fill the descriptors for a plan placed at `scratch`.
void fill_descs(const unison_trace *const *traces, const unison_replay_params *params, int n_replays,
                const ReplayPlan &P, char *scratch, unison_replay_result *res, unison_decision *log_dev,
                uint64_t log_cap, std::vector<ComboDesc> &hc, std::vector<ReplayDesc> &hd,
                std::vector<uint32_t> &order) {
  hc.resize(P.combos.size());
  for (size_t c = 0; c < P.combos.size(); c++) {
    const unison_trace *tr = traces[std::get<0>(P.combos[c])];
    ComboDesc &d = hc[c];
    d.turn_ev = tr->d<uint32_t>(tr->off_turn_ev);
    d.turn_t = tr->d<uint32_t>(tr->off_turn_t);
    d.turn_off = tr->d<uint32_t>(tr->off_turn_off);
    d.tps = tr->d<uint32_t>(tr->off_tps);
    d.n_sessions = tr->n_sessions;
    d.n_events = (uint32_t)tr->n_events;
    d.ema_num = std::get<1>(P.combos[c]);
    d.ema_den = std::get<2>(P.combos[c]);
    d.bucket = std::get<3>(P.combos[c]);
    d.signals = std::get<5>(P.combos[c]);
    d.penalty_q = std::get<4>(P.combos[c]);
    d.sigma = reinterpret_cast<uint16_t *>(scratch + P.off_lut[c]);
    d.t2 = reinterpret_cast<uint64_t *>(scratch + P.off_lut[c] + 128);
    d.pkey = reinterpret_cast<uint64_t *>(scratch + P.off_stream[c]);
    d.gq = reinterpret_cast<uint32_t *>(scratch + P.off_stream[c] + 8 * tr->n_events);
    d.pkb = reinterpret_cast<uint64_t *>(scratch + P.off_stream[c] + align_up(12 * tr->n_events, 8));
  }
  hd.resize(n_replays);
  for (int r = 0; r < n_replays; r++) {
    const unison_replay_params &p = params[r];
    const unison_trace *tr = traces[p.trace_idx];
    ReplayDesc &d = hd[r];
    d.ev = tr->d<uint4>(tr->off_ev);
    d.prev_out = tr->d<uint32_t>(tr->off_prev_out);
    d.nref = tr->d<uint32_t>(tr->off_nref);
    d.prev_ev = tr->d<uint32_t>(tr->off_prev_ev);
    d.pkey = P.replay_combo[r] >= 0 ? hc[P.replay_combo[r]].pkey : nullptr;
    d.gq = P.replay_combo[r] >= 0 ? hc[P.replay_combo[r]].gq : nullptr;
    d.pkb = P.replay_combo[r] >= 0 ? hc[P.replay_combo[r]].pkb : nullptr;
    d.ttft = reinterpret_cast<uint64_t *>(scratch + P.off_ttft[r]);
    d.glist = P.off_glist[r] ? reinterpret_cast<uint32_t *>(scratch + P.off_glist[r]) : nullptr;
    d.log = log_dev ? log_dev + (uint64_t)r * log_cap : nullptr;
    d.log_cap = log_dev ? log_cap : 0;
    d.result = res + r;
    d.cap_s = p.cap_fast_bytes / p.kv_bytes_per_token;
    d.cap_h = p.cap_hbm_bytes / p.kv_bytes_per_token;
    d.dma = p.dma_bytes_per_us;
    d.prefill_ns = p.t_p_ps_per_tok / 1000;
    d.n_events = (uint32_t)tr->n_events;
    d.n_turns = (uint32_t)tr->n_turns;
    d.n_sessions = tr->n_sessions;
    d.policy = p.policy;
    d.max_sessions = p.max_sessions;
    d.kvb = p.kv_bytes_per_token;
    d.ttl = p.ttl_us;
    d.load = p.ttft_load;
    d.rcap_s = P.rcap_s[r];
    d.rcap_h = P.rcap_h[r];
    d.tmap = P.tmap[r];
    d.bucket = p.hazard_bucket;
    d.penalty = p.penalty_q;
    d.t2 = P.replay_combo[r] >= 0 ? hc[P.replay_combo[r]].t2 : nullptr;
    d.stale_sync = p.stale_sync;
    d.stale_m = p.stale_m;
  }
  order.clear();
  for (const auto *g : {&P.in_st, &P.in_mix, &P.in_gst, &P.in_gmix, &P.in_online, &P.in_stale})
    order.insert(order.end(), g->begin(), g->end());
  // A launch lasts as long as its slowest replay, and CTAs start in index
  // order: the SPEAR+TIDE launch takes its replays by predicted cost,
  // largest first, so the long ones start early and the short ones fill in.
  // The predictor is the product of the tiers' capacities (the larger both
  // tiers, the more tier moves a replay makes); decisions do not depend on
  // the order.
  std::stable_sort(order.begin(), order.begin() + P.in_st.size(), [&](uint32_t a, uint32_t b) {
    return (double)hd[a].cap_s * (double)hd[a].cap_h > (double)hd[b].cap_s * (double)hd[b].cap_h;
  });
}

// Side streams for the replay groups of one call, one set per device, made
// on first use.  The caller holds the lock while it forks and joins, so two
// host threads never interleave their events.
constexpr int kSideStreams = 5;
struct SideStreams {
  cudaStream_t s[kSideStreams] = {};
  cudaEvent_t fork = nullptr, join[kSideStreams] = {};
  bool ready = false;
};
std::mutex g_side_mu;
SideStreams g_side[64];

SideStreams *side_streams(std::unique_lock<std::mutex> &hold) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
    cudaGetLastError();
    return nullptr;
  }
  hold = std::unique_lock<std::mutex>(g_side_mu);
  SideStreams &g = g_side[dev];
  if (!g.ready) {
    // handles made by an earlier, failed try are kept and not made again
    bool ok = g.fork || cudaEventCreateWithFlags(&g.fork, cudaEventDisableTiming) == cudaSuccess;
    for (int i = 0; ok && i < kSideStreams; i++) {
      ok = g.s[i] || cudaStreamCreateWithFlags(&g.s[i], cudaStreamNonBlocking) == cudaSuccess;
      ok = ok && (g.join[i] || cudaEventCreateWithFlags(&g.join[i], cudaEventDisableTiming) == cudaSuccess);
    }
    if (!ok) {
      cudaGetLastError();
      return nullptr;
    }
    g.ready = true;
  }
  return &g;
}

// Queue the kernels of a planned batch on `stream`.
int launch_replays(const ReplayPlan &P, char *scratch, const std::vector<ComboDesc> &hc,
                   const std::vector<ReplayDesc> &hd, const std::vector<uint32_t> &order, int n_replays,
                   cudaStream_t stream, bool profile, bool logged) {
  int rc = UNISON_OK;
  auto ck = [&](cudaError_t e) {
    if (e != cudaSuccess && rc == UNISON_OK) rc = UNISON_ERR_CUDA;
  };
  ReplayDesc *d_desc = reinterpret_cast<ReplayDesc *>(scratch + P.off_desc);
  uint32_t *d_order = reinterpret_cast<uint32_t *>(scratch + P.off_order);
  ComboDesc *d_combo = reinterpret_cast<ComboDesc *>(scratch + P.off_combo);
  ck(cudaMemcpyAsync(d_desc, hd.data(), sizeof(ReplayDesc) * n_replays, cudaMemcpyHostToDevice, stream));
  ck(cudaMemcpyAsync(d_order, order.data(), sizeof(uint32_t) * order.size(), cudaMemcpyHostToDevice, stream));
  if (!P.combos.empty()) {
    ck(cudaMemcpyAsync(d_combo, hc.data(), sizeof(ComboDesc) * P.combos.size(), cudaMemcpyHostToDevice, stream));
    hazard_lut_kernel<<<(unsigned)P.combos.size(), 256, 0, stream>>>(d_combo);
    count_launches(1);
    uint32_t max_s = 0;
    for (auto &c : hc) max_s = std::max(max_s, c.n_sessions);
    {
      ProfSpan span(profile ? "key_stream" : "", stream);
      // one grid row per combination; a grid has at most 65,535 rows
      constexpr size_t kRows = 65535;
      for (size_t c0 = 0; c0 < P.combos.size(); c0 += kRows) {
        const unsigned rows = (unsigned)std::min(kRows, P.combos.size() - c0);
        key_stream_kernel<<<dim3((max_s + 127) / 128, rows), 128, 0, stream>>>(d_combo + c0);
        count_launches(1);
      }
    }
    ck(cudaGetLastError());
  }
  {
    ProfSpan span(profile ? "replay" : "", stream);
    // one launch per non-empty group, in the order of `order`
    struct Launch {
      ReplayKernel k;
      size_t n, smem;
    };
    const Launch all[] = {
        {st_kernel(P, logged), P.in_st.size(), P.max_smem_st},
        {replay_kernel<false, kKeyStream, -1, false>, P.in_mix.size(), P.max_smem_mix},
        {replay_kernel<true, kKeyStream, UNISON_SPEAR_TIDE, false>, P.in_gst.size(), 0},
        {replay_kernel<true, kKeyStream, -1, false>, P.in_gmix.size(), 0},
        {replay_kernel<false, kKeyOnline, -1, false>, P.in_online.size(), P.max_smem_online},
        {replay_kernel<false, kKeyStale, -1, false>, P.in_stale.size(), P.max_smem_stale}};
    std::vector<Launch> ls;
    std::vector<size_t> first;
    size_t off = 0;
    for (const Launch &l : all) {
      if (l.n) {
        ls.push_back(l);
        first.push_back(off);
      }
      off += l.n;
    }
    // the first group runs on the caller's stream, the others on side
    // streams forked from it and joined back before the TTFT medians
    std::unique_lock<std::mutex> hold;
    SideStreams *side = nullptr;
    if (ls.size() > 1) {
      side = side_streams(hold);
      if (!side) rc = UNISON_ERR_CUDA;
      if (side) ck(cudaEventRecord(side->fork, stream));
    }
    for (size_t i = 0; i < ls.size() && rc == UNISON_OK; i++) {
      cudaStream_t s = i == 0 ? stream : side->s[i - 1];
      if (i > 0) ck(cudaStreamWaitEvent(s, side->fork, 0));
      if (ls[i].smem) ck(cudaFuncSetAttribute(ls[i].k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ls[i].smem));
      ls[i].k<<<(unsigned)ls[i].n, 32, ls[i].smem, s>>>(d_desc, d_order + first[i]);
      count_launches(1);
      ck(cudaGetLastError());
      if (i > 0) {
        ck(cudaEventRecord(side->join[i - 1], s));
        ck(cudaStreamWaitEvent(stream, side->join[i - 1], 0));
      }
    }
  }
  {
    ProfSpan span(profile ? "ttft_median" : "", stream);
    ttft_median_kernel<<<(unsigned)n_replays, 256, 0, stream>>>(d_desc, (uint32_t)n_replays);
  }
  count_launches(1);
  ck(cudaGetLastError());
  return rc;
}

int check_batch(const unison_trace *const *traces, int n_traces, const unison_replay_params *params, int n_replays,
                int &dev, size_t &smem_limit) {
  if (!traces || n_traces <= 0 || !params || n_replays < 0) return UNISON_ERR_ARG;
  if (cudaGetDevice(&dev) != cudaSuccess) return UNISON_ERR_CUDA;
  for (int i = 0; i < n_traces; i++)
    if (!traces[i] || !traces[i]->d_block || traces[i]->device != dev) return UNISON_ERR_ARG;
  for (int r = 0; r < n_replays; r++) {
    const int rc = check_params(params[r], n_traces);
    if (rc != UNISON_OK) return rc;
  }
  int smem_optin = 0;
  cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  smem_limit = (size_t)smem_optin > 1024 ? (size_t)smem_optin - 1024 : 0;
  return UNISON_OK;
}

}  // namespace

extern "C" int unison_replay_batch(const unison_trace *const *traces, int n_traces,
                                   const unison_replay_params *params, int n_replays,
                                   unison_replay_result *results_dev, unison_replay_result *results_host,
                                   unison_decision *log_dev, uint64_t log_capacity_per_replay, void *cuda_stream) {
  int dev = 0;
  size_t smem_limit = 0;
  int rc = check_batch(traces, n_traces, params, n_replays, dev, smem_limit);
  if (rc != UNISON_OK) return rc;
  if (n_replays == 0) return UNISON_OK;
  if (!results_dev && !results_host) return UNISON_ERR_ARG;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  ReplayPlan P;
  size_t off_res = 0;
  rc = plan_replays(traces, params, n_replays, smem_limit, results_dev == nullptr, P, off_res);
  if (rc != UNISON_OK) return rc;
  char *scratch = nullptr;
  if (unison_fault_alloc() || cudaMallocAsync(reinterpret_cast<void **>(&scratch), P.bytes, stream) != cudaSuccess) {
    cudaGetLastError();
    return UNISON_ERR_OOM;
  }
  unison_replay_result *res = results_dev ? results_dev : reinterpret_cast<unison_replay_result *>(scratch + off_res);
  std::vector<ComboDesc> hc;
  std::vector<ReplayDesc> hd;
  std::vector<uint32_t> order;
  fill_descs(traces, params, n_replays, P, scratch, res, log_dev, log_capacity_per_replay, hc, hd, order);
  rc = launch_replays(P, scratch, hc, hd, order, n_replays, stream, true, log_dev != nullptr);
  if (results_host &&
      cudaMemcpyAsync(results_host, res, sizeof(unison_replay_result) * n_replays, cudaMemcpyDeviceToHost, stream) !=
          cudaSuccess &&
      rc == UNISON_OK)
    rc = UNISON_ERR_CUDA;
  if (cudaFreeAsync(scratch, stream) != cudaSuccess && rc == UNISON_OK) rc = UNISON_ERR_CUDA;
  if (results_host && cudaStreamSynchronize(stream) != cudaSuccess && rc == UNISON_OK) rc = UNISON_ERR_CUDA;
  return rc;
}

extern "C" int unison_stats(const unison_replay_result *r, const unison_replay_params *p, unison_stats_t *out) {
  if (!r || !p || !out) return UNISON_ERR_ARG;
  const double R = (double)r->req_warm;
  out->hit_rate = R > 0 ? (double)(r->hit_s + r->hit_h) / R : 0.0;
  const long double amat = (long double)p->t_s_ps_per_tok * r->tok_hit_s +
                           (long double)p->t_h_ps_per_tok * r->tok_hit_h +
                           (long double)p->t_p_ps_per_tok * r->tok_miss;
  out->amat_ps = R > 0 ? (double)(amat / R) : 0.0;
  out->prered = r->tok_needed ? 1.0 - (double)r->tok_computed / (double)r->tok_needed : 0.0;
  out->prefetch_acc = r->promote ? (double)r->promoted_then_hit_s / (double)r->promote : 0.0;
  const long double sum = (long double)r->ttft_sum_hi * 18446744073709551616.0L + (long double)r->ttft_sum_lo;
  out->ttft_mean_ns = r->ttft_n ? (double)(sum / r->ttft_n) : 0.0;
  out->ttft_p50_ns = (double)r->ttft_p50_ns;
  return UNISON_OK;
}

// Eq. (ase), accumulated as a mean of logarithms (many datasets would
// underflow a plain product).
extern "C" int unison_ase(const unison_stats_t *stats, int n_configs, int n_datasets, double *ase_out) {
  if (!stats || !ase_out || n_configs < 1 || n_datasets < 1) return UNISON_ERR_ARG;
  const size_t nc = (size_t)n_configs, nd = (size_t)n_datasets;
  for (size_t i = 0; i < nc * nd; i++) {
    const unison_stats_t &x = stats[i];
    if (!std::isfinite(x.hit_rate) || !std::isfinite(x.amat_ps) || !std::isfinite(x.ttft_mean_ns) ||
        x.hit_rate < 0 || x.amat_ps < 0 || x.ttft_mean_ns < 0)
      return UNISON_ERR_RANGE;
  }
  std::vector<double> logsum(nc, 0.0);
  std::vector<char> zero(nc, 0);
  for (size_t d = 0; d < nd; d++) {
    double hr_max = 0.0, amat_min = INFINITY, ttft_min = INFINITY;
    for (size_t c = 0; c < nc; c++) {
      const unison_stats_t &x = stats[c * nd + d];
      hr_max = std::max(hr_max, x.hit_rate);
      amat_min = std::min(amat_min, x.amat_ps);
      ttft_min = std::min(ttft_min, x.ttft_mean_ns);
    }
    // factor num/den of one metric: 0/0 counts as 1, 0/positive as 0
    auto factor = [&](size_t c, double num, double den) {
      if (den == 0.0) return;  // then num == 0 as well (num <= den): 1
      if (num == 0.0) {
        zero[c] = 1;
        return;
      }
      logsum[c] += std::log(num / den);
    };
    for (size_t c = 0; c < nc; c++) {
      const unison_stats_t &x = stats[c * nd + d];
      factor(c, x.hit_rate, hr_max);
      factor(c, amat_min, x.amat_ps);
      factor(c, ttft_min, x.ttft_mean_ns);
    }
  }
  for (size_t c = 0; c < nc; c++) ase_out[c] = zero[c] ? 0.0 : std::exp(logsum[c] / (3.0 * (double)nd));
  return UNISON_OK;
}

// Eq. (attainment) over windows of observed sessions.  Every event's window
// comes from the trace's host event array (a final completion has the edge
// flag); each log then adds its warm requests, and hits, to their windows.
extern "C" int unison_attainment(const unison_trace *trace, const unison_decision *log_online, uint64_t len_online,
                                 const unison_decision *log_offline, uint64_t len_offline,
                                 const unison_decision *log_lru, uint64_t len_lru, uint32_t n_points,
                                 unison_attainment_point *out) {
  if (!trace || !trace->h_block || !out || (len_online && !log_online) || (len_offline && !log_offline) ||
      (len_lru && !log_lru))
    return UNISON_ERR_ARG;
  const uint64_t N = trace->n_sessions, E = trace->n_events;
  if (n_points == 0 || n_points > N) return UNISON_ERR_RANGE;
  const uint4 *ev = trace->h<uint4>(trace->off_ev);
  std::vector<uint32_t> window(E);
  uint64_t seen = 0;
  uint32_t j = 0;  // windows only advance: seen grows with the event index
  for (uint64_t e = 0; e < E; e++) {
    while (j + 1 < n_points && (uint64_t)(j + 1) * N / n_points <= seen) j++;
    window[e] = j;
    const uint32_t w1 = ev[e].y;
    if (!(w1 & kEvArrival) && (w1 & kEvEdge)) seen++;
  }
  const unison_decision *logs[3] = {log_online, log_offline, log_lru};
  const uint64_t lens[3] = {len_online, len_offline, len_lru};
  std::vector<uint64_t> warm(3 * (size_t)n_points, 0), hits(3 * (size_t)n_points, 0);
  for (int r = 0; r < 3; r++)
    for (uint64_t i = 0; i < lens[r]; i++) {
      const unison_decision &d = logs[r][i];
      const uint32_t kind = d.kind_session >> 24;
      if (d.event >= E) return UNISON_ERR_FORMAT;
      if (kind == UNISON_KIND_HIT_S || kind == UNISON_KIND_HIT_H || kind == UNISON_KIND_MISS) {
        const size_t w = (size_t)r * n_points + window[d.event];
        warm[w]++;
        hits[w] += kind != UNISON_KIND_MISS;
      }
    }
  for (uint32_t k = 0; k < n_points; k++) {
    const uint64_t n = warm[k];
    if (warm[n_points + k] != n || warm[2 * (size_t)n_points + k] != n) return UNISON_ERR_FORMAT;
    unison_attainment_point &o = out[k];
    o.sessions_seen = (uint32_t)((uint64_t)k * N / n_points);
    o.reserved = 0;
    o.warm = n;
    o.hr_online = n ? (double)hits[k] / (double)n : NAN;
    o.hr_offline = n ? (double)hits[n_points + k] / (double)n : NAN;
    o.hr_lru = n ? (double)hits[2 * (size_t)n_points + k] / (double)n : NAN;
    o.attainment = (n && o.hr_offline != o.hr_lru) ? (o.hr_online - o.hr_lru) / (o.hr_offline - o.hr_lru) : NAN;
  }
  return UNISON_OK;
}

// ---------------------------------------------------------------------------
// Replay without device allocation.
//
// The scratch this entry point needs (descriptors, hazard tables, key
// streams, TTFT values, global resident lists) lives in one file-scope device
// array instead of memory from cudaMallocAsync.  Host code must not use the
// array's name as an address: for host code it names a host-side shadow, so
// its device address is fetched with cudaGetSymbolAddress once per device
// (with that device current) and passed to the kernels.
// ---------------------------------------------------------------------------
static __device__ __align__(256) unsigned char g_unison_noalloc_scratch[UNISON_NOALLOC_SCRATCH_BYTES];

namespace {
constexpr int kNoAllocMaxDevices = 64;
std::mutex g_noalloc_mu;
char *g_noalloc_addr[kNoAllocMaxDevices] = {};

// Device address of the scratch array on the current device.
int noalloc_scratch_address(char **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return UNISON_ERR_CUDA;
  }
  if (dev < 0 || dev >= kNoAllocMaxDevices) return UNISON_ERR_ARG;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_addr[dev]) {
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_unison_noalloc_scratch);
    if (e != cudaSuccess || p == nullptr) {
      cudaGetLastError();
      return UNISON_ERR_CUDA;
    }
    g_noalloc_addr[dev] = static_cast<char *>(p);
  }
  *out = g_noalloc_addr[dev];
  return UNISON_OK;
}
}  // namespace

extern "C" int unison_replay_batch_noalloc(const unison_trace *const *traces, int n_traces,
                                           const unison_replay_params *params, int n_replays,
                                           unison_replay_result *results_dev, unison_replay_result *results_host,
                                           unison_decision *log_dev, uint64_t log_capacity_per_replay,
                                           void *cuda_stream) {
  int dev = 0;
  size_t smem_limit = 0;
  int rc = check_batch(traces, n_traces, params, n_replays, dev, smem_limit);
  if (rc != UNISON_OK) return rc;
  if (n_replays == 0) return UNISON_OK;
  if (!results_dev) return UNISON_ERR_ARG;  // the caller provides the output buffer
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  char *scratch = nullptr;
  rc = noalloc_scratch_address(&scratch);
  if (rc != UNISON_OK) return rc;
  ReplayPlan P;
  size_t off_res = 0;
  rc = plan_replays(traces, params, n_replays, smem_limit, false, P, off_res);
  if (rc != UNISON_OK) return rc;
  if (P.bytes > UNISON_NOALLOC_SCRATCH_BYTES) return UNISON_ERR_RANGE;  // batch too large for the fixed scratch
  // Every scratch region is written before it is read within one call (the
  // descriptors by the copies in launch_replays, the tables and streams by
  // their kernels, TTFT values and lists by the event loop), so nothing left
  // by an earlier call is ever read and no region needs clearing.
  std::vector<ComboDesc> hc;
  std::vector<ReplayDesc> hd;
  std::vector<uint32_t> order;
  fill_descs(traces, params, n_replays, P, scratch, results_dev, log_dev, log_capacity_per_replay, hc, hd, order);
  rc = launch_replays(P, scratch, hc, hd, order, n_replays, stream, false, log_dev != nullptr);
  if (results_host) {
    if (cudaMemcpyAsync(results_host, results_dev, sizeof(unison_replay_result) * n_replays, cudaMemcpyDeviceToHost,
                        stream) != cudaSuccess &&
        rc == UNISON_OK)
      rc = UNISON_ERR_CUDA;
    if (cudaStreamSynchronize(stream) != cudaSuccess && rc == UNISON_OK) rc = UNISON_ERR_CUDA;
  }
  return rc;
}
