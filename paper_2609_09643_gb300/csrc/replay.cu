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
//   replay_kernel       Algorithm 1: one warp per replay, resident sessions of
//                       each tier held structure-of-arrays in shared memory,
//                       every decision a warp-wide scan + shuffle/redux argmax
//                       (or argmin) over the packed 64-bit keys.
//   ttft_median_kernel  Sec. V-A TTFT p50: radix select of the lower median
//                       over each replay's per-request TTFT values.
#include <algorithm>
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
constexpr uint32_t kAuxPinned = 1u, kAuxPromoted = 2u;
constexpr uint16_t kMapNone = 0xFFFFu;
constexpr uint32_t kEntryBytes = 20;  // hi, lo, size, aux, ret (u32 each)

struct ComboDesc {
  const uint32_t *turn_ev;   // [2T]
  const uint32_t *turn_t;    // [2T]
  const uint32_t *turn_off;  // [S+1]
  const uint32_t *tps;       // [S]
  uint32_t n_sessions, n_events;
  uint32_t ema_num, ema_den, bucket, pad;
  uint64_t penalty_q;
  uint16_t *sigma;  // [51]
  uint64_t *t2;     // [51]
  uint64_t *pkey;   // [E]
  uint32_t *gq;     // [E]
};

struct ReplayDesc {
  const uint4 *ev;
  const uint32_t *prev_out;
  const uint32_t *nref;
  const uint64_t *pkey;  // key stream (SPEAR policies) or null
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
  uint32_t rcap_s, rcap_h, use_map, pad;
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
  __shared__ uint32_t sig[kLutN];
  __shared__ unsigned long long t2[kLutN];
  for (uint32_t i = threadIdx.x; i < kLutN; i += blockDim.x) {
    sig[i] = c.sigma[i];
    t2[i] = c.t2[i];
  }
  __syncthreads();
  const uint32_t s = blockIdx.x * blockDim.x + threadIdx.x;
  if (s >= c.n_sessions) return;
  const uint32_t b = c.turn_off[s], ts = c.tps[s];
  const uint64_t a_num = c.ema_num, a_rest = c.ema_den - c.ema_num, a_den = c.ema_den;
  uint64_t g = 0;
  uint32_t prev_c = 0;
  for (uint32_t k = 0; k < ts; k++) {
    const uint32_t ti = b + k;
    const uint32_t ta = c.turn_t[2 * ti], tc = c.turn_t[2 * ti + 1];
    if (k) {
      const uint64_t gap = (uint32_t)(ta - prev_c);
      g = (a_num * gap + a_rest * g) / a_den;
    }
    prev_c = tc;
    const uint32_t t = k < kTMax ? k : kTMax;
    const uint64_t key = (g * kLambda) / sig[t] + t2[t];
    const uint64_t pk = pack_key(key, s);
    const uint32_t ea = c.turn_ev[2 * ti], ec = c.turn_ev[2 * ti + 1];
    c.pkey[ea] = pk;
    c.gq[ea] = (uint32_t)g;
    c.pkey[ec] = (k + 1 == ts) ? pack_key(kKeyMax40, s) : pk;
    c.gq[ec] = (uint32_t)g;
  }
}

// --------------------------------------------------------------------------
// Resident lists: one per tier, structure of arrays, unordered (removal
// swaps in the last entry).  All list state is warp-uniform; lane 0 writes.
// --------------------------------------------------------------------------
struct TierList {
  uint32_t *hi, *lo, *size, *aux, *ret;
  uint32_t n, cap;
  uint64_t used, pinned;  // tokens resident / tokens of pinned residents
};

struct Pick {
  int slot;
  uint64_t pk;
};

__device__ __forceinline__ uint64_t entry_key(const TierList &L, uint32_t i) {
  return ((uint64_t)L.hi[i] << 32) | L.lo[i];
}

// Most evictable unpinned entry (largest packed key); slot -1 if none.
__device__ __forceinline__ Pick argmax_unpinned(const TierList &L, int lane) {
  uint64_t best = 0;
  int bi = -1;
  for (uint32_t i = lane; i < L.n; i += 32) {
    const uint32_t a = L.aux[i];
    const uint64_t k = entry_key(L, i);
    if (!(a & kAuxPinned) && k > best) {
      best = k;
      bi = (int)i;
    }
  }
  const uint32_t h = (uint32_t)(best >> 32);
  const uint32_t mh = __reduce_max_sync(kFull, h);
  const uint32_t l = (h == mh) ? (uint32_t)best : 0u;
  const uint32_t ml = __reduce_max_sync(kFull, l);
  const uint64_t m = ((uint64_t)mh << 32) | ml;
  Pick p{-1, 0};
  if (m == 0) return p;  // valid packed keys are never 0 (inverted id >= 1)
  const uint32_t who = __ballot_sync(kFull, bi >= 0 && best == m);
  p.slot = __shfl_sync(kFull, bi, __ffs(who) - 1);
  p.pk = m;
  return p;
}

// Least evictable unpinned entry (smallest packed key); slot -1 if none.
__device__ __forceinline__ Pick argmin_unpinned(const TierList &L, int lane) {
  uint64_t best = ~0ull;
  int bi = -1;
  for (uint32_t i = lane; i < L.n; i += 32) {
    const uint32_t a = L.aux[i];
    const uint64_t k = entry_key(L, i);
    if (!(a & kAuxPinned) && (bi < 0 || k < best)) {
      best = k;
      bi = (int)i;
    }
  }
  Pick p{-1, 0};
  const uint32_t any = __ballot_sync(kFull, bi >= 0);
  if (!any) return p;
  const uint32_t h = bi >= 0 ? (uint32_t)(best >> 32) : kFull;
  const uint32_t mh = __reduce_min_sync(kFull, h);
  const uint32_t l = (bi >= 0 && h == mh) ? (uint32_t)best : kFull;
  const uint32_t ml = __reduce_min_sync(kFull, l);
  const uint64_t m = ((uint64_t)mh << 32) | ml;
  const uint32_t who = __ballot_sync(kFull, bi >= 0 && best == m);
  p.slot = __shfl_sync(kFull, bi, __ffs(who) - 1);
  p.pk = m;
  return p;
}

struct ReplayState {
  TierList S, H;
  uint16_t *map;  // session -> (tier bit 15 | slot), or null
  unison_decision *log;
  uint64_t log_cap;
  uint32_t e;  // current event index
  int status;
  uint32_t pinned_cnt;
  // counters
  unison_replay_result c;
};

__device__ __forceinline__ void log_dec(ReplayState &st, uint32_t kind, uint32_t s, int lane) {
  const uint64_t w = ((uint64_t)st.e << 32) | ((uint64_t)kind << 24) | s;
  st.c.decision_hash = (st.c.decision_hash ^ w) * kFnvPrime;
  if (st.log) {
    if (st.c.log_len < st.log_cap) {
      if (lane == 0) {
        unison_decision d;
        d.event = st.e;
        d.kind_session = (kind << 24) | s;
        st.log[st.c.log_len] = d;
      }
    } else if (st.status == UNISON_OK) {
      st.status = UNISON_ERR_LOG_FULL;
    }
  }
  st.c.log_len++;
}

__device__ __forceinline__ bool tl_append(ReplayState &st, TierList &L, uint32_t tier, uint64_t pk, uint32_t size,
                                          uint32_t aux, uint32_t ret, int lane) {
  if (L.n >= L.cap) {
    st.status = UNISON_ERR_CAPACITY;
    return false;
  }
  const uint32_t i = L.n;
  if (lane == 0) {
    L.hi[i] = (uint32_t)(pk >> 32);
    L.lo[i] = (uint32_t)pk;
    L.size[i] = size;
    L.aux[i] = aux;
    L.ret[i] = ret;
    if (st.map) st.map[packed_id(pk)] = (uint16_t)((tier == kTierH ? 0x8000u : 0u) | i);
  }
  L.n++;
  L.used += size;
  if (aux & kAuxPinned) L.pinned += size;
  __syncwarp();
  return true;
}

__device__ __forceinline__ void tl_remove(ReplayState &st, TierList &L, uint32_t tier, uint32_t i, int lane) {
  const uint32_t last = L.n - 1;
  const uint32_t sz = L.size[i], ax = L.aux[i], lo = L.lo[i];
  const uint32_t lhi = L.hi[last], llo = L.lo[last], lsz = L.size[last], lax = L.aux[last], lret = L.ret[last];
  __syncwarp();
  if (lane == 0) {
    if (i != last) {
      L.hi[i] = lhi;
      L.lo[i] = llo;
      L.size[i] = lsz;
      L.aux[i] = lax;
      L.ret[i] = lret;
      if (st.map) st.map[(~llo) & kIdMask] = (uint16_t)((tier == kTierH ? 0x8000u : 0u) | i);
    }
    if (st.map) st.map[(~lo) & kIdMask] = kMapNone;
  }
  L.n = last;
  L.used -= sz;
  if (ax & kAuxPinned) L.pinned -= sz;
  __syncwarp();
}

// Where session s is resident: tier (0 none) and slot.
__device__ __forceinline__ void locate(const ReplayState &st, uint32_t s, uint32_t &tier, uint32_t &slot, int lane) {
  if (st.map) {
    const uint16_t v = st.map[s];
    if (v == kMapNone) {
      tier = kTierNone;
      slot = 0;
    } else {
      tier = (v & 0x8000u) ? kTierH : kTierS;
      slot = v & 0x7FFFu;
    }
    return;
  }
  const uint32_t want = (~s) & kIdMask;
  int mine = -1;
  for (uint32_t i = lane; i < st.S.n; i += 32)
    if ((st.S.lo[i] & kIdMask) == want) mine = (int)i;
  uint32_t b = __ballot_sync(kFull, mine >= 0);
  if (b) {
    tier = kTierS;
    slot = (uint32_t)__shfl_sync(kFull, mine, __ffs(b) - 1);
    return;
  }
  for (uint32_t i = lane; i < st.H.n; i += 32)
    if ((st.H.lo[i] & kIdMask) == want) mine = (int)i;
  b = __ballot_sync(kFull, mine >= 0);
  if (b) {
    tier = kTierH;
    slot = (uint32_t)__shfl_sync(kFull, mine, __ffs(b) - 1);
    return;
  }
  tier = kTierNone;
  slot = 0;
}

// Evict entry `slot` of a tier (log EVICT / EXPIRE).
__device__ __forceinline__ void evict_entry(ReplayState &st, TierList &L, uint32_t tier, uint32_t slot, uint32_t kind,
                                            int lane) {
  const uint32_t id = (~L.lo[slot]) & kIdMask;
  tl_remove(st, L, tier, slot, lane);
  log_dec(st, kind, id, lane);
  if (kind == UNISON_KIND_EXPIRE)
    st.c.expire++;
  else
    st.c.evict++;
}

// A session demoted out of the fast tier enters HBM, displacing the most
// evictable unpinned HBM sessions, or is dropped when it is itself the most
// evictable of (unpinned HBM) + {itself}.
__device__ __forceinline__ bool admit_demoted(ReplayState &st, const ReplayDesc &D, uint64_t pk, uint32_t size,
                                              uint32_t aux, uint32_t ret, int lane) {
  const uint32_t id = packed_id(pk);
  if (st.H.pinned > D.cap_h || size > D.cap_h - st.H.pinned) {
    log_dec(st, UNISON_KIND_EVICT, id, lane);
    st.c.evict++;
    return true;
  }
  while (st.H.used + size > D.cap_h) {
    const Pick v = argmax_unpinned(st.H, lane);
    if (v.slot < 0 || pk > v.pk) {
      log_dec(st, UNISON_KIND_EVICT, id, lane);
      st.c.evict++;
      return true;
    }
    evict_entry(st, st.H, kTierH, (uint32_t)v.slot, UNISON_KIND_EVICT, lane);
  }
  if (!tl_append(st, st.H, kTierH, pk, size, aux, ret, lane)) return false;
  log_dec(st, UNISON_KIND_DEMOTE, id, lane);
  st.c.demote++;
  return true;
}

// Placement of the arriving (pinned) session s with n tokens.
__device__ __forceinline__ bool place(ReplayState &st, const ReplayDesc &D, uint32_t s, uint64_t pk, uint32_t n,
                                      int lane) {
  if (D.max_sessions && st.pinned_cnt >= D.max_sessions) {
    log_dec(st, UNISON_KIND_BYPASS, s, lane);
    st.c.bypass++;
    return true;
  }
  if (st.S.pinned <= D.cap_s && n <= D.cap_s - st.S.pinned) {
    while (st.S.used + n > D.cap_s) {
      const Pick d = argmax_unpinned(st.S, lane);
      if (d.slot < 0) {
        st.status = UNISON_ERR_CAPACITY;
        return false;
      }
      const uint32_t sd = st.S.size[d.slot], ad = st.S.aux[d.slot], rd = st.S.ret[d.slot];
      tl_remove(st, st.S, kTierS, (uint32_t)d.slot, lane);
      if (!admit_demoted(st, D, d.pk, sd, ad, rd, lane)) return false;
    }
    if (!tl_append(st, st.S, kTierS, pk, n, kAuxPinned, 0u, lane)) return false;
    log_dec(st, UNISON_KIND_PLACE_S, s, lane);
    st.c.place_s++;
  } else if (st.H.pinned <= D.cap_h && n <= D.cap_h - st.H.pinned) {
    while (st.H.used + n > D.cap_h) {
      const Pick v = argmax_unpinned(st.H, lane);
      if (v.slot < 0) {
        st.status = UNISON_ERR_CAPACITY;
        return false;
      }
      evict_entry(st, st.H, kTierH, (uint32_t)v.slot, UNISON_KIND_EVICT, lane);
    }
    if (!tl_append(st, st.H, kTierH, pk, n, kAuxPinned, 0u, lane)) return false;
    log_dec(st, UNISON_KIND_PLACE_H, s, lane);
    st.c.place_h++;
  } else {
    log_dec(st, UNISON_KIND_BYPASS, s, lane);
    st.c.bypass++;
    return true;
  }
  st.pinned_cnt++;
  if (D.max_sessions) {
    while (st.S.n + st.H.n > D.max_sessions) {
      const Pick a = argmax_unpinned(st.S, lane);
      const Pick b = argmax_unpinned(st.H, lane);
      if (a.slot < 0 && b.slot < 0) {
        st.status = UNISON_ERR_CAPACITY;
        return false;
      }
      if (b.slot < 0 || (a.slot >= 0 && a.pk > b.pk))
        evict_entry(st, st.S, kTierS, (uint32_t)a.slot, UNISON_KIND_EVICT, lane);
      else
        evict_entry(st, st.H, kTierH, (uint32_t)b.slot, UNISON_KIND_EVICT, lane);
    }
  }
  return true;
}

// Move entry `slot` from one tier list to the other, keeping its fields.
__device__ __forceinline__ bool move_entry(ReplayState &st, TierList &from, uint32_t from_tier, TierList &to,
                                           uint32_t to_tier, uint32_t slot, uint32_t aux_or, int lane) {
  const uint64_t pk = entry_key(from, slot);
  const uint32_t sz = from.size[slot], ax = from.aux[slot], rt = from.ret[slot];
  tl_remove(st, from, from_tier, slot, lane);
  return tl_append(st, to, to_tier, pk, sz, ax | aux_or, rt, lane);
}

// TIDE at a gap_start with budget bytes: promotions into free fast-tier space
// (least evictable HBM sessions first), then the pair loop of Algorithm 1.
__device__ __forceinline__ uint64_t tide(ReplayState &st, const ReplayDesc &D, uint64_t budget, int lane) {
  uint64_t rem = budget;
  const uint64_t kvb = D.kvb;
  for (;;) {
    const Pick p = argmin_unpinned(st.H, lane);
    if (p.slot < 0) break;
    const uint32_t sz = st.H.size[p.slot];
    const uint64_t by = (uint64_t)sz * kvb;
    if (by > rem || st.S.used + sz > D.cap_s) break;
    rem -= by;
    if (!move_entry(st, st.H, kTierH, st.S, kTierS, (uint32_t)p.slot, kAuxPromoted, lane)) return budget - rem;
    log_dec(st, UNISON_KIND_PROMOTE, packed_id(p.pk), lane);
    st.c.promote++;
  }
  for (;;) {
    const Pick p = argmin_unpinned(st.H, lane);
    const Pick d = argmax_unpinned(st.S, lane);
    if (p.slot < 0 || d.slot < 0) break;
    if (!(d.pk > p.pk)) break;  // the demoted session must be strictly more evictable
    const uint32_t sp = st.H.size[p.slot], sd = st.S.size[d.slot];
    const uint64_t by = ((uint64_t)sp + sd) * kvb;
    if (by > rem) break;
    if (st.S.used - sd + sp > D.cap_s) break;
    if (st.H.used - sp + sd > D.cap_h) break;
    rem -= by;
    if (!move_entry(st, st.H, kTierH, st.S, kTierS, (uint32_t)p.slot, kAuxPromoted, lane)) return budget - rem;
    // the promoted entry was appended at the end of S; d's slot is unchanged
    if (!move_entry(st, st.S, kTierS, st.H, kTierH, (uint32_t)d.slot, 0u, lane)) return budget - rem;
    log_dec(st, UNISON_KIND_PROMOTE, packed_id(p.pk), lane);
    log_dec(st, UNISON_KIND_TIDE_DEMOTE, packed_id(d.pk), lane);
    st.c.promote++;
    st.c.tide_demote++;
  }
  return budget - rem;
}

// Timeout: expire unpinned residents idle >= ttl, smallest session id first.
__device__ __forceinline__ void expire_idle(ReplayState &st, uint32_t now, uint32_t ttl, int lane) {
  for (;;) {
    uint32_t bid = kFull, bslot = 0, btier = 0;
    for (uint32_t i = lane; i < st.S.n; i += 32) {
      const uint32_t id = (~st.S.lo[i]) & kIdMask;
      if (!(st.S.aux[i] & kAuxPinned) && now - st.S.ret[i] >= ttl && id < bid) {
        bid = id;
        bslot = i;
        btier = kTierS;
      }
    }
    for (uint32_t i = lane; i < st.H.n; i += 32) {
      const uint32_t id = (~st.H.lo[i]) & kIdMask;
      if (!(st.H.aux[i] & kAuxPinned) && now - st.H.ret[i] >= ttl && id < bid) {
        bid = id;
        bslot = i;
        btier = kTierH;
      }
    }
    const uint32_t m = __reduce_min_sync(kFull, bid);
    if (m == kFull) return;
    const int src = __ffs(__ballot_sync(kFull, bid == m)) - 1;
    const uint32_t slot = __shfl_sync(kFull, bslot, src), tier = __shfl_sync(kFull, btier, src);
    if (tier == kTierS)
      evict_entry(st, st.S, kTierS, slot, UNISON_KIND_EXPIRE, lane);
    else
      evict_entry(st, st.H, kTierH, slot, UNISON_KIND_EXPIRE, lane);
  }
}

// Completion of a resident session's turn: unpin, refresh its key, stamp
// its last return time.
__device__ __forceinline__ void unpin(ReplayState &st, TierList &L, uint32_t slot, bool spear_keys, bool belady,
                                      uint64_t cu_pk, uint32_t j, uint32_t e, uint32_t s, uint32_t now, int lane) {
  const uint32_t ax = L.aux[slot], sz = L.size[slot];
  uint64_t pk = entry_key(L, slot);
  const uint64_t spk = __shfl_sync(kFull, cu_pk, j);
  if (spear_keys)
    pk = spk;
  else if (!belady)
    pk = pack_key(0xFFFFFFFFull - e, s);
  __syncwarp();
  if (lane == 0) {
    L.aux[slot] = ax & ~kAuxPinned;
    L.ret[slot] = now;
    L.hi[slot] = (uint32_t)(pk >> 32);
    L.lo[slot] = (uint32_t)pk;
  }
  if (ax & kAuxPinned) {
    L.pinned -= sz;
    st.pinned_cnt--;
  }
  __syncwarp();
}

__device__ __forceinline__ bool has_tide(uint32_t policy) {
  return policy == UNISON_SPEAR_TIDE || policy == UNISON_LRU_TIDE;
}

template <bool kGlobalLists>
__global__ void __launch_bounds__(32) replay_kernel(const ReplayDesc *descs, const uint32_t *order) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int lane = threadIdx.x & 31;
  const ReplayDesc D = descs[order[blockIdx.x]];

  ReplayState st;
  unsigned char *base = kGlobalLists ? reinterpret_cast<unsigned char *>(D.glist) : smem;
  {
    uint32_t *p = reinterpret_cast<uint32_t *>(base);
    const uint32_t cs = D.rcap_s, ch = D.rcap_h;
    st.S.hi = p; p += cs;
    st.S.lo = p; p += cs;
    st.S.size = p; p += cs;
    st.S.aux = p; p += cs;
    st.S.ret = p; p += cs;
    st.H.hi = p; p += ch;
    st.H.lo = p; p += ch;
    st.H.size = p; p += ch;
    st.H.aux = p; p += ch;
    st.H.ret = p; p += ch;
    st.map = D.use_map ? reinterpret_cast<uint16_t *>(p) : nullptr;
    st.S.n = st.H.n = 0;
    st.S.cap = cs;
    st.H.cap = ch;
    st.S.used = st.S.pinned = st.H.used = st.H.pinned = 0;
  }
  if (st.map) {
    for (uint32_t i = lane; i < D.n_sessions; i += 32) st.map[i] = kMapNone;
    __syncwarp();
  }
  st.log = D.log;
  st.log_cap = D.log_cap;
  st.status = UNISON_OK;
  st.pinned_cnt = 0;
  {
    unison_replay_result z = {};
    st.c = z;
  }
  st.c.decision_hash = kFnvOffset;

  const uint32_t policy = D.policy;
  const bool spear_keys = policy == UNISON_SPEAR || policy == UNISON_SPEAR_TIDE;
  const bool tide_on = has_tide(policy);
  const bool belady = policy == UNISON_BELADY;
  const bool timeout = policy == UNISON_TIMEOUT && D.ttl != 0xFFFFFFFFu;

  // TTFT queue (Sec. V-A): arrivals compressed by the load factor.
  uint64_t rel_us = 0, q_free = 0;
  uint32_t prev_now = 0, n_arr = 0;
  unsigned long long s_lo = 0, s_hi = 0;
  bool dma_busy = false;
  uint32_t busy_until = 0;

  // Event prefetch: lane i holds event base + i of the current batch.
  const uint32_t E = D.n_events;
  uint4 nx_ev = make_uint4(0, 0, 0, 0);
  uint32_t nx_prev = 0, nx_nref = kNoRef, nx_gq = 0;
  uint64_t nx_pk = 0;
  auto fetch = [&](uint32_t b) {
    const uint32_t i = b + lane;
    if (i < E) {
      nx_ev = __ldg(&D.ev[i]);
      nx_prev = __ldg(&D.prev_out[i]);
      if (belady) nx_nref = __ldg(&D.nref[i]);
      if (spear_keys) nx_pk = __ldg(&D.pkey[i]);
      if (tide_on) nx_gq = __ldg(&D.gq[i]);
    }
  };
  fetch(0);
  if (E) prev_now = __shfl_sync(kFull, nx_ev.x, 0);

  for (uint32_t b = 0; b < E && st.status != UNISON_ERR_CAPACITY; b += 32) {
    const uint4 cu_ev = nx_ev;
    const uint32_t cu_prev = nx_prev, cu_nref = nx_nref, cu_gq = nx_gq;
    const uint64_t cu_pk = nx_pk;
    if (b + 32 < E) fetch(b + 32);
    const uint32_t cnt = min(32u, E - b);
    for (uint32_t j = 0; j < cnt; j++) {
      const uint32_t e = b + j;
      const uint32_t now = __shfl_sync(kFull, cu_ev.x, j);
      const uint32_t w1 = __shfl_sync(kFull, cu_ev.y, j);
      const uint32_t s = w1 & kIdMask;
      const bool arrival = (w1 & kEvArrival) != 0;
      const bool edge = (w1 & kEvEdge) != 0;
      st.e = e;
      st.c.events++;
      rel_us += (uint32_t)(now - prev_now);
      prev_now = now;
      if (timeout) expire_idle(st, now, D.ttl, lane);
      if (dma_busy && (int32_t)(now - busy_until) >= 0) dma_busy = false;

      uint32_t tier, slot;
      locate(st, s, tier, slot, lane);
      if (arrival) {
        const uint32_t in = __shfl_sync(kFull, cu_ev.z, j);
        const uint32_t out = __shfl_sync(kFull, cu_ev.w, j);
        const uint32_t prev = __shfl_sync(kFull, cu_prev, j);
        uint64_t prefill;
        if (edge) {
          log_dec(st, UNISON_KIND_COLD, s, lane);
          st.c.cold++;
          prefill = in;
        } else {
          st.c.req_warm++;
          st.c.tok_needed += in;
          if (tier == kTierS) {
            log_dec(st, UNISON_KIND_HIT_S, s, lane);
            st.c.hit_s++;
            st.c.tok_hit_s += prev;
            prefill = in - prev;
            if (st.S.aux[slot] & kAuxPromoted) st.c.promoted_then_hit_s++;
          } else if (tier == kTierH) {
            log_dec(st, UNISON_KIND_HIT_H, s, lane);
            st.c.hit_h++;
            st.c.tok_hit_h += prev;
            prefill = in - prev;
          } else {
            log_dec(st, UNISON_KIND_MISS, s, lane);
            st.c.miss++;
            st.c.tok_miss += prev;
            prefill = in;
          }
          st.c.tok_computed += prefill;
        }
        {
          const uint64_t arr = rel_us * 1000ull / D.load;
          if (q_free < arr) q_free = arr;
          q_free += prefill * D.prefill_ns;
          const uint64_t v = q_free - arr;
          if (lane == 0 && n_arr < D.n_turns) D.ttft[n_arr] = v;
          n_arr++;
          const unsigned long long lo2 = s_lo + v;
          s_hi += (lo2 < s_lo);
          s_lo = lo2;
        }
        if (tier == kTierS)
          tl_remove(st, st.S, kTierS, slot, lane);
        else if (tier == kTierH)
          tl_remove(st, st.H, kTierH, slot, lane);
        uint64_t pk;
        if (spear_keys)
          pk = __shfl_sync(kFull, cu_pk, j);
        else if (belady) {
          const uint32_t nr = __shfl_sync(kFull, cu_nref, j);
          pk = pack_key(nr == kNoRef ? kKeyMax40 : (uint64_t)nr, s);
        } else
          pk = pack_key(0xFFFFFFFFull - e, s);
        if (!place(st, D, s, pk, out, lane)) break;
      } else {
        if (tier == kTierS)
          unpin(st, st.S, slot, spear_keys, belady, cu_pk, j, e, s, now, lane);
        else if (tier == kTierH)
          unpin(st, st.H, slot, spear_keys, belady, cu_pk, j, e, s, now, lane);
        if (!edge && tide_on && !dma_busy) {
          const uint64_t g = __shfl_sync(kFull, cu_gq, j);
          const uint64_t budget = g * D.dma;
          st.c.tide_calls++;
          const uint64_t moved = tide(st, D, budget, lane);
          st.c.dma_bytes += moved;
          if (moved > 0 && D.dma > 0) {
            dma_busy = true;
            busy_until = now + (uint32_t)((moved + D.dma - 1) / D.dma);
          }
          if (st.status == UNISON_ERR_CAPACITY) break;
        }
      }
    }
  }
  st.c.ttft_n = n_arr;
  st.c.ttft_sum_lo = s_lo;
  st.c.ttft_sum_hi = s_hi;
  st.c.ttft_p50_ns = 0;
  st.c.status = st.status;
  if (lane == 0) *D.result = st.c;
}

// Lower median (element floor((n-1)/2) in sorted order) by MSB-first radix select.
__global__ void __launch_bounds__(256) ttft_median_kernel(const ReplayDesc *descs, uint32_t n_replays) {
  const ReplayDesc &D = descs[blockIdx.x];
  __shared__ unsigned int hist[256];
  __shared__ unsigned long long red[8];
  __shared__ unsigned int sel_digit;
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
  uint64_t target = (n - 1) / 2, prefix = 0, mask = 0;
  for (int b = top; b >= 0; b--) {
    for (uint32_t i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (uint64_t i = threadIdx.x; i < n; i += blockDim.x) {
      const uint64_t x = v[i];
      if ((x & mask) == prefix) atomicAdd(&hist[(x >> (8 * b)) & 0xFF], 1u);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      uint64_t cum = 0;
      uint32_t d = 0;
      for (; d < 256; d++) {
        if (cum + hist[d] > target) break;
        cum += hist[d];
      }
      sel_digit = d < 256 ? d : 255;
      sel_target = target - cum;
    }
    __syncthreads();
    prefix |= (uint64_t)sel_digit << (8 * b);
    mask |= 0xFFull << (8 * b);
    target = sel_target;
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

extern "C" int unison_replay_batch(const unison_trace *const *traces, int n_traces,
                                   const unison_replay_params *params, int n_replays,
                                   unison_replay_result *results_dev, unison_replay_result *results_host,
                                   unison_decision *log_dev, uint64_t log_capacity_per_replay, void *cuda_stream) {
  if (!traces || n_traces <= 0 || !params || n_replays < 0) return UNISON_ERR_ARG;
  if (n_replays == 0) return UNISON_OK;
  if (!results_dev && !results_host) return UNISON_ERR_ARG;
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return UNISON_ERR_CUDA;
  for (int i = 0; i < n_traces; i++)
    if (!traces[i] || !traces[i]->d_block || traces[i]->device != dev) return UNISON_ERR_ARG;
  for (int r = 0; r < n_replays; r++) {
    const int rc = check_params(params[r], n_traces);
    if (rc != UNISON_OK) return rc;
  }
  int smem_optin = 0;
  cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  const size_t smem_limit = (size_t)smem_optin > 1024 ? (size_t)smem_optin - 1024 : 0;

  // Key streams: one per (trace, EMA weight, bucket, P_Z) used by a policy that needs them.
  std::map<std::tuple<uint32_t, uint32_t, uint32_t, uint32_t, uint64_t>, int> combo_of;
  std::vector<std::tuple<uint32_t, uint32_t, uint32_t, uint32_t, uint64_t>> combos;
  std::vector<int> replay_combo(n_replays, -1);
  for (int r = 0; r < n_replays; r++) {
    const unison_replay_params &p = params[r];
    if (!needs_stream(p.policy)) continue;
    auto key = std::make_tuple(p.trace_idx, p.ema_num, p.ema_den, p.hazard_bucket, p.penalty_q);
    auto it = combo_of.find(key);
    if (it == combo_of.end()) {
      it = combo_of.emplace(key, (int)combos.size()).first;
      combos.push_back(key);
    }
    replay_combo[r] = it->second;
  }

  // Scratch layout.
  size_t off = 0;
  const size_t off_desc = off;
  off = align_up(off + sizeof(ReplayDesc) * n_replays, 256);
  const size_t off_order = off;
  off = align_up(off + sizeof(uint32_t) * 2 * n_replays, 256);
  const size_t off_combo = off;
  off = align_up(off + sizeof(ComboDesc) * combos.size() + 1, 256);
  std::vector<size_t> off_lut(combos.size()), off_stream(combos.size());
  for (size_t c = 0; c < combos.size(); c++) {
    off_lut[c] = off;
    off = align_up(off + 128 + 51 * 8, 256);
    const uint64_t E = traces[std::get<0>(combos[c])]->n_events;
    off_stream[c] = off;
    off = align_up(off + 12 * E, 256);
  }
  std::vector<size_t> off_ttft(n_replays), off_glist(n_replays, 0);
  std::vector<uint32_t> rcap_s(n_replays), rcap_h(n_replays), use_map(n_replays), smem_bytes(n_replays);
  std::vector<uint32_t> in_smem, in_global;
  size_t max_smem = 0;
  for (int r = 0; r < n_replays; r++) {
    const unison_replay_params &p = params[r];
    const unison_trace *tr = traces[p.trace_idx];
    const uint64_t cs = p.cap_fast_bytes / p.kv_bytes_per_token, ch = p.cap_hbm_bytes / p.kv_bytes_per_token;
    const uint64_t mo = std::max<uint32_t>(tr->min_out_tok, 1);
    rcap_s[r] = (uint32_t)std::min<uint64_t>(tr->n_sessions, cs / mo) + 1;
    rcap_h[r] = (uint32_t)std::min<uint64_t>(tr->n_sessions, ch / mo) + 1;
    const size_t lists = (size_t)kEntryBytes * (rcap_s[r] + rcap_h[r]);
    const size_t map_b = align_up(2ull * tr->n_sessions, 16);
    const bool map_ok = rcap_s[r] <= 0x7FFF && rcap_h[r] <= 0x7FFF;
    if (map_ok && lists + map_b <= smem_limit && map_b <= 32768) {
      use_map[r] = 1;
      smem_bytes[r] = (uint32_t)(lists + map_b);
    } else {
      use_map[r] = 0;
      smem_bytes[r] = (uint32_t)lists;
    }
    if (smem_bytes[r] <= smem_limit) {
      in_smem.push_back((uint32_t)r);
      max_smem = std::max<size_t>(max_smem, smem_bytes[r]);
    } else {
      use_map[r] = 0;
      in_global.push_back((uint32_t)r);
      off_glist[r] = off;
      off = align_up(off + lists, 256);
    }
    off_ttft[r] = off;
    off = align_up(off + 8 * (tr->n_turns + 1), 256);
  }
  size_t off_res = 0;
  if (!results_dev) {
    off_res = off;
    off = align_up(off + sizeof(unison_replay_result) * n_replays, 256);
  }
  char *scratch = nullptr;
  if (cudaMallocAsync(reinterpret_cast<void **>(&scratch), off, stream) != cudaSuccess) {
    cudaGetLastError();
    return UNISON_ERR_OOM;
  }
  unison_replay_result *res = results_dev ? results_dev : reinterpret_cast<unison_replay_result *>(scratch + off_res);

  std::vector<ComboDesc> hc(combos.size());
  for (size_t c = 0; c < combos.size(); c++) {
    const unison_trace *tr = traces[std::get<0>(combos[c])];
    ComboDesc &d = hc[c];
    d.turn_ev = tr->d<uint32_t>(tr->off_turn_ev);
    d.turn_t = tr->d<uint32_t>(tr->off_turn_t);
    d.turn_off = tr->d<uint32_t>(tr->off_turn_off);
    d.tps = tr->d<uint32_t>(tr->off_tps);
    d.n_sessions = tr->n_sessions;
    d.n_events = (uint32_t)tr->n_events;
    d.ema_num = std::get<1>(combos[c]);
    d.ema_den = std::get<2>(combos[c]);
    d.bucket = std::get<3>(combos[c]);
    d.pad = 0;
    d.penalty_q = std::get<4>(combos[c]);
    d.sigma = reinterpret_cast<uint16_t *>(scratch + off_lut[c]);
    d.t2 = reinterpret_cast<uint64_t *>(scratch + off_lut[c] + 128);
    d.pkey = reinterpret_cast<uint64_t *>(scratch + off_stream[c]);
    d.gq = reinterpret_cast<uint32_t *>(scratch + off_stream[c] + 8 * tr->n_events);
  }
  std::vector<ReplayDesc> hd(n_replays);
  for (int r = 0; r < n_replays; r++) {
    const unison_replay_params &p = params[r];
    const unison_trace *tr = traces[p.trace_idx];
    ReplayDesc &d = hd[r];
    d.ev = tr->d<uint4>(tr->off_ev);
    d.prev_out = tr->d<uint32_t>(tr->off_prev_out);
    d.nref = tr->d<uint32_t>(tr->off_nref);
    d.pkey = replay_combo[r] >= 0 ? hc[replay_combo[r]].pkey : nullptr;
    d.gq = replay_combo[r] >= 0 ? hc[replay_combo[r]].gq : nullptr;
    d.ttft = reinterpret_cast<uint64_t *>(scratch + off_ttft[r]);
    d.glist = off_glist[r] ? reinterpret_cast<uint32_t *>(scratch + off_glist[r]) : nullptr;
    d.log = log_dev ? log_dev + (uint64_t)r * log_capacity_per_replay : nullptr;
    d.log_cap = log_dev ? log_capacity_per_replay : 0;
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
    d.rcap_s = rcap_s[r];
    d.rcap_h = rcap_h[r];
    d.use_map = use_map[r];
    d.pad = 0;
  }
  std::vector<uint32_t> order;
  order.insert(order.end(), in_smem.begin(), in_smem.end());
  order.insert(order.end(), in_global.begin(), in_global.end());

  int rc = UNISON_OK;
  auto ck = [&](cudaError_t e) {
    if (e != cudaSuccess && rc == UNISON_OK) rc = UNISON_ERR_CUDA;
  };
  ReplayDesc *d_desc = reinterpret_cast<ReplayDesc *>(scratch + off_desc);
  uint32_t *d_order = reinterpret_cast<uint32_t *>(scratch + off_order);
  ComboDesc *d_combo = reinterpret_cast<ComboDesc *>(scratch + off_combo);
  ck(cudaMemcpyAsync(d_desc, hd.data(), sizeof(ReplayDesc) * n_replays, cudaMemcpyHostToDevice, stream));
  ck(cudaMemcpyAsync(d_order, order.data(), sizeof(uint32_t) * order.size(), cudaMemcpyHostToDevice, stream));
  if (!combos.empty()) {
    ck(cudaMemcpyAsync(d_combo, hc.data(), sizeof(ComboDesc) * combos.size(), cudaMemcpyHostToDevice, stream));
    hazard_lut_kernel<<<(unsigned)combos.size(), 256, 0, stream>>>(d_combo);
    uint32_t max_s = 0;
    for (auto &c : hc) max_s = std::max(max_s, c.n_sessions);
    dim3 g((max_s + 127) / 128, (unsigned)combos.size());
    {
      ProfSpan span("key_stream", stream);
      key_stream_kernel<<<g, 128, 0, stream>>>(d_combo);
    }
    count_launches(2);
    ck(cudaGetLastError());
  }
  {
    ProfSpan span("replay", stream);
    if (!in_smem.empty()) {
      ck(cudaFuncSetAttribute(replay_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)max_smem));
      replay_kernel<false><<<(unsigned)in_smem.size(), 32, max_smem, stream>>>(d_desc, d_order);
      count_launches(1);
      ck(cudaGetLastError());
    }
    if (!in_global.empty()) {
      replay_kernel<true><<<(unsigned)in_global.size(), 32, 0, stream>>>(d_desc, d_order + in_smem.size());
      count_launches(1);
      ck(cudaGetLastError());
    }
  }
  {
    ProfSpan span("ttft_median", stream);
    ttft_median_kernel<<<(unsigned)n_replays, 256, 0, stream>>>(d_desc, (uint32_t)n_replays);
  }
  count_launches(1);
  ck(cudaGetLastError());
  if (results_host)
    ck(cudaMemcpyAsync(results_host, res, sizeof(unison_replay_result) * n_replays, cudaMemcpyDeviceToHost, stream));
  ck(cudaFreeAsync(scratch, stream));
  if (results_host) ck(cudaStreamSynchronize(stream));
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
  if (!traces || n_traces <= 0 || !params || n_replays < 0) return UNISON_ERR_ARG;
  if (n_replays == 0) return UNISON_OK;
  if (!results_dev) return UNISON_ERR_ARG;  // the caller provides the output buffer
  cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return UNISON_ERR_CUDA;
  for (int i = 0; i < n_traces; i++)
    if (!traces[i] || !traces[i]->d_block || traces[i]->device != dev) return UNISON_ERR_ARG;
  for (int r = 0; r < n_replays; r++) {
    const int rc = check_params(params[r], n_traces);
    if (rc != UNISON_OK) return rc;
  }
  char *scratch = nullptr;
  {
    const int rc = noalloc_scratch_address(&scratch);
    if (rc != UNISON_OK) return rc;
  }
  int smem_optin = 0;
  cudaDeviceGetAttribute(&smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  const size_t smem_limit = (size_t)smem_optin > 1024 ? (size_t)smem_optin - 1024 : 0;

  std::map<std::tuple<uint32_t, uint32_t, uint32_t, uint32_t, uint64_t>, int> combo_of;
  std::vector<std::tuple<uint32_t, uint32_t, uint32_t, uint32_t, uint64_t>> combos;
  std::vector<int> replay_combo(n_replays, -1);
  for (int r = 0; r < n_replays; r++) {
    const unison_replay_params &p = params[r];
    if (!needs_stream(p.policy)) continue;
    auto key = std::make_tuple(p.trace_idx, p.ema_num, p.ema_den, p.hazard_bucket, p.penalty_q);
    auto it = combo_of.find(key);
    if (it == combo_of.end()) {
      it = combo_of.emplace(key, (int)combos.size()).first;
      combos.push_back(key);
    }
    replay_combo[r] = it->second;
  }

  // Same layout as unison_replay_batch, without the results region.
  size_t off = 0;
  const size_t off_desc = off;
  off = align_up(off + sizeof(ReplayDesc) * n_replays, 256);
  const size_t off_order = off;
  off = align_up(off + sizeof(uint32_t) * 2 * n_replays, 256);
  const size_t off_combo = off;
  off = align_up(off + sizeof(ComboDesc) * combos.size() + 1, 256);
  std::vector<size_t> off_lut(combos.size()), off_stream(combos.size());
  for (size_t c = 0; c < combos.size(); c++) {
    off_lut[c] = off;
    off = align_up(off + 128 + 51 * 8, 256);
    const uint64_t E = traces[std::get<0>(combos[c])]->n_events;
    off_stream[c] = off;
    off = align_up(off + 12 * E, 256);
  }
  std::vector<size_t> off_ttft(n_replays), off_glist(n_replays, 0);
  std::vector<uint32_t> rcap_s(n_replays), rcap_h(n_replays), use_map(n_replays), smem_bytes(n_replays);
  std::vector<uint32_t> in_smem, in_global;
  size_t max_smem = 0;
  for (int r = 0; r < n_replays; r++) {
    const unison_replay_params &p = params[r];
    const unison_trace *tr = traces[p.trace_idx];
    const uint64_t cs = p.cap_fast_bytes / p.kv_bytes_per_token, ch = p.cap_hbm_bytes / p.kv_bytes_per_token;
    const uint64_t mo = std::max<uint32_t>(tr->min_out_tok, 1);
    rcap_s[r] = (uint32_t)std::min<uint64_t>(tr->n_sessions, cs / mo) + 1;
    rcap_h[r] = (uint32_t)std::min<uint64_t>(tr->n_sessions, ch / mo) + 1;
    const size_t lists = (size_t)kEntryBytes * (rcap_s[r] + rcap_h[r]);
    const size_t map_b = align_up(2ull * tr->n_sessions, 16);
    const bool map_ok = rcap_s[r] <= 0x7FFF && rcap_h[r] <= 0x7FFF;
    if (map_ok && lists + map_b <= smem_limit && map_b <= 32768) {
      use_map[r] = 1;
      smem_bytes[r] = (uint32_t)(lists + map_b);
    } else {
      use_map[r] = 0;
      smem_bytes[r] = (uint32_t)lists;
    }
    if (smem_bytes[r] <= smem_limit) {
      in_smem.push_back((uint32_t)r);
      max_smem = std::max<size_t>(max_smem, smem_bytes[r]);
    } else {
      use_map[r] = 0;
      in_global.push_back((uint32_t)r);
      off_glist[r] = off;
      off = align_up(off + lists, 256);
    }
    off_ttft[r] = off;
    off = align_up(off + 8 * (tr->n_turns + 1), 256);
  }
  if (off > UNISON_NOALLOC_SCRATCH_BYTES) return UNISON_ERR_RANGE;  // batch too large for the fixed scratch

  // Every scratch region is written before it is read within one call (the
  // descriptors by the copies below, the tables and streams by their kernels,
  // TTFT values and lists by the event loop), so nothing left by an earlier
  // call is ever read and no region needs clearing.
  std::vector<ComboDesc> hc(combos.size());
  for (size_t c = 0; c < combos.size(); c++) {
    const unison_trace *tr = traces[std::get<0>(combos[c])];
    ComboDesc &d = hc[c];
    d.turn_ev = tr->d<uint32_t>(tr->off_turn_ev);
    d.turn_t = tr->d<uint32_t>(tr->off_turn_t);
    d.turn_off = tr->d<uint32_t>(tr->off_turn_off);
    d.tps = tr->d<uint32_t>(tr->off_tps);
    d.n_sessions = tr->n_sessions;
    d.n_events = (uint32_t)tr->n_events;
    d.ema_num = std::get<1>(combos[c]);
    d.ema_den = std::get<2>(combos[c]);
    d.bucket = std::get<3>(combos[c]);
    d.pad = 0;
    d.penalty_q = std::get<4>(combos[c]);
    d.sigma = reinterpret_cast<uint16_t *>(scratch + off_lut[c]);
    d.t2 = reinterpret_cast<uint64_t *>(scratch + off_lut[c] + 128);
    d.pkey = reinterpret_cast<uint64_t *>(scratch + off_stream[c]);
    d.gq = reinterpret_cast<uint32_t *>(scratch + off_stream[c] + 8 * tr->n_events);
  }
  std::vector<ReplayDesc> hd(n_replays);
  for (int r = 0; r < n_replays; r++) {
    const unison_replay_params &p = params[r];
    const unison_trace *tr = traces[p.trace_idx];
    ReplayDesc &d = hd[r];
    d.ev = tr->d<uint4>(tr->off_ev);
    d.prev_out = tr->d<uint32_t>(tr->off_prev_out);
    d.nref = tr->d<uint32_t>(tr->off_nref);
    d.pkey = replay_combo[r] >= 0 ? hc[replay_combo[r]].pkey : nullptr;
    d.gq = replay_combo[r] >= 0 ? hc[replay_combo[r]].gq : nullptr;
    d.ttft = reinterpret_cast<uint64_t *>(scratch + off_ttft[r]);
    d.glist = off_glist[r] ? reinterpret_cast<uint32_t *>(scratch + off_glist[r]) : nullptr;
    d.log = log_dev ? log_dev + (uint64_t)r * log_capacity_per_replay : nullptr;
    d.log_cap = log_dev ? log_capacity_per_replay : 0;
    d.result = results_dev + r;
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
    d.rcap_s = rcap_s[r];
    d.rcap_h = rcap_h[r];
    d.use_map = use_map[r];
    d.pad = 0;
  }
  std::vector<uint32_t> order;
  order.insert(order.end(), in_smem.begin(), in_smem.end());
  order.insert(order.end(), in_global.begin(), in_global.end());

  int rc = UNISON_OK;
  auto ck = [&](cudaError_t e) {
    if (e != cudaSuccess && rc == UNISON_OK) rc = UNISON_ERR_CUDA;
  };
  ReplayDesc *d_desc = reinterpret_cast<ReplayDesc *>(scratch + off_desc);
  uint32_t *d_order = reinterpret_cast<uint32_t *>(scratch + off_order);
  ComboDesc *d_combo = reinterpret_cast<ComboDesc *>(scratch + off_combo);
  ck(cudaMemcpyAsync(d_desc, hd.data(), sizeof(ReplayDesc) * n_replays, cudaMemcpyHostToDevice, stream));
  ck(cudaMemcpyAsync(d_order, order.data(), sizeof(uint32_t) * order.size(), cudaMemcpyHostToDevice, stream));
  if (!combos.empty()) {
    ck(cudaMemcpyAsync(d_combo, hc.data(), sizeof(ComboDesc) * combos.size(), cudaMemcpyHostToDevice, stream));
    hazard_lut_kernel<<<(unsigned)combos.size(), 256, 0, stream>>>(d_combo);
    uint32_t max_s = 0;
    for (auto &c : hc) max_s = std::max(max_s, c.n_sessions);
    dim3 g((max_s + 127) / 128, (unsigned)combos.size());
    key_stream_kernel<<<g, 128, 0, stream>>>(d_combo);
    count_launches(2);
    ck(cudaGetLastError());
  }
  if (!in_smem.empty()) {
    ck(cudaFuncSetAttribute(replay_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)max_smem));
    replay_kernel<false><<<(unsigned)in_smem.size(), 32, max_smem, stream>>>(d_desc, d_order);
    count_launches(1);
    ck(cudaGetLastError());
  }
  if (!in_global.empty()) {
    replay_kernel<true><<<(unsigned)in_global.size(), 32, 0, stream>>>(d_desc, d_order + in_smem.size());
    count_launches(1);
    ck(cudaGetLastError());
  }
  ttft_median_kernel<<<(unsigned)n_replays, 256, 0, stream>>>(d_desc, (uint32_t)n_replays);
  count_launches(1);
  ck(cudaGetLastError());
  if (results_host) {
    ck(cudaMemcpyAsync(results_host, results_dev, sizeof(unison_replay_result) * n_replays, cudaMemcpyDeviceToHost,
                       stream));
    ck(cudaStreamSynchronize(stream));
  }
  return rc;
}
