/*
 * UNISON CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, single-threaded restatement of the paper's method
 * (UNISON, arXiv 2609.09643): the SPEAR survival-penalty score (Sec. III-B,
 * fixed point per Sec. IV-C), the TIDE idle-window fill (Sec. III-C) and the
 * joint event loop (Algorithm 1), replayed over one session trace, plus the
 * standalone ranking of a live set.  It exists so that tests and the
 * benchmark's CPU baseline can check the CUDA library against something a
 * reader can verify by eye.  Only tests/, __graft_entry__.smoke() and
 * bench.py's CPU-baseline leg may load it; the library never does, and the
 * two share no code, header, table or constant generator.
 *
 * Style: every decision is a linear scan, every ranking is recomputed from
 * the register file at the moment it is needed, and all arithmetic is
 * integer.  Times are absolute unsigned 64-bit microseconds.
 *
 * Readings of points the paper leaves open (each one named where used):
 *   R1  open-loop trace: arrivals and completions come from the trace.
 *   R2  event order: (time, COMPLETION before ARRIVAL, session id).
 *   R5  hazard LUT: 0-based turns, n(t)=#{T_s>=t+1}, d(t)=#{T_s=t+1},
 *       t=0..50, pooled over buckets of width w, h_q by exact integer
 *       rounding; indexed by the register turn min(t,50).
 *   R6  EMA weight a_num/a_den ((3,10) in the paper; window W -> (2,W+1)).
 *   R7  gap average starts at 0.
 *   R8  one total order "more evictable" = larger key, then smaller id.
 *   R9  placement: remove, then place S-first with a demote cascade into H,
 *       else H, else bypass.
 *   R10 request accounting (warm = turn >= 1).
 *   R11 TIDE budget in bytes = g_q(us) * dma bytes per us.
 *   R25 ASE: a metric ratio 0/0 counts as 1.
 *   R26 online hazard table (Sec. V-F): starts with no sessions; at the final
 *       completion of a session its turn count T_s is added and the table is
 *       rebuilt with the quantizer of R5; every later key uses it.
 *   R28 stale snapshot of a dual design (Sec. IV-B eq. stale, Tab. org): the
 *       ranking decisions (make-room victims, slot-limit evictions, TIDE's
 *       promotions and demotions) score every session from a copy of its
 *       register row (g_q, turn, done) taken at the last sync point, after
 *       that event's own decisions; residency, sizes and pins stay live.  Rows
 *       start at zero.  Sync points: every event, every m-th arrival, or
 *       every gap_start.  Vict!= (Prom!=) counts the acted-upon victim
 *       (promotion) choices whose session differs from the choice by the
 *       live rows over the same candidates.
 *   R29 signal leave-one-out (Sec. V-D, Fig. signal): without the gap
 *       recurrence signal the score sees g_q = 0; without the hazard signal
 *       it sees sigma_q = Lambda (zero hazard, so T2 = 0 as well).
 *   R27 attainment A(n) (eq. attainment): "after n observed sessions" is a
 *       window of the trace, the warm requests arriving while the online
 *       table holds n_j <= n < n_{j+1} sessions, n_j = floor(j N / P) for P
 *       points (the last window includes n = N); H is a replay's hit rate
 *       over that window.
 *   R12 a completed session stays resident with the maximal key.
 *   R13 DMA busy until now + ceil(moved / dma bytes per us).
 *   R14 TIDE phase 1 (promotion into free fast-tier space) then phase 2
 *       (the paper's promote/demote pair loop).
 *   R15 session-slot limit: evict the global most evictable resident.
 *   R16 Timeout: LRU order plus expiry of residents idle >= TTL.
 *   R17 TTFT: one FIFO prefill server, arrivals compressed by the load
 *       factor.
 *   R19 prefetch accuracy: promoted sessions whose next request hits the
 *       fast tier.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ---- constants of the locked format, eq. (lock): (b_h,b_g,b_s,tau,P_Z) -- */
#define OR_LAMBDA 4095u            /* Lambda_{b_h} = 2^12 - 1, eq. (uq)       */
#define OR_EPS_Q 41u               /* floor(0.01 * 4095 + 1/2), eq. (survq)   */
#define OR_T_MAX 50u               /* hazard table covers t = 0..50, eq. (hazard) */
#define OR_SCORE_MAX UINT64_MAX    /* 2^{b_s} - 1 for a completed session     */

enum { OR_LRU = 0, OR_TIMEOUT = 1, OR_SPEAR = 2, OR_SPEAR_TIDE = 3, OR_BELADY = 4, OR_LRU_TIDE = 5 };
enum { OR_NONE = 0, OR_S = 1, OR_H = 2 };
enum { OR_ARRIVAL = 1, OR_COMPLETION = 0 };
enum {
  K_COLD = 0, K_HIT_S = 1, K_HIT_H = 2, K_MISS = 3, K_PLACE_S = 4, K_PLACE_H = 5, K_BYPASS = 6,
  K_DEMOTE = 7, K_EVICT = 8, K_PROMOTE = 9, K_TIDE_DEMOTE = 10, K_EXPIRE = 11
};
enum {
  OR_OK = 0, OR_ERR_ARG = -1, OR_ERR_FORMAT = -3, OR_ERR_RANGE = -4, OR_ERR_OOM = -6,
  OR_ERR_LOG_FULL = -7, OR_ERR_INVARIANT = -20, OR_ERR_TIDE_FORMS = -21
};

typedef struct {
  uint32_t n_sessions;
  uint32_t pad0;
  uint64_t n_turns;
  const uint64_t *turn_off;      /* [n_sessions + 1] */
  const uint64_t *arrival_us;    /* [n_turns] */
  const uint64_t *completion_us; /* [n_turns] */
  const uint32_t *in_tok;        /* [n_turns] */
  const uint32_t *out_tok;       /* [n_turns] */
} or_trace;

typedef struct {
  uint32_t policy;
  uint32_t hazard_bucket;        /* w >= 1 */
  uint64_t cap_s_bytes;
  uint64_t cap_h_bytes;
  uint32_t kv_bytes_per_token;
  uint32_t max_sessions;         /* 0 = no slot limit */
  uint32_t ema_num, ema_den;     /* (3,10) */
  uint64_t penalty_q;            /* P_Z */
  uint32_t ttl_us;               /* Timeout */
  uint32_t ttft_load;            /* load factor L */
  uint64_t dma_bytes_per_us;
  uint64_t prefill_ns_per_tok;   /* t_p in ns per token, for TTFT */
  uint32_t debug;                /* 1: check invariants and both TIDE forms every event */
  uint32_t hazard_online;        /* 1: the hazard table starts empty and grows as sessions complete (R26) */
  uint32_t stale_sync;           /* R28: 0 live; 1 every event; 2 every stale_m arrivals; 3 every gap_start */
  uint32_t stale_m;
  uint32_t signals;              /* R29: bit 1 drops the gap signal, bit 2 the hazard signal */
  uint32_t pad3;
} or_params;

enum { OR_NO_GAP = 2, OR_NO_HAZARD = 4 };

enum { OR_SYNC_LIVE = 0, OR_SYNC_EVENT = 1, OR_SYNC_ARRIVALS = 2, OR_SYNC_GAP_START = 3 };

typedef struct {
  uint64_t events, req_warm, cold, hit_s, hit_h, miss, bypass, place_s, place_h;
  uint64_t evict, demote, promote, tide_demote, expire;
  uint64_t tok_hit_s, tok_hit_h, tok_miss, tok_computed, tok_needed;
  uint64_t dma_bytes, tide_calls, promoted_then_hit_s;
  uint64_t ttft_sum_lo, ttft_sum_hi, ttft_p50_ns, ttft_n;
  uint64_t decision_hash, log_len;
  uint64_t vict_n, vict_diff, prom_n, prom_diff; /* R28 */
  int32_t status;
  uint32_t pad2;
} or_result;

typedef struct { uint32_t event; uint32_t kind_session; } or_logrec;

/* ====================================================================== */
/* Hazard table, eqs. (hazard), (surv), (uq), (hq), (survq); reading R5.   */
/* ====================================================================== */

/* Turn counts -> per-t h_q and sigma_q for bucket width w. */
int or_hazard_lut(const uint32_t *turns_per_session, uint64_t n_sessions, uint32_t w,
                  uint16_t *h_q, uint16_t *sigma_q) {
  uint64_t n[OR_T_MAX + 1], d[OR_T_MAX + 1];
  if (w == 0) return OR_ERR_ARG;
  for (uint32_t t = 0; t <= OR_T_MAX; t++) {
    n[t] = 0;
    d[t] = 0;
    for (uint64_t s = 0; s < n_sessions; s++) {
      uint64_t ts = turns_per_session[s];
      if (ts >= (uint64_t)t + 1) n[t]++;   /* live at turn t */
      if (ts == (uint64_t)t + 1) d[t]++;   /* completes at turn t */
    }
  }
  for (uint32_t t = 0; t <= OR_T_MAX; t++) {
    uint64_t nn = 0, dd = 0;
    for (uint32_t u = 0; u <= OR_T_MAX; u++)
      if (u / w == t / w) { nn += n[u]; dd += d[u]; }
    /* Q_{12}(d/n) = floor(x*Lambda + 1/2) = floor((2*d*Lambda + n) / (2n)) */
    uint64_t hq = 0;
    if (nn > 0) {
      hq = (2 * dd * OR_LAMBDA + nn) / (2 * nn);
      if (hq > OR_LAMBDA) hq = OR_LAMBDA;
    }
    uint64_t sq = OR_LAMBDA - hq;
    if (sq < OR_EPS_Q) sq = OR_EPS_Q;
    h_q[t] = (uint16_t)hq;
    sigma_q[t] = (uint16_t)sq;
  }
  return OR_OK;
}

/* score_q, eqs. (t1), (t2), (scoreq): sat64(floor(g*L/s) + floor((L-s)*P/L)). */
uint64_t or_spear_score(uint64_t g_q, uint32_t sigma_q, uint64_t penalty_q, int done) {
  if (done) return OR_SCORE_MAX;
  uint64_t t1 = (g_q * OR_LAMBDA) / sigma_q;
  uint64_t t2 = ((uint64_t)(OR_LAMBDA - sigma_q) * penalty_q) / OR_LAMBDA;
  uint64_t s = t1 + t2;
  if (s < t1) s = OR_SCORE_MAX; /* saturate */
  return s;
}

/* eq. (ema-int) with weight a_num/a_den (paper: 3/10). */
uint64_t or_ema(uint64_t g_q, uint64_t g_new, uint32_t a_num, uint32_t a_den) {
  return ((uint64_t)a_num * g_new + (uint64_t)(a_den - a_num) * g_q) / a_den;
}

/* ====================================================================== */
/* Replay state                                                             */
/* ====================================================================== */

typedef struct {
  uint64_t time;
  uint32_t session;
  uint32_t turn;
  uint32_t type;
} or_event;

typedef struct {
  uint64_t g_q;        /* gap average, us */
  uint64_t last_ret;   /* completion time of the last turn */
  uint32_t turn;       /* register turn t */
  uint32_t tier;       /* OR_NONE / OR_S / OR_H */
  uint32_t pinned, done, promoted;
  uint64_t size;       /* resident tokens while in a tier */
  uint64_t last_touch; /* event index of the last event (LRU) */
  uint64_t next_ref;   /* event index of the next arrival (Belady) */
} or_sess;

typedef struct {
  const or_trace *tr;
  const or_params *p;
  or_result *res;
  or_sess *S;
  uint16_t sigma_q[OR_T_MAX + 1];
  int stale;           /* R28: rank from the snapshot rows below */
  uint64_t *snap_g;
  uint32_t *snap_turn, *snap_done;
  uint32_t *resident;  /* ids of sessions in a tier, unordered */
  uint64_t n_resident;
  uint64_t cap_s, cap_h;  /* tokens */
  uint64_t used_s, used_h; /* tokens resident per tier (running totals) */
  uint64_t now;
  uint64_t e;             /* current event index */
  or_logrec *log;
  uint64_t log_cap;
} or_state;

static int cmp_event(const void *a, const void *b) {
  const or_event *x = (const or_event *)a, *y = (const or_event *)b;
  if (x->time != y->time) return x->time < y->time ? -1 : 1;
  if (x->type != y->type) return x->type < y->type ? -1 : 1; /* COMPLETION first */
  if (x->session != y->session) return x->session < y->session ? -1 : 1;
  return 0;
}

/* SPEAR key of a register row (g_q, turn, done), with the signals of R29. */
static uint64_t spear_key(const or_state *st, uint64_t g_q, uint32_t turn, uint32_t done) {
  uint32_t t = turn < OR_T_MAX ? turn : OR_T_MAX;
  uint64_t g = (st->p->signals & OR_NO_GAP) ? 0 : g_q;
  uint32_t sigma = (st->p->signals & OR_NO_HAZARD) ? OR_LAMBDA : st->sigma_q[t];
  return or_spear_score(g, sigma, st->p->penalty_q, (int)done);
}

/* Policy key of session s from its live register row (R8); larger = more
 * evictable. */
static uint64_t live_key_of(const or_state *st, uint32_t s) {
  const or_sess *x = &st->S[s];
  switch (st->p->policy) {
    case OR_SPEAR:
    case OR_SPEAR_TIDE:
      return spear_key(st, x->g_q, x->turn, x->done);
    case OR_BELADY:
      return x->next_ref;
    default: /* LRU, Timeout, LRU+TIDE: older last touch = more evictable */
      return UINT64_MAX - x->last_touch;
  }
}

/* The key decisions rank by: the live row, or the snapshot row (R28). */
static uint64_t key_of(const or_state *st, uint32_t s) {
  if (!st->stale) return live_key_of(st, s);
  return spear_key(st, st->snap_g[s], st->snap_turn[s], st->snap_done[s]);
}

/* a more evictable than b: larger key, then smaller id. */
static int more_evictable(const or_state *st, uint32_t a, uint32_t b) {
  uint64_t ka = key_of(st, a), kb = key_of(st, b);
  if (ka != kb) return ka > kb;
  return a < b;
}

static int more_evictable_live(const or_state *st, uint32_t a, uint32_t b) {
  uint64_t ka = live_key_of(st, a), kb = live_key_of(st, b);
  if (ka != kb) return ka > kb;
  return a < b;
}

static void log_decision(or_state *st, uint32_t kind, uint32_t s) {
  uint64_t w = (st->e << 32) | ((uint64_t)kind << 24) | (uint64_t)s;
  st->res->decision_hash = (st->res->decision_hash ^ w) * 0x100000001B3ull;
  if (st->log) {
    if (st->res->log_len < st->log_cap) {
      st->log[st->res->log_len].event = (uint32_t)st->e;
      st->log[st->res->log_len].kind_session = (kind << 24) | s;
    } else if (st->res->status == OR_OK) {
      st->res->status = OR_ERR_LOG_FULL;
    }
  }
  st->res->log_len++;
}

static uint64_t used_of(const or_state *st, uint32_t tier, int pinned_only) {
  uint64_t u = 0;
  for (uint64_t i = 0; i < st->n_resident; i++) {
    const or_sess *x = &st->S[st->resident[i]];
    if (x->tier == tier && (!pinned_only || x->pinned)) u += x->size;
  }
  return u;
}

static uint64_t *used_ref(or_state *st, uint32_t tier) { return tier == OR_S ? &st->used_s : &st->used_h; }

static void res_add(or_state *st, uint32_t s, uint32_t tier, uint64_t size) {
  st->S[s].tier = tier;
  st->S[s].size = size;
  st->resident[st->n_resident++] = s;
  *used_ref(st, tier) += size;
}

static void res_remove(or_state *st, uint32_t s) {
  for (uint64_t i = 0; i < st->n_resident; i++)
    if (st->resident[i] == s) {
      st->resident[i] = st->resident[--st->n_resident];
      break;
    }
  if (st->S[s].tier != OR_NONE) *used_ref(st, st->S[s].tier) -= st->S[s].size;
  st->S[s].tier = OR_NONE;
  st->S[s].size = 0;
}

static void evict(or_state *st, uint32_t s, uint32_t kind) {
  if (st->S[s].pinned) st->res->status = OR_ERR_INVARIANT; /* never evict a pinned session */
  res_remove(st, s);
  log_decision(st, kind, s);
  if (kind == K_EXPIRE) st->res->expire++; else st->res->evict++;
}

/* Most evictable unpinned resident of a tier (tier 0: any tier); -1 if none. */
static int64_t argmax_unpinned(const or_state *st, uint32_t tier) {
  int64_t best = -1;
  for (uint64_t i = 0; i < st->n_resident; i++) {
    uint32_t s = st->resident[i];
    const or_sess *x = &st->S[s];
    if (x->pinned || (tier != 0 && x->tier != tier)) continue;
    if (best < 0 || more_evictable(st, s, (uint32_t)best)) best = s;
  }
  return best;
}

/* Least evictable unpinned resident of a tier; -1 if none. */
static int64_t argmin_unpinned(const or_state *st, uint32_t tier) {
  int64_t best = -1;
  for (uint64_t i = 0; i < st->n_resident; i++) {
    uint32_t s = st->resident[i];
    const or_sess *x = &st->S[s];
    if (x->pinned || x->tier != tier) continue;
    if (best < 0 || more_evictable(st, (uint32_t)best, s)) best = s;
  }
  return best;
}

/* Most / least evictable unpinned resident of a tier by the live rows. */
static int64_t argmax_unpinned_live(const or_state *st, uint32_t tier) {
  int64_t best = -1;
  for (uint64_t i = 0; i < st->n_resident; i++) {
    uint32_t s = st->resident[i];
    const or_sess *x = &st->S[s];
    if (x->pinned || (tier != 0 && x->tier != tier)) continue;
    if (best < 0 || more_evictable_live(st, s, (uint32_t)best)) best = s;
  }
  return best;
}

static int64_t argmin_unpinned_live(const or_state *st, uint32_t tier) {
  int64_t best = -1;
  for (uint64_t i = 0; i < st->n_resident; i++) {
    uint32_t s = st->resident[i];
    const or_sess *x = &st->S[s];
    if (x->pinned || x->tier != tier) continue;
    if (best < 0 || more_evictable_live(st, (uint32_t)best, s)) best = s;
  }
  return best;
}

/* R28: one acted-upon victim (promotion) choice against the live choice. */
static void count_victim(or_state *st, uint32_t chosen, int64_t live) {
  if (!st->stale) return;
  st->res->vict_n++;
  st->res->vict_diff += live != (int64_t)chosen;
}

static void count_promotion(or_state *st, uint32_t chosen, int64_t live) {
  if (!st->stale) return;
  st->res->prom_n++;
  st->res->prom_diff += live != (int64_t)chosen;
}

/* R9: admit a session demoted from the fast tier into the HBM tier. */
static void admit_demoted(or_state *st, uint32_t d, uint64_t size) {
  uint64_t pinned_h = used_of(st, OR_H, 1);
  if (pinned_h > st->cap_h || size > st->cap_h - pinned_h) {
    log_decision(st, K_EVICT, d);
    st->res->evict++;
    return;
  }
  while (st->used_h + size > st->cap_h) {
    int64_t v = argmax_unpinned(st, OR_H);
    /* v = most evictable of (unpinned H) u {d}; if that is d, drop d. */
    if (st->stale) {
      int64_t lv = argmax_unpinned_live(st, OR_H);
      int64_t live = (lv < 0 || more_evictable_live(st, d, (uint32_t)lv)) ? (int64_t)d : lv;
      count_victim(st, (v < 0 || more_evictable(st, d, (uint32_t)v)) ? d : (uint32_t)v, live);
    }
    if (v < 0 || more_evictable(st, d, (uint32_t)v)) {
      log_decision(st, K_EVICT, d);
      st->res->evict++;
      return;
    }
    evict(st, (uint32_t)v, K_EVICT);
  }
  res_add(st, d, OR_H, size);
  log_decision(st, K_DEMOTE, d);
  st->res->demote++;
}

/* R9 (placement of the arriving session s with n tokens) and R15. */
static void place(or_state *st, uint32_t s, uint64_t n) {
  const or_params *p = st->p;
  if (p->max_sessions > 0) {
    uint64_t pinned_cnt = 0;
    for (uint64_t i = 0; i < st->n_resident; i++) pinned_cnt += st->S[st->resident[i]].pinned;
    if (pinned_cnt >= p->max_sessions) {
      log_decision(st, K_BYPASS, s);
      st->res->bypass++;
      return;
    }
  }
  uint64_t pinned_s = used_of(st, OR_S, 1), pinned_h = used_of(st, OR_H, 1);
  if (pinned_s <= st->cap_s && n <= st->cap_s - pinned_s) {
    /* (i) fast tier: demote the most evictable unpinned fast-tier sessions. */
    while (st->used_s + n > st->cap_s) {
      int64_t d = argmax_unpinned(st, OR_S);
      if (d < 0) { st->res->status = OR_ERR_INVARIANT; return; }
      if (st->stale) count_victim(st, (uint32_t)d, argmax_unpinned_live(st, OR_S));
      uint64_t sz = st->S[d].size;
      res_remove(st, (uint32_t)d);
      admit_demoted(st, (uint32_t)d, sz);
    }
    res_add(st, s, OR_S, n);
    log_decision(st, K_PLACE_S, s);
    st->res->place_s++;
  } else if (pinned_h <= st->cap_h && n <= st->cap_h - pinned_h) {
    /* (ii) HBM tier: evict the most evictable unpinned HBM sessions. */
    while (st->used_h + n > st->cap_h) {
      int64_t v = argmax_unpinned(st, OR_H);
      if (v < 0) { st->res->status = OR_ERR_INVARIANT; return; }
      if (st->stale) count_victim(st, (uint32_t)v, argmax_unpinned_live(st, OR_H));
      evict(st, (uint32_t)v, K_EVICT);
    }
    res_add(st, s, OR_H, n);
    log_decision(st, K_PLACE_H, s);
    st->res->place_h++;
  } else {
    /* (iii) larger than what either tier can free: serve, do not retain. */
    log_decision(st, K_BYPASS, s);
    st->res->bypass++;
    return;
  }
  if (p->max_sessions > 0) {
    while (st->n_resident > p->max_sessions) {
      int64_t v = argmax_unpinned(st, 0);
      if (v < 0) { st->res->status = OR_ERR_INVARIANT; return; }
      if (st->stale) count_victim(st, (uint32_t)v, argmax_unpinned_live(st, 0));
      evict(st, (uint32_t)v, K_EVICT);
    }
  }
}

/* ---- TIDE, R14, list form (no mutation): fills the move lists ------------ */

static const or_state *g_sort_state; /* qsort has no context argument */

static int cmp_asc(const void *a, const void *b) { /* least evictable first */
  uint32_t x = *(const uint32_t *)a, y = *(const uint32_t *)b;
  if (x == y) return 0;
  return more_evictable(g_sort_state, y, x) ? -1 : 1;
}
static int cmp_desc(const void *a, const void *b) { /* most evictable first */
  uint32_t x = *(const uint32_t *)a, y = *(const uint32_t *)b;
  if (x == y) return 0;
  return more_evictable(g_sort_state, x, y) ? -1 : 1;
}

typedef struct { uint32_t n1, n2; uint32_t *p1, *p2, *d2; uint64_t moved; } or_tide_moves;

static void tide_list_form(or_state *st, uint64_t budget, or_tide_moves *mv) {
  uint64_t kvB = st->p->kv_bytes_per_token;
  uint32_t *P = (uint32_t *)malloc(sizeof(uint32_t) * (st->n_resident + 1));
  uint32_t *D = (uint32_t *)malloc(sizeof(uint32_t) * (st->n_resident + 1));
  uint64_t np = 0, nd = 0;
  for (uint64_t i = 0; i < st->n_resident; i++) {
    uint32_t s = st->resident[i];
    if (st->S[s].pinned) continue;
    if (st->S[s].tier == OR_H) P[np++] = s;
    else if (st->S[s].tier == OR_S) D[nd++] = s;
  }
  g_sort_state = st;
  qsort(P, np, sizeof(uint32_t), cmp_asc);
  uint64_t used_s = st->used_s, used_h = st->used_h, rem = budget;
  uint64_t j = 0;
  mv->n1 = mv->n2 = 0;
  /* phase 1: promotions into free fast-tier space, ascending key order */
  while (j < np) {
    uint64_t sz = st->S[P[j]].size, by = sz * kvB;
    if (by > rem || used_s + sz > st->cap_s) break;
    rem -= by;
    used_s += sz;
    used_h -= sz;
    mv->p1[mv->n1++] = P[j];
    D[nd++] = P[j];
    j++;
  }
  qsort(D, nd, sizeof(uint32_t), cmp_desc);
  /* phase 2: pair P[j] (ascending HBM) with D[i] (descending fast tier) */
  for (uint64_t i = 0; j < np && i < nd; i++, j++) {
    uint32_t pp = P[j], dd = D[i];
    uint64_t sp = st->S[pp].size, sd = st->S[dd].size, by = (sp + sd) * kvB;
    if (!more_evictable(st, dd, pp)) break;
    if (by > rem) break;
    if (used_s - sd + sp > st->cap_s) break;
    if (used_h - sp + sd > st->cap_h) break;
    rem -= by;
    used_s = used_s - sd + sp;
    used_h = used_h - sp + sd;
    mv->p2[mv->n2] = pp;
    mv->d2[mv->n2] = dd;
    mv->n2++;
  }
  mv->moved = budget - rem;
  free(P);
  free(D);
}

/* ---- TIDE, R14, loop form (Algorithm 1, the WHILE over legal pairs) ------ */
static uint64_t tide_loop_form(or_state *st, uint64_t budget, or_tide_moves *rec) {
  uint64_t kvB = st->p->kv_bytes_per_token, rem = budget;
  rec->n1 = rec->n2 = 0;
  /* phase 1 */
  for (;;) {
    int64_t p = argmin_unpinned(st, OR_H);
    if (p < 0) break;
    uint64_t sz = st->S[p].size, by = sz * kvB;
    if (by > rem || st->used_s + sz > st->cap_s) break;
    if (st->stale) count_promotion(st, (uint32_t)p, argmin_unpinned_live(st, OR_H));
    rem -= by;
    res_remove(st, (uint32_t)p);
    res_add(st, (uint32_t)p, OR_S, sz);
    st->S[p].promoted = 1;
    log_decision(st, K_PROMOTE, (uint32_t)p);
    st->res->promote++;
    rec->p1[rec->n1++] = (uint32_t)p;
  }
  /* phase 2: p = argmin over H, d = argmax over S (eqs. promote, demote) */
  for (;;) {
    int64_t p = argmin_unpinned(st, OR_H), d = argmax_unpinned(st, OR_S);
    if (p < 0 || d < 0) break;
    uint64_t sp = st->S[p].size, sd = st->S[d].size, by = (sp + sd) * kvB;
    if (!more_evictable(st, (uint32_t)d, (uint32_t)p)) break;
    if (by > rem) break;
    if (st->used_s - sd + sp > st->cap_s) break;
    if (st->used_h - sp + sd > st->cap_h) break;
    if (st->stale) {
      count_promotion(st, (uint32_t)p, argmin_unpinned_live(st, OR_H));
      count_victim(st, (uint32_t)d, argmax_unpinned_live(st, OR_S));
    }
    rem -= by;
    res_remove(st, (uint32_t)p);
    res_remove(st, (uint32_t)d);
    res_add(st, (uint32_t)p, OR_S, sp);
    res_add(st, (uint32_t)d, OR_H, sd);
    st->S[p].promoted = 1;
    log_decision(st, K_PROMOTE, (uint32_t)p);
    log_decision(st, K_TIDE_DEMOTE, (uint32_t)d);
    st->res->promote++;
    st->res->tide_demote++;
    rec->p2[rec->n2] = (uint32_t)p;
    rec->d2[rec->n2] = (uint32_t)d;
    rec->n2++;
  }
  return budget - rem;
}

static void check_invariants(or_state *st) {
  uint64_t us = used_of(st, OR_S, 0), uh = used_of(st, OR_H, 0);
  if (us != st->used_s || uh != st->used_h) st->res->status = OR_ERR_INVARIANT;
  if (us > st->cap_s || uh > st->cap_h) st->res->status = OR_ERR_INVARIANT;
  if (st->p->max_sessions > 0 && st->n_resident > st->p->max_sessions) st->res->status = OR_ERR_INVARIANT;
  uint64_t cnt = 0;
  for (uint32_t s = 0; s < st->tr->n_sessions; s++) cnt += st->S[s].tier != OR_NONE;
  if (cnt != st->n_resident) st->res->status = OR_ERR_INVARIANT;
}

static int cmp_u64(const void *a, const void *b) {
  uint64_t x = *(const uint64_t *)a, y = *(const uint64_t *)b;
  return x < y ? -1 : (x > y ? 1 : 0);
}

static int has_tide(uint32_t policy) { return policy == OR_SPEAR_TIDE || policy == OR_LRU_TIDE; }

/* Validate a trace: session-major turns in time order, gaps below 2^31 us,
 * consecutive events (in R2 order) less than 2^31 us apart, sessions numbered
 * in order of first arrival (R3), and prefixes that never shrink. */
int or_validate(const or_trace *tr, or_event **events_out) {
  uint64_t T = tr->n_turns, S = tr->n_sessions;
  if (tr->turn_off[0] != 0 || tr->turn_off[S] != T) return OR_ERR_FORMAT;
  if (S >= (1u << 24)) return OR_ERR_RANGE;
  if (T >= (1ull << 31)) return OR_ERR_RANGE;
  for (uint64_t s = 0; s < S; s++) {
    uint64_t a = tr->turn_off[s], b = tr->turn_off[s + 1];
    if (b <= a) return OR_ERR_FORMAT; /* at least one turn */
    if (b - a >= 65536) return OR_ERR_RANGE;
    if (s > 0 && tr->arrival_us[a] < tr->arrival_us[tr->turn_off[s - 1]]) return OR_ERR_FORMAT;
    for (uint64_t i = a; i < b; i++) {
      if (tr->completion_us[i] <= tr->arrival_us[i]) return OR_ERR_FORMAT;
      if (tr->completion_us[i] - tr->arrival_us[i] >= (1ull << 31)) return OR_ERR_RANGE;
      if (tr->out_tok[i] < tr->in_tok[i] || tr->in_tok[i] == 0) return OR_ERR_FORMAT;
      if (i > a) {
        if (tr->arrival_us[i] <= tr->completion_us[i - 1]) return OR_ERR_FORMAT;
        if (tr->arrival_us[i] - tr->completion_us[i - 1] >= (1ull << 31)) return OR_ERR_RANGE;
        if (tr->in_tok[i] < tr->out_tok[i - 1]) return OR_ERR_FORMAT;
      }
    }
  }
  or_event *ev = (or_event *)malloc(sizeof(or_event) * (2 * T + 1));
  if (!ev) return OR_ERR_OOM;
  uint64_t m = 0;
  for (uint32_t s = 0; s < S; s++)
    for (uint64_t i = tr->turn_off[s]; i < tr->turn_off[s + 1]; i++) {
      uint32_t k = (uint32_t)(i - tr->turn_off[s]);
      ev[m++] = (or_event){tr->arrival_us[i], s, k, OR_ARRIVAL};
      ev[m++] = (or_event){tr->completion_us[i], s, k, OR_COMPLETION};
    }
  qsort(ev, m, sizeof(or_event), cmp_event);
  for (uint64_t i = 1; i < m; i++)
    if (ev[i].time - ev[i - 1].time >= (1ull << 31)) { free(ev); return OR_ERR_RANGE; }
  *events_out = ev;
  return OR_OK;
}

/* One replay of Algorithm 1 over a trace. */
int or_replay(const or_trace *tr, const or_params *p, or_result *res, or_logrec *log,
              uint64_t log_cap, uint64_t *ttft_out) {
  memset(res, 0, sizeof(*res));
  res->decision_hash = 0xCBF29CE484222325ull;
  if (!tr || !p || p->hazard_bucket == 0 || p->ema_den == 0 || p->ema_num > p->ema_den ||
      p->kv_bytes_per_token == 0 || p->kv_bytes_per_token > (1u << 24) || p->ttft_load == 0 ||
      p->policy > OR_LRU_TIDE || p->penalty_q >= (1ull << 32) ||
      (p->ttl_us != UINT32_MAX && p->ttl_us >= (1u << 31)) || p->dma_bytes_per_us >= (1ull << 32) ||
      p->stale_sync > OR_SYNC_GAP_START || (p->stale_sync == OR_SYNC_ARRIVALS && p->stale_m == 0) ||
      (p->stale_sync != OR_SYNC_LIVE &&
       (p->hazard_online || (p->policy != OR_SPEAR && p->policy != OR_SPEAR_TIDE))) ||
      (p->signals & ~(uint32_t)(OR_NO_GAP | OR_NO_HAZARD)) ||
      (p->signals && (p->hazard_online || (p->policy != OR_SPEAR && p->policy != OR_SPEAR_TIDE))))
    return res->status = OR_ERR_ARG;
  or_event *ev = NULL;
  int rc = or_validate(tr, &ev);
  if (rc != OR_OK) return res->status = rc;

  uint64_t S = tr->n_sessions, T = tr->n_turns, E = 2 * T;
  or_state st;
  memset(&st, 0, sizeof(st));
  st.tr = tr;
  st.p = p;
  st.res = res;
  st.S = (or_sess *)calloc(S + 1, sizeof(or_sess));
  st.stale = p->stale_sync != OR_SYNC_LIVE;
  st.snap_g = (uint64_t *)calloc(S + 1, sizeof(uint64_t)); /* R28: rows start at zero */
  st.snap_turn = (uint32_t *)calloc(S + 1, sizeof(uint32_t));
  st.snap_done = (uint32_t *)calloc(S + 1, sizeof(uint32_t));
  st.resident = (uint32_t *)malloc(sizeof(uint32_t) * (S + 1));
  uint64_t *ttft = (uint64_t *)malloc(sizeof(uint64_t) * (T + 1));
  uint64_t *next_arr = (uint64_t *)malloc(sizeof(uint64_t) * (E + 1));
  uint32_t *tps = (uint32_t *)malloc(sizeof(uint32_t) * (S + 1));
  or_tide_moves m1, m2;
  memset(&m1, 0, sizeof(m1));
  memset(&m2, 0, sizeof(m2));
  m1.p1 = (uint32_t *)malloc(sizeof(uint32_t) * (S + 1));
  m1.p2 = (uint32_t *)malloc(sizeof(uint32_t) * (S + 1));
  m1.d2 = (uint32_t *)malloc(sizeof(uint32_t) * (S + 1));
  m2.p1 = (uint32_t *)malloc(sizeof(uint32_t) * (S + 1));
  m2.p2 = (uint32_t *)malloc(sizeof(uint32_t) * (S + 1));
  m2.d2 = (uint32_t *)malloc(sizeof(uint32_t) * (S + 1));
  if (!st.S || !st.snap_g || !st.snap_turn || !st.snap_done || !st.resident || !ttft || !next_arr || !tps || !m1.p1 || !m1.p2 || !m1.d2 ||
      !m2.p1 || !m2.p2 || !m2.d2) {
    rc = OR_ERR_OOM;
    goto done;
  }
  st.cap_s = p->cap_s_bytes / p->kv_bytes_per_token;
  st.cap_h = p->cap_h_bytes / p->kv_bytes_per_token;
  st.log = log;
  st.log_cap = log_cap;

  /* Offline hazard table fitted on all sessions of the trace (R5), or (R26,
   * Sec. V-F) an online table that starts empty: tps then lists the turn
   * counts of the sessions completed so far. */
  uint16_t h_q[OR_T_MAX + 1];
  uint64_t n_done = 0;
  for (uint64_t s = 0; s < S; s++) tps[s] = (uint32_t)(tr->turn_off[s + 1] - tr->turn_off[s]);
  or_hazard_lut(tps, p->hazard_online ? 0 : S, p->hazard_bucket, h_q, st.sigma_q);

  /* Belady next reference: event index of each session's next arrival. */
  {
    uint64_t *last_arr_of = (uint64_t *)malloc(sizeof(uint64_t) * (S + 1));
    for (uint64_t s = 0; s < S; s++) last_arr_of[s] = UINT64_MAX;
    for (uint64_t i = E; i-- > 0;) {
      next_arr[i] = UINT64_MAX;
      if (ev[i].type == OR_ARRIVAL) {
        next_arr[i] = last_arr_of[ev[i].session];
        last_arr_of[ev[i].session] = i;
      }
    }
    free(last_arr_of);
  }

  uint64_t t0 = E ? ev[0].time : 0, q_free = 0, n_ttft = 0, n_arrivals = 0;
  unsigned __int128 ttft_sum = 0;
  uint64_t dma_busy_until = 0;
  int dma_busy = 0;

  for (uint64_t e = 0; e < E; e++) {
    const or_event *x = &ev[e];
    uint32_t s = x->session;
    uint64_t ti = tr->turn_off[s] + x->turn;
    or_sess *R = &st.S[s];
    st.now = x->time;
    st.e = e;
    res->events++;

    /* R16: Timeout expiry before the event, in ascending session id. */
    if (p->policy == OR_TIMEOUT && p->ttl_us != UINT32_MAX) { /* UINT32_MAX: no expiry */
      for (uint32_t v = 0; v < S; v++) {
        or_sess *y = &st.S[v];
        if (y->tier != OR_NONE && !y->pinned && st.now - y->last_ret >= p->ttl_us) evict(&st, v, K_EXPIRE);
      }
    }
    if (dma_busy && st.now >= dma_busy_until) dma_busy = 0;

    if (x->type == OR_ARRIVAL) {
      uint32_t k = x->turn;
      uint64_t in = tr->in_tok[ti], out = tr->out_tok[ti];
      uint64_t out_prev = k ? tr->out_tok[ti - 1] : 0;
      /* gap_end: eq. (gap) then eq. (ema-int) */
      if (k >= 1) {
        uint64_t g_new = tr->arrival_us[ti] - tr->completion_us[ti - 1];
        R->g_q = or_ema(R->g_q, g_new, p->ema_num, p->ema_den);
      }
      /* classify and account (R10) */
      uint64_t prefill;
      if (k == 0) {
        log_decision(&st, K_COLD, s);
        res->cold++;
        prefill = in;
      } else {
        res->req_warm++;
        res->tok_needed += in;
        if (R->tier == OR_S) {
          log_decision(&st, K_HIT_S, s);
          res->hit_s++;
          res->tok_hit_s += out_prev;
          prefill = in - out_prev;
          if (R->promoted) res->promoted_then_hit_s++;
        } else if (R->tier == OR_H) {
          log_decision(&st, K_HIT_H, s);
          res->hit_h++;
          res->tok_hit_h += out_prev;
          prefill = in - out_prev;
        } else {
          log_decision(&st, K_MISS, s);
          res->miss++;
          res->tok_miss += out_prev;
          prefill = in;
        }
        res->tok_computed += prefill;
      }
      R->promoted = 0;
      /* TTFT queue (R17) */
      {
        uint64_t arr = (st.now - t0) * 1000ull / p->ttft_load;
        if (q_free < arr) q_free = arr;
        q_free += prefill * p->prefill_ns_per_tok;
        uint64_t v = q_free - arr;
        ttft[n_ttft++] = v;
        ttft_sum += v;
      }
      /* write e into R */
      R->turn = k;
      R->pinned = 1;
      R->last_touch = e;
      R->next_ref = next_arr[e];
      if (R->tier != OR_NONE) res_remove(&st, s);
      place(&st, s, out);
    } else {
      R->pinned = 0;
      R->last_ret = x->time;
      R->last_touch = e;
      int final = (x->turn + 1 == tr->turn_off[s + 1] - tr->turn_off[s]);
      if (final) {
        R->done = 1; /* R12: stays resident with the maximal key */
        if (p->hazard_online) {
          /* R26: the session's turn count joins the table; every later key
           * uses the rebuilt sigma */
          tps[n_done++] = x->turn + 1;
          or_hazard_lut(tps, n_done, p->hazard_bucket, h_q, st.sigma_q);
        }
      } else if (has_tide(p->policy) && !dma_busy) {
        /* gap_start with DMA free: TIDE with budget = Delta * B (R11) */
        uint64_t budget = R->g_q * p->dma_bytes_per_us;
        res->tide_calls++;
        if (p->debug) tide_list_form(&st, budget, &m1);
        uint64_t moved = tide_loop_form(&st, budget, &m2);
        if (p->debug) {
          int same = m1.n1 == m2.n1 && m1.n2 == m2.n2 && m1.moved == moved;
          for (uint32_t i = 0; same && i < m1.n1; i++) same = m1.p1[i] == m2.p1[i];
          for (uint32_t i = 0; same && i < m1.n2; i++) same = m1.p2[i] == m2.p2[i] && m1.d2[i] == m2.d2[i];
          if (!same) res->status = OR_ERR_TIDE_FORMS;
        }
        res->dma_bytes += moved;
        if (moved > 0 && p->dma_bytes_per_us > 0) {
          dma_busy = 1;
          dma_busy_until = st.now + (moved + p->dma_bytes_per_us - 1) / p->dma_bytes_per_us;
        }
      }
    }
    /* R28: a sync point copies every live row into the snapshot, after the
     * event's own decisions */
    if (st.stale) {
      int sync = p->stale_sync == OR_SYNC_EVENT;
      if (x->type == OR_ARRIVAL && p->stale_sync == OR_SYNC_ARRIVALS) sync = ++n_arrivals % p->stale_m == 0;
      if (x->type == OR_COMPLETION && p->stale_sync == OR_SYNC_GAP_START)
        sync = x->turn + 1 != tr->turn_off[s + 1] - tr->turn_off[s];
      if (sync)
        for (uint64_t v = 0; v < S; v++) {
          st.snap_g[v] = st.S[v].g_q;
          st.snap_turn[v] = st.S[v].turn;
          st.snap_done[v] = st.S[v].done;
        }
    }
    if (p->debug) check_invariants(&st);
  }

  res->ttft_n = n_ttft;
  res->ttft_sum_lo = (uint64_t)ttft_sum;
  res->ttft_sum_hi = (uint64_t)(ttft_sum >> 64);
  if (ttft_out) memcpy(ttft_out, ttft, sizeof(uint64_t) * n_ttft);
  if (n_ttft) {
    qsort(ttft, n_ttft, sizeof(uint64_t), cmp_u64);
    res->ttft_p50_ns = ttft[(n_ttft - 1) / 2]; /* lower median */
  }
  rc = res->status;

done:
  free(ev);
  free(st.S);
  free(st.snap_g);
  free(st.snap_turn);
  free(st.snap_done);
  free(st.resident);
  free(ttft);
  free(next_arr);
  free(tps);
  free(m1.p1); free(m1.p2); free(m1.d2);
  free(m2.p1); free(m2.p2); free(m2.d2);
  if (rc != OR_OK && res->status == OR_OK) res->status = rc;
  return res->status;
}

/* ====================================================================== */
/* Standalone ranking of a live set (the scan of Sec. IV-D plus TIDE).     */
/* ====================================================================== */

typedef struct {
  const uint32_t *gap_q;
  const uint32_t *last_ret;
  const uint16_t *turn;
  const uint32_t *kv_tok;
  const uint8_t *tier;
  const uint8_t *flags; /* bit0 pinned, bit1 done */
  uint64_t n;
} or_records;

static const uint64_t *g_rank_keys;

static int rank_more(uint32_t a, uint32_t b) {
  if (g_rank_keys[a] != g_rank_keys[b]) return g_rank_keys[a] > g_rank_keys[b];
  return a < b;
}
static int cmp_rank_desc(const void *a, const void *b) {
  uint32_t x = *(const uint32_t *)a, y = *(const uint32_t *)b;
  if (x == y) return 0;
  return rank_more(x, y) ? -1 : 1;
}
static int cmp_rank_asc(const void *a, const void *b) { return -cmp_rank_desc(a, b); }

/* Every key of a live set; then the k most evictable unpinned records
 * (victims), and the TIDE fill for one budget: phase-1 promotions into
 * free_s_tok, then the pair loop.  Move lists hold at most max_moves. */
int or_rank(const or_records *r, const uint16_t *sigma_q51, uint64_t penalty_q, uint32_t k,
            uint64_t budget_bytes, uint32_t kv_bytes_per_token, uint64_t free_s_tok,
            uint64_t free_h_tok, uint32_t *victims, uint32_t *n_victims, uint32_t *promote,
            uint32_t *n_promote, uint32_t *demote, uint32_t *n_demote, uint64_t *moved_bytes,
            uint64_t *keys_out, uint32_t max_moves) {
  uint64_t n = r->n;
  uint64_t *key = (uint64_t *)malloc(sizeof(uint64_t) * (n + 1));
  uint32_t *all = (uint32_t *)malloc(sizeof(uint32_t) * (n + 1));
  uint32_t *P = (uint32_t *)malloc(sizeof(uint32_t) * (n + 1));
  uint32_t *D = (uint32_t *)malloc(sizeof(uint32_t) * (n + 1));
  if (!key || !all || !P || !D) { free(key); free(all); free(P); free(D); return OR_ERR_OOM; }
  uint64_t na = 0, np = 0, nd = 0;
  for (uint64_t i = 0; i < n; i++) {
    uint32_t t = r->turn[i] < OR_T_MAX ? r->turn[i] : OR_T_MAX;
    key[i] = or_spear_score(r->gap_q[i], sigma_q51[t], penalty_q, (r->flags[i] & 2) != 0);
    if (keys_out) keys_out[i] = key[i];
    if (r->flags[i] & 1) continue; /* pinned: never a victim, never moved */
    if (r->tier[i] == OR_S || r->tier[i] == OR_H) all[na++] = (uint32_t)i;
    if (r->tier[i] == OR_H) P[np++] = (uint32_t)i;
    if (r->tier[i] == OR_S) D[nd++] = (uint32_t)i;
  }
  g_rank_keys = key;
  qsort(all, na, sizeof(uint32_t), cmp_rank_desc);
  uint64_t nv = k < na ? k : na;
  for (uint64_t i = 0; i < nv; i++) victims[i] = all[i];
  *n_victims = (uint32_t)nv;

  qsort(P, np, sizeof(uint32_t), cmp_rank_asc);
  /* Free space is tracked exactly (128 bits): the capacity tests are on the
   * integers, whatever the free space passed in. */
  unsigned __int128 fs = free_s_tok, fh = free_h_tok;
  uint64_t rem = budget_bytes, j = 0, npro = 0, ndem = 0;
  while (j < np && npro < max_moves) { /* phase 1 */
    uint64_t sz = r->kv_tok[P[j]], by = sz * kv_bytes_per_token;
    if (by > rem || sz > fs) break;
    rem -= by;
    fs -= sz;
    fh += sz;
    promote[npro++] = P[j];
    D[nd++] = P[j];
    j++;
  }
  qsort(D, nd, sizeof(uint32_t), cmp_rank_desc);
  for (uint64_t i = 0; j < np && i < nd && npro < max_moves; i++, j++) { /* phase 2 */
    uint32_t pp = P[j], dd = D[i];
    uint64_t sp = r->kv_tok[pp], sd = r->kv_tok[dd], by = (sp + sd) * kv_bytes_per_token;
    if (!rank_more(dd, pp)) break;
    if (by > rem) break;
    if (sp > fs + sd) break;  /* fast tier would exceed its capacity */
    if (sd > fh + sp) break;  /* HBM tier would exceed its capacity */
    rem -= by;
    fs = fs + sd - sp;
    fh = fh + sp - sd;
    promote[npro++] = pp;
    demote[ndem++] = dd;
  }
  *n_promote = (uint32_t)npro;
  *n_demote = (uint32_t)ndem;
  *moved_bytes = budget_bytes - rem;
  free(key);
  free(all);
  free(P);
  free(D);
  return OR_OK;
}

/* ====================================================================== */
/* Kendall tau-b between two score vectors (reporting; Sec. IV-C, Eq. lock) */
/* ====================================================================== */

/* Brute force O(n^2): concordant minus discordant over sqrt of untied pairs. */
double or_kendall_brute(const double *x, const double *y, uint64_t n) {
  double c = 0, d = 0, tx = 0, ty = 0;
  for (uint64_t i = 0; i < n; i++)
    for (uint64_t j = i + 1; j < n; j++) {
      double a = (x[i] > x[j]) - (x[i] < x[j]);
      double b = (y[i] > y[j]) - (y[i] < y[j]);
      if (a == 0 && b == 0) continue;
      if (a == 0) { tx++; continue; }
      if (b == 0) { ty++; continue; }
      if (a * b > 0) c++; else d++;
    }
  double n0 = c + d + tx, n1 = c + d + ty;
  if (n0 == 0 || n1 == 0) return 0.0;
  return (c - d) / __builtin_sqrt(n0 * n1);
}

/* ====================================================================== */
/* Agent Serving Effectiveness (Sec. IV-E, Eq. ase)                        */
/* ====================================================================== */

/* ASE of each configuration c over datasets d: the 3*nd-th root of the
 * product, over d, of HR_cd/HR_d^max, AMAT_d^min/AMAT_cd, TTFT_d^min/TTFT_cd
 * (extremes over the configurations).  Arrays are [nc][nd].  Reading R25: a
 * ratio 0/0 (every configuration at 0 on that metric) counts as 1. */
void or_ase(const double *hr, const double *amat, const double *ttft, int nc, int nd, double *out) {
  for (int c = 0; c < nc; c++) {
    double prod = 1.0;
    for (int d = 0; d < nd; d++) {
      double hr_max = 0.0, amat_min = amat[d], ttft_min = ttft[d];
      for (int c2 = 0; c2 < nc; c2++) {
        if (hr[c2 * nd + d] > hr_max) hr_max = hr[c2 * nd + d];
        if (amat[c2 * nd + d] < amat_min) amat_min = amat[c2 * nd + d];
        if (ttft[c2 * nd + d] < ttft_min) ttft_min = ttft[c2 * nd + d];
      }
      prod *= hr_max == 0.0 ? 1.0 : hr[c * nd + d] / hr_max;
      prod *= amat[c * nd + d] == 0.0 ? 1.0 : amat_min / amat[c * nd + d];
      prod *= ttft[c * nd + d] == 0.0 ? 1.0 : ttft_min / ttft[c * nd + d];
    }
    out[c] = pow(prod, 1.0 / (3.0 * nd));
  }
}

/* Attainment (Sec. V-F, eq. attainment) of an online-table replay against the
 * offline-table and LRU replays of the same trace, from their decision logs
 * (kinds HIT_S, HIT_H, MISS mark warm requests).  Windows per reading R27.
 * out[6j .. 6j+5] = n_j, warm requests in window j, H_on, H_off, H_LRU,
 * A_j = (H_on - H_LRU) / (H_off - H_LRU); A_j is NaN when the window holds no
 * warm request or H_off = H_LRU.  The three logs must list the same warm
 * requests (else OR_ERR_FORMAT). */
int or_attainment(const or_trace *tr, const or_logrec *const *logs, const uint64_t *lens, uint32_t P,
                  double *out) {
  if (!tr || !logs || !lens || !out) return OR_ERR_ARG;
  const uint64_t N = tr->n_sessions;
  if (P == 0 || P > N) return OR_ERR_RANGE;
  or_event *ev = NULL;
  int rc = or_validate(tr, &ev);
  if (rc != OR_OK) return rc;
  const uint64_t E = 2 * tr->n_turns;
  /* window of every event: sessions completed before it, then the largest
   * j with floor(j N / P) <= that count */
  uint32_t *win = (uint32_t *)malloc(sizeof(uint32_t) * (E + 1));
  uint64_t *warm = (uint64_t *)calloc(3 * (size_t)P, sizeof(uint64_t));
  uint64_t *hit = (uint64_t *)calloc(3 * (size_t)P, sizeof(uint64_t));
  if (!win || !warm || !hit) {
    free(ev), free(win), free(warm), free(hit);
    return OR_ERR_OOM;
  }
  uint64_t done = 0;
  for (uint64_t e = 0; e < E; e++) {
    uint32_t j = 0;
    while (j + 1 < P && (j + 1) * N / P <= done) j++;
    win[e] = j;
    const or_event *x = &ev[e];
    if (x->type == OR_COMPLETION && x->turn + 1 == tr->turn_off[x->session + 1] - tr->turn_off[x->session]) done++;
  }
  for (int r = 0; r < 3 && rc == OR_OK; r++) {
    for (uint64_t i = 0; i < lens[r]; i++) {
      const uint32_t e = logs[r][i].event, kind = logs[r][i].kind_session >> 24;
      if (e >= E) {
        rc = OR_ERR_FORMAT;
        break;
      }
      if (kind == K_HIT_S || kind == K_HIT_H || kind == K_MISS) {
        warm[r * P + win[e]]++;
        if (kind != K_MISS) hit[r * P + win[e]]++;
      }
    }
  }
  for (uint32_t j = 0; j < P && rc == OR_OK; j++) {
    if (warm[j] != warm[P + j] || warm[j] != warm[2 * P + j]) {
      rc = OR_ERR_FORMAT;
      break;
    }
    double h[3];
    for (int r = 0; r < 3; r++) h[r] = warm[j] ? (double)hit[r * P + j] / (double)warm[j] : NAN;
    double *o = out + 6 * (size_t)j;
    o[0] = (double)((uint64_t)j * N / P);
    o[1] = (double)warm[j];
    o[2] = h[0];
    o[3] = h[1];
    o[4] = h[2];
    o[5] = (warm[j] && h[1] != h[2]) ? (h[0] - h[2]) / (h[1] - h[2]) : NAN;
  }
  free(ev), free(win), free(warm), free(hit);
  return rc;
}
