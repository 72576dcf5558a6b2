/*
 * unison.h -- C ABI of the GB300 implementation of UNISON's shared live
 * ranking (SPEAR score + TIDE fill) and its batched trace replay.
 *
 * Method: UNISON (arXiv 2609.09643).  Sec. III-A (problem statement:
 * sessions, turns, gaps, tiers, capacities, eqs. gap, reuse, cap), Sec. III-B
 * (SPEAR score, eqs. ema, hazard, surv, esp), Sec. III-C (TIDE, eqs. budget,
 * promote, demote), Sec. III-D (Algorithm 1, the joint event loop), Sec. IV-C
 * (the integer contract, eqs. uq, hq, survq, gapq, t1, t2, scoreq, ema-int,
 * lock) and Sec. V-A (metrics, eqs. hr-amat, prered, br).
 *
 * Conventions for every entry point:
 *  - Every function returns an int status: UNISON_OK (0) or a negative
 *    UNISON_ERR_* code.  Nothing aborts, traps or throws; a device-side
 *    problem is reported through the per-replay / per-set status word.
 *  - "host" pointers are ordinary CPU memory read during the call only;
 *    "device" pointers are CUDA global memory owned by the caller and must
 *    stay valid until the work queued on the stream has finished.
 *  - cuda_stream is a cudaStream_t (NULL = the legacy default stream).  Work
 *    is queued asynchronously on it, except where a host output is
 *    requested, in which case the call synchronises that stream.
 *  - Handles (unison_trace) are thread-compatible, not thread-safe.
 *  - Times are microseconds.  On the device they are 32-bit and wrap modulo
 *    2^32; every duration is a wrapping difference, which is exact because a
 *    loaded trace never has two consecutive events, a turn or a gap 2^31 us
 *    or more apart.
 */
#ifndef UNISON_H
#define UNISON_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---------------------------------------------------------------- status */
enum {
  UNISON_OK = 0,
  UNISON_ERR_ARG = -1,      /* null pointer, bad enum, inconsistent sizes      */
  UNISON_ERR_IO = -2,       /* file could not be opened or read                */
  UNISON_ERR_FORMAT = -3,   /* trace breaks its ordering rules                 */
  UNISON_ERR_RANGE = -4,    /* value beyond a documented limit (2^31 us gaps,  */
                            /* 2^24 sessions, 2^32 penalty, ...)               */
  UNISON_ERR_CUDA = -5,     /* a CUDA runtime call failed                      */
  UNISON_ERR_OOM = -6,      /* host or device allocation failed                */
  UNISON_ERR_LOG_FULL = -7, /* decision log capacity exceeded (replay goes on, */
                            /* counters and hash stay exact)                   */
  UNISON_ERR_TIMEOUT = -8,  /* a bounded device wait gave up                   */
  UNISON_ERR_CAPACITY = -9  /* internal resident-list bound exceeded           */
};

/* Human-readable text for a status code (static storage, never NULL). */
const char *unison_strerror(int code);

/* ABI version: major * 10000 + minor * 100 + patch. */
int unison_version(void);

/* ================================================================ traces */
/*
 * A trace is a set of agent sessions (Sec. III-A): session s has T_s turns;
 * turn k arrives at a_{s,k}, completes at c_{s,k}, needs in_tok tokens of
 * KV (l^in) and leaves out_tok resident (l^out, the prefix the next turn
 * reuses).  The tool gap before turn k is g_{s,k} = a_{s,k} - c_{s,k-1}
 * (eq. gap).
 *
 * Layout of unison_turns (host, caller-owned, read during the call):
 *   turn_off[n_sessions+1]  session s owns turns [turn_off[s], turn_off[s+1])
 *   arrival_us, completion_us [n_turns]  absolute times, u64 microseconds
 *   in_tok, out_tok [n_turns]
 * Rules (UNISON_ERR_FORMAT / _RANGE otherwise): 1 <= T_s < 65536;
 * n_sessions < 2^24 - 1; n_turns < 2^31; sessions are numbered in order of
 * first arrival; within a session a_k < c_k < a_{k+1}; c_k - a_k, gaps and
 * the spacing of consecutive events (in event order) are below 2^31 us;
 * 0 < in_tok_k <= out_tok_k and in_tok_k >= out_tok_{k-1}.
 *
 * Event order (a reading; the paper does not fix ties): by time, then
 * completions before arrivals, then session id.  A completion of a
 * non-final turn is a gap_start, an arrival of turn k >= 1 a gap_end
 * (Algorithm 1).
 */
typedef struct {
  uint32_t n_sessions;
  uint32_t reserved;
  uint64_t n_turns;
  const uint64_t *turn_off;
  const uint64_t *arrival_us;
  const uint64_t *completion_us;
  const uint32_t *in_tok;
  const uint32_t *out_tok;
} unison_turns;

typedef struct unison_trace unison_trace; /* opaque, library-owned */

/* Validate and order a trace on the host (events, per-turn event indices,
 * next-arrival indices).  *out receives a new handle; free it with
 * unison_trace_free.  No device memory is touched; the host copy is
 * page-locked (cudaMallocHost) when a CUDA driver is present, else ordinary
 * memory. */
int unison_trace_create(const unison_turns *turns, unison_trace **out);

/* Read a .utr file (little endian: "UTR1", u32 n_sessions, u64 n_turns,
 * u64 turn_off[S+1], u64 arrival[T], u64 completion[T], u32 in[T],
 * u32 out[T]) and create a trace from it. */
int unison_trace_load(const char *path, unison_trace **out);

/* Copy the trace's event arrays to device memory owned by the handle
 * (allocated on first upload, reused afterwards), asynchronously on
 * cuda_stream from page-locked host staging.  Must precede replay. */
int unison_trace_upload(unison_trace *tr, void *cuda_stream);

/* Release host and device memory of a trace (synchronises the device
 * memory's last stream).  NULL is ignored. */
void unison_trace_free(unison_trace *tr);

/* Sizes of a trace; any output pointer may be NULL. */
int unison_trace_info(const unison_trace *tr, uint32_t *n_sessions, uint64_t *n_turns,
                      uint64_t *n_events);

/* Bytes an upload copies host-to-device for this trace (the size of its
 * device block, fixed when the trace is created). */
uint64_t unison_trace_device_bytes(const unison_trace *tr);

/* ================================================================ replay */
typedef enum {
  UNISON_LRU = 0,        /* recency (Tab. main baseline)                       */
  UNISON_TIMEOUT = 1,    /* recency plus expiry of sessions idle >= ttl_us     */
  UNISON_SPEAR = 2,      /* SPEAR eviction only (Sec. III-B)                   */
  UNISON_SPEAR_TIDE = 3, /* UNISON: SPEAR + TIDE (Algorithm 1)                 */
  UNISON_BELADY = 4,     /* offline oracle: farthest next arrival (Sec. III-A) */
  UNISON_LRU_TIDE = 5    /* recency keys with TIDE migration (ablation)        */
} unison_policy;

/* Per-replay parameters (host array in unison_replay_batch). */
typedef struct {
  uint32_t policy;             /* unison_policy                                   */
  uint32_t trace_idx;          /* index into the traces[] argument                */
  uint64_t cap_fast_bytes;     /* C_S of eq. (cap), bytes                         */
  uint64_t cap_hbm_bytes;      /* C_H of eq. (cap), bytes                         */
  uint32_t kv_bytes_per_token; /* 1 .. 2^24; capacities count whole tokens        */
  uint32_t max_sessions;       /* N_sess of eq. (cap); 0 = no slot limit          */
  uint32_t ema_num, ema_den;   /* gap-average weight, eq. (ema-int): (3,10);      */
                               /* a window W reads as (2, W+1)                    */
  uint32_t hazard_bucket;      /* turns pooled per hazard entry; 1 = eq. (hazard) */
  uint32_t ttl_us;             /* Timeout idle limit < 2^31; 0xFFFFFFFF = none    */
  uint64_t penalty_q;          /* P_Z of eq. (t2), < 2^32; 5e8 = eq. (lock)       */
  uint64_t dma_bytes_per_us;   /* TIDE budget rate B (eq. budget) in bytes/us,    */
                               /* < 2^32                                          */
  uint64_t t_s_ps_per_tok;     /* AMAT per-token costs (eq. hr-amat), picoseconds */
  uint64_t t_h_ps_per_tok;
  uint64_t t_p_ps_per_tok;     /* prefill cost; TTFT uses t_p / 1000 ns per token */
  uint32_t ttft_load;          /* arrival compression factor of the TTFT queue    */
  uint32_t flags;              /* UNISON_HAZARD_ONLINE, UNISON_SIGNAL_*, or 0     */
  uint32_t stale_sync;         /* UNISON_SYNC_*: dual-design ablation, or 0       */
  uint32_t stale_m;            /* arrivals per sync for UNISON_SYNC_ARRIVALS      */
} unison_replay_params;

/* Stale-snapshot replays (Sec. IV-B eq. stale, Tab. org): the ranking of a
 * dual design whose engines copy the register file only at sync points.
 * Every ranking decision (make-room victims, slot-limit evictions, TIDE's
 * promotions and demotions) scores each session from its register row
 * (gap average, turn, done) as of the last sync; rows start at zero; a sync
 * copies every row after that event's own decisions; residency, sizes and
 * pins stay live.  Each acted-upon victim (promotion) choice is compared
 * with the choice by the live rows over the same candidates: the result's
 * vict_n / vict_diff (prom_n / prom_diff) count them.  UNISON_SYNC_EVENT
 * decides exactly as the live replay.  SPEAR and SPEAR+TIDE only, not with
 * UNISON_HAZARD_ONLINE, stale_m >= 1 for UNISON_SYNC_ARRIVALS (else
 * UNISON_ERR_ARG); the same shared-memory and session limits as the online
 * table apply, with 20 bytes per session (tier, pin slot, live and snapshot
 * keys, a changed flag) beside the power-of-two lists (else
 * UNISON_ERR_RANGE). */
#define UNISON_SYNC_LIVE 0u      /* no snapshot: the live ranking          */
#define UNISON_SYNC_EVENT 1u     /* copy after every event                 */
#define UNISON_SYNC_ARRIVALS 2u  /* copy after every stale_m-th arrival    */
#define UNISON_SYNC_GAP_START 3u /* copy after every non-final completion  */

/* Online hazard table (Sec. V-F, eq. attainment): instead of the table fitted
 * on the whole trace, the table starts with no sessions, and the turn count
 * of each session joins it at that session's final completion, which then
 * re-ranks every resident under the rebuilt table before the next event.
 * SPEAR and SPEAR+TIDE only (else UNISON_ERR_ARG); the trace must have at
 * most 32,768 sessions and the replay's resident lists, rounded up to powers
 * of two, plus 9 bytes per session (tier, pin slot, gap average, arrival
 * count) and the table must fit in shared memory (else UNISON_ERR_RANGE).
 * A bit of `flags` not defined here is UNISON_ERR_ARG. */
#define UNISON_HAZARD_ONLINE 1u

/* Signal leave-one-out (Sec. V-D, Fig. signal), SPEAR and SPEAR+TIDE only,
 * not with UNISON_HAZARD_ONLINE (else UNISON_ERR_ARG): the score drops one
 * of its two signals.  Without the gap recurrence it sees a gap average of 0
 * (score = T2 of the turn); without the hazard it sees sigma_q = Lambda, a
 * zero hazard (score = g_q).  TIDE's budget keeps the true gap average. */
#define UNISON_SIGNAL_NO_GAP 2u
#define UNISON_SIGNAL_NO_HAZARD 4u

/* Per-replay counters (written by the device). */
typedef struct {
  uint64_t events, req_warm, cold, hit_s, hit_h, miss, bypass, place_s, place_h;
  uint64_t evict, demote, promote, tide_demote, expire;
  uint64_t tok_hit_s, tok_hit_h, tok_miss; /* sums of l_i = l^out_{k-1} per class */
  uint64_t tok_computed, tok_needed;       /* prefill tokens vs tokens needed (warm) */
  uint64_t dma_bytes, tide_calls, promoted_then_hit_s;
  uint64_t ttft_sum_lo, ttft_sum_hi;       /* 128-bit sum of TTFT, ns              */
  uint64_t ttft_p50_ns, ttft_n;            /* lower median over all requests       */
  uint64_t decision_hash;                  /* see UNISON_KIND_* below              */
  uint64_t log_len;                        /* decisions made (logged or not)       */
  uint64_t vict_n, vict_diff;              /* stale snapshot: victim choices, and  */
  uint64_t prom_n, prom_diff;              /* promotions, unlike the live choice   */
  int32_t status;
  uint32_t reserved;
} unison_replay_result;

/* Decision kinds.  Each decision is logged as {event index, kind << 24 |
 * session}; decision_hash folds the stream in order, starting from
 * 0xCBF29CE484222325 and applying h = (h ^ w) * 0x100000001B3 (mod 2^64)
 * with w = event << 32 | kind << 24 | session.  Within one event the order
 * is: expiries (ascending session), the request class, then placement
 * decisions in the order they are taken, or the TIDE moves. */
enum {
  UNISON_KIND_COLD = 0, UNISON_KIND_HIT_S = 1, UNISON_KIND_HIT_H = 2, UNISON_KIND_MISS = 3,
  UNISON_KIND_PLACE_S = 4, UNISON_KIND_PLACE_H = 5, UNISON_KIND_BYPASS = 6,
  UNISON_KIND_DEMOTE = 7, UNISON_KIND_EVICT = 8, UNISON_KIND_PROMOTE = 9,
  UNISON_KIND_TIDE_DEMOTE = 10, UNISON_KIND_EXPIRE = 11
};
typedef struct {
  uint32_t event;
  uint32_t kind_session;
} unison_decision;

/*
 * Replay n_replays independent (trace, policy, parameters) combinations,
 * each one a literal run of Algorithm 1 over its trace's events:
 *  - gap_end: EMA update of the session's gap average (eq. ema-int);
 *  - every decision ranks the live sessions by one total order: larger key
 *    is more evictable, ties go to the smaller session id.  SPEAR keys are
 *    score_q (eq. scoreq; a completed session has the maximal key) from the
 *    offline hazard table fitted on the trace (Sec. V-E);
 *  - placement when a request arrives: the session leaves its tier and is
 *    placed in the fast tier if its l^out fits beside the pinned sessions,
 *    demoting the most evictable unpinned fast-tier sessions into HBM
 *    (where each displaces the most evictable unpinned HBM session, or is
 *    dropped itself if it is the most evictable); else in HBM, evicting the
 *    most evictable unpinned HBM sessions; else it is served and not kept.
 *    With max_sessions > 0, the global most evictable resident is evicted
 *    while the slot limit is exceeded.  A session is pinned from its
 *    arrival to its completion and never moved while pinned;
 *  - gap_start with TIDE and the DMA free: budget = g_q * dma_bytes_per_us
 *    (eq. budget); first the least evictable HBM sessions are promoted into
 *    free fast-tier space, then pairs (argmin over HBM, argmax over the
 *    fast tier; eqs. promote, demote) are swapped while the demoted one is
 *    strictly more evictable, the pair fits the remaining budget and both
 *    tiers stay within capacity.  The DMA is then busy for
 *    ceil(moved / dma_bytes_per_us) us.
 * Per-replay variants (definitions above): UNISON_HAZARD_ONLINE (the table
 * grows as sessions complete), UNISON_SIGNAL_NO_GAP / _NO_HAZARD (the score
 * without one signal), stale_sync (decisions on a register-file snapshot).
 * Replays of one call may mix policies and variants; each runs in the
 * launch for its kind, and a launch whose replays share the policy and
 * simple settings runs a kernel specialised for them.  SPEAR+TIDE replays
 * always run in their own launch.  The launches of one call are independent
 * and run concurrently: the first on cuda_stream, the others on side
 * streams the library owns (one set per device, made on the first call that
 * needs them), forked from cuda_stream and joined back to it before the
 * call's last kernel.  The call's work therefore stays ordered on
 * cuda_stream.  The call is not meant for stream capture: it copies its
 * descriptors from host memory that it frees when it returns.
 *
 * traces[n_traces]: uploaded handles (host array of pointers).
 * params[n_replays]: host array.
 * results_dev: device array [n_replays] written by the device (may be NULL
 *   if results_host is given).
 * results_host: host array [n_replays]; if non-NULL the call copies the
 *   results back and synchronises cuda_stream.
 * log_dev: device array [n_replays * log_capacity_per_replay] or NULL; replay
 *   r writes its decisions at log_dev + r * log_capacity_per_replay and sets
 *   status UNISON_ERR_LOG_FULL if it makes more.
 * Scratch (key streams, TTFT values, descriptors) is allocated
 * stream-ordered on cuda_stream and released before the call returns its
 * work to the stream.
 */
int unison_replay_batch(const unison_trace *const *traces, int n_traces,
                        const unison_replay_params *params, int n_replays,
                        unison_replay_result *results_dev, unison_replay_result *results_host,
                        unison_decision *log_dev, uint64_t log_capacity_per_replay,
                        void *cuda_stream);

/* Replay for callers that cannot allocate device memory.  The paper has no
 * counterpart to this entry point; it exists for the library's users.
 *
 * Some callers must not allocate: a serving runtime whose memory manager
 * reserves the device's whole budget up front and refuses allocations made
 * behind its back, or a latency-critical control loop that cannot afford an
 * allocator call (cudaMalloc and cudaFree may synchronise the device, and an
 * allocation can fail in the middle of a run).  This entry point replays
 * exactly like unison_replay_batch (same arguments, same results) but takes
 * its scratch from one fixed device array compiled into the library,
 * UNISON_NOALLOC_SCRATCH_BYTES long.  It calls no cudaMalloc, cudaFree or
 * other allocating routine.
 *  - When the array and other set-up come into being: CUDA loads a library's
 *    device code lazily by default, so the array is created on a device when
 *    the library first launches a kernel or looks up the array there (this
 *    entry point's first call on the device at the latest), and that device
 *    holds it until the process exits.  The first call on a device whose
 *    batch needs more than one launch group (policies other than SPEAR+TIDE
 *    beside it, online-table or stale-snapshot replays) also creates the
 *    library's side streams and their events there.  A caller whose memory
 *    manager will later own the whole device should therefore make its first
 *    call, with the kinds of replays it will run, during start-up.
 *  - results_dev is required (the caller provides the output buffer);
 *    results_host, log_dev and the traces are as in unison_replay_batch.
 *    The traces must already be uploaded (unison_trace_upload allocates, so
 *    upload them beforehand).
 *  - A batch whose scratch (descriptors, hazard tables, 12 B per event per
 *    key stream, 8 B per request per replay, resident lists that do not fit
 *    in shared memory) exceeds UNISON_NOALLOC_SCRATCH_BYTES is rejected with
 *    UNISON_ERR_RANGE before anything is queued.
 *  - The first call on a device looks up the array's device address on that
 *    device (cudaGetSymbolAddress, with that device current).  Like
 *    unison_replay_batch, the call is not meant for stream capture.
 *  - All calls share the one array, which keeps what the last call left in
 *    it; each call writes every region it reads before reading it, so no
 *    region needs clearing.  Calls whose work overlaps on the GPU (on
 *    different streams or from different threads) race on the array: queue
 *    them on one stream or order them. */
#define UNISON_NOALLOC_SCRATCH_BYTES (32ull << 20)
int unison_replay_batch_noalloc(const unison_trace *const *traces, int n_traces,
                                const unison_replay_params *params, int n_replays,
                                unison_replay_result *results_dev, unison_replay_result *results_host,
                                unison_decision *log_dev, uint64_t log_capacity_per_replay,
                                void *cuda_stream);

/* Host-side summary of one replay (Sec. V-A): hit rate HR = (H_S + H_H)/R,
 * AMAT = (t_s sum_S + t_h sum_H + t_p sum_M)/R in ps (eq. hr-amat), prefill
 * reduction 1 - computed/needed (eq. prered), prefetch accuracy = promoted
 * sessions whose next request hit the fast tier / promotions, TTFT mean and
 * p50 in ns.  Ratios with an empty denominator are 0. */
typedef struct {
  double hit_rate, amat_ps, prered, prefetch_acc, ttft_mean_ns, ttft_p50_ns;
} unison_stats_t;
int unison_stats(const unison_replay_result *r, const unison_replay_params *p, unison_stats_t *out);

/* Agent Serving Effectiveness (Sec. IV-E, eq. ase) of n_configs
 * configurations compared over n_datasets datasets (traces):
 *   ASE_c = ( prod_d  HR_cd / HR_d^max  *  AMAT_d^min / AMAT_cd
 *                     *  TTFT_d^min / TTFT_cd ) ^ (1 / (3 n_datasets)),
 * the extremes taken over the n_configs configurations of dataset d.
 * stats: host array [n_configs][n_datasets] of unison_stats outputs (TTFT is
 * ttft_mean_ns); ase_out: host double[n_configs], each in [0, 1].  Readings:
 * a ratio 0/0 (every configuration at 0) counts as 1; a zero AMAT or TTFT
 * minimum against a positive value gives a factor 0, so ASE_c = 0.
 * n_configs, n_datasets >= 1, else UNISON_ERR_ARG; a negative or non-finite
 * metric gives UNISON_ERR_RANGE. */
int unison_ase(const unison_stats_t *stats, int n_configs, int n_datasets, double *ase_out);

/* Attainment A(n) (Sec. V-F, eq. attainment) of an online-table replay
 * (UNISON_HAZARD_ONLINE) against the offline-table and LRU replays of the
 * same trace:  A = (H_on - H_LRU) / (H_off - H_LRU), H a hit rate.  Reading:
 * "after n observed sessions" is a window of the trace, the warm requests
 * (decisions HIT_S, HIT_H, MISS) arriving while n_j <= n < n_{j+1} sessions
 * have completed, n_j = floor(j N / n_points), j = 0 .. n_points-1, N the
 * trace's sessions; the last window runs to the end of the trace.  Window j
 * fills out[j]: n_j, its warm requests, the three hit rates over them, and A
 * (NaN when the window holds no warm request or H_off = H_LRU).
 * trace: a handle from unison_trace_create/_load (host data only is read);
 * logs: host copies of the three replays' complete decision logs (len =
 * the result's log_len, which must not exceed the capacity used).
 * Errors: a null pointer -> UNISON_ERR_ARG; n_points = 0 or > N ->
 * UNISON_ERR_RANGE; an event index outside the trace, or logs that disagree
 * on which events are warm requests -> UNISON_ERR_FORMAT. */
typedef struct {
  uint32_t sessions_seen;  /* n_j */
  uint32_t reserved;
  uint64_t warm;           /* warm requests in the window */
  double hr_online, hr_offline, hr_lru;
  double attainment;
} unison_attainment_point;

int unison_attainment(const unison_trace *trace, const unison_decision *log_online, uint64_t len_online,
                      const unison_decision *log_offline, uint64_t len_offline, const unison_decision *log_lru,
                      uint64_t len_lru, uint32_t n_points, unison_attainment_point *out);

/* Device self-check of the division every score of eq. (t1) uses:
 * floor(x / s) as the high word of x times a magic number (Granlund and
 * Montgomery), for x < 2^43 and 2 <= s < 2^12.  Checks every divisor s in
 * [2, 4095] at every x < 2^20 and at x = q*s - 1, q*s, q*s + s - 1 for 2^16
 * quotients q per divisor spread up to the largest below 2^43, each against
 * q*s <= x < (q+1)*s.  *mismatches (host) receives the number of failures;
 * the call synchronises cuda_stream.  NULL mismatches: UNISON_ERR_ARG. */
int unison_selftest_division(uint64_t *mismatches, void *cuda_stream);

/* Fault injection for error-path tests (host side only): the next n device
 * allocations the library makes -- a replay call's scratch, the ranking
 * scratch when it grows, a trace's device block at its first upload -- fail
 * as if the device were out of memory, and those calls return
 * UNISON_ERR_OOM.  n <= 0 clears pending faults. */
void unison_debug_fail_allocations(int n);

/* ============================================================ hazard LUT */
/* The survival table of eqs. (hazard), (hq), (survq) built on the device
 * from turns-per-session counts: n(t) = #{T_s >= t+1}, d(t) = #{T_s = t+1}
 * for t = 0..50, pooled over buckets of `bucket` consecutive turns,
 * h_q = round-half-up(4095 d / n) (0 where n = 0), sigma_q = max(41,
 * 4095 - h_q).  turns_dev: device u32[n_sessions]; sigma_q_dev: device
 * u16[51] output (h_q_dev, device u16[51], may be NULL). */
int unison_hazard_lut(const uint32_t *turns_dev, uint64_t n_sessions, uint32_t bucket,
                      uint16_t *sigma_q_dev, uint16_t *h_q_dev, void *cuda_stream);

/* ================================================================ ranking */
/* A live set of n session records, structure of arrays, device memory
 * (caller-owned).  gap_q: gap average in us (eq. gapq, < 2^31: the device
 * does not check it, and a larger value gives an unspecified key); last_ret:
 * last completion time (carried, not read by the score); turn: register turn
 * t; kv_tok: resident tokens; tier: 1 fast, 2 HBM, other = not resident;
 * flags: bit0 pinned (mid-turn), bit1 done (completed session).  1 <= n <= 2^24
 * (the index is packed into 24 bits of the ranking key); gap_q, turn, tier
 * and flags must start on 16-byte boundaries (they are streamed with bulk
 * copies), else UNISON_ERR_ARG. */
typedef struct {
  const uint32_t *gap_q;
  const uint32_t *last_ret;
  const uint16_t *turn;
  const uint32_t *kv_tok;
  const uint8_t *tier;
  const uint8_t *flags;
  uint64_t n;
} unison_records;

typedef struct {
  uint16_t sigma_q[51];        /* survival table (unison_hazard_lut), host copy  */
  uint16_t reserved0;
  uint32_t k;                  /* victims wanted, 0 .. 4096 (else _RANGE)        */
  uint64_t penalty_q;          /* P_Z, < 2^32                                    */
  uint64_t budget_bytes;       /* TIDE budget for this set                       */
  uint32_t kv_bytes_per_token; /* 1 .. 2^24                                      */
  uint32_t max_moves;          /* cap on promotions (and on promote[] / demote[] */
                               /* capacity), 0 .. 4096                           */
  uint64_t free_fast_tok;      /* free fast-tier capacity, tokens                */
  uint64_t free_hbm_tok;       /* free HBM capacity, tokens                      */
} unison_rank_params;

/* Device outputs of one set (caller-owned). */
typedef struct {
  uint32_t *victims;     /* [k]: most evictable unpinned resident records first */
  uint32_t *promote;     /* [max_moves]: HBM -> fast, in move order             */
  uint32_t *demote;      /* [max_moves]: fast -> HBM, paired with promotions    */
                         /* after the free-space promotions                     */
  uint32_t *counts;      /* [4]: n_victims, n_promote, n_demote, status         */
  uint64_t *moved_bytes; /* [1]                                                 */
  uint64_t *keys;        /* [n] score_q of every record, or NULL                */
} unison_rank_out;

/*
 * Rank n_sets live sets in one pass over their records (the scan of
 * eq. pipe/scan with the victim argmax generalised to a top-k, and one TIDE
 * fill per set with the selections of eqs. promote/demote).  Keys are
 * score_q (eq. scoreq); order as in replay (larger key, then smaller index,
 * is more evictable).  Results are exact: candidate thresholds come from a
 * sample, and a set whose candidates fall short is re-selected exactly on
 * the device.  sets, params, outs: host arrays [n_sets].  Asynchronous: the
 * call queues one upload of its descriptors and one cooperative kernel on
 * cuda_stream (every CTA of the grid resident at once; each set is ranked
 * by a group of CTAs, or, with more sets than resident CTAs, each CTA takes
 * whole sets in turn).  Any n_sets >= 0 that fits in memory is accepted.
 * Memory: the call's device scratch (about 1.7 MB per set) is kept per
 * (device, stream) and grown when a call needs more, and the per-call
 * descriptors go up from a small pinned host ring; both are held for the
 * life of the process.  Calls on one stream run in order and share that
 * stream's scratch; calls on different streams use different scratch.  The
 * scratch is found by the stream's handle, so a stream must outlive the
 * ranking calls queued on it.
 * Errors: UNISON_ERR_ARG (null or misaligned arrays), UNISON_ERR_RANGE
 * (limits above), UNISON_ERR_OOM (scratch or staging), UNISON_ERR_CUDA
 * (launch; a device without cooperative launch); a bounded device wait that
 * gives up sets counts[3] of its set to UNISON_ERR_TIMEOUT.
 */
int unison_rank_batch(const unison_records *sets, const unison_rank_params *params,
                      const unison_rank_out *outs, int n_sets, void *cuda_stream);

/* One live set: the ranking of Sec. IV-D and the TIDE fill of Sec. III-C
 * (eqs. scoreq, pipe/scan, promote, demote, budget) for a single set, with
 * the same arguments, outputs, limits and errors as unison_rank_batch with
 * n_sets = 1 (records, params and out point to one element each). */
int unison_rank(const unison_records *records, const unison_rank_params *params,
                const unison_rank_out *out, void *cuda_stream);

/* Record-sharded ranking of one live set over several GPUs (Sec. IV-D's
 * scan and Sec. III-C's selections, eqs. promote/demote, split by records).
 * Each GPU ranks its slice -- records [index_offset, index_offset + n) of
 * the whole set, 16-byte-aligned device arrays as for unison_rank -- and
 * writes its candidate lists to cands_dev: its k most evictable unpinned
 * records (V), its max_moves most evictable unpinned fast-tier records (D)
 * and its max_moves least evictable unpinned HBM records (P), each in
 * ranking order with its KV size, keyed by its index in the whole set.  The
 * global top-k of V, and the first max_moves of D and of P, lie in the union
 * of the slices' lists, so after one all-gather of the fixed-size buffers
 * (n_shards x unison_rank_cands_bytes(k, max_moves), in any order) every GPU
 * runs unison_rank_merge, which selects the global lists and runs the TIDE
 * fill exactly as unison_rank does for the whole set: the outputs are equal.
 * params must be the same on every GPU (budget and free tier capacities are
 * the whole set's).  index_offset + n <= 2^24 (the index is packed into 24
 * bits of the ranking key), else UNISON_ERR_RANGE.  cands_dev: device,
 * caller-owned, 256-byte aligned, at least unison_rank_cands_bytes(k,
 * max_moves) bytes; gathered_dev: n_shards such buffers back to back.
 * Errors as for unison_rank_batch; asynchronous on cuda_stream. */
uint64_t unison_rank_cands_bytes(uint32_t k, uint32_t max_moves);
int unison_rank_shard(const unison_records *slice, uint64_t index_offset, const unison_rank_params *params,
                      void *cands_dev, void *cuda_stream);
int unison_rank_merge(const void *gathered_dev, int n_shards, const unison_rank_params *params,
                      const unison_rank_out *out, void *cuda_stream);

/* ============================================================ measurement */
/* While enabled (on != 0), every replay and ranking call records a pair of
 * CUDA events on its own stream around each launch of its main kernels
 * ("replay" = the event loop, "key_stream", "ttft_median", "rank" = the
 * whole ranking kernel).  Not thread-safe; meant for benchmarks. */
int unison_profile_enable(int on);

/* Synchronise the recorded events of one kernel name and return the summed
 * device time (ms) and the number of timed launches since the last reset;
 * reset != 0 then discards that kernel's records.  Unknown names give 0. */
int unison_profile_read(const char *kernel, double *total_ms, uint64_t *launches, int reset);

/* Number of kernels this library has launched since it was loaded. */
uint64_t unison_launch_count(void);

#ifdef __cplusplus
}
#endif
#endif /* UNISON_H */
