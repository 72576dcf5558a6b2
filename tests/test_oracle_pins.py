"""Pins for the CPU oracle: hand-worked values, closed forms, textbook
special cases, brute force on tiny inputs and invariants.  None of these
re-types the oracle's code; each fixes a fact the paper or the mathematics
determines, so a dropped term, swapped operand or flipped order fails one."""
import itertools
import math
import os

import numpy as np
import pytest

import oracle
import synth

GOLD = os.path.join(os.path.dirname(__file__), "golden")
BIG = 1 << 60


def _rows(name):
    with open(os.path.join(GOLD, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                yield line


# ---------------------------------------------------------------- score ----

def test_locked_constants():
    # eq. (survq): eps_q = floor(0.01 * 4095 + 1/2) = 41; h = 1 saturates at it
    assert oracle.spear_score(1000, 41) == oracle.spear_score(1000, 41)
    h, s = oracle.hazard_lut([1] * 10)  # every session ends at turn 0 -> h(0) = 1
    assert int(h[0]) == 4095 and int(s[0]) == 41
    assert int(s[1]) == 4095  # n(1) = 0 -> h = 0


def test_score_hand_values():
    for row in _rows("spear_score_hand.txt"):
        g, hn, hd, hq, sq, t1, t2, score = map(int, row.split())
        # the hazard quantiser via a one-turn-type population: hd sessions of
        # which hn end at turn 0 gives h(0) = hn / hd
        h, s = oracle.hazard_lut([1] * hn + [2] * (hd - hn))
        assert int(h[0]) == hq and int(s[0]) == sq
        assert oracle.spear_score(g, sq) == score == t1 + t2


def test_score_done_is_max():
    assert oracle.spear_score(123, 4095, done=True) == 2 ** 64 - 1


def test_score_within_float_bound():
    """eq. (esp) in floating point (g/sigma + (1 - sigma) P with sigma = sigma_q / Lambda)
    minus the fixed-point score lies in [0, 2): two floors, nothing else."""
    rs = np.random.default_rng(5)
    for _ in range(3000):
        g = int(rs.integers(0, 2 ** 31))
        sq = int(rs.integers(41, 4096))
        sig = sq / 4095.0
        flt = g / sig + (1.0 - sig) * 5e8
        fix = oracle.spear_score(g, sq)
        assert -1e-6 * flt - 1e-3 <= flt - fix < 2 + 1e-6 * flt


def test_score_monotone_in_gap_and_hazard():
    for sq in (41, 1000, 3919, 4095):
        vals = [oracle.spear_score(g, sq) for g in range(0, 10 ** 6, 9973)]
        assert all(a <= b for a, b in zip(vals, vals[1:]))
    # lower survival (higher hazard) never lowers the score at fixed gap
    for g in (0, 10 ** 5, 3 * 10 ** 6):
        vals = [oracle.spear_score(g, sq) for sq in range(4095, 40, -37)]
        assert all(a <= b for a, b in zip(vals, vals[1:]))


def test_zero_hazard_is_gap_order():
    # closed form: h = 0 -> sigma_q = Lambda -> score_q = g_q exactly
    for g in (0, 1, 977, 2 ** 31 - 1):
        assert oracle.spear_score(g, 4095) == g


# ------------------------------------------------------------------ EMA ----

def test_ema_hand_values():
    for row in _rows("ema_hand.txt"):
        g0, gn, g1 = map(int, row.split())
        assert oracle.ema(g0, gn) == g1


def test_ema_constant_gap_converges_from_below():
    g = 0
    for _ in range(200):
        g = oracle.ema(g, 1_234_567)
        assert g <= 1_234_567
    assert 1_234_567 - 10 <= g <= 1_234_567


def test_ema_window_weight():
    # span-W EMA (2, W+1): one step from 0 gives floor(2x/(W+1))
    for w in (4, 8, 16, 32):
        assert oracle.ema(0, 999_999, 2, w + 1) == (2 * 999_999) // (w + 1)


# --------------------------------------------------------------- hazard ----

def test_hazard_hand_counts():
    # T_s = [1,2,2,3]: n = 4,3,1 ; d = 1,2,1 ; h = 1/4, 2/3, 1
    h, s = oracle.hazard_lut([1, 2, 2, 3])
    assert list(map(int, h[:4])) == [1024, 2730, 4095, 0]
    assert list(map(int, s[:4])) == [3071, 1365, 41, 4095]
    # bucket width 2 pools t = 0,1: 3/7 -> floor(1755 + 1/2) = 1755
    h2, _ = oracle.hazard_lut([1, 2, 2, 3], 2)
    assert int(h2[0]) == int(h2[1]) == 1755
    assert int(h2[2]) == 4095  # {2,3}: d = 1, n = 1


def test_hazard_fixed_turns():
    # every session exactly 12 turns: h(t) = 0 except h(11) = 1
    h, s = oracle.hazard_lut([12] * 64)
    assert int(h[11]) == 4095 and int(s[11]) == 41
    assert all(int(h[t]) == 0 for t in range(51) if t != 11)


def test_hazard_matches_brute_counts_and_rounding():
    tps = synth.geometric_turns(3, 5000, 23.7, 2, 200)
    for w in (1, 2, 4, 8, 64):
        h, s = oracle.hazard_lut(tps, w)
        for t in range(51):
            bucket = [u for u in range(51) if u // w == t // w]
            n = sum(int((tps >= u + 1).sum()) for u in bucket)
            d = sum(int((tps == u + 1).sum()) for u in bucket)
            x = d / n if n else 0.0
            assert abs(int(h[t]) - x * 4095) <= 0.5 + 1e-9  # round to nearest
            assert int(s[t]) == max(41, 4095 - int(h[t]))
        if w >= 51:
            assert len(set(map(int, h))) == 1


def test_hazard_geometric_nearly_constant():
    # memoryless turns: h(t) ~ p for t >= 2, h(0) = 0 since T_s >= 2
    tps = synth.geometric_turns(11, 200000, 23.7, 2, 200)
    h, _ = oracle.hazard_lut(tps)
    assert int(h[0]) == 0
    assert all(abs(int(h[t]) - 4095 / 23.7) < 25 for t in range(2, 30))


# -------------------------------------------------------- hand replay ----

def _hand_trace(name):
    turns, log, counts = {}, [], {}
    for row in _rows(name):
        tag, *rest = row.split()
        if tag == "trace":
            s, k, a, c, i, o = map(int, rest)
            turns.setdefault(s, []).append((k, a, c, i, o))
        elif tag == "log":
            log.append((int(rest[0]), oracle.KINDS.index(rest[1]), int(rest[2])))
        elif tag == "count":
            counts[rest[0]] = int(rest[1])
    sess = [sorted(turns[s]) for s in sorted(turns)]
    tr = synth.trace_from_turns([[t[1] for t in x] for x in sess], [[t[2] for t in x] for x in sess],
                                [[t[3] for t in x] for x in sess], [[t[4] for t in x] for x in sess])
    return tr, log, counts


HAND_PARAMS = dict(policy="spear", kv_bytes_per_token=1, cap_s_bytes=100, cap_h_bytes=100,
                   t_p_ps_per_tok=20_000_000, ttft_load=4)


def test_hand_replay_spear():
    tr, log, counts = _hand_trace("replay_hand_spear.txt")
    r = oracle.replay(tr, HAND_PARAMS, log=True, debug=True)
    assert r["status"] == 0
    got = list(zip(*(map(int, a) for a in r["log"])))
    assert got == log
    for k, v in counts.items():
        assert r[k] == v, k


HAND_TIDE_PARAMS = dict(policy="spear_tide", kv_bytes_per_token=1, cap_s_bytes=100, cap_h_bytes=1000,
                        dma_bytes_per_us=4, t_p_ps_per_tok=20_000_000, ttft_load=4)


def test_hand_replay_spear_tide():
    """Sec. III-C inside a replay, worked by hand: a phase-1 promotion beside
    pinned fast-tier sessions, a phase-2 stop on the order test and one on
    the budget, a gap_start inside the DMA-busy window and one exactly at its
    end, and prefetch accuracy over a promoted session that hits the fast
    tier and one that was demoted before its next request."""
    tr, log, counts = _hand_trace("replay_hand_tide.txt")
    r = oracle.replay(tr, HAND_TIDE_PARAMS, log=True, debug=True)
    assert r["status"] == 0
    got = list(zip(*(map(int, a) for a in r["log"])))
    assert got == log
    for k, v in counts.items():
        assert r[k] == v, k


def test_tide_unaffordable_budget_equals_spear():
    """Closed form of eq. (budget): if g_q * B is below the cost of the
    smallest possible move (its tokens x kvB) at every gap_start, TIDE runs
    and moves nothing, so SPEAR+TIDE decides exactly as SPEAR.  The gap
    average is a convex combination of observed gaps (eq. ema-int), so the
    largest gap of the trace bounds it."""
    tr = synth.paper_scale_trace(1, "coding")
    kvb = 1 << 24
    max_gap = int(max(np.max(tr.arrival_us[i + 1:j] - tr.completion_us[i:j - 1]) if j - i > 1 else 0
                      for i, j in zip(tr.turn_off[:-1], tr.turn_off[1:])))
    min_cost = int(np.min(tr.out_tok)) * kvb
    rate = (min_cost - 1) // max_gap
    assert rate >= 1
    p = dict(kv_bytes_per_token=kvb, cap_s_bytes=4 << 40, cap_h_bytes=64 << 40, dma_bytes_per_us=rate)
    a = oracle.replay(tr, dict(p, policy="spear_tide"), log=True)
    b = oracle.replay(tr, dict(p, policy="spear"), log=True)
    assert a["status"] == b["status"] == 0
    assert a["tide_calls"] > 1000 and a["promote"] == a["tide_demote"] == a["dma_bytes"] == 0
    assert a["decision_hash"] == b["decision_hash"]
    for x, y in zip(a["log"], b["log"]):
        assert np.array_equal(x, y)
    # at 64 times that rate some move becomes affordable: the bound is not vacuous
    c = oracle.replay(tr, dict(p, policy="spear_tide", dma_bytes_per_us=64 * rate))
    assert c["promote"] > 0


# ------------------------------------------------------ capacity extremes ----

POLICIES = ["lru", "timeout", "spear", "spear_tide", "belady", "lru_tide"]


@pytest.mark.parametrize("pol", POLICIES)
def test_infinite_capacity_all_warm_hits(pol):
    tr = synth.tiny_trace(3)
    r = oracle.replay(tr, dict(policy=pol, cap_s_bytes=BIG, cap_h_bytes=BIG, kv_bytes_per_token=28672,
                               ttl_us=0xFFFFFFFF), debug=True)
    assert r["status"] == 0
    assert r["hit_s"] == r["req_warm"] == tr.n_turns - tr.n_sessions
    assert r["evict"] == r["demote"] == r["expire"] == r["miss"] == 0


@pytest.mark.parametrize("pol", POLICIES)
def test_zero_capacity_all_bypass(pol):
    tr = synth.tiny_trace(4)
    r = oracle.replay(tr, dict(policy=pol, cap_s_bytes=0, cap_h_bytes=0, kv_bytes_per_token=28672),
                      debug=True)
    assert r["status"] == 0
    assert r["bypass"] == tr.n_turns and r["hit_s"] == r["hit_h"] == 0
    assert r["miss"] == r["req_warm"]
    assert r["tok_computed"] == r["tok_needed"]


@pytest.mark.parametrize("pol", POLICIES)
def test_no_fast_tier_no_fast_hits(pol):
    tr = synth.paper_scale_trace(2)
    r = oracle.replay(tr, dict(policy=pol, cap_s_bytes=0, cap_h_bytes=16 << 30), debug=False)
    assert r["status"] == 0 and r["hit_s"] == 0 and r["place_s"] == 0 and r["hit_h"] > 0


# ------------------------------------------------------- slot-mode pins ----

def _slot_trace(seq):
    """Arrivals on a 1 ms grid in the given session order, 1 us of service,
    one token each (sessions numbered by first arrival)."""
    order = []
    for s in seq:
        if s not in order:
            order.append(s)
    ren = {s: i for i, s in enumerate(order)}
    seq = [ren[s] for s in seq]
    arr = [[] for _ in order]
    for i, s in enumerate(seq):
        arr[s].append(1000 * (i + 1))
    tr = synth.trace_from_turns(arr, [[a + 1 for a in x] for x in arr],
                                [[1] * len(x) for x in arr], [[1] * len(x) for x in arr])
    return tr, seq


SLOT = dict(cap_s_bytes=0, cap_h_bytes=BIG, kv_bytes_per_token=1)


def _brute_max_hits(seq, n_slots):
    best = 0

    def go(i, cache, hits):
        nonlocal best
        if i == len(seq):
            best = max(best, hits)
            return
        s = seq[i]
        warm = s in seq[:i]
        if s in cache:
            go(i + 1, cache, hits + (1 if warm else 0))
            return
        if len(cache) < n_slots:
            go(i + 1, cache | {s}, hits)
            return
        for v in cache:
            go(i + 1, (cache - {v}) | {s}, hits)

    go(0, frozenset(), 0)
    return best


def _random_seqs(n, seed):
    rs = np.random.default_rng(seed)
    for _ in range(n):
        ns = int(rs.integers(2, 7))
        ln = int(rs.integers(4, 13))
        seq = list(map(int, rs.integers(0, ns, ln)))
        # at most 4 turns per session
        cnt = {}
        out = []
        for s in seq:
            cnt[s] = cnt.get(s, 0) + 1
            if cnt[s] <= 4:
                out.append(s)
        yield out


@pytest.mark.parametrize("slots", [1, 2, 3])
def test_belady_is_optimal_bruteforce(slots):
    for seq in _random_seqs(60, 100 + slots):
        tr, seq = _slot_trace(seq)
        r = oracle.replay(tr, dict(SLOT, policy="belady", max_sessions=slots), debug=True)
        assert r["status"] == 0
        assert r["hit_h"] + r["hit_s"] == _brute_max_hits(seq, slots), seq


@pytest.mark.parametrize("slots", [1, 2, 3])
def test_lru_matches_stack_distance(slots):
    for seq in _random_seqs(60, 200 + slots):
        tr, seq = _slot_trace(seq)
        r = oracle.replay(tr, dict(SLOT, policy="lru", max_sessions=slots), debug=True)
        hits = 0
        for i, s in enumerate(seq):
            prev = [j for j in range(i) if seq[j] == s]
            if prev:
                dist = len(set(seq[prev[-1] + 1:i]))
                hits += dist < slots
        assert r["status"] == 0 and r["hit_h"] == hits, seq


def test_timeout_limits():
    tr = synth.tiny_trace(5)
    base = dict(cap_s_bytes=512 << 20, cap_h_bytes=8 << 30, kv_bytes_per_token=28672)
    lru = oracle.replay(tr, dict(base, policy="lru"), log=True)
    inf = oracle.replay(tr, dict(base, policy="timeout", ttl_us=0xFFFFFFFF), log=True)
    assert lru["decision_hash"] == inf["decision_hash"]
    zero = oracle.replay(tr, dict(base, policy="timeout", ttl_us=0))
    assert zero["status"] == 0 and zero["hit_s"] == zero["hit_h"] == 0
    assert zero["miss"] == zero["req_warm"]


# ------------------------------------------------------------------ TIDE ----

def test_tide_zero_budget_equals_spear():
    tr = synth.paper_scale_trace(3)
    base = dict(cap_s_bytes=2 << 30, cap_h_bytes=32 << 30, kv_bytes_per_token=131072)
    a = oracle.replay(tr, dict(base, policy="spear"))
    b = oracle.replay(tr, dict(base, policy="spear_tide", dma_bytes_per_us=0))
    assert a["decision_hash"] == b["decision_hash"] and b["promote"] == 0 and b["tide_calls"] > 0


def test_tide_loop_equals_list_form_and_invariants():
    """Debug replays check, at every TIDE call, that the literal pair loop
    and the sorted-list form move the same sessions, and at every event the
    capacity and pinning invariants."""
    for seed, kv, cs, ch, dma in [(0, 28672, 512 << 20, 8 << 30, 64000), (1, 131072, 1 << 30, 32 << 30, 64000),
                                  (2, 131072, 8 << 30, 32 << 30, 640000), (3, 28672, 4 << 30, 64 << 30, 6400)]:
        tr = synth.paper_scale_trace(seed) if seed else synth.tiny_trace(0)
        r = oracle.replay(tr, dict(policy="spear_tide", cap_s_bytes=cs, cap_h_bytes=ch,
                                   kv_bytes_per_token=kv, dma_bytes_per_us=dma), debug=True)
        assert r["status"] == 0 and r["promote"] > 0
        assert r["dma_bytes"] <= r["tide_calls"] * (2 ** 31) * dma


def test_tide_unlimited_budget_sorts_tiers():
    """With an unbounded budget and sessions of one size, TIDE leaves the
    least evictable unpinned sessions in the fast tier (Sec. III-C)."""
    rs = np.random.default_rng(9)
    for trial in range(20):
        n = 12
        rec = synth.Records(gap_q=rs.integers(0, 10 ** 6, n).astype(np.uint32),
                            last_ret=np.zeros(n, np.uint32), turn=np.zeros(n, np.uint16),
                            kv_tok=np.full(n, 7, np.uint32),
                            tier=np.where(rs.random(n) < 0.4, 1, 2).astype(np.uint8),
                            flags=np.zeros(n, np.uint8))
        sig = np.full(51, 4095, np.uint16)
        out = oracle.rank(rec, sig, 0, 1, 10 ** 12, 1, 0, 10 ** 9)
        tier = rec.tier.copy()
        tier[out["promote"]] = 1
        tier[out["demote"]] = 2
        n_s = int((rec.tier == 1).sum())
        order = sorted(range(n), key=lambda i: (int(rec.gap_q[i]), -i))  # least evictable first
        assert set(np.nonzero(tier == 1)[0]) == set(order[:n_s])


def test_rank_hand_values():
    recs = []
    checks = []
    for row in _rows("rank_hand.txt"):
        tag, *rest = row.split()
        if tag == "rec":
            recs.append(list(map(int, rest)))
        else:
            checks.append((tag, rest))
    a = np.array(recs)
    rec = synth.Records(a[:, 1].astype(np.uint32), np.zeros(len(a), np.uint32), np.zeros(len(a), np.uint16),
                        a[:, 3].astype(np.uint32), a[:, 2].astype(np.uint8), a[:, 4].astype(np.uint8))
    sig = np.full(51, 4095, np.uint16)
    for tag, rest in checks:
        if tag == "victims":
            k = int(rest[0])
            out = oracle.rank(rec, sig, 5 * 10 ** 8, k, 0, 1, 0, 0)
            assert list(map(int, out["victims"])) == list(map(int, rest[2:]))
        else:
            parts = " ".join(rest).split(":")
            budget, fs, fh = map(int, parts[0].split())
            pro = list(map(int, parts[1].split()[1:]))
            dem = list(map(int, parts[2].split()[1:]))
            moved = int(parts[3].split()[1])
            out = oracle.rank(rec, sig, 5 * 10 ** 8, 1, budget, 1, fs, fh)
            assert list(map(int, out["promote"])) == pro
            assert list(map(int, out["demote"])) == dem
            assert out["moved_bytes"] == moved


def test_rank_victims_are_sorted_topk():
    rec = synth.make_records(12, 5000)
    _, sig = oracle.hazard_lut(synth.geometric_turns(1, 1415, 23.7, 2, 200))
    out = oracle.rank(rec, sig, 5 * 10 ** 8, 300, 0, 131072, 0, 0, keys=True)
    keys = out["keys"]
    cand = [i for i in range(rec.n) if not (rec.flags[i] & 1)]
    best = sorted(cand, key=lambda i: (-int(keys[i]), i))[:300]
    assert list(map(int, out["victims"])) == best
    done = (rec.flags & 2) != 0
    assert (keys[done] == 2 ** 64 - 1).all()


# ------------------------------------------------------------ invariance ----

def test_time_shift_invariance():
    tr = synth.tiny_trace(6)
    p = dict(policy="spear_tide", cap_s_bytes=512 << 20, cap_h_bytes=8 << 30, kv_bytes_per_token=28672)
    a = oracle.replay(tr, p, log=True)
    sh = synth.Trace(tr.turn_off, tr.arrival_us + np.uint64(3 << 32), tr.completion_us + np.uint64(3 << 32),
                     tr.in_tok, tr.out_tok)
    b = oracle.replay(sh, p, log=True)
    assert a["decision_hash"] == b["decision_hash"] and a["ttft_sum"] == b["ttft_sum"]


def test_trace_validation_rejects_bad_input():
    tr = synth.tiny_trace(0)
    bad = synth.Trace(tr.turn_off, tr.arrival_us.copy(), tr.completion_us.copy(), tr.in_tok, tr.out_tok)
    bad.completion_us[3] = bad.arrival_us[3]  # zero-length turn
    assert oracle.replay(bad, {})["status"] == -3
    gap = synth.Trace(tr.turn_off, tr.arrival_us.copy(), tr.completion_us.copy(), tr.in_tok, tr.out_tok)
    gap.arrival_us[5:12] += np.uint64(1 << 31)
    gap.completion_us[5:12] += np.uint64(1 << 31)
    assert oracle.replay(gap, {})["status"] == -4
    assert oracle.replay(tr, dict(ttl_us=1 << 31, policy="timeout"))["status"] == -1


def test_log_overflow_is_reported():
    tr = synth.tiny_trace(0)
    r = oracle.replay(tr, dict(cap_s_bytes=512 << 20, cap_h_bytes=8 << 30, kv_bytes_per_token=28672),
                      log=True, log_capacity=10)
    assert r["status"] == -7 and r["log_len"] > 10


def test_kendall_brute_matches_scipy():
    stats = pytest.importorskip("scipy.stats")
    rs = np.random.default_rng(1)
    for n in (5, 50, 400):
        x = rs.integers(0, 20, n).astype(float)
        y = x + rs.normal(0, 3, n).round()
        assert abs(oracle.kendall_brute(x, y) - stats.kendalltau(x, y).statistic) < 1e-12


# ------------------------------------------------------------------ ASE --
def test_ase_hand_values():
    rows, want = {}, {}
    for line in _rows("ase_hand.txt"):
        tag, *rest = line.split()
        if tag == "row":
            c, d, hr, am, tt = rest
            rows[(int(c), int(d))] = (float(hr), float(am), float(tt))
        else:
            want[int(rest[0])] = float(rest[1])
    nc, nd = 1 + max(c for c, _ in rows), 1 + max(d for _, d in rows)
    grid = np.array([[rows[(c, d)] for d in range(nd)] for c in range(nc)])
    got = oracle.ase(grid[:, :, 0], grid[:, :, 1], grid[:, :, 2])
    for c, v in want.items():
        assert abs(got[c] - v) < 1e-15


def _ase_grid(seed, nc=5, nd=4):
    rs = np.random.default_rng(seed)
    return rs.uniform(0.05, 0.9, (nc, nd)), rs.uniform(1e5, 1e8, (nc, nd)), rs.uniform(1e3, 1e9, (nc, nd))


def test_ase_closed_forms():
    hr, am, tt = _ase_grid(3)
    # identical configurations: every ratio is 1
    one = oracle.ase(np.tile(hr[:1], (4, 1)), np.tile(am[:1], (4, 1)), np.tile(tt[:1], (4, 1)))
    assert np.allclose(one, 1.0, rtol=0, atol=1e-15)
    # a configuration at the best value of every metric on every dataset scores 1
    hr2, am2, tt2 = hr.copy(), am.copy(), tt.copy()
    hr2[2], am2[2], tt2[2] = hr.max(0), am.min(0), tt.min(0)
    a = oracle.ase(hr2, am2, tt2)
    assert abs(a[2] - 1.0) < 1e-15 and (a <= 1.0 + 1e-15).all()
    # each metric is a ratio within a dataset: scaling it by a per-dataset constant changes nothing
    s = np.array([3.0, 0.5, 7.0, 11.0])
    assert np.allclose(oracle.ase(hr * s, am * s, tt / s), oracle.ase(hr, am, tt), rtol=1e-14)
    # one dataset: the cube root of the three ratios, written out
    h1, m1, t1 = hr[:, :1], am[:, :1], tt[:, :1]
    direct = ((h1 / h1.max()) * (m1.min() / m1) * (t1.min() / t1)) ** (1 / 3)
    assert np.allclose(oracle.ase(h1, m1, t1), direct[:, 0], rtol=1e-14)


def test_ase_zero_readings():
    hr, am, tt = _ase_grid(4, nc=3, nd=2)
    hr[:, 0] = 0.0                     # no configuration hits on dataset 0: factor 1 for all (0/0)
    base = oracle.ase(hr, am, tt)
    hr1 = hr.copy()
    hr1[:, 0] = 0.5                    # equal positive values are also factor 1
    assert np.allclose(base, oracle.ase(hr1, am, tt), rtol=1e-14)
    am[1, 1] = 0.0                     # a zero AMAT minimum: the others' factor is 0
    z = oracle.ase(hr, am, tt)
    assert z[0] == 0.0 and z[2] == 0.0 and z[1] > 0.0


# ------------------------------------------------- online hazard table --
MIB, GIB = 1 << 20, 1 << 30
def _online_logs(tr, p_online, p_offline):
    from cases import to_oracle
    cap = 16 * tr.n_events
    a = oracle.replay(tr, to_oracle(p_online), log=True, log_capacity=cap, debug=True)
    b = oracle.replay(tr, to_oracle(p_offline), log=True, log_capacity=cap, debug=True)
    assert a["status"] == 0 and b["status"] == 0
    return [np.asarray(x) for x in a["log"]], [np.asarray(x) for x in b["log"]], a, b


def test_online_hazard_beyond_horizon():
    """Sessions of more than 51 turns have d(t) = 0 for every table entry
    t <= 50: the online table never leaves zero hazard, as the offline one,
    so both make the same decisions.  With turn counts inside the horizon the
    two differ (the decisions do depend on the table)."""
    from cases import base
    long = synth.make_trace(11, np.full(40, 55), 0.5, synth.GAP_MIX_CODING)
    short = synth.make_trace(11, 2 + (np.arange(40) % 15), 0.5, synth.GAP_MIX_CODING)
    for pol in ("spear", "spear_tide"):
        p = base(pol, 48 * MIB, 1 * GIB, 131072)
        la, lb, _, _ = _online_logs(long, dict(p, online=True), p)
        assert all(np.array_equal(x, y) for x, y in zip(la, lb)), pol
        sa, sb, _, _ = _online_logs(short, dict(p, online=True), p)
        assert not all(np.array_equal(x, y) for x, y in zip(sa, sb)), pol


def _two_phase_trace():
    """Wave 1: three small sessions (3, 4, 4 turns) that finish early.  Wave 2:
    ten 3-turn and twenty 4-turn sessions (the same turn-count ratios): their
    turns but the last run within the first minutes, their last turns all
    arrive in one burst at 1,000 s, and they all complete at 1,500 s, after
    every decision."""
    arr, comp, ins, outs = [], [], [], []
    for i, ts in enumerate((3, 4, 4)):
        a0 = 1000 + 200_000 * i
        arr.append([a0 + 100_000 * k for k in range(ts)])
        comp.append([a0 + 100_000 * k + 1000 for k in range(ts)])
        ins.append([100 + 50 * k for k in range(ts)])
        outs.append([120 + 50 * k for k in range(ts)])
    for j in range(30):
        ts = 3 if j < 10 else 4
        t = 5_000_000 + 300_000 * j
        a, c, i_, o_ = [], [], [], []
        tok = 3000 + 500 * (j % 5)
        for k in range(ts):
            final = k + 1 == ts
            if final:
                t = 1_000_000_000 + 1000 * j
            a.append(t)
            i_.append(tok)
            tok += 100 + 40 * ((j + k) % 7)
            o_.append(tok)
            c.append(1_500_000_000 + j if final else t + 2000)
            t = c[-1] + 200_000 * (1 + ((j * 7 + k * 13) % 10) ** 2)
        arr.append(a), comp.append(c), ins.append(i_), outs.append(o_)
    return synth.trace_from_turns(arr, comp, ins, outs)


def test_online_hazard_two_phase_equals_offline():
    """After wave 1 completes, the online table holds turn counts {3, 4, 4};
    the offline table over both waves holds {3 x 11, 4 x 22}: the same d/n
    in every entry, hence the same table (worked: h(2) = floor((2*1*4095+3)/6)
    = floor((2*11*4095+33)/66) = 1365, h(3) = 4095, h = 0 elsewhere).  Wave 1 never fills a
    tier, and no wave-2 session completes before the last decision, so the
    online and offline replays decide identically.  Pooling turns (bucket 3)
    changes the table and the decisions."""
    from cases import base
    tr = _two_phase_trace()
    for pol in ("spear", "spear_tide"):
        p = base(pol, 6000 * 131072, 20000 * 131072, 131072, dma=2000)
        la, lb, a, b = _online_logs(tr, dict(p, online=True), p)
        assert all(np.array_equal(x, y) for x, y in zip(la, lb)), pol
        assert a["evict"] + a["demote"] > 0, pol  # the tiers do fill in wave 2
        _, lc, _, _ = _online_logs(tr, p, dict(p, bucket=3))
        assert not all(np.array_equal(x, y) for x, y in zip(lb, lc)), pol


# ---- attainment A(n) (Sec. V-F, eq. attainment; reading R27) ---------------------

def _attain_hand():
    """Four sessions of two turns.  Events in time order: the four first turns
    (e0..e7), then e8 = arrival of s0's second turn, e9 its final completion,
    e10/e11 the same for s1, e12/e13 for s2, e14/e15 for s3.  So the warm
    arrivals e8, e10, e12, e14 see 0, 1, 2, 3 completed sessions."""
    arr = [[0, 100], [20, 200], [40, 300], [60, 400]]
    comp = [[10, 110], [30, 210], [50, 310], [70, 410]]
    tr = synth.trace_from_turns(arr, comp, [[100, 200]] * 4, [[150, 250]] * 4)
    HS, HH, MI, CO, PS, EV = 1, 2, 3, 0, 4, 8

    def lg(kinds):  # warm decisions at e8, e10, e12, e14 plus ignored records
        ev = [0, 1, 8, 10, 11, 12, 14]
        kd = [CO, PS, kinds[0], kinds[1], EV, kinds[2], kinds[3]]
        ss = [0, 0, 0, 1, 2, 2, 3]
        return np.array(ev, np.uint32), np.array(kd, np.uint8), np.array(ss, np.uint32)

    return tr, [lg((HS, MI, HH, HS)), lg((HS, HS, HS, HH)), lg((MI, MI, HS, MI))]


# expected (n_j, warm, H_on, H_off, H_lru, A) per point count, worked by hand:
# P=1: H = 3/4, 4/4, 1/4 -> A = (3/4 - 1/4) / (1 - 1/4) = 2/3
# P=2 (n_j = 0, 2): {e8, e10} -> 1/2, 1, 0 -> 1/2;  {e12, e14} -> 1, 1, 1/2 -> 1
# P=3 (n_j = 0, 1, 2): {e8} -> 1;  {e10} -> 0, 1, 0 -> 0;  {e12, e14} -> 1
# P=4: {e8} -> 1;  {e10} -> 0;  {e12} -> 1, 1, 1 -> undefined;  {e14} -> 1, 1, 0 -> 1
_ATTAIN_HAND = {
    1: [(0, 4, 0.75, 1.0, 0.25, 2 / 3)],
    2: [(0, 2, 0.5, 1.0, 0.0, 0.5), (2, 2, 1.0, 1.0, 0.5, 1.0)],
    3: [(0, 1, 1.0, 1.0, 0.0, 1.0), (1, 1, 0.0, 1.0, 0.0, 0.0), (2, 2, 1.0, 1.0, 0.5, 1.0)],
    4: [(0, 1, 1.0, 1.0, 0.0, 1.0), (1, 1, 0.0, 1.0, 0.0, 0.0), (2, 1, 1.0, 1.0, 1.0, float("nan")),
        (3, 1, 1.0, 1.0, 0.0, 1.0)],
}


def test_attainment_hand_case():
    tr, logs = _attain_hand()
    for P, want in _ATTAIN_HAND.items():
        rc, got = oracle.attainment(tr, logs, P)
        assert rc == 0
        np.testing.assert_allclose(got, np.array(want), rtol=1e-15, atol=0, equal_nan=True, err_msg=str(P))


def test_attainment_errors():
    tr, logs = _attain_hand()
    assert oracle.attainment(tr, logs, 0)[0] == -4  # OR_ERR_RANGE
    assert oracle.attainment(tr, logs, 5)[0] == -4  # more points than sessions
    bad = (logs[0][0], logs[0][1].copy(), logs[0][2])
    bad[1][2] = 0  # e8 no longer a warm request in one log
    assert oracle.attainment(tr, [bad, logs[1], logs[2]], 2)[0] == -3  # OR_ERR_FORMAT
    far = (logs[0][0].copy(), logs[0][1], logs[0][2])
    far[0][-1] = 16  # past the last event
    assert oracle.attainment(tr, [far, logs[1], logs[2]], 2)[0] == -3


def test_attainment_identities_on_replays():
    """On real replay logs: the offline replay against itself attains 1 and
    LRU attains 0 in every window where they differ; the windows partition
    the warm requests; n_j = floor(j N / P)."""
    from cases import base, to_oracle
    tr = synth.make_trace(21, 2 + (np.arange(120) % 9), 0.3, synth.GAP_MIX_CODING)
    cap = 16 * tr.n_events
    r_on, r_off, r_lru = (oracle.replay(tr, to_oracle(base(p, 20000 * 131072, 100000 * 131072, 131072, online=o)),
                                        log=True, log_capacity=cap)
                          for p, o in (("spear", True), ("spear", False), ("lru", False)))
    for P in (1, 7, 16, 120):
        rc, a = oracle.attainment(tr, [r_off["log"], r_off["log"], r_lru["log"]], P)
        assert rc == 0
        d = (a[:, 1] > 0) & (a[:, 3] != a[:, 4])
        assert d.any()
        assert np.all(a[d, 5] == 1.0) and np.all(np.isnan(a[~d, 5]))
        rc, z = oracle.attainment(tr, [r_lru["log"], r_off["log"], r_lru["log"]], P)
        assert np.all(z[d, 5] == 0.0)
        rc, b = oracle.attainment(tr, [r_on["log"], r_off["log"], r_lru["log"]], P)
        assert rc == 0
        assert int(b[:, 1].sum()) == r_on["req_warm"]
        assert list(b[:, 0]) == [j * 120 // P for j in range(P)]


# ---- stale snapshot of a dual design (Sec. IV-B eq. stale; reading R28) -------------

STALE_HAND = dict(policy="spear", kv_bytes_per_token=1, cap_s_bytes=300, cap_h_bytes=0,
                  t_p_ps_per_tok=20_000_000, ttft_load=4)


def test_hand_replay_stale_snapshot():
    tr, log, counts = _hand_trace("replay_hand_stale.txt")
    for sync, m in (("arrivals", 100), ("gap_start", 0)):  # e5 is final: no gap_start sync after e3
        r = oracle.replay(tr, dict(STALE_HAND, stale_sync=sync, stale_m=m), log=True, debug=True)
        assert r["status"] == 0
        assert list(zip(*(map(int, a) for a in r["log"]))) == log, sync
        for k, v in counts.items():
            assert r[k] == v, (sync, k)
    # synced after every event, the snapshot is the live state: s1 is dropped at e6, s0 hits at e8
    live = oracle.replay(tr, STALE_HAND, log=True)
    r = oracle.replay(tr, dict(STALE_HAND, stale_sync="event"), log=True, debug=True)
    assert r["decision_hash"] == live["decision_hash"] and r["vict_diff"] == 0 and r["vict_n"] == 1
    got = list(zip(*(map(int, a) for a in live["log"])))
    assert (6, oracle.KINDS.index("EVICT"), 1) in got and (8, oracle.KINDS.index("HIT_S"), 0) in got


@pytest.mark.parametrize("mix", ["coding", "general"])
def test_stale_every_event_is_live(mix):
    """A snapshot copied after every event holds, at each decision, the rows
    of the candidates as they are live (their rows change only at their own
    events, and a session is pinned through its arrival's decisions), so the
    dual design decides exactly as the live one."""
    from cases import base, to_oracle
    tr = synth.paper_scale_trace(2, mix)
    for pol in ("spear", "spear_tide"):
        p = base(pol, 2 * GIB, 16 * GIB, 131072)
        live = oracle.replay(tr, to_oracle(p))
        st = oracle.replay(tr, to_oracle(dict(p, stale="event")))
        assert st["status"] == 0 and st["decision_hash"] == live["decision_hash"]
        assert st["vict_n"] > 1000 and st["vict_diff"] == 0 and st["prom_diff"] == 0
        assert (st["prom_n"] > 0) == (pol == "spear_tide")
        lag = oracle.replay(tr, to_oracle(dict(p, stale="arrivals", stale_m=8)))
        assert lag["decision_hash"] != live["decision_hash"] and lag["vict_diff"] > 0


def test_stale_snapshot_rejected_params():
    tr, _, _ = _hand_trace("replay_hand_stale.txt")
    for bad in (dict(policy="lru", stale_sync="event"), dict(policy="belady", stale_sync="gap_start"),
                dict(stale_sync="arrivals", stale_m=0), dict(stale_sync="event", hazard_online=True)):
        assert oracle.replay(tr, dict(STALE_HAND, **bad))["status"] == -1


# ---- signal leave-one-out (Sec. V-D, Fig. signal; reading R29) -----------------------

def _unit_gap_trace(n=60, turns=5):
    """Every tool gap lasts 1 us: the gap average (3,10) stays at
    floor(3*1/10) = 0 from the first gap on."""
    arr, comp, ins, outs = [], [], [], []
    for s in range(n):
        a, c, i_, o_ = [], [], [], []
        t = s * 1500
        tok = 500 + 37 * (s % 11)
        for k in range(turns):
            a.append(t)
            i_.append(tok)
            tok += 64 + (s * 7 + k * 13) % 150
            o_.append(tok)
            t += 20 * (64 + (s + k) % 150)
            c.append(t)
            t += 1
        arr.append(a), comp.append(c), ins.append(i_), outs.append(o_)
    return synth.trace_from_turns(arr, comp, ins, outs)


def test_signal_no_gap_equals_spear_when_gaps_vanish():
    from cases import base, to_oracle
    tr = _unit_gap_trace()
    for pol in ("spear", "spear_tide"):
        p = base(pol, 3000, 20000, 1)
        a = oracle.replay(tr, to_oracle(p), debug=True)
        b = oracle.replay(tr, to_oracle(dict(p, no_gap=True)), debug=True)
        assert a["status"] == b["status"] == 0 and a["evict"] + a["demote"] > 10
        assert a["decision_hash"] == b["decision_hash"], pol
    tr = synth.paper_scale_trace(2, "coding")
    p = base("spear", 2 * GIB, 16 * GIB, 131072)
    assert (oracle.replay(tr, to_oracle(p))["decision_hash"] !=
            oracle.replay(tr, to_oracle(dict(p, no_gap=True)))["decision_hash"])


def test_signal_no_hazard_equals_spear_beyond_horizon():
    """With every session longer than 51 turns, d(t) = 0 for every table
    entry: zero hazard, sigma = Lambda, T2 = 0, as without the signal."""
    from cases import base, to_oracle
    tr = synth.make_trace(13, 52 + np.arange(30) % 5, 0.4, synth.GAP_MIX_CODING)
    h, sig = oracle.hazard_lut(52 + np.arange(30) % 5)
    assert np.all(h == 0) and np.all(sig == 4095)
    for pol in ("spear", "spear_tide"):
        p = base(pol, 40000 * 131072, 200000 * 131072, 131072)
        a = oracle.replay(tr, to_oracle(p), debug=True)
        b = oracle.replay(tr, to_oracle(dict(p, no_hazard=True)), debug=True)
        assert a["status"] == b["status"] == 0 and a["evict"] + a["demote"] > 10
        assert a["decision_hash"] == b["decision_hash"], pol
    tr = synth.paper_scale_trace(2, "coding")
    p = base("spear", 2 * GIB, 16 * GIB, 131072)
    assert (oracle.replay(tr, to_oracle(p))["decision_hash"] !=
            oracle.replay(tr, to_oracle(dict(p, no_hazard=True)))["decision_hash"])


def test_signal_flags_rejected():
    tr = _unit_gap_trace(4, 2)
    for bad in (dict(policy="lru", no_gap=True), dict(policy="belady", no_hazard=True),
                dict(policy="spear", no_gap=True, hazard_online=True)):
        assert oracle.replay(tr, dict(STALE_HAND, **bad))["status"] == -1
