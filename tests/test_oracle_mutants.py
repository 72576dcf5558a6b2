"""The TIDE pins have teeth: each test plants one plausible mistake in a
copy of the oracle's C source, compiles it, and checks that the hand-worked
SPEAR+TIDE replay (tests/golden/replay_hand_tide.txt) no longer matches.
The mistakes are the ones a reading of Sec. III-C and Algorithm 1 invites:
the budget taken from the gap just closed instead of the gap average (R11),
a strict test for a free DMA engine or a floor in its busy time (R13), a
phase-1 promotion that ignores the pinned sessions' share of the fast tier
(R14), and prefetch accuracy counted on hits other than a promoted session's
fast-tier hit (R19).  The copies run without the oracle's self-check of the
two TIDE forms, so only the golden file can reject them."""
import pytest

import oracle
from test_oracle_pins import HAND_TIDE_PARAMS, _hand_trace

MUTANTS = {
    "budget_from_last_gap": (
        "uint64_t budget = R->g_q * p->dma_bytes_per_us;",
        "uint64_t budget = (x->turn ? tr->arrival_us[ti] - tr->completion_us[ti - 1] : 0) * p->dma_bytes_per_us;"),
    "dma_free_strict": (
        "if (dma_busy && st.now >= dma_busy_until) dma_busy = 0;",
        "if (dma_busy && st.now > dma_busy_until) dma_busy = 0;"),
    "busy_time_floor": (
        "dma_busy_until = st.now + (moved + p->dma_bytes_per_us - 1) / p->dma_bytes_per_us;",
        "dma_busy_until = st.now + moved / p->dma_bytes_per_us;"),
    "phase1_ignores_pinned": (
        "if (by > rem || st->used_s + sz > st->cap_s) break;",
        "if (by > rem || st->used_s - used_of(st, OR_S, 1) + sz > st->cap_s) break;"),
    "prefetch_hit_on_hbm_hit": (
        "res->tok_hit_h += out_prev;",
        "res->tok_hit_h += out_prev;\n          if (R->promoted) res->promoted_then_hit_s++;"),
    "prefetch_hit_on_any_fast_hit": (
        "if (R->promoted) res->promoted_then_hit_s++;",
        "res->promoted_then_hit_s++;"),
}


def _matches_golden(r, log, counts):
    got = list(zip(*(map(int, a) for a in r["log"])))
    return r["status"] == 0 and got == log and all(r[k] == v for k, v in counts.items())


def test_unmodified_copy_matches(tmp_path):
    L = oracle.build_variant(oracle.source(), str(tmp_path))
    tr, log, counts = _hand_trace("replay_hand_tide.txt")
    assert _matches_golden(oracle.replay(tr, HAND_TIDE_PARAMS, log=True, lib_=L), log, counts)


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_fails_the_golden(name, tmp_path):
    old, new = MUTANTS[name]
    src = oracle.source()
    assert src.count(old) == 1, name  # the planted mistake replaces exactly one statement
    L = oracle.build_variant(src.replace(old, new), str(tmp_path))
    tr, log, counts = _hand_trace("replay_hand_tide.txt")
    r = oracle.replay(tr, HAND_TIDE_PARAMS, log=True, lib_=L)
    assert not _matches_golden(r, log, counts), name
