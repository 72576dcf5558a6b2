"""GPU parity of the standalone ranking (victims, TIDE fill, keys) against the
CPU oracle: bit-exact on every output index and key."""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu

P_Z = 500_000_000
KVB = 131072
GIB = 1 << 30


@pytest.fixture(scope="module")
def B():
    from paper_2609_09643_gb300 import native
    native.build()
    from paper_2609_09643_gb300 import binding
    return binding


@pytest.fixture(scope="module")
def sigma():
    _, s = oracle.hazard_lut(synth.geometric_turns(1, 1415, 23.7, 2, 200))
    return s


def run(B, recs, params, keys=False):
    import torch
    devs = [B.records_to_device(r) for r in recs]
    outs = [B.rank_outputs(r.n, p["k"], p["max_moves"], keys) for r, p in zip(recs, params)]
    B.rank_batch(devs, params, outs)
    torch.cuda.synchronize()
    return [B.rank_result(o) for o in outs]


def check(r, rec, p, keys=False):
    o = oracle.rank(rec, p["sigma_q"], p["penalty_q"], p["k"], p["budget_bytes"], p["kv_bytes_per_token"],
                    p["free_fast_tok"], p["free_hbm_tok"], keys=keys, max_moves=max(p["max_moves"], 1))
    compare(r, o, p, keys)


def compare(r, o, p, keys=False):
    if p["max_moves"] == 0:
        o["promote"] = o["promote"][:0]
        o["demote"] = o["demote"][:0]
        o["moved_bytes"] = 0
    assert r["status"] == 0
    assert np.array_equal(r["victims"], o["victims"]), "victims"
    assert np.array_equal(r["promote"], o["promote"]), ("promote", r["promote"][:8], o["promote"][:8])
    assert np.array_equal(r["demote"], o["demote"]), ("demote", r["demote"][:8], o["demote"][:8])
    assert r["moved_bytes"] == o["moved_bytes"], "moved"
    if keys:
        assert np.array_equal(r["keys"], o["keys"]), "keys"


def prm(sig, k=1024, budget=16 * GIB, max_moves=1024, free_s=0, free_h=1 << 40):
    return dict(sigma_q=sig, k=k, penalty_q=P_Z, budget_bytes=budget, kv_bytes_per_token=KVB, max_moves=max_moves,
                free_fast_tok=free_s, free_hbm_tok=free_h)


def test_sigma_from_device_table(B):
    """The chain the library offers end to end: the survival table built on
    the device from turn counts (unison_hazard_lut, eqs. hazard/hq/survq)
    feeds the ranking call, and the victims and fill equal the oracle's with
    the oracle's own table."""
    import torch
    tps = synth.geometric_turns(2, 5000, 23.7, 2, 200)
    turns = torch.from_numpy(np.asarray(tps, dtype=np.int32)).to("cuda")
    sig_dev, _ = B.hazard_lut(turns)
    sig = sig_dev.cpu().numpy().view(np.uint16)
    _, sig_oracle = oracle.hazard_lut(tps)
    assert np.array_equal(sig, sig_oracle)
    rec = synth.make_records(21, 300_000)
    ps = [prm(sig, k=k, budget=b, free_s=fs) for k, b, fs in [(1024, 8 * GIB, 0), (64, 64 * GIB, 50_000)]]
    res = run(B, [rec] * len(ps), ps)
    for r, p in zip(res, ps):
        o = oracle.rank(rec, sig_oracle, p["penalty_q"], p["k"], p["budget_bytes"], p["kv_bytes_per_token"],
                        p["free_fast_tok"], p["free_hbm_tok"], max_moves=p["max_moves"])
        compare(r, o, p)


@pytest.mark.parametrize("n", [1, 7, 1000, 2047, 2049, 4096, 16384])
def test_small_sets_all_candidates(B, sigma, n):
    rec = synth.make_records(n, n)
    ps = [prm(sigma, k=k, budget=b, free_s=fs) for k, b, fs in
          [(1, 1 * GIB, 0), (5, 64 * GIB, 0), (1024, 4 * GIB, 30000), (4096, 1 << 50, 10 ** 7)]]
    res = run(B, [rec] * len(ps), ps, keys=True)
    for r, p in zip(res, ps):
        check(r, rec, p, keys=True)


@pytest.mark.parametrize("n", [16385, 1 << 17, 1 << 18, 1 << 20])
def test_sampled_sizes(B, sigma, n):
    rec = synth.make_records(11, n)
    ps = [prm(sigma, k=k, budget=b) for k, b in [(1, 1 * GIB), (64, 8 * GIB), (1024, 64 * GIB)]]
    res = run(B, [rec] * len(ps), ps, keys=(n <= (1 << 18)))
    for r, p in zip(res, ps):
        check(r, rec, p, keys=(n <= (1 << 18)))


def test_full_size_2p24(B, sigma):
    """The largest live set (2^24 records): victims, fill and every key."""
    rec = synth.make_records(4, 1 << 24)
    p = prm(sigma, k=1024, budget=64 * GIB)
    r = run(B, [rec], [p], keys=True)[0]
    check(r, rec, p, keys=True)


def test_bench_launch_seven_sets(B, sigma):
    """The benchmark's ranking launch: seven copies of one 2^24-record live
    set with TIDE budgets 1..64 GiB and k = 1,024, in one call.  Every set's
    victims, moves and moved bytes equal the oracle's (a spawn pool runs the
    seven oracle rankings, each worker building the set itself)."""
    import multiprocessing as mp
    from cases import oracle_rank_job
    rec = synth.make_records(4, 1 << 24)
    ps = [prm(sigma, k=1024, budget=b * GIB) for b in (1, 2, 4, 8, 16, 32, 64)]
    res = run(B, [rec] * len(ps), ps)
    with mp.get_context("spawn").Pool(len(ps)) as pool:
        ores = pool.map(oracle_rank_job, [(4, 1 << 24, p) for p in ps], chunksize=1)
    for r, o, p in zip(res, ores, ps):
        compare(r, o, p)


def _sorted_records(n, ascending=True):
    rec = synth.make_records(5, n)
    order = np.argsort(rec.gap_q.astype(np.int64), kind="stable")
    if not ascending:
        order = order[::-1]
    f = lambda a: np.ascontiguousarray(a[order])
    rec2 = synth.Records(f(rec.gap_q), f(rec.last_ret), np.zeros(n, np.uint16), f(rec.kv_tok), f(rec.tier),
                         (f(rec.flags) & 1).astype(np.uint8))
    return rec2


@pytest.mark.parametrize("asc", [True, False])
def test_adversarial_order(B, sigma, asc):
    """Records sorted by key put every top record in one region: the sampled
    thresholds miss and the exact re-selection must still give the answer."""
    rec = _sorted_records(1 << 20, asc)
    ps = [prm(sigma, k=1024, budget=64 * GIB), prm(sigma, k=3000, budget=1 << 50, max_moves=4096)]
    for r, p in zip(run(B, [rec] * 2, ps), ps):
        check(r, rec, p)


def test_massive_ties(B, sigma):
    n = 300000
    rec = synth.make_records(6, n)
    rec = synth.Records(np.zeros(n, np.uint32), rec.last_ret, np.zeros(n, np.uint16), rec.kv_tok, rec.tier,
                        np.zeros(n, np.uint8))
    ps = [prm(sigma, k=777, budget=64 * GIB), prm(sigma, k=4096, budget=1 << 45, free_s=50000, max_moves=4096)]
    for r, p in zip(run(B, [rec] * 2, ps, keys=True), ps):
        check(r, rec, p, keys=True)


def test_crowded_buckets(B, sigma):
    """A few records whose keys sit far above thousands of equal ones: below
    the candidates' common prefix every equal-key record falls in one bucket,
    so the finish's bucket cut keeps them all (the radix select when they
    exceed 4,096) and the bucket sort declines for the sorting network."""
    n = 300000
    base = synth.make_records(11, n)
    gap = np.zeros(n, np.uint32)
    gap[np.arange(0, n, n // 7)[:7]] = 1 << 30  # seven far larger gap averages
    rec = synth.Records(gap, base.last_ret, np.zeros(n, np.uint16), base.kv_tok, base.tier, np.zeros(n, np.uint8))
    ps = [prm(sigma, k=1024, budget=64 * GIB), prm(sigma, k=4096, budget=1 << 45, free_s=50000, max_moves=4096)]
    for r, p in zip(run(B, [rec] * 2, ps), ps):
        check(r, rec, p)


def test_degenerate_sets(B, sigma):
    n = 50000
    base = synth.make_records(8, n)
    all_pinned = synth.Records(base.gap_q, base.last_ret, base.turn, base.kv_tok, base.tier,
                               np.ones(n, np.uint8))
    all_fast = synth.Records(base.gap_q, base.last_ret, base.turn, base.kv_tok, np.ones(n, np.uint8), base.flags)
    none_res = synth.Records(base.gap_q, base.last_ret, base.turn, base.kv_tok, np.zeros(n, np.uint8), base.flags)
    cases = [(all_pinned, prm(sigma)), (all_fast, prm(sigma)), (none_res, prm(sigma)),
             (base, prm(sigma, k=0, budget=0, max_moves=0)), (base, prm(sigma, budget=0)),
             (base, prm(sigma, max_moves=3)), (base, prm(sigma, free_h=0)), (base, prm(sigma, budget=1))]
    res = run(B, [c[0] for c in cases], [c[1] for c in cases])
    for r, (rec, p) in zip(res, cases):
        check(r, rec, p)


def test_phase1_promotions(B, sigma):
    rec = synth.make_records(9, 200000)
    ps = [prm(sigma, budget=b, free_s=fs, max_moves=mm) for b, fs, mm in
          [(64 * GIB, 60000, 1024), (1 << 50, 10 ** 6, 4096), (1 << 50, 10 ** 9, 64), (2 * GIB, 10 ** 9, 4096)]]
    for r, p in zip(run(B, [rec] * 4, ps), ps):
        check(r, rec, p)


def test_fill_byte_sums_beyond_2p64(B, sigma):
    """Sizes near 2^32 tokens at 2^24 bytes per token and the largest budget:
    the running byte sums pass 2^64 within a few hundred moves, in phase 1
    (free fast-tier space, random sizes) and in the pair loop (equal sizes,
    one promotion's worth of free space)."""
    n = 100000
    base = synth.make_records(10, n)
    big = synth.rng.randint(11, 0, np.arange(n, dtype=np.uint64), 1 << 31, (1 << 32) - 1).astype(np.uint32)
    rnd = synth.Records(base.gap_q, base.last_ret, base.turn, big, base.tier, base.flags)
    flat = synth.Records(base.gap_q, base.last_ret, base.turn, np.full(n, 0xFFFFFFFF, np.uint32), base.tier,
                         base.flags)
    top = (1 << 64) - 1
    cases = [(rnd, 1 << 62, 1 << 62), (rnd, top, top), (flat, 0xFFFFFFFF, 1 << 62), (flat, 0, top)]
    recs, ps = [], []
    for rec, fs, fh in cases:
        p = prm(sigma, k=64, budget=top, max_moves=4096, free_s=fs, free_h=fh)
        p["kv_bytes_per_token"] = 1 << 24
        recs.append(rec)
        ps.append(p)
    res = run(B, recs, ps)
    for r, rec, p in zip(res, recs, ps):
        check(r, rec, p)
    assert len(res[0]["promote"]) > 100 and len(res[2]["demote"]) > 100


def test_more_sets_than_filter_ctas(B, sigma):
    """600 sampled sets (more than the filter's resident CTAs): every CTA
    deals tiles from all sets instead of owning one set's group."""
    n = 20000
    recs = [synth.make_records(1000 + i, n) for i in range(600)]
    ks = [1, 7, 64, 1024]
    ps = [prm(sigma, k=ks[i % 4], budget=(1 << (i % 7)) * GIB, max_moves=(64, 1024)[i % 2]) for i in range(600)]
    res = run(B, recs, ps)
    for i in list(range(0, 600, 37)) + [599]:
        check(res[i], recs[i], ps[i])


def test_batch_of_mixed_sets(B, sigma):
    recs = [synth.make_records(20 + i, n) for i, n in enumerate([100, 20000, 1 << 18, 3000, 1 << 19])]
    ps = [prm(sigma, k=k, budget=(1 << i) * GIB) for i, k in enumerate([3, 50, 1024, 4096, 700])]
    for r, rec, p in zip(run(B, recs, ps, keys=True), recs, ps):
        check(r, rec, p, keys=True)


def test_keys_exact_at_division_boundaries(B):
    """Every sigma in [41, 4095] (through a table of 51 distinct values per
    run), gaps at multiples of sigma and just below, and the largest gap."""
    import torch
    rs = np.random.default_rng(3)
    for run_i in range(4):
        sig = np.sort(rs.choice(np.arange(41, 4096), size=51, replace=False))[::-1].astype(np.uint16)
        if run_i == 0:
            sig[0], sig[1] = 4095, 41
        gs, ts = [], []
        for t in range(51):
            s = int(sig[t])
            q = rs.integers(0, (2 ** 31 - 1) * 4095 // s, 200)
            for x in np.concatenate([q * s, q * s + s - 1]):
                g = int(x) // 4095
                for dg in (-1, 0, 1):
                    if 0 <= g + dg < 2 ** 31:
                        gs.append(g + dg)
                        ts.append(t)
            gs += [0, 1, 2 ** 31 - 1]
            ts += [t, t, t]
        n = len(gs)
        rec = synth.Records(np.array(gs, np.uint32), np.zeros(n, np.uint32), np.array(ts, np.uint16),
                            np.full(n, 100, np.uint32), np.full(n, 2, np.uint8), np.zeros(n, np.uint8))
        p = dict(sigma_q=sig, k=10, penalty_q=(1 << 32) - 1, budget_bytes=0, kv_bytes_per_token=1, max_moves=0,
                 free_fast_tok=0, free_hbm_tok=0)
        r = run(B, [rec], [p], keys=True)[0]
        o = oracle.rank(rec, sig, p["penalty_q"], 10, 0, 1, 0, 0, keys=True)
        assert np.array_equal(r["keys"], o["keys"])


def test_rank_rejects_bad_args(B, sigma):
    import torch
    rec = synth.make_records(1, 100)
    d = B.records_to_device(rec)
    for bad in (dict(k=5000), dict(max_moves=5000), dict(penalty_q=1 << 32), dict(kv_bytes_per_token=0)):
        p = prm(sigma)
        p.update(bad)
        with pytest.raises(B.UnisonError):
            B.rank_batch([d], [p], [B.rank_outputs(100, 5000, 5000)])
    bad_sig = prm(np.full(51, 40, np.uint16))
    with pytest.raises(B.UnisonError):
        B.rank_batch([d], [bad_sig], [B.rank_outputs(100, 1024, 1024)])
    off = dict(d, gap_q=d["gap_q"][1:])  # misaligned
    with pytest.raises(B.UnisonError):
        B.rank_batch([off], [prm(sigma)], [B.rank_outputs(99, 1024, 1024)])
    empty = {k: v[:0] for k, v in d.items()}  # a live set needs at least one record
    with pytest.raises(B.UnisonError):
        B.rank_batch([empty], [prm(sigma)], [B.rank_outputs(1, 1024, 1024)])


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_random_sets_and_parameters(B, seed):
    """Ten live sets per call with random sizes (1 to 2^20 records), random
    shares of pinned, completed and fast-tier records, gap averages with many
    ties, and random k, move limit, DMA budget, free space, P_Z, KV size and
    hazard table: victims, fill and moved bytes equal the oracle's."""
    rng = np.random.default_rng(1000 + seed)
    recs, ps = [], []
    for j in range(10):
        n = int(rng.choice([1, 3, 100, 2047, 4097, 30000, 200000, 1 << 20]))
        base = synth.make_records(100 * seed + j, n)
        u = rng.random(n)
        p_pin, p_done = rng.choice([0.0, 1 / 64, 0.3]), rng.choice([0.0, 0.05, 0.5])
        flags = np.where(u < p_pin, 1, np.where(u < p_pin + p_done, 2, 0)).astype(np.uint8)
        tier = np.where(rng.random(n) < rng.choice([0.0, 1 / 16, 0.5, 1.0]), 1, 2).astype(np.uint8)
        tier[rng.random(n) < rng.choice([0.0, 0.1])] = 0
        gap = base.gap_q.astype(np.int64)
        if rng.random() < 0.5:  # coarse gaps: many equal keys, ties broken by index
            gap = (gap // 1_000_000) * 1_000_000
        gap = np.clip(gap, 0, (1 << 31) - 1).astype(np.uint32)
        recs.append(synth.Records(gap, base.last_ret, base.turn, base.kv_tok, tier, flags))
        sig = rng.integers(41, 4096, size=51).astype(np.uint16)
        ps.append(dict(sigma_q=sig, k=int(rng.integers(0, 4097)), penalty_q=int(rng.integers(0, 1 << 32)),
                       budget_bytes=int(rng.choice([0, 1 << 30, 1 << 36, 1 << 40, 1 << 44, (1 << 63) + 5])),
                       kv_bytes_per_token=int(rng.choice([1, 1024, 28672, 131072, 1 << 24])),
                       max_moves=int(rng.integers(0, 4097)),
                       free_fast_tok=int(rng.choice([0, 1000, 1 << 20, (1 << 64) - 1])),
                       free_hbm_tok=int(rng.choice([0, 5000, 1 << 40, (1 << 64) - 1]))))
    for r, rec, p in zip(run(B, recs, ps), recs, ps):
        check(r, rec, p)


def test_single_set_entry_point(B, sigma):
    """unison_rank, the one-set form, against the oracle and against the batch
    call on the same set."""
    import torch
    rec = synth.make_records(31, 1 << 20)
    dev = B.records_to_device(rec)
    for p in (prm(sigma), prm(sigma, k=3, budget=2 * GIB, max_moves=64, free_s=20_000)):
        out = B.rank_outputs(rec.n, p["k"], p["max_moves"])
        B.rank(dev, p, out)
        torch.cuda.synchronize()
        r = B.rank_result(out)
        check(r, rec, p)
        (rb,) = run(B, [rec], [p])
        for key in ("victims", "promote", "demote"):
            assert np.array_equal(r[key], rb[key]), key


def test_bounded_waits_report_timeout_and_recover(B, sigma):
    """The test library's short waits: a threshold wait on a flag that nothing
    sets and a tile wait on a barrier that nothing arrives at each run out,
    record UNISON_ERR_TIMEOUT in their set's counts[3] and let the kernel
    finish (the other outputs are still exact).  The next ordinary call on
    the same stream then ranks every set exactly, with status OK."""
    import torch
    from paper_2609_09643_gb300 import native
    native.build_debug()
    D = B.debug_lib()
    recs = [synth.make_records(41 + i, 300_000) for i in range(3)]
    ps = [prm(sigma, k=256, budget=4 * GIB, max_moves=128) for _ in recs]
    devs = [B.records_to_device(r) for r in recs]
    outs = [B.rank_outputs(r.n, p["k"], p["max_moves"]) for r, p in zip(recs, ps)]
    call = B.RankCall(devs, ps, outs, lib_=D)
    stream = torch.cuda.current_stream()
    try:
        assert D.unison_debug_rank_wait_hooks(0, 2) == B.OK
        call.run(stream)
        torch.cuda.synchronize()
        res = [B.rank_result(o) for o in outs]
        assert [r["status"] for r in res] == [B.ERR_TIMEOUT, 0, B.ERR_TIMEOUT]
        for r, rec, p in zip(res, recs, ps):
            r["status"] = 0
            check(r, rec, p)
    finally:
        assert D.unison_debug_rank_wait_hooks(-1, -1) == B.OK
    for o in outs:
        o["counts"].zero_()
    call.run(stream)
    torch.cuda.synchronize()
    for o, rec, p in zip(outs, recs, ps):
        check(B.rank_result(o), rec, p)


@pytest.mark.parametrize("world", [2, 4])
def test_record_sharded_ranking_equals_whole_set(B, sigma, world):
    """Sec. IV-D's scan split by records: each slice ranked into its candidate
    lists (global indices), the lists gathered (here: concatenated on one
    GPU, as the all-gather lays them out) and merged; the victims, moves and
    moved bytes equal the oracle's for the whole set."""
    import torch
    from paper_2609_09643_gb300 import shard
    n = 1 << 22
    rec = synth.make_records(51, n)
    dev = B.records_to_device(rec)
    for p in (prm(sigma, k=1024, budget=16 * GIB, max_moves=1024),
              prm(sigma, k=37, budget=3 * GIB, max_moves=300, free_s=40_000)):
        parts = []
        for r in range(world):
            off, cnt = shard.record_slice(n, r, world)
            c = B.rank_cands(p["k"], p["max_moves"])
            B.rank_shard({k: v[off:off + cnt] for k, v in dev.items()}, off, p, c)
            parts.append(c)
        out = B.rank_outputs(n, p["k"], p["max_moves"])
        B.rank_merge(torch.cat(parts), world, p, out)
        torch.cuda.synchronize()
        check(B.rank_result(out), rec, p)
