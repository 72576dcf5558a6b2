"""Host-side checks of the C ABI (no GPU needed): the library loads, exports
every symbol include/unison.h declares, and its host logic (trace
validation, status strings, stats) behaves as documented."""
import ctypes as C
import os
import re

import numpy as np
import pytest

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def B():
    from paper_2609_09643_gb300 import native
    native.build()
    from paper_2609_09643_gb300 import binding
    return binding


def declared_symbols(header="unison.h"):
    src = open(os.path.join(ROOT, "include", header)).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(unison_[a-z0-9_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(B):
    lib = C.CDLL(B.lib_path())
    decl = declared_symbols()
    assert len(decl) >= 10
    for name in decl:
        assert hasattr(lib, name), name
    assert sorted(B.EXPORTS) == decl


def test_debug_library_exports_its_hooks(B):
    """The ranking test library (include/unison_debug.h) builds for sm_103a
    and exports its hooks beside the ranking calls; the default library does
    not contain them."""
    from paper_2609_09643_gb300 import native
    path = native.build_debug()
    dbg = C.CDLL(path)
    decl = declared_symbols("unison_debug.h")
    assert decl == sorted(B.DEBUG_EXPORTS)
    for name in decl + ["unison_rank_batch", "unison_rank", "unison_strerror"]:
        assert hasattr(dbg, name), name
    lib = C.CDLL(B.lib_path())
    for name in decl:
        assert not hasattr(lib, name), name


def test_strerror_and_version(B):
    assert B.strerror(0) == "ok"
    assert "argument" in B.strerror(-1)
    assert B.strerror(-9999) == "unknown status"
    assert B.lib().unison_version() >= 10000


def test_trace_create_and_info(B):
    tr = synth.tiny_trace(0)
    t = B.Trace(tr)
    assert t.info() == (64, 768, 1536)
    assert t.device_bytes > 16 * 1536
    t.close()


def _bad(tr, **mods):
    arrs = dict(turn_off=tr.turn_off.copy(), arrival_us=tr.arrival_us.copy(), completion_us=tr.completion_us.copy(),
                in_tok=tr.in_tok.copy(), out_tok=tr.out_tok.copy())
    for k, f in mods.items():
        f(arrs[k])
    return synth.Trace(**arrs)


def test_trace_validation_errors(B):
    tr = synth.tiny_trace(1)

    def code(t):
        with pytest.raises(B.UnisonError) as e:
            B.Trace(t)
        return e.value.code

    def zero_len(a):
        a[3] = 0

    assert code(_bad(tr, completion_us=lambda a: a.__setitem__(3, tr.arrival_us[3]))) == B.ERR_FORMAT
    assert code(_bad(tr, in_tok=zero_len)) == B.ERR_FORMAT
    assert code(_bad(tr, out_tok=lambda a: a.__setitem__(5, 1))) == B.ERR_FORMAT  # out < in

    def long_gap(a):
        a[5:12] += np.uint64(1 << 31)

    assert code(_bad(tr, arrival_us=long_gap, completion_us=long_gap)) == B.ERR_RANGE

    def swap_sessions(a):
        a[0:12] += np.uint64(10 ** 9)  # session 0 first arrives after session 1

    assert code(_bad(tr, arrival_us=swap_sessions, completion_us=swap_sessions)) == B.ERR_FORMAT


def test_trace_load_file(B, tmp_path):
    tr = synth.tiny_trace(2)
    p = str(tmp_path / "t.utr")
    synth.save_utr(tr, p)
    assert B.Trace(path=p).info() == (64, 768, 1536)
    with pytest.raises(B.UnisonError) as e:
        B.Trace(path=str(tmp_path / "missing.utr"))
    assert e.value.code == B.ERR_IO
    with open(p, "r+b") as f:
        f.write(b"XXXX")
    with pytest.raises(B.UnisonError) as e:
        B.Trace(path=p)
    assert e.value.code == B.ERR_FORMAT


def test_stats_definitions(B):
    r = dict((f, 0) for f in B.RESULT_FIELDS)
    r.update(req_warm=4, hit_s=1, hit_h=1, miss=2, tok_hit_s=100, tok_hit_h=200, tok_miss=300,
             tok_needed=1000, tok_computed=600, promote=4, promoted_then_hit_s=1, ttft_n=4,
             ttft_sum_lo=40, ttft_sum_hi=0, ttft_p50_ns=7)
    p = dict(t_s_ps_per_tok=10, t_h_ps_per_tok=20, t_p_ps_per_tok=1000)
    s = B.stats(r, p)
    assert s["hit_rate"] == 0.5
    assert s["amat_ps"] == (10 * 100 + 20 * 200 + 1000 * 300) / 4  # eq. (hr-amat)
    assert s["prered"] == pytest.approx(0.4)                       # eq. (prered)
    assert s["prefetch_acc"] == 0.25
    assert s["ttft_mean_ns"] == 10.0 and s["ttft_p50_ns"] == 7.0
    r2 = dict(r, ttft_sum_hi=1, ttft_sum_lo=0)  # 128-bit sum
    assert B.stats(r2, p)["ttft_mean_ns"] == pytest.approx(2.0 ** 64 / 4)


def test_oracle_library_loads_standalone():
    import oracle
    assert oracle.spear_score(3_000_000, 41) == 794_628_040


def test_ase_library_matches_oracle(B):
    """unison_ase (host function of the library) against the oracle's plain
    product, and its argument checks."""
    import oracle
    rs = np.random.default_rng(7)
    for nc, nd in ((1, 1), (3, 6), (17, 8)):
        hr = rs.uniform(0.0, 1.0, (nc, nd))
        am = rs.uniform(1e5, 1e9, (nc, nd))
        tt = rs.uniform(1e3, 1e9, (nc, nd))
        if nc > 2:
            hr[:, 0] = 0.0
            am[1, -1] = 0.0
        grid = [[dict(hit_rate=hr[c, d], amat_ps=am[c, d], ttft_mean_ns=tt[c, d]) for d in range(nd)]
                for c in range(nc)]
        got = np.array(B.ase(grid))
        want = oracle.ase(hr, am, tt)
        assert np.allclose(got, want, rtol=1e-12, atol=0), (nc, nd, got, want)
    with pytest.raises(B.UnisonError):
        B.ase([[dict(hit_rate=-1.0, amat_ps=1.0, ttft_mean_ns=1.0)]])
    with pytest.raises(B.UnisonError):
        B.ase([])


def test_attainment_library_matches_oracle(B):
    """unison_attainment (host function over a trace handle) against the
    oracle's on the worked hand case and on three replays' logs; errors."""
    import oracle
    from cases import base, to_oracle
    from test_oracle_pins import _attain_hand, _ATTAIN_HAND
    tr, logs = _attain_hand()
    h = B.Trace(tr)
    for P, want in _ATTAIN_HAND.items():
        got = B.attainment(h, logs, P)
        arr = np.array([[g["sessions_seen"], g["warm"], g["hr_online"], g["hr_offline"], g["hr_lru"],
                         g["attainment"]] for g in got])
        np.testing.assert_array_equal(arr, oracle.attainment(tr, logs, P)[1])
        np.testing.assert_allclose(arr, np.array(want), rtol=1e-15, atol=0, equal_nan=True)
    for P in (0, 5):
        with pytest.raises(B.UnisonError) as ei:
            B.attainment(h, logs, P)
        assert ei.value.code == B.ERR_RANGE
    bad = (logs[0][0], logs[0][1].copy(), logs[0][2])
    bad[1][2] = 0
    with pytest.raises(B.UnisonError) as ei:
        B.attainment(h, [bad, logs[1], logs[2]], 2)
    assert ei.value.code == B.ERR_FORMAT
    far = (logs[0][0].copy(), logs[0][1], logs[0][2])
    far[0][-1] = 16
    with pytest.raises(B.UnisonError) as ei:
        B.attainment(h, [far, logs[1], logs[2]], 2)
    assert ei.value.code == B.ERR_FORMAT

    tr = synth.make_trace(21, 2 + (np.arange(120) % 9), 0.3, synth.GAP_MIX_CODING)
    cap = 16 * tr.n_events
    lg = [oracle.replay(tr, to_oracle(base(p, 20000 * 131072, 100000 * 131072, 131072, online=o)), log=True,
                        log_capacity=cap)["log"] for p, o in (("spear", True), ("spear", False), ("lru", False))]
    h = B.Trace(tr)
    for P in (1, 7, 16, 120):
        got = B.attainment(h, lg, P)
        arr = np.array([[g["sessions_seen"], g["warm"], g["hr_online"], g["hr_offline"], g["hr_lru"],
                         g["attainment"]] for g in got])
        np.testing.assert_array_equal(arr, oracle.attainment(tr, lg, P)[1])
