"""Pins for the CPU oracle: it is checked against values the paper fixes, hand
derivations from the paper's definitions, brute force, library routines and
invariants -- never against the CUDA path.  CPU only."""
import math
import os
import shutil
import subprocess

import numpy as np
import pytest

import oracle
import tracegen

NC = oracle.N_COUNTERS


def _op(v):
    return {"STRUCTURAL": oracle.STRUCTURAL, "NONOP": oracle.NONOP}.get(v, v)


def worked_arrays(g):
    r, k, n = g["ranges"], g["kernels"], g["ncu"]
    ranges = (np.array(r["stream"], np.uint8), np.array(r["start"], np.int64), np.array(r["end"], np.int64),
              np.array(r["depth"], np.uint8), np.array([_op(x) for x in r["op"]], np.uint32))
    kern = (np.array(k["stream"], np.uint8), np.array(k["start"], np.int64), np.array(k["dur"], np.int64),
            np.array(k["name"], np.uint32))
    counters = np.array([[np.nan if v is None else v for v in row] for row in n["counters"]], np.float32)
    return ranges, kern, np.array(n["name"], np.uint32), counters


def assert_agg(expected, got, rtol=1e-12):
    for e, g in zip(expected, got):
        if e is None:
            assert math.isnan(g), (expected, got)
        else:
            assert g == pytest.approx(e, rel=rtol, abs=0), (expected, got)


# ---------------------------------------------------------------- worked trace

@pytest.mark.parametrize("mode", ["brute", "indexed"])
def test_worked_enclosure(golden, mode):
    g = golden("worked.json")
    (rs, rt, re, rd, ro), (ks, kt, kd, kn), _, _ = worked_arrays(g)
    st, rk, nop = oracle.enclose(ks, kt, rs, rt, re, rd, ro, mode=mode)
    assert st == oracle.OK
    assert rk.tolist() == g["expect"]["range_of_kernel"]
    assert nop.tolist() == g["expect"]["n_op_enclosing"]


@pytest.mark.parametrize("mode", ["skip_name", "prefix", "error"])
@pytest.mark.parametrize("brute", [False, True])
def test_worked_match_and_aggregate(golden, mode, brute):
    g = golden("worked.json")
    (rs, rt, re, rd, ro), (ks, kt, kd, kn), ncu_name, counters = worked_arrays(g)
    exp = g["expect"][mode]
    st, idx, kind, summ = oracle.match(ks, kt, kn, ncu_name, mode=mode, brute=brute)
    assert st == exp["status"]
    if mode == "error":
        return
    assert idx.tolist() == exp["ncu_idx"]
    assert kind.tolist() == [1 if i >= 0 else 0 for i in exp["ncu_idx"]]
    if mode == "skip_name":
        assert summ["names_mismatched"] == exp["names_mismatched"]
    rk = np.array(g["expect"]["range_of_kernel"], np.int32)
    st, ops, tot = oracle.aggregate(kd, rk, ro, counters, idx, g["n_ops"])
    assert st == oracle.OK
    for key in ("kernel_count", "total_duration_ns", "matched_count"):
        assert ops[key].tolist() == exp["ops"][key]
    assert_agg(exp["ops"]["c1_sum"], ops["agg"][0])
    assert_agg(exp["ops"]["c4_dw"], ops["agg"][3])
    assert_agg(exp["ops"]["c5_dw"], ops["agg"][4])
    assert_agg(exp["ops"]["c18_max"], ops["agg"][17])
    for c in set(range(NC)) - {0, 3, 4, 17}:            # every other counter is null in every row
        assert np.isnan(ops["agg"][c]).all()
    t = g["expect"]["totals"]
    assert (tot["total_ns"], tot["attributed_ns"], tot["unattributed_ns"]) == (
        t["total_ns"], t["attributed_ns"], t["unattributed_ns"])
    assert tot["attributed_frac"] == pytest.approx(37 / 68, rel=1e-15)


@pytest.mark.parametrize("mode", ["skip_name", "prefix"])
def test_worked_permuted(golden, mode):
    # The same trace with kernel and range arrays permuted: every kernel start
    # is distinct, so time order -- and with it every output -- only follows
    # the permutation (kernel i of the new arrays is kernel kp[i] of the old).
    g = golden("worked.json")
    (rs, rt, re, rd, ro), (ks, kt, kd, kn), ncu_name, counters = worked_arrays(g)
    kp = np.array([9, 3, 7, 0, 5, 1, 8, 2, 6, 4])
    rp = np.array([4, 8, 0, 6, 2, 7, 1, 5, 3])
    inv_r = np.argsort(rp)
    exp_rk = [int(inv_r[x]) if x >= 0 else -1 for x in np.array(g["expect"]["range_of_kernel"])[kp]]
    for emode in ("brute", "indexed"):
        st, rk, nop = oracle.enclose(ks[kp], kt[kp], rs[rp], rt[rp], re[rp], rd[rp], ro[rp], mode=emode)
        assert st == oracle.OK and rk.tolist() == exp_rk
        assert nop.tolist() == np.array(g["expect"]["n_op_enclosing"])[kp].tolist()
    st, idx, kind, summ = oracle.match(ks[kp], kt[kp], kn[kp], ncu_name, mode=mode)
    assert st == g["expect"][mode]["status"]
    assert idx.tolist() == np.array(g["expect"][mode]["ncu_idx"])[kp].tolist()


@pytest.mark.parametrize("brute", [False, True])
def test_per_stream_ordinals(brute):
    # Limitations paragraph (Sec. 5): Nsight Compute replays a multi-stream
    # workload one stream per run, so its rows come as per-stream runs and
    # the k-th launch of a name must be counted per (name, stream).
    # Launches in time order: t0 A on s0, t1 A on s1, t2 A on s0, t3 B on s1.
    # Rows: the s0 run (A, A), then the s1 run (A, B).
    ks = np.array([0, 1, 0, 1], np.uint8)
    kt = np.array([0, 1, 2, 3], np.int64)
    kn = np.array([7, 7, 7, 9], np.uint32)
    nn = np.array([7, 7, 7, 9], np.uint32)
    ns = np.array([0, 0, 1, 1], np.uint8)
    st, idx, kind, summ = oracle.match(ks, kt, kn, nn, ncu_stream=ns, brute=brute)
    assert st == oracle.OK and idx.tolist() == [0, 2, 1, 3] and kind.tolist() == [1, 1, 1, 1]
    # the per-name reading pairs the rows with the wrong launches
    st, idx, kind, summ = oracle.match(ks, kt, kn, nn, brute=brute)
    assert idx.tolist() == [0, 1, 2, 3]
    # a run missing one launch: skip-name drops only that (name, stream)
    st, idx, kind, summ = oracle.match(ks, kt, kn, nn[[0, 2, 3]], ncu_stream=ns[[0, 2, 3]], brute=brute)
    assert st == oracle.W_COUNT_MISMATCH and idx.tolist() == [-1, 1, -1, 2]
    assert summ["names_mismatched"] == 1 and summ["count_unmatched"] == 2
    # names must fit beside the stream in one 32-bit key
    st, _, _, _ = oracle.match(ks, kt, np.array([7, 7, 1 << 24, 9], np.uint32), nn, ncu_stream=ns, brute=brute)
    assert st == oracle.E_INVALID_ARG


def test_per_stream_runs_generator():
    # tracegen.per_stream_runs regroups one-row-per-kernel traces into runs:
    # with per-stream ordinals every kernel gets its own row back
    t = tracegen.generate("gpt2")
    u = tracegen.per_stream_runs(t)
    st, idx, kind, summ = oracle.match(u.k_stream, u.k_start, u.k_name, u.ncu_name, ncu_stream=u.ncu_stream)
    assert st == oracle.OK and (kind == 1).all()
    assert np.array_equal(u.counters[idx], t.counters)
    assert np.array_equal(u.ncu_stream[idx], u.k_stream)


@pytest.mark.parametrize("name,shuffle", [("dedup", False), ("gpt2", True), ("dedup", True)])
def test_per_stream_runs_generator_dedup_shuffled(name, shuffle):
    # with layer classes the rows are the replayed kernels only, and with
    # shuffled kernel arrays the rows still follow kernel time order: per-
    # stream ordinals give every replayed kernel the row the time-ordered
    # join gave it
    t = tracegen.generate(name, shuffle=shuffle)
    u = tracegen.per_stream_runs(t)
    dd = bool(t.config.get("dedup")) and t.k_layer is not None
    args = dict(k_layer=t.k_layer, class_of_layer=t.class_of_layer, rep_of_class=t.rep_of_class, dedup=dd)
    st0, idx0, kind0, _ = oracle.match(t.k_stream, t.k_start, t.k_name, t.ncu_name, **args)
    st1, idx1, kind1, _ = oracle.match(u.k_stream, u.k_start, u.k_name, u.ncu_name, ncu_stream=u.ncu_stream, **args)
    assert st0 == oracle.OK and st1 == oracle.OK
    assert np.array_equal(kind0, kind1)
    m = idx0 >= 0
    assert np.array_equal(idx1 >= 0, m)
    assert np.array_equal(u.counters[idx1[m]], t.counters[idx0[m]])
    assert np.array_equal(u.ncu_stream[idx1[kind1 == 1]], u.k_stream[kind1 == 1])


def test_table8_rules():
    # Table 8: SUM for #1 #2 #3 #11 #15 #19, MAX for #18 #20, DW-mean for the rest
    sums, maxes = {1, 2, 3, 11, 15, 19}, {18, 20}
    want = [oracle.SUM if c + 1 in sums else oracle.MAX if c + 1 in maxes else oracle.DW for c in range(NC)]
    assert oracle.agg_rules() == want


# ---------------------------------------------------------------- dedup, Fig. 3, single kernel

@pytest.mark.parametrize("brute", [False, True])
def test_dedup_mini(golden, brute):
    g = golden("dedup_mini.json")
    k = g["kernels"]
    args = (np.array(k["stream"], np.uint8), np.array(k["start"], np.int64))
    layer = np.array(k["layer"], np.int32)
    col, roc = np.array(g["class_of_layer"], np.int32), np.array(g["rep_of_class"], np.int32)
    ncu = np.array(g["ncu_name"], np.uint32)
    st, idx, kind, summ = oracle.match(*args, np.array(k["name"], np.uint32), ncu, layer, col, roc, dedup=True,
                                       brute=brute)
    e = g["expect"]
    assert st == oracle.OK
    assert idx.tolist() == e["ncu_idx"] and kind.tolist() == e["match_kind"]
    assert summ["replayed"] == e["replayed"] == len(ncu)
    assert summ["replayed"] * 4 == len(layer) * 2            # N/K = 4/2 replay reduction
    st, idx, kind, summ = oracle.match(*args, np.array(e["swapped_names"], np.uint32), ncu, layer, col, roc,
                                       dedup=True, brute=brute)
    assert st == e["swapped_status"]
    assert idx.tolist() == e["swapped_ncu_idx"]
    assert summ["dedup_mismatch"] == e["swapped_dedup_mismatch"]


def test_clock_domain_order_not_time(golden):
    g = golden("clock_domain.json")
    ns, nc = np.array(g["nsys_t"]), np.array(g["ncu_t"])
    # the figure's failure mode: a nearest-timestamp join sends K_D to K_C's row
    assert int(np.argmin(np.abs(nc - ns[3]))) == g["expect"]["nearest_timestamp_join_of_K_D"]
    names = np.array(g["names"], np.uint32)
    for scale, shift in [(1000, 0), (1000, 50_000), (7, 3)]:
        kt = (ns * scale).astype(np.int64) + shift
        st, idx, _, _ = oracle.match(np.zeros(5, np.uint8), kt, names, names)
        assert st == oracle.OK and idx.tolist() == g["expect"]["ncu_idx"]


def test_single_kernel_operator(golden):
    g = golden("single_kernel.json")
    row = np.full((1, NC), np.nan, np.float32)
    for num, v in g["counters"].items():
        row[0, int(num) - 1] = np.nan if v is None else v
    st, ops, tot = oracle.aggregate(np.array([g["duration_ns"]]), np.array([0], np.int32),
                                    np.array([0], np.uint32), row, np.array([0], np.int32), 1)
    assert st == oracle.OK
    assert ops["total_duration_ns"][0] == g["expect"]["total_duration_ns"]
    assert ops["kernel_count"][0] == g["expect"]["kernel_count"]
    for num, v in g["counters"].items():
        got = ops["agg"][int(num) - 1][0]
        if v is None:
            assert math.isnan(got)
        else:
            assert got == float(np.float32(v))                # n = 1: the aggregate is the raw value


# ---------------------------------------------------------------- validation

def _v(ranges, mode):
    s, a, b, d = zip(*ranges)
    return oracle.validate_ranges(np.array(s), np.array(a), np.array(b), np.array(d), mode=mode)


@pytest.mark.parametrize("mode", ["brute", "indexed"])
def test_validation(mode):
    ok = [(0, 0, 10, 0), (0, 2, 5, 1), (0, 5, 5, 1), (0, 5, 8, 1), (0, 5, 5, 2), (0, 5, 5, 2)]
    assert _v(ok, mode) == oracle.OK
    assert _v([(0, 0, 10, 0), (0, 5, 12, 0)], mode) == oracle.E_NOT_NESTED       # same-depth overlap
    assert _v([(0, 0, 10, 0), (0, 5, 12, 1)], mode) == oracle.E_NOT_NESTED       # sticks out of parent
    assert _v([(0, 0, 10, 0), (1, 2, 5, 1)], mode) == oracle.E_NOT_NESTED        # parent on another stream
    assert _v([(0, 0, 10, 0), (0, 2, 5, 2)], mode) == oracle.E_NOT_NESTED        # depth gap
    assert _v([(0, 0, 10, 0), (0, 0, 10, 0)], mode) == oracle.E_NOT_NESTED       # positive-length twins
    assert _v([(0, 0, 10, 32)], mode) == oracle.E_DEPTH
    assert _v([(0, 5, 4, 0)], mode) == oracle.E_INVALID_ARG
    assert _v([(0, 0, 10, 0), (0, 10, 20, 0), (0, 10, 10, 0)], mode) == oracle.OK  # touching + zero length


def test_empty_and_uncovered():
    e64, e8, e32 = np.zeros(0, np.int64), np.zeros(0, np.uint8), np.zeros(0, np.uint32)
    st, rk, nop = oracle.enclose(e8, e64, e8, e64, e64, e8, e32)
    assert st == 0 and rk.size == 0
    ks, kt = np.array([0, 1, 3], np.uint8), np.array([5, 6, 7], np.int64)
    st, rk, nop = oracle.enclose(ks, kt, e8, e64, e64, e8, e32)
    assert st == 0 and rk.tolist() == [-1, -1, -1] and nop.tolist() == [0, 0, 0]
    st, ops, tot = oracle.aggregate(np.array([4, 5, 6]), rk, e32, np.zeros((0, NC), np.float32),
                                    np.full(3, -1, np.int32), 0)
    assert st == 0 and tot["total_ns"] == 15 and tot["unattributed_ns"] == 15 and tot["attributed_frac"] == 0.0
    st, ops, tot = oracle.aggregate(e64, np.zeros(0, np.int32), e32, np.zeros((0, NC), np.float32),
                                    np.zeros(0, np.int32), 3)
    assert st == 0 and math.isnan(tot["attributed_frac"]) and ops["kernel_count"].tolist() == [0, 0, 0]
    assert np.isnan(ops["agg"]).all()


def test_walk_cases():
    # one stream, nested chain: STRUCT(0) > OP a(1) > NONOP(2) > OP b(3) > STRUCT(4) > OP c(5)
    rs = np.zeros(6, np.uint8)
    rt = np.array([0, 1, 2, 3, 4, 5], np.int64)
    re = np.array([100, 90, 80, 70, 60, 50], np.int64)
    rd = np.arange(6, dtype=np.uint8)
    ro = np.array([oracle.STRUCTURAL, 0, oracle.NONOP, 1, oracle.STRUCTURAL, 2], np.uint32)
    kt = np.array([0, 1, 2, 3, 4, 5, 55, 65, 75, 85, 95, 200], np.int64)
    st, rk, nop = oracle.enclose(np.zeros(len(kt), np.uint8), kt, rs, rt, re, rd, ro, mode="brute")
    assert st == 0
    # T=3: b, skip the non-op, a, stop -> (b, 2); T=4 and T=55: the innermost range is
    # structural, so the walk stops before any operator; T=5: c, then the cut -> (c, 1)
    assert rk.tolist() == [-1, 1, 1, 3, -1, 5, -1, 3, 1, 1, -1, -1]
    assert nop.tolist() == [0, 1, 1, 2, 0, 1, 0, 2, 1, 1, 0, 0]


# ---------------------------------------------------------------- brute force vs indexed / Algorithm 1

@pytest.mark.parametrize("seed", range(300))
def test_enclosure_brute_vs_indexed(seed):
    t = tracegen.small_random(seed, n_streams=1 + seed % 3, n_events=20 + seed % 50, max_depth=1 + seed % 6)
    a = oracle.enclose(t.k_stream, t.k_start, t.r_stream, t.r_start, t.r_end, t.r_depth, t.r_op, mode="brute")
    b = oracle.enclose(t.k_stream, t.k_start, t.r_stream, t.r_start, t.r_end, t.r_depth, t.r_op, mode="indexed")
    c = oracle.enclose(t.k_stream, t.k_start, t.r_stream, t.r_start, t.r_end, t.r_depth, t.r_op, mode="brute_chain")
    assert a[0] == b[0] == c[0] == oracle.OK
    assert a[1].tolist() == b[1].tolist() == c[1].tolist() and a[2].tolist() == b[2].tolist() == c[2].tolist()
    # the chosen range contains T on the kernel's stream and is an operator
    for k in np.nonzero(a[1] >= 0)[0]:
        r = a[1][k]
        assert t.r_stream[r] == t.k_stream[k] and t.r_start[r] <= t.k_start[k] <= t.r_end[r]
        assert t.r_op[r] < t.n_ops


@pytest.mark.parametrize("seed", range(200))
def test_validation_brute_vs_indexed(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 12))
    s = rng.integers(0, 2, n)
    a = rng.integers(0, 8, n)
    b = a + rng.integers(0, 4, n)
    d = rng.integers(0, 3, n)
    assert oracle.validate_ranges(s, a, b, d, "brute") == oracle.validate_ranges(s, a, b, d, "indexed")


@pytest.mark.parametrize("seed", range(150))
@pytest.mark.parametrize("mode", ["skip_name", "prefix", "error"])
def test_match_brute_vs_algorithm1(seed, mode):
    t = tracegen.small_random(seed, n_events=60, n_names=2 + seed % 4)
    rng = np.random.default_rng(seed + 1000)
    ncu = t.ncu_name.copy()
    if seed % 3 == 1 and len(ncu):             # drop rows: count mismatches
        ncu = np.delete(ncu, rng.integers(0, len(ncu), 1 + seed % 3))
    elif seed % 3 == 2 and len(ncu):           # an extra row and a swap
        ncu = np.append(ncu, ncu[0])
        i, j = rng.integers(0, len(ncu), 2)
        ncu[i], ncu[j] = ncu[j], ncu[i]
    a = oracle.match(t.k_stream, t.k_start, t.k_name, ncu, mode=mode, brute=True)
    b = oracle.match(t.k_stream, t.k_start, t.k_name, ncu, mode=mode, brute=False)
    assert a[0] == b[0]
    if a[0] >= 0:
        assert a[1].tolist() == b[1].tolist() and a[2].tolist() == b[2].tolist() and a[3] == b[3]
        used = a[1][a[1] >= 0]
        assert len(np.unique(used)) == len(used)                    # no row is used twice
        assert (ncu[used] == t.k_name[a[1] >= 0]).all()             # a row carries its kernel's name


@pytest.mark.parametrize("seed", range(40))
def test_dedup_brute_vs_algorithm1(seed):
    cfg = tracegen.config("dedup", seed=100 + seed, n_streams=1 + seed % 3, n_iters=2, n_slots=3 + seed % 4,
                          n_classes=1 + seed % 3, tmpl_len=(4 + seed % 5, 3, 6, 0, 0, 0, 0, 0))
    t = tracegen.generate(cfg)
    name = t.k_name.copy()
    if seed % 4 == 3:
        name[np.random.default_rng(seed).integers(0, t.K)] += 1
    args = (t.k_stream, t.k_start, name, t.ncu_name, t.k_layer, t.class_of_layer, t.rep_of_class)
    a = oracle.match(*args, dedup=True, brute=True)
    b = oracle.match(*args, dedup=True, brute=False)
    assert a[0] == b[0] and a[1].tolist() == b[1].tolist() and a[3] == b[3]
    if seed % 4 != 3:
        assert a[0] == oracle.OK and a[3]["unmatched"] == 0


# ---------------------------------------------------------------- aggregation vs numpy

@pytest.mark.parametrize("seed", range(30))
def test_aggregate_vs_numpy(seed):
    rng = np.random.default_rng(seed)
    K, R, M, O = 500, 60, 400, 25
    r_op = rng.integers(0, O, R).astype(np.uint32)
    r_op[rng.random(R) < 0.1] = oracle.STRUCTURAL
    ops_ok = np.nonzero(r_op < O)[0]
    rk = np.where(rng.random(K) < 0.8, rng.choice(ops_ok, K), -1).astype(np.int32)
    idx = np.where(rng.random(K) < 0.9, rng.integers(0, M, K), -1).astype(np.int32)
    dur = rng.integers(0, 10**6, K).astype(np.int64)
    cnt = rng.uniform(0, 1000, (M, NC)).astype(np.float32)
    cnt[rng.random((M, NC)) < 0.05] = np.nan
    st, ops, tot = oracle.aggregate(dur, rk, r_op, cnt, idx, O)
    assert st == 0
    att = rk >= 0
    op = r_op[rk[att]].astype(np.int64)
    assert ops["kernel_count"].tolist() == np.bincount(op, minlength=O).tolist()
    assert ops["total_duration_ns"].tolist() == np.bincount(op, weights=dur[att], minlength=O).astype(np.int64).tolist()
    m_att = att & (idx >= 0)
    op_m = r_op[rk[m_att]].astype(np.int64)
    assert ops["matched_count"].tolist() == np.bincount(op_m, minlength=O).tolist()
    rules = oracle.agg_rules()
    for c in range(NC):
        v = cnt[idx[m_att], c].astype(np.float64)
        d = dur[m_att].astype(np.float64)
        ok = ~np.isnan(v)
        n = np.bincount(op_m[ok], minlength=O)
        if rules[c] == oracle.SUM:
            want = np.bincount(op_m[ok], weights=v[ok], minlength=O)
        elif rules[c] == oracle.DW:
            den = np.bincount(op_m[ok], weights=d[ok], minlength=O)
            with np.errstate(invalid="ignore", divide="ignore"):
                want = np.bincount(op_m[ok], weights=v[ok] * d[ok], minlength=O) / den
            want[den == 0] = np.nan
        else:
            want = np.full(O, -np.inf)
            np.maximum.at(want, op_m[ok], v[ok])
        want[n == 0] = np.nan
        np.testing.assert_allclose(ops["agg"][c], want, rtol=1e-12, equal_nan=True)
    assert tot["total_ns"] == dur.sum() and tot["attributed_ns"] == dur[att].sum()


def test_aggregate_rejects():
    one = np.array([0], np.int32)
    good = np.ones((1, NC), np.float32)
    bad = good.copy(); bad[0, 5] = np.inf
    assert oracle.aggregate([1], one, [0], bad, one, 1)[0] == oracle.E_INVALID_ARG
    assert oracle.aggregate([-1], one, [0], good, one, 1)[0] == oracle.E_INVALID_ARG
    assert oracle.aggregate([1], one, [oracle.STRUCTURAL], good, one, 1)[0] == oracle.E_INVALID_ARG
    assert oracle.aggregate([1], one, [3], good, one, 2)[0] == oracle.E_INVALID_ARG
    assert oracle.aggregate([1], np.array([1], np.int32), [0], good, one, 1)[0] == oracle.E_INVALID_ARG
    assert oracle.aggregate([1], one, [0], good, np.array([1], np.int32), 1)[0] == oracle.E_INVALID_ARG


# ---------------------------------------------------------------- invariants on the configurations

@pytest.mark.parametrize("name", ["tiny", "gpt2", "gpt2_dedup", "dedup"])
def test_config_invariants(name):
    t = tracegen.generate(name)
    res = oracle.run(t)
    assert res["enclose_status"] == oracle.OK and res["aggregate_status"] == oracle.OK
    assert res["match_status"] == oracle.OK
    rk, idx, ops, tot = res["range_of_kernel"], res["ncu_idx"], res["ops"], res["totals"]
    att = rk >= 0
    assert (t.r_op[rk[att]] < t.n_ops).all()                                   # an operator range
    assert (t.r_stream[rk[att]] == t.k_stream[att]).all()
    assert ((t.r_start[rk[att]] <= t.k_start[att]) & (t.k_start[att] <= t.r_end[rk[att]])).all()
    assert tot["attributed_ns"] + tot["unattributed_ns"] == tot["total_ns"] == t.k_dur.sum()
    assert ops["kernel_count"].sum() == att.sum()
    assert ops["total_duration_ns"].sum() == tot["attributed_ns"]
    direct = idx[res["match_kind"] == 1]
    assert len(np.unique(direct)) == len(direct)                                # no row matched twice
    assert res["summary"]["unmatched"] == 0
    # weighted means lie between the per-operator min and max of the counter
    rules = oracle.agg_rules()
    m = att & (idx >= 0)
    op = t.r_op[rk[m]].astype(np.int64)
    for c in [c for c in range(NC) if rules[c] == oracle.DW][:4]:
        v = t.counters[idx[m], c].astype(np.float64)
        lo = np.full(t.n_ops, np.inf); hi = np.full(t.n_ops, -np.inf)
        np.minimum.at(lo, op, v); np.maximum.at(hi, op, v)
        dw = ops["agg"][c]
        has = ~np.isnan(dw)
        assert (dw[has] >= lo[has] * (1 - 1e-12)).all() and (dw[has] <= hi[has] * (1 + 1e-12)).all()
    if t.class_of_layer is not None and t.config.get("dedup"):
        # replay count reduced by exactly N/K for layer kernels
        n_layers, n_classes = len(t.class_of_layer), len(t.rep_of_class)
        in_layer = t.k_layer >= 0
        assert res["summary"]["replayed"] * n_layers == (
            (~in_layer).sum() * n_layers + in_layer.sum() * n_classes)
        assert res["summary"]["replayed"] == t.M


# ---------------------------------------------------------------- attribution tiers (Fig. 2)

def _tiers_args(g):
    k = g["kernels"]
    kern = (np.array(k["stream"], np.uint8), np.array(k["start"], np.int64), np.array(k["name"], np.uint32),
            np.array(k["range_of_kernel"], np.int32), np.array(k["n_op_enclosing"], np.uint8))
    corr = tuple(np.array(g["corr"][f], np.uint32) for f in ("name", "invocation", "op"))
    fusion = (np.array(g["fusion"]["op_of_name"], np.uint32), np.array(g["fusion"]["list_len"], np.uint8))
    return kern, np.array(g["r_op"], np.uint32), g["n_ops"], corr, fusion


@pytest.mark.parametrize("brute", [True, False])
def test_tiers_worked(golden, brute):
    g = golden("tiers.json")
    (ks, kt, kn, rk, nop), r_op, n_ops, corr, fusion = _tiers_args(g)
    st, op, tier, fw, fz, summ = oracle.attribute(ks, kt, kn, rk, nop, r_op, n_ops, corr, fusion, brute=brute)
    e = g["expect"]
    assert st == oracle.OK
    assert op.tolist() == e["op_of_kernel"]
    assert tier.tolist() == e["tier"]
    assert fw.tolist() == e["fused_with"]
    assert fz.tolist() == e["is_fused"]
    assert summ == e["summary"]


def test_tiers_rejects(golden):
    g = golden("tiers.json")
    (ks, kt, kn, rk, nop), r_op, n_ops, corr, fusion = _tiers_args(g)
    # a repeated pair that names a launch (B, 2 -> k6)
    dup = tuple(np.append(a, v).astype(np.uint32) for a, v in zip(corr, (1, 2, 3)))
    assert oracle.attribute(ks, kt, kn, rk, nop, r_op, n_ops, dup, fusion)[0] == oracle.E_INVALID_ARG
    big = (corr[0], corr[1], np.where(np.arange(len(corr[2])) == 4, n_ops, corr[2]).astype(np.uint32))
    assert oracle.attribute(ks, kt, kn, rk, nop, r_op, n_ops, big, fusion)[0] == oracle.E_INVALID_ARG
    fbig = (np.array([n_ops, 15, 16, 16], np.uint32), fusion[1])
    assert oracle.attribute(ks, kt, kn, rk, nop, r_op, n_ops, corr, fbig)[0] == oracle.E_INVALID_ARG
    rbad = rk.copy(); rbad[1] = len(r_op)
    assert oracle.attribute(ks, kt, kn, rbad, nop, r_op, n_ops, corr, fusion)[0] == oracle.E_INVALID_ARG
    nonop = np.array([10, oracle.NONOP, 12], np.uint32)                 # an attributed range must be an operator
    assert oracle.attribute(ks, kt, kn, rk, nop, nonop, n_ops, corr, fusion)[0] == oracle.E_INVALID_ARG


@pytest.mark.parametrize("seed", range(0, 60, 4))
def test_tiers_brute_vs_indexed(seed):
    # invocation indices by rescanning every earlier kernel and map lookups by
    # scanning the whole map, against per-name counters and the sorted map
    t = tracegen.small_random(seed, n_streams=1 + seed % 4, n_events=10 + (seed * 7) % 90, max_depth=1 + seed % 7,
                              n_names=2 + seed % 5)
    u = tracegen.with_tiers(t, seed=seed, p_corr=[0.0, 0.3, 0.7, 1.0][seed % 4], p_fused=0.4)
    a = oracle.run_tiers(u, enclose_mode="brute", brute=True)
    b = oracle.run_tiers(u, enclose_mode="indexed", brute=False)
    assert a["attribute_status"] == b["attribute_status"] == oracle.OK
    for k in ("op_of_kernel", "tier", "fused_with", "is_fused"):
        assert np.array_equal(a[k], b[k]), k
    assert a["tier_summary"] == b["tier_summary"]


@pytest.mark.parametrize("name", ["tiny", "gpt2", "dedup"])
def test_tiers_reduce_to_enclosure(name):
    # without either map every kernel takes its enclosing operator (NVTX) or
    # none, and aggregating by operator equals aggregating by range
    t = tracegen.generate(name)
    r = oracle.run(t)
    q = oracle.run_tiers(t, use_corr=False, use_fusion=False)
    rk = r["range_of_kernel"]
    want = np.where(rk >= 0, t.r_op[np.maximum(rk, 0)], oracle.OP_NONE).astype(np.uint32)
    assert np.array_equal(q["op_of_kernel"], want)
    assert np.array_equal(q["tier"], np.where(rk >= 0, oracle.TIER_NVTX, oracle.TIER_NONE))
    assert np.array_equal(q["is_fused"], (r["n_op_enclosing"] > 1).astype(np.uint8))
    for k in ("kernel_count", "total_duration_ns", "matched_count"):
        assert np.array_equal(q["ops"][k], r["ops"][k])
    assert np.array_equal(np.isnan(q["ops"]["agg"]), np.isnan(r["ops"]["agg"]))
    m = ~np.isnan(r["ops"]["agg"])
    assert np.array_equal(q["ops"]["agg"][m], r["ops"]["agg"][m])
    assert q["totals"] == r["totals"]


@pytest.mark.parametrize("name", ["tiny", "gpt2"])
def test_tiers_full_map(name):
    # a map entry for every launch: every kernel is HIGH, and its operator is
    # the entry for (its name, the number of earlier launches of that name)
    t = tracegen.with_tiers(tracegen.generate(name), p_corr=1.0, p_stray=0.0)
    q = oracle.run_tiers(t)
    assert (q["tier"] == oracle.TIER_HIGH).all()
    order = np.lexsort((np.arange(t.K), t.k_stream.astype(np.int64), t.k_start))
    seen = {}
    lookup = {(int(n), int(i)): int(o) for n, i, o in zip(t.corr_name, t.corr_inv, t.corr_op)}
    for k in order[:2000]:
        n = int(t.k_name[k])
        i = seen.get(n, 0)
        seen[n] = i + 1
        assert q["op_of_kernel"][k] == lookup[(n, i)]


# ---------------------------------------------------------------- class roll-up

@pytest.mark.parametrize("name", ["tiny", "gpt2", "dedup"])
def test_rollup_from_operator_records(name):
    # the class records follow from the operator records and the operators'
    # matched durations alone: counts and durations add up, SUM counters add
    # up, MAX counters take the maximum, and a duration-weighted mean is the
    # mean of its operators' means weighted by their matched duration (no
    # null counters in these traces)
    t = tracegen.generate(name)
    r = oracle.run(t)
    rk, idx = r["range_of_kernel"], r["ncu_idx"]
    op = np.where(rk >= 0, t.r_op[np.maximum(rk, 0)], oracle.OP_NONE).astype(np.uint32)
    C = 9
    cm = tracegen.op_classes(t, n_classes=C, seed=3)
    st, cr, _ = oracle.rollup(t.k_dur, op, t.counters, idx, cm, C)
    assert st == oracle.OK
    ops = r["ops"]
    has = cm != oracle.OP_NONE
    cl = cm[has].astype(np.int64)
    for k in ("kernel_count", "total_duration_ns", "matched_count"):
        assert np.array_equal(cr[k], np.bincount(cl, ops[k][has], minlength=C).astype(np.int64))
    att = (op != oracle.OP_NONE) & (idx >= 0)
    wop = np.bincount(op[att].astype(np.int64), t.k_dur[att].astype(np.float64), minlength=t.n_ops)
    rules = oracle.agg_rules()
    for c in range(NC):
        v = ops["agg"][c][has]
        ok = ~np.isnan(v)
        if rules[c] == oracle.SUM:
            want = np.bincount(cl[ok], v[ok], minlength=C)
        elif rules[c] == oracle.MAX:
            want = np.full(C, -np.inf)
            np.maximum.at(want, cl[ok], v[ok])
        else:
            w = wop[has][ok]
            want = np.bincount(cl[ok], v[ok] * w, minlength=C) / np.bincount(cl[ok], w, minlength=C)
        got = cr["agg"][c]
        m = np.bincount(cl[ok], minlength=C) > 0
        assert np.all(np.isnan(got[~m]))
        np.testing.assert_allclose(got[m], want[m], rtol=1e-12, err_msg=f"counter {c}")


def test_rollup_one_class_per_op():
    # classes equal to operators: the roll-up is the operator aggregation
    t = tracegen.generate("tiny")
    r = oracle.run(t)
    rk = r["range_of_kernel"]
    op = np.where(rk >= 0, t.r_op[np.maximum(rk, 0)], oracle.OP_NONE).astype(np.uint32)
    st, cr, _ = oracle.rollup(t.k_dur, op, t.counters, r["ncu_idx"], np.arange(t.n_ops, dtype=np.uint32), t.n_ops)
    assert st == oracle.OK
    for k in ("kernel_count", "total_duration_ns", "matched_count"):
        assert np.array_equal(cr[k], r["ops"][k])
    assert np.array_equal(np.isnan(cr["agg"]), np.isnan(r["ops"]["agg"]))


# ---------------------------------------------------------------- the pins catch planted mistakes

MUTATIONS = [
    ("half-open interval", "r_start[i] <= T && T <= r_end[i]", "r_start[i] <= T && T < r_end[i]"),
    ("structural range skipped, not a stop", "if (op == OP_STRUCTURAL) break;", "if (op == OP_STRUCTURAL) continue;"),
    ("walk outermost first", "for (int d = MAX_DEPTH - 1; d >= 0; --d) {", "for (int d = 0; d < MAX_DEPTH; ++d) {"),
    ("representative by smallest start", "if (r->start[a] != r->start[b]) return r->start[a] > r->start[b];",
     "if (r->start[a] != r->start[b]) return r->start[a] < r->start[b];"),
    ("unweighted mean", "nadd(&num[at], m * (double)d); den[at] += d;", "nadd(&num[at], m); den[at] += 1;"),
    ("minimum for MAX counters", "(m > mx[at] ? m : mx[at])", "(m < mx[at] ? m : mx[at])"),
    ("ordinal over array order", "int64_t k = order[a];\n            if (replayed[k]) ord_k[k]",
     "int64_t k = a;\n            if (replayed[k]) ord_k[k]"),
    ("prefix rule in skip-name mode", "mode == MODE_SKIP_NAME ? (cnt_k[n] == cnt_j[n]) : (ord_k[k] < cnt_j[n])",
     "(ord_k[k] < cnt_j[n])"),
    ("dedup source from the kernel's own layer", "int64_t src = p < lay_cnt[rep] ? lay_kern[rep][p] : -1;",
     "int64_t src = p < lay_cnt[k_layer[k]] ? lay_kern[k_layer[k]][p] : -1;"),
    ("SUM and DW swapped for counter #1", "    AGG_SUM, AGG_SUM, AGG_SUM,                  /* 1 gpu time",
     "    AGG_DW, AGG_SUM, AGG_SUM,                  /* 1 gpu time"),
    ("attributed time counts every kernel", "att += d; natt++;", "natt++;"),
    ("invocation index over array order", "int64_t k = order[a];\n            inv[k] = ",
     "int64_t k = a;\n            inv[k] = "),
    ("NVTX before HIGH", "if (hits == 1) { op = c_op[hit]; t = TIER_HIGH; }\n        else if (rok[k] >= 0)",
     "if (rok[k] >= 0 && 0) { }\n        else if (rok[k] >= 0) { op = r_op[rok[k]]; t = TIER_NVTX; }\n"
     "        else if (hits == 1) { op = c_op[hit]; t = TIER_HIGH; }\n        else if (0)"),
    ("fusion overrides NVTX", "else if (rok[k] >= 0) { op = r_op[rok[k]]; t = TIER_NVTX; }\n        else if (fo != OP_NONE)",
     "else if (fo != OP_NONE) { op = fo; t = TIER_INDUCTOR; }\n        else if (rok[k] >= 0) { op = r_op[rok[k]]; t = TIER_NVTX; }\n        else if (0)"),
    ("fused list length ignored", "(fo != OP_NONE && fl > 1)", "(fo != OP_NONE)"),
    ("walk count marks every tier fused", "(t == TIER_NVTX && nop && nop[k] > 1)", "(nop && nop[k] > 1)"),
]


def _all_pins(golden):
    """Run every hand-derived pin; return the list of failures (names)."""
    failures = []
    for fn, args in [(test_worked_enclosure, ("brute",)), (test_worked_enclosure, ("indexed",)),
                     (test_worked_match_and_aggregate, ("skip_name", False)),
                     (test_worked_match_and_aggregate, ("prefix", False)),
                     (test_worked_match_and_aggregate, ("prefix", True)),
                     (test_worked_permuted, ("skip_name",)), (test_worked_permuted, ("prefix",)),
                     (test_dedup_mini, (False,)), (test_table8_rules, ()), (test_single_kernel_operator, ()),
                     (test_walk_cases, ()), (test_clock_domain_order_not_time, ()), (test_tiers_worked, (True,)),
                     (test_tiers_worked, (False,))]:
        try:
            if fn in (test_table8_rules, test_walk_cases):
                fn()
            else:
                fn(golden, *args)
        except AssertionError:
            failures.append(fn.__name__)
    return failures


@pytest.mark.parametrize("label,old,new", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_pins_catch_mutation(tmp_path, golden, label, old, new):
    src = open(oracle._SRC).read()
    assert src.count(old) == 1, f"mutation anchor not found: {label}"
    mutant = tmp_path / "oracle_mut.c"
    mutant.write_text(src.replace(old, new))
    so = tmp_path / "liboracle_mut.so"
    subprocess.run(["gcc", "-O1", "-std=c11", "-shared", "-fPIC", str(mutant), "-o", str(so), "-lm"], check=True)
    assert _all_pins(golden) == []                   # the real oracle passes every pin
    with oracle.use_library(str(so)):
        failures = _all_pins(golden)
    assert failures, f"no pin caught the planted mistake: {label}"


@pytest.mark.parametrize("name,kw", [("tiny", {}), ("gpt2", {}), ("gpt2_dedup", {}), ("dedup", {}),
                                     ("large", dict(n_kernels=150_000)),
                                     ("adversarial", dict(n_kernels=150_000))])
def test_threaded_oracle_equals_single_thread(name, kw):
    """The CPU baseline's threaded run (streams, names and op blocks split
    over host threads) gives the single-thread oracle's outputs bit for bit."""
    from oracle.parallel import run_threads
    t = tracegen.generate(name, **kw)
    a = oracle.run(t, enclose_mode="indexed")
    b = run_threads(t, 5)
    for k in ("enclose_status", "match_status", "aggregate_status", "summary"):
        assert a[k] == b[k], k
    for k in ("range_of_kernel", "n_op_enclosing", "ncu_idx", "match_kind"):
        np.testing.assert_array_equal(a[k], b[k], err_msg=k)
    for k in ("kernel_count", "total_duration_ns", "matched_count"):
        np.testing.assert_array_equal(a["ops"][k], b["ops"][k], err_msg=k)
    assert np.array_equal(a["ops"]["agg"].view(np.int64), b["ops"]["agg"].view(np.int64))
    for k, v in a["totals"].items():
        assert v == b["totals"][k] or (v != v and b["totals"][k] != b["totals"][k]), k
