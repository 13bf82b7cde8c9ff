"""GPU parity: the CUDA path, called through the C ABI, against the CPU oracle
on the same seeded inputs.  Integer outputs bit-exact, floating-point
aggregates within 1e-9 relative."""
import json
import os

import numpy as np
import pytest

import oracle
import tracegen
from gpu_util import RTOL, assert_close, assert_parity, assert_parity_tiers, gpu_run, gpu_run_tiers

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


@pytest.fixture(scope="module")
def opa():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_11938_gb300 as m
    m.build()
    return m


def worked_trace():
    g = json.load(open(os.path.join(GOLDEN, "worked.json")))
    conv = {"STRUCTURAL": oracle.STRUCTURAL, "NONOP": oracle.NONOP}
    r, k, n = g["ranges"], g["kernels"], g["ncu"]
    counters = np.array([[np.nan if v is None else v for v in row] for row in n["counters"]], np.float32)
    t = tracegen.Trace(
        k_stream=np.array(k["stream"], np.uint8), k_start=np.array(k["start"], np.int64),
        k_dur=np.array(k["dur"], np.int64), k_name=np.array(k["name"], np.uint32), k_layer=None,
        r_stream=np.array(r["stream"], np.uint8), r_start=np.array(r["start"], np.int64),
        r_end=np.array(r["end"], np.int64), r_depth=np.array(r["depth"], np.uint8),
        r_op=np.array([conv.get(x, x) for x in r["op"]], np.uint32), n_ops=g["n_ops"],
        ncu_name=np.array(n["name"], np.uint32), counters=counters)
    return g, t


@pytest.mark.parametrize("mode", ["skip_name", "prefix"])
def test_worked_example(opa, mode):
    g, t = worked_trace()
    res = gpu_run(t, mode=mode)
    e = g["expect"]
    assert res["range_of_kernel"].tolist() == e["range_of_kernel"]
    assert res["n_op_enclosing"].tolist() == e["n_op_enclosing"]
    assert res["ncu_idx"].tolist() == e[mode]["ncu_idx"]
    assert res["match_status"] == e[mode]["status"]
    ops = res["ops"]
    for key in ("kernel_count", "total_duration_ns", "matched_count"):
        assert ops[key].tolist() == e[mode]["ops"][key]
    for col, key in ((0, "c1_sum"), (3, "c4_dw"), (4, "c5_dw"), (17, "c18_max")):
        want = np.array([np.nan if v is None else v for v in e[mode]["ops"][key]])
        assert_close(ops["agg"][col], want, rtol=1e-12, what=key)
    assert res["totals"]["attributed_ns"] == 37 and res["totals"]["total_ns"] == 68
    assert_parity(res, oracle.run(t, mode=mode, enclose_mode="brute"))


def test_worked_error_mode(opa):
    _, t = worked_trace()
    ctx = opa.Context(0, mismatch="error")
    tr = opa.to_device(t)
    with pytest.raises(opa.OpattrError) as ei:
        ctx.match(tr)
    assert ei.value.status == opa.E_COUNT_MISMATCH
    # the context stays usable after an error status
    st, rk, nop = ctx.enclose(tr)
    assert st == opa.OK and rk.cpu().tolist() == [-1, 2, 8, 2, 4, 5, -1, -1, 7, -1]
    ctx.close()


@pytest.mark.parametrize("seed", range(160))
def test_small_random(opa, seed):
    t = tracegen.small_random(seed, n_streams=1 + seed % 4, n_events=10 + (seed * 7) % 90,
                              max_depth=1 + seed % 7, shuffle=seed % 2 == 0, n_names=2 + seed % 5)
    if seed % 5 == 3 and t.M > 1:              # force the general match path and count mismatches
        t.ncu_name = t.ncu_name[1:].copy()
        t.counters = t.counters[1:].copy()
    if seed % 7 == 4:
        t.counters[np.random.default_rng(seed).random(t.counters.shape) < 0.2] = np.nan
    mode = ["skip_name", "prefix"][seed % 2]
    assert_parity(gpu_run(t, mode=mode), oracle.run(t, mode=mode, enclose_mode="brute"))


@pytest.mark.parametrize("name", ["tiny", "gpt2", "gpt2_dedup", "dedup"])
@pytest.mark.parametrize("shuffle", [False, True])
def test_configs(opa, name, shuffle):
    t = tracegen.generate(name, shuffle=shuffle)
    g = gpu_run(t)
    o = oracle.run(t, enclose_mode="brute" if name in ("tiny", "gpt2") else "indexed")
    assert_parity(g, o)
    assert g["match_status"] == opa.OK and g["summary"]["unmatched"] == 0
    # rows follow the replayed launches in time order, shuffled kernel arrays
    # or not: one pass pairs them, through the time order when it is needed
    assert g["summary"]["fast_path"] == 1


@pytest.mark.parametrize("mode", ["skip_name", "prefix", "error"])
def test_gpt2_count_mismatch(opa, mode):
    t = tracegen.generate("gpt2")
    rng = np.random.default_rng(7)
    drop = rng.choice(t.M, 25, replace=False)
    keep = np.setdiff1d(np.arange(t.M), drop)
    t.ncu_name, t.counters = t.ncu_name[keep].copy(), t.counters[keep].copy()
    o = oracle.run(t, mode=mode, enclose_mode="indexed")
    if mode == "error":
        import paper_2609_11938_gb300 as m
        ctx = m.Context(0, mismatch="error")
        with pytest.raises(m.OpattrError) as ei:
            ctx.match(m.to_device(t))
        assert ei.value.status == m.E_COUNT_MISMATCH == o["match_status"]
        ctx.close()
        return
    g = gpu_run(t, mode=mode)
    assert g["match_status"] == opa.W_COUNT_MISMATCH
    assert_parity(g, o)


def test_dedup_swapped_names(opa):
    t = tracegen.generate("dedup")
    # rename one kernel of a duplicate layer: its broadcast source no longer matches
    dup = np.nonzero((t.k_layer >= 0) & (t.rep_of_class[t.class_of_layer[np.maximum(t.k_layer, 0)]] != t.k_layer))[0]
    t.k_name = t.k_name.copy()
    t.k_name[dup[::997]] += 1
    g = gpu_run(t)
    o = oracle.run(t)
    assert g["match_status"] == o["match_status"] == opa.W_DEDUP_MISMATCH
    assert_parity(g, o)


def test_nan_counters(opa):
    t = tracegen.generate("gpt2", nan_frac=0.1, nan_mask=1 << 12)
    g, o = gpu_run(t), oracle.run(t, enclose_mode="indexed")
    assert np.isnan(g["ops"]["agg"][12]).all()
    assert_parity(g, o)


def test_empty_inputs(opa):
    t = tracegen.small_random(3)
    z = lambda a: a[:0].copy()
    for cut in ("kernels", "ranges", "ncu", "all"):
        u = tracegen.small_random(3)
        if cut in ("kernels", "all"):
            u.k_stream, u.k_start, u.k_dur, u.k_name = z(t.k_stream), z(t.k_start), z(t.k_dur), z(t.k_name)
        if cut in ("ranges", "all"):
            u.r_stream, u.r_start, u.r_end, u.r_depth, u.r_op = (z(t.r_stream), z(t.r_start), z(t.r_end),
                                                                z(t.r_depth), z(t.r_op))
            u.n_ops = 0
        if cut in ("ncu", "all"):
            u.ncu_name, u.counters = z(t.ncu_name), z(t.counters)
        assert_parity(gpu_run(u), oracle.run(u, enclose_mode="brute"))


def test_error_statuses(opa):
    import torch
    t = tracegen.small_random(11, n_events=80, max_depth=4)
    ctx = opa.Context(0)
    # depth above 31
    u = tracegen.small_random(11, n_events=80, max_depth=4)
    u.r_depth = u.r_depth.copy(); u.r_depth[0] = 32
    with pytest.raises(opa.OpattrError) as ei:
        ctx.enclose(opa.to_device(u))
    assert ei.value.status == opa.E_DEPTH
    # end before start
    u = tracegen.small_random(11, n_events=80, max_depth=4)
    u.r_end = u.r_end.copy(); u.r_end[0] = u.r_start[0] - 1
    with pytest.raises(opa.OpattrError) as ei:
        ctx.enclose(opa.to_device(u))
    assert ei.value.status == opa.E_INVALID_ARG
    # two overlapping ranges at one depth
    u = tracegen.small_random(11, n_events=80, max_depth=4)
    u.r_stream = np.append(u.r_stream, [0, 0]).astype(np.uint8)
    u.r_start = np.append(u.r_start, [100, 105]).astype(np.int64)
    u.r_end = np.append(u.r_end, [110, 120]).astype(np.int64)
    u.r_depth = np.append(u.r_depth, [0, 0]).astype(np.uint8)
    u.r_op = np.append(u.r_op, [u.n_ops, u.n_ops + 1]).astype(np.uint32)
    assert oracle.validate_ranges(u.r_stream, u.r_start, u.r_end, u.r_depth) == oracle.E_NOT_NESTED
    with pytest.raises(opa.OpattrError) as ei:
        ctx.enclose(opa.to_device(u))
    assert ei.value.status == opa.E_NOT_NESTED
    # aggregate: out-of-range index, infinite counter, negative duration
    tr = opa.to_device(t)
    st, rk, _ = ctx.enclose(tr)
    st, idx, _, _ = ctx.match(tr)
    bad = rk.clone(); bad[0] = t.R
    with pytest.raises(opa.OpattrError):
        ctx.aggregate(tr, bad, idx)
    att = int(np.nonzero(rk.cpu().numpy() >= 0)[0][0])   # an attributed kernel's row index past the rows
    bad = idx.clone(); bad[att] = t.M
    with pytest.raises(opa.OpattrError) as ei:
        ctx.aggregate(tr, rk, bad)
    assert ei.value.status == opa.E_INVALID_ARG
    u = tracegen.small_random(11, n_events=80, max_depth=4)
    u.counters = u.counters.copy(); u.counters[:, 4] = np.inf
    res = oracle.run(u)
    if (res["range_of_kernel"] >= 0).any():
        with pytest.raises(opa.OpattrError) as ei:
            ctx.aggregate(opa.to_device(u), rk, idx)
        assert ei.value.status == opa.E_INVALID_ARG == res["aggregate_status"]
    u = tracegen.small_random(11, n_events=80, max_depth=4)
    u.k_dur = u.k_dur.copy(); u.k_dur[-1] = -5
    with pytest.raises(opa.OpattrError):
        ctx.aggregate(opa.to_device(u), rk, idx)
    # still usable afterwards
    assert_parity(gpu_run(t, ctx=ctx), oracle.run(t, enclose_mode="brute"))
    ctx.close()


def test_oom_injection(opa, monkeypatch):
    t = tracegen.generate("tiny")
    monkeypatch.setenv("OPATTR_FAULT", "alloc")
    ctx = opa.Context(0)
    with pytest.raises(opa.OpattrError) as ei:
        ctx.enclose(opa.to_device(t))
    assert ei.value.status == opa.E_OOM
    monkeypatch.delenv("OPATTR_FAULT")
    assert_parity(gpu_run(t, ctx=ctx), oracle.run(t, enclose_mode="brute"))
    ctx.close()


def test_lookback_wait_bound(opa, monkeypatch):
    """Scans out of place chain their tiles' prefixes by decoupled look-back,
    whose wait is bounded by the context's spin limit.  With every status word
    reading as silent (OPATTR_FAULT=lookback) each tile gives up after that
    many polls and sums the silent tiles' input itself: the call returns
    E_TIMEOUT and its outputs are still exact."""
    import torch
    t = tracegen.generate("dedup")
    assert t.n_ops + 1 > 32 * 1024            # the per-op offsets take the multi-tile scan
    ctx = opa.Context(0, spin_limit=64)
    tr = opa.to_device(t)
    _, rk, _ = ctx.enclose(tr)
    _, idx, _, _ = ctx.match(tr, dedup=True)
    _, want, want_tot = ctx.aggregate(tr, rk, idx)
    got = ctx.alloc_ops(t.n_ops)
    monkeypatch.setenv("OPATTR_FAULT", "lookback")
    with pytest.raises(opa.OpattrError) as ei:
        ctx.aggregate(tr, rk, idx, ops=got)
    assert ei.value.status == opa.E_TIMEOUT
    monkeypatch.delenv("OPATTR_FAULT")
    torch.cuda.synchronize()
    for key in want:
        np.testing.assert_array_equal(got[key].cpu().numpy(), want[key].cpu().numpy(), err_msg=key)
    # the context goes on as before
    st, again, tot = ctx.aggregate(tr, rk, idx)
    assert st >= 0 and tot == want_tot
    np.testing.assert_array_equal(again["agg"].cpu().numpy(), want["agg"].cpu().numpy())
    ctx.close()


def _agg_inputs(seed, K, seg_lens, n_small_ops, nan_frac=0.0, counter_dist="uniform", dur_sigma=1.2,
                dur_median=8000.0):
    """Aggregation-only inputs: ops 0..len(seg_lens)-1 get seg_lens[i] kernels,
    the rest of the kernels fall on n_small_ops more ops or stay unattributed;
    kernel order is shuffled so that every op's kernels are scattered.
    Counters uniform on [0, 100] or log-uniform on [1e-3, 1e3]; durations
    log-normal with the given median and sigma."""
    rng = np.random.default_rng(seed)
    n_ops = len(seg_lens) + n_small_ops
    op_of = np.full(K, -1, np.int64)
    pos = 0
    for i, n in enumerate(seg_lens):
        op_of[pos:pos + n] = i
        pos += n
    rest = K - pos
    op_of[pos:] = np.where(rng.random(rest) < 0.9, len(seg_lens) + rng.integers(0, n_small_ops, rest), -1)
    op_of = op_of[rng.permutation(K)]
    # one range per op id plus a few ranges sharing op ids (duplicates aggregate together)
    r_op = np.concatenate([np.arange(n_ops), rng.integers(0, n_ops, 64)]).astype(np.uint32)
    dup_of_op = {int(r_op[n_ops + q]): n_ops + q for q in range(64)}
    rk = np.where(op_of >= 0, op_of, -1).astype(np.int32)
    for k in np.nonzero(op_of >= 0)[0][::7]:              # some kernels through the duplicate ranges
        if int(op_of[k]) in dup_of_op:
            rk[k] = dup_of_op[int(op_of[k])]
    dur = rng.lognormal(np.log(dur_median), dur_sigma, K).astype(np.int64)
    M = K
    if counter_dist == "loguniform":
        counters = np.exp(rng.uniform(np.log(1e-3), np.log(1e3), (M, 20))).astype(np.float32)
    else:
        counters = rng.uniform(0, 100, (M, 20)).astype(np.float32)
    if nan_frac:
        counters[rng.random((M, 20)) < nan_frac] = np.nan
    idx = np.where(rng.random(K) < 0.95, np.arange(K), -1).astype(np.int32)
    R = len(r_op)
    t = tracegen.Trace(np.zeros(K, np.uint8), np.arange(K, dtype=np.int64), dur, np.zeros(K, np.uint32), None,
                       np.zeros(R, np.uint8), np.arange(R, dtype=np.int64), np.arange(R, dtype=np.int64),
                       np.zeros(R, np.uint8), r_op, n_ops, np.zeros(M, np.uint32), counters)
    return t, rk, idx


def _gpu_aggregate(opa, t, rk, idx, ctx=None):
    import torch
    own = ctx is None
    ctx = ctx or opa.Context(0)
    try:
        tr = opa.to_device(t)
        st, ops, tot = ctx.aggregate(tr, torch.from_numpy(rk).cuda(), torch.from_numpy(idx).cuda())
        return st, {k: v.cpu().numpy() for k, v in ops.items()}, tot
    finally:
        if own:
            ctx.close()


def _check_aggregate(g, o):
    gst, gops, gtot = g
    ost, oops, otot = o
    assert gst == ost
    for k in ("kernel_count", "total_duration_ns", "matched_count"):
        np.testing.assert_array_equal(gops[k], oops[k])
    for c in range(20):
        assert_close(gops["agg"][c], oops["agg"][c], what=f"counter {c}")
    for k in ("total_ns", "attributed_ns", "kernels", "attributed_kernels", "matched_kernels"):
        assert gtot[k] == otot[k], k


@pytest.mark.parametrize("nan_frac", [0.0, 0.02])
def test_aggregate_segment_lengths(opa, nan_frac):
    """Ops whose kernels are walked by selection (<= 48), after an in-place
    sort (49 .. 16384) and in list order (above), with kernels scattered over
    the array, duplicate op ids and null counters: against the oracle."""
    seg_lens = [1, 2, 48, 49, 64, 65, 100, 256, 257, 300, 1024, 1025, 5000, 16384, 16385, 40000]
    t, rk, idx = _agg_inputs(7, 200_000, seg_lens, 20_000, nan_frac)
    o = oracle.aggregate(t.k_dur, rk, t.r_op, t.counters, idx, t.n_ops)
    _check_aggregate(_gpu_aggregate(opa, t, rk, idx), o)


@pytest.mark.parametrize("rows", ["identity", "swapped", "unmatched", "last"])
def test_aggregate_identity_rows(opa, rows):
    """Row index k for every kernel k (the ops pass skips the row-index
    gather) and near misses that must take the gather: two kernels' rows
    swapped, one kernel without a row, the last kernel's row moved."""
    t, rk, _ = _agg_inputs(9, 150_000, [3, 64, 65, 300, 5000], 20_000)
    K = len(rk)
    idx = np.arange(K, dtype=np.int32)
    if rows == "swapped":
        idx[[10, 70_000]] = idx[[70_000, 10]]
    elif rows == "unmatched":
        idx[12_345] = -1
    elif rows == "last":
        idx[K - 1] = 0
    o = oracle.aggregate(t.k_dur, rk, t.r_op, t.counters, idx, t.n_ops)
    _check_aggregate(_gpu_aggregate(opa, t, rk, idx), o)


def test_aggregate_reproducible(opa):
    """Two runs give bit-identical records although the count pass orders each
    op's kernel list by atomics: segments are walked in ascending index."""
    t, rk, idx = _agg_inputs(8, 300_000, [3000, 700], 40_000)
    ctx = opa.Context(0)
    a = _gpu_aggregate(opa, t, rk, idx, ctx)[1]
    b = _gpu_aggregate(opa, t, rk, idx, ctx)[1]
    ctx.close()
    for k in a:
        assert np.array_equal(a[k].view(np.int64), b[k].view(np.int64)), k
    assert_parity(gpu_run(t), oracle.run(t, enclose_mode="indexed"))


def test_large_full_parity(opa):
    """The 20M-kernel benchmark trace, in the configuration the benchmark runs,
    against the oracle on every output."""
    t = tracegen.generate("large")
    g = gpu_run(t)
    assert g["summary"]["fast_path"] == 1
    o = oracle.run(t, enclose_mode="indexed")
    assert_parity(g, o)


def _endpoint_kernels(t):
    """Kernels whose T equals the start or end of some range on their stream."""
    ep = np.zeros(t.K, bool)
    for s in np.unique(t.k_stream):
        km = np.nonzero(t.k_stream == s)[0]
        rm = t.r_stream == s
        e = np.unique(np.concatenate([t.r_start[rm], t.r_end[rm]]))
        if len(e) == 0:
            continue
        T = t.k_start[km]
        p = np.minimum(np.searchsorted(e, T), len(e) - 1)
        ep[km[e[p] == T]] = True
    return ep


def test_adversarial_full_parity(opa):
    """The 50M-kernel adversarial trace (64 streams, depth up to 32, zero-length
    and identical-endpoint ranges, 85% of runtime outside every range) against
    the indexed oracle on every output of every kernel and op; in addition a
    sample of the kernels that sit exactly on a range endpoint (the closed
    interval and tie rules of Algorithm 2) and a 1-in-10^4 sample of all
    kernels against the brute-force chain."""
    t = tracegen.generate("adversarial")
    g = gpu_run(t)
    assert g["summary"]["fast_path"] == 1
    o = oracle.run(t, enclose_mode="indexed")
    assert_parity(g, o)
    ep = _endpoint_kernels(t)
    assert ep.mean() > 0.01                           # the configuration's >= 1 % of endpoint kernels
    rng = np.random.default_rng(4)
    pick = np.union1d(rng.choice(np.nonzero(ep)[0], 20_000, replace=False), np.arange(0, t.K, 10_000))
    st, b_rk, b_nop = oracle.enclose(t.k_stream[pick], t.k_start[pick], t.r_stream, t.r_start, t.r_end, t.r_depth,
                                     t.r_op, mode="brute_chain")
    assert st == 0
    np.testing.assert_array_equal(g["range_of_kernel"][pick], b_rk)
    np.testing.assert_array_equal(g["n_op_enclosing"][pick], b_nop)


@pytest.mark.parametrize("name,order", [("gpt2", None), ("gpt2", "reversed"), ("large2m", None)])
def test_per_stream_runs(opa, name, order):
    """ncu rows as per-stream replay runs, tagged with their stream: ordinals
    per (name, stream), against the oracle; every kernel gets its own row."""
    t = tracegen.generate("large", n_kernels=2_000_000) if name == "large2m" else tracegen.generate(name)
    streams = np.unique(t.k_stream)
    u = tracegen.per_stream_runs(t, None if order is None else streams[::-1])
    g = gpu_run(u)
    assert_parity(g, oracle.run(u, enclose_mode="indexed"))
    assert (g["match_kind"] == 1).all()
    assert g["summary"]["fast_path"] == 1
    np.testing.assert_array_equal(u.counters[g["ncu_idx"]], t.counters)


@pytest.mark.parametrize("name,shuffle", [("dedup", False), ("gpt2", True), ("dedup", True), ("gpt2_dedup", False)])
def test_per_stream_partition_paths(opa, name, shuffle):
    """Per-stream rows with layer classes (the rows are the replayed kernels,
    gathered by stream) and with kernel arrays out of time order: the
    stream-partitioned pairing gives the oracle's answer."""
    t = tracegen.generate(name, shuffle=shuffle)
    u = tracegen.per_stream_runs(t)
    g = gpu_run(u)
    assert_parity(g, oracle.run(u, enclose_mode="indexed"))
    assert g["summary"]["fast_path"] == 1
    assert g["summary"]["unmatched"] == 0


@pytest.mark.parametrize("mode", ["skip_name", "prefix", "error"])
def test_per_stream_swapped_rows(opa, mode):
    """Two rows of different names swapped inside one stream's run: the
    stream-partitioned pairing no longer holds and the general ordinal join
    decides, name by name."""
    t = tracegen.generate("gpt2")
    u = tracegen.per_stream_runs(t)
    s0 = np.nonzero(u.ncu_stream == u.ncu_stream[0])[0]
    j = s0[1 + np.nonzero(u.ncu_name[s0[1:]] != u.ncu_name[s0[0]])[0][0]]
    for a in (u.ncu_name, u.counters):
        a[[s0[0], j]] = a[[j, s0[0]]]
    g = gpu_run(u, mode=mode)
    assert_parity(g, oracle.run(u, mode=mode, enclose_mode="indexed"))
    assert g["summary"]["fast_path"] == 0


@pytest.mark.parametrize("seed", range(0, 40, 3))
def test_per_stream_small_random(opa, seed):
    """Random traces with rows as per-stream runs, some rows dropped so the
    mismatch modes see per-(name, stream) count differences."""
    t = tracegen.small_random(seed, n_streams=1 + seed % 4, n_events=10 + (seed * 7) % 90, max_depth=1 + seed % 7,
                              n_names=2 + seed % 5)
    if t.M != t.K:
        pytest.skip("needs one row per kernel")
    u = tracegen.per_stream_runs(t)
    if seed % 2 and u.M > 2:
        keep = np.ones(u.M, bool)
        keep[[0, u.M // 2]] = False
        u.ncu_name, u.counters, u.ncu_stream = u.ncu_name[keep], u.counters[keep], u.ncu_stream[keep]
    mode = ["skip_name", "prefix"][seed % 2]
    assert_parity(gpu_run(u, mode=mode), oracle.run(u, mode=mode, enclose_mode="brute"))


def test_per_stream_name_limit(opa):
    """With stream-tagged rows a name id must fit in 24 bits."""
    t = tracegen.per_stream_runs(tracegen.generate("tiny"))
    t.k_name = t.k_name.copy()
    t.k_name[5] = 1 << 24
    ctx = opa.Context(0)
    with pytest.raises(opa.OpattrError) as ei:
        ctx.match(opa.to_device(t))
    assert ei.value.status == opa.E_INVALID_ARG
    ctx.close()


def test_launch_time_query(opa):
    """Algorithm 2 queries at the host launch timestamp, which precedes the
    GPU start by a variable lag: the enclosure takes those times as its query
    points (kernels then out of time order) while matching keeps GPU order."""
    import torch
    t = tracegen.generate("gpt2")
    rng = np.random.default_rng(3)
    launch = t.k_start - rng.integers(0, 4000, t.K)
    st, want_rk, want_nop = oracle.enclose(t.k_stream, launch, t.r_stream, t.r_start, t.r_end, t.r_depth, t.r_op,
                                           mode="indexed")
    assert st == oracle.OK
    ctx = opa.Context(0)
    tr = opa.to_device(t)
    tq = opa.to_device(t)
    tq.k_start = torch.from_numpy(launch).cuda()
    st, rk, nop = ctx.enclose(tq)
    np.testing.assert_array_equal(rk.cpu().numpy(), want_rk)
    np.testing.assert_array_equal(nop.cpu().numpy(), want_nop)
    st, idx, kind, _ = ctx.match(tr)
    st, ops, tot = ctx.aggregate(tr, rk, idx)
    o = oracle.aggregate(t.k_dur, want_rk, t.r_op, t.counters, idx.cpu().numpy(), t.n_ops)
    for k in ("kernel_count", "total_duration_ns", "matched_count"):
        np.testing.assert_array_equal(ops[k].cpu().numpy(), o[1][k])
    assert_close(ops["agg"].cpu().numpy(), o[1]["agg"], what="agg")
    ctx.close()


# ---------------------------------------------------------------- attribution tiers (Fig. 2)

def test_tiers_worked(opa):
    """The hand-derived tiers example (tests/golden/tiers.json) through the C ABI."""
    import torch
    g = json.load(open(os.path.join(GOLDEN, "tiers.json")))
    k = g["kernels"]
    dev = "cuda:0"
    t = lambda a, dt: torch.tensor(np.array(a, dt), device=dev)
    K = len(k["start"])
    tr = opa.DeviceTrace(t(k["stream"], np.uint8), t(k["start"], np.int64), t([1] * K, np.int64),
                         t(k["name"], np.int32), None, None, t([0] * 3, np.int64), t([0] * 3, np.int64), None,
                         t(g["r_op"], np.int32), g["n_ops"], t([], np.int32), None,
                         corr_name=t(g["corr"]["name"], np.int32), corr_inv=t(g["corr"]["invocation"], np.int32),
                         corr_op=t(g["corr"]["op"], np.int32),
                         fusion_op=t(np.array(g["fusion"]["op_of_name"], np.uint32).view(np.int32), np.int32),
                         fusion_len=t(g["fusion"]["list_len"], np.uint8))
    ctx = opa.Context(0)
    st, op, tier, fw, fz, summ = ctx.attribute(tr, t(k["range_of_kernel"], np.int32), t(k["n_op_enclosing"], np.uint8))
    e = g["expect"]
    assert st == 0
    assert op.cpu().numpy().view(np.uint32).tolist() == e["op_of_kernel"]
    assert tier.cpu().numpy().tolist() == e["tier"]
    assert fw.cpu().numpy().view(np.uint32).tolist() == e["fused_with"]
    assert fz.cpu().numpy().tolist() == e["is_fused"]
    assert summ == e["summary"]
    # a repeated pair that names a launch is rejected; the context stays usable
    tr.corr_name = t(g["corr"]["name"] + [1], np.int32)
    tr.corr_inv = t(g["corr"]["invocation"] + [2], np.int32)
    tr.corr_op = t(g["corr"]["op"] + [3], np.int32)
    with pytest.raises(opa.OpattrError) as ei:
        ctx.attribute(tr, t(k["range_of_kernel"], np.int32), t(k["n_op_enclosing"], np.uint8))
    assert ei.value.status == opa.E_INVALID_ARG
    tr.corr_op = t(g["corr"]["op"] + [g["n_ops"]], np.int32)
    tr.corr_name = t(g["corr"]["name"] + [1], np.int32)
    tr.corr_inv = t(g["corr"]["invocation"] + [7], np.int32)       # names no launch, but its operator is invalid
    with pytest.raises(opa.OpattrError) as ei:
        ctx.attribute(tr, t(k["range_of_kernel"], np.int32), t(k["n_op_enclosing"], np.uint8))
    assert ei.value.status == opa.E_INVALID_ARG
    ctx.close()


@pytest.mark.parametrize("name,shuffle,p_corr", [("tiny", False, 0.5), ("gpt2", False, 0.5), ("gpt2", True, 0.5),
                                                ("gpt2_dedup", False, 1.0), ("dedup", False, 0.3),
                                                ("dedup", True, 0.0)])
def test_tiers_configs(opa, name, shuffle, p_corr):
    """The tiers on the generator's configurations (kernels in and out of time
    order), against the oracle on every output, aggregation by operator included."""
    t = tracegen.with_tiers(tracegen.generate(name, shuffle=shuffle), p_corr=p_corr)
    assert_parity_tiers(gpu_run_tiers(t), oracle.run_tiers(t))


@pytest.mark.parametrize("seed", range(0, 80, 3))
def test_tiers_small_random(opa, seed):
    t = tracegen.small_random(seed, n_streams=1 + seed % 4, n_events=10 + (seed * 7) % 90, max_depth=1 + seed % 7,
                              n_names=2 + seed % 5)
    u = tracegen.with_tiers(t, seed=seed, p_corr=[0.0, 0.3, 0.7, 1.0][seed % 4], p_fused=[0.0, 0.4, 1.0][seed % 3])
    use_corr, use_fusion = seed % 5 != 1, seed % 7 != 2
    assert_parity_tiers(gpu_run_tiers(u, use_corr=use_corr, use_fusion=use_fusion),
                        oracle.run_tiers(u, use_corr=use_corr, use_fusion=use_fusion, enclose_mode="brute", brute=True))


def test_tiers_large(opa):
    """The 20 M-kernel trace with a correlation map for half of the launches and
    fusion entries for a tenth of the names, against the indexed oracle."""
    t = tracegen.with_tiers(tracegen.generate("large"))
    assert_parity_tiers(gpu_run_tiers(t), oracle.run_tiers(t))


# ---------------------------------------------------------------- class roll-up

def _rollup_case(opa, t, C, seed=3, tiers=False):
    import torch
    cm = tracegen.op_classes(t, n_classes=C, seed=seed)
    ctx = opa.Context(0)
    tr = opa.to_device(t)
    st, rk, nop = ctx.enclose(tr)
    st, idx, kind, summ = ctx.match(tr)
    dcm = torch.from_numpy(cm.view(np.int32)).cuda()
    if tiers:
        st, op, tier, fw, fz, ts = ctx.attribute(tr, rk, nop)
        st, cr = ctx.rollup(tr, None, idx, dcm, C, op_of_kernel=op)
        op_h = op.cpu().numpy().view(np.uint32)
    else:
        st, cr = ctx.rollup(tr, rk, idx, dcm, C)
        rk_h = rk.cpu().numpy()
        op_h = np.where(rk_h >= 0, t.r_op[np.maximum(rk_h, 0)], oracle.OP_NONE).astype(np.uint32)
    torch.cuda.synchronize()
    g = {k: v.cpu().numpy() for k, v in cr.items()}
    ctx.close()
    o_st, o, _ = oracle.rollup(t.k_dur, op_h, t.counters, idx.cpu().numpy(), cm, C)
    assert st == o_st == 0
    for k in ("kernel_count", "total_duration_ns", "matched_count"):
        np.testing.assert_array_equal(g[k], o[k], err_msg=k)
    assert_close(g["agg"], o["agg"], what="rollup agg")


@pytest.mark.parametrize("name,C", [("tiny", 5), ("gpt2", 64), ("dedup", 300), ("gpt2", 1)])
def test_rollup_configs(opa, name, C):
    """Per-class records against the oracle's aggregation by class (empty and
    left-out classes included)."""
    _rollup_case(opa, tracegen.generate(name), C)


def test_rollup_tiers(opa):
    """Roll-up of the tiered attribution (operators given per kernel)."""
    _rollup_case(opa, tracegen.with_tiers(tracegen.generate("gpt2")), 40, tiers=True)


def test_rollup_large(opa):
    """The 20 M-kernel trace rolled up to 64 classes."""
    _rollup_case(opa, tracegen.generate("large"), 64)


def test_rollup_rejects(opa):
    import torch
    t = tracegen.generate("tiny")
    ctx = opa.Context(0)
    tr = opa.to_device(t)
    st, rk, nop = ctx.enclose(tr)
    st, idx, kind, summ = ctx.match(tr)
    cm = np.zeros(t.n_ops, np.uint32)
    cm[3] = 7
    with pytest.raises(opa.OpattrError) as ei:
        ctx.rollup(tr, rk, idx, torch.from_numpy(cm.view(np.int32)).cuda(), 7)
    assert ei.value.status == opa.E_INVALID_ARG
    ctx.close()


# ---------------------------------------------------------------- profile.json

def test_profile_from_gpu(opa, tmp_path):
    """profile.json written from the GPU join's outputs against the one written
    from the oracle's: the same operators, kernels and tiers; aggregated
    counters within 1e-9."""
    t = tracegen.with_tiers(tracegen.generate("gpt2"))
    g = gpu_run_tiers(t)
    o = oracle.run_tiers(t)
    docs = []
    for r, tag in ((g, "gpu"), (o, "oracle")):
        path = tmp_path / f"{tag}.json"
        opa.write_profile(path, t.k_stream, t.k_dur, t.k_name, r["op_of_kernel"], r["ncu_idx"], t.counters, r["ops"],
                          tier=r["tier"], is_fused=r["is_fused"], fused_with=r["fused_with"])
        docs.append(json.load(open(path)))
    a, b = docs
    assert len(a["operators"]) == len(b["operators"]) and a["unattributed_kernels"] == b["unattributed_kernels"]
    for x, y in zip(a["operators"], b["operators"]):
        assert {k: v for k, v in x.items() if k != "aggregated"} == {k: v for k, v in y.items() if k != "aggregated"}
        for k, v in x["aggregated"].items():
            w = y["aggregated"][k]
            assert (v is None) == (w is None), k
            if v is not None:
                assert abs(v - w) <= RTOL * abs(w), (k, v, w)


@pytest.mark.parametrize("kids,p_kernel", [(1.2, 0.3), (2.0, 0.55), (3.0, 0.7)])
def test_enclose_dense_ranges(opa, kids, p_kernel):
    """Range-dense traces (about one range per kernel and fewer): tiles whose
    range windows outgrow the compact shared-memory layout are deferred to the
    wide layout, some or all of them; the result is the oracle's."""
    t = tracegen.generate("large", n_kernels=200_000, n_streams=2, max_depth=8, kids_mean=kids,
                          p_kernel_child=p_kernel, uncovered_frac=0.0)
    g = gpu_run(t)
    o = oracle.run(t, enclose_mode="indexed")
    np.testing.assert_array_equal(g["range_of_kernel"], o["range_of_kernel"])
    np.testing.assert_array_equal(g["n_op_enclosing"], o["n_op_enclosing"])


def _nesting_trace(case):
    """Ranges over several 4,096-range tiles for the laminar checks: stream 0
    parents each followed by one child (the parent in the child's tile),
    stream 1 one long parent over 9,000 children (the parent tiles back),
    stream 3 a child among 6,000 zero-length parents with its start (equal
    starts across a tile boundary), and per case one defect."""
    T = 500_000_000
    st, s, e, d = [], [], [], []

    def add(stream, a, b, depth):
        st.append(stream); s.append(a); e.append(b); d.append(depth)
    for i in range(6000):
        add(0, i * 100, i * 100 + 90, 0)
        add(0, i * 100 + 10, i * 100 + (95 if case == "past_near_parent" and i == 5000 else 50), 1)
    add(1, 0, 1_000_000_000, 0)
    for j in range(9000):
        add(1, j * 100 + 5, 1_000_000_001 if case == "past_far_parent" and j == 8999 else j * 100 + 55, 1)
    for q in range(6001):
        if q == 3000:
            add(3, T, T + (1 if case == "tie_past_parent" else 0), 1)
        else:
            add(3, T, T, 0)
    if case == "orphan":
        add(2, 500, 600, 1)
    order = np.argsort(np.asarray(s, np.int64), kind="stable")
    r_stream = np.asarray(st, np.uint8)[order]
    r_start = np.asarray(s, np.int64)[order]
    r_end = np.asarray(e, np.int64)[order]
    r_depth = np.asarray(d, np.uint8)[order]
    R = len(r_start)
    rng = np.random.default_rng(5)
    K = 3000
    k_start = np.sort(rng.integers(0, 1_000_000_100, K)).astype(np.int64)
    k_start[:5] = T                                   # a few kernels at the tied instant
    k_start.sort()
    k_stream = rng.integers(0, 4, K).astype(np.uint8)
    return tracegen.Trace(k_stream, k_start, np.full(K, 1000, np.int64), np.zeros(K, np.uint32), None,
                          r_stream, r_start, r_end, r_depth, np.arange(R, dtype=np.uint32), R,
                          np.zeros(K, np.uint32), np.zeros((K, 20), np.float32))


@pytest.mark.parametrize("case", ["valid", "past_near_parent", "past_far_parent", "orphan", "tie_valid",
                                  "tie_past_parent"])
def test_nesting_checks_across_tiles(opa, case):
    """The laminar checks of the level lists -- parent found in the child's
    tile, in an earlier tile, in a later tile through equal starts, or
    missing -- give the oracle's status; valid traces give its enclosure."""
    t = _nesting_trace(case)
    want = oracle.validate_ranges(t.r_stream, t.r_start, t.r_end, t.r_depth)
    assert (want == 0) == (case in ("valid", "tie_valid"))
    ctx = opa.Context(0)
    try:
        if want != 0:
            with pytest.raises(opa.OpattrError) as ei:
                ctx.enclose(opa.to_device(t))
            assert ei.value.status == want
        else:
            st, rk, nop = ctx.enclose(opa.to_device(t))
            ost, ork, onop = oracle.enclose(t.k_stream, t.k_start, t.r_stream, t.r_start, t.r_end, t.r_depth,
                                            t.r_op)
            assert st == ost == 0
            np.testing.assert_array_equal(rk.cpu().numpy(), ork)
            np.testing.assert_array_equal(nop.cpu().numpy(), onop)
    finally:
        ctx.close()


@pytest.mark.parametrize("shuffle,per_stream", [(False, False), (True, False), (False, True)])
def test_max_streams_and_depth(opa, shuffle, per_stream):
    """Every stream id (0..255) and every depth (0..31): thousands of levels
    (the radix-sorted level lists and the wide enclosure layout), in time
    order and permuted, and with per-stream ncu rows: against the oracle."""
    t = tracegen.generate("adversarial", n_kernels=400_000, n_streams=256, seed=21, shuffle=shuffle)
    assert len(np.unique(t.r_stream)) == 256 and int(t.r_depth.max()) == 31
    if per_stream:
        t = tracegen.per_stream_runs(t)
    assert_parity(gpu_run(t), oracle.run(t, enclose_mode="indexed"))


def _join_cases(name):
    if name == "large1m":
        return tracegen.generate("large", n_kernels=1_000_000)
    if name == "gpt2_shuffled":
        return tracegen.generate("gpt2", shuffle=True)
    if name == "dedup_per_stream":
        return tracegen.per_stream_runs(tracegen.generate("dedup"))
    if name == "gpt2_count_mismatch":
        t = tracegen.generate("gpt2")
        keep = np.setdiff1d(np.arange(t.M), np.random.default_rng(7).choice(t.M, 25, replace=False))
        t.ncu_name, t.counters = t.ncu_name[keep].copy(), t.counters[keep].copy()
        return t
    if name == "gpt2_rows_swapped":
        # as many rows as kernels, in time order except two rows of different
        # names swapped: the identity pairing that runs beside the enclosure
        # finds names that differ, and the ordinal join decides
        t = tracegen.generate("gpt2")
        names = t.ncu_name
        i = 100
        j = int(np.nonzero(names[i + 1:] != names[i])[0][0]) + i + 1
        order = np.arange(t.M)
        order[[i, j]] = order[[j, i]]
        t.ncu_name, t.counters = names[order].copy(), t.counters[order].copy()
        assert t.K == t.M
        return t
    return tracegen.generate(name)


@pytest.mark.parametrize("name", ["large1m", "gpt2_shuffled", "dedup", "dedup_per_stream", "gpt2_count_mismatch",
                                  "gpt2_rows_swapped", "tiny"])
def test_join_matches_three_calls(opa, name):
    """opattr_join gives the three calls' outputs bit for bit (the order
    verdict shared between enclosure and matching, sorted or not), their
    warning, and the oracle's results."""
    t = _join_cases(name)
    tr = opa.to_device(t)
    dd = bool(t.config.get("dedup")) and t.k_layer is not None     # as the oracle decides
    ctx = opa.Context(0)
    try:
        st, out, ops, summ, tot = ctx.join(tr, dedup=dd)
        e_st, rk, nop = ctx.enclose(tr)
        m_st, idx, kind, msumm = ctx.match(tr, dedup=dd)
        a_st, ops3, tot3 = ctx.aggregate(tr, rk, idx)
    finally:
        ctx.close()
    assert st == (m_st if m_st > 0 else a_st)
    np.testing.assert_array_equal(out["range_of_kernel"].cpu().numpy(), rk.cpu().numpy())
    np.testing.assert_array_equal(out["n_op_enclosing"].cpu().numpy(), nop.cpu().numpy())
    np.testing.assert_array_equal(out["ncu_idx"].cpu().numpy(), idx.cpu().numpy())
    np.testing.assert_array_equal(out["match_kind"].cpu().numpy(), kind.cpu().numpy())
    for k in ops:
        assert np.array_equal(ops[k].cpu().numpy().view(np.int64), ops3[k].cpu().numpy().view(np.int64)), k
    assert summ == msumm and tot == tot3
    o = oracle.run(t, enclose_mode="indexed")
    np.testing.assert_array_equal(out["range_of_kernel"].cpu().numpy(), o["range_of_kernel"])
    np.testing.assert_array_equal(out["ncu_idx"].cpu().numpy(), o["ncu_idx"])


def test_join_stops_at_the_first_error(opa):
    """A nesting error in the enclosure ends the join with that error; the
    context stays usable."""
    u = _nesting_trace("orphan")
    ctx = opa.Context(0)
    try:
        with pytest.raises(opa.OpattrError) as ei:
            ctx.join(opa.to_device(u))
        assert ei.value.status == opa.E_NOT_NESTED
        t = tracegen.generate("tiny")
        st, out, ops, summ, tot = ctx.join(opa.to_device(t))
        o = oracle.run(t, enclose_mode="brute")
        np.testing.assert_array_equal(out["range_of_kernel"].cpu().numpy(), o["range_of_kernel"])
    finally:
        ctx.close()


def test_join_nesting_error_with_deferred_status(opa):
    """A join whose matching is the identity pairing run beside the
    enclosure (kernels in (start, stream) order, one row per kernel with the
    same name) reads the enclosure's status with the aggregation's; a
    nesting error found there is still the join's status, and the context
    goes on."""
    u = _nesting_trace("orphan")
    order = np.lexsort((u.k_stream, u.k_start))          # strict time order: the deferred path
    u.k_stream, u.k_start = u.k_stream[order].copy(), u.k_start[order].copy()
    assert u.K == u.M
    ctx = opa.Context(0)
    try:
        with pytest.raises(opa.OpattrError) as ei:
            ctx.join(opa.to_device(u))
        assert ei.value.status == opa.E_NOT_NESTED
        t = tracegen.generate("tiny")
        st, out, ops, summ, tot = ctx.join(opa.to_device(t))
        o = oracle.run(t, enclose_mode="brute")
        np.testing.assert_array_equal(out["range_of_kernel"].cpu().numpy(), o["range_of_kernel"])
        np.testing.assert_array_equal(out["ncu_idx"].cpu().numpy(), o["ncu_idx"])
        assert summ["fast_path"] == 1
    finally:
        ctx.close()


def _equal_starts_trace():
    """Ranges sorted by start whose equal-start pairs at one depth are not in
    (start, end) order -- a long range listed before a zero-length one at the
    same instant -- with children below the long ones, over several tiles."""
    st, s, e, d = [], [], [], []
    for i in range(3000):
        a = i * 1000
        st += [0, 0, 0]
        s += [a, a, a + 10]
        e += [a + 500, a, a + 20]
        d += [0, 0, 1]
    R = len(s)
    rng = np.random.default_rng(9)
    K = 20_000
    k_start = np.sort(np.concatenate([rng.integers(0, 3_000_000, K - 3000), np.arange(3000) * 1000])).astype(np.int64)
    K = len(k_start)
    return tracegen.Trace(np.zeros(K, np.uint8), k_start, np.full(K, 100, np.int64),
                          rng.integers(0, 50, K).astype(np.uint32), None,
                          np.asarray(st, np.uint8), np.asarray(s, np.int64), np.asarray(e, np.int64),
                          np.asarray(d, np.uint8), np.arange(R, dtype=np.uint32), R,
                          rng.integers(0, 50, K).astype(np.uint32), rng.uniform(0, 100, (K, 20)).astype(np.float32))


def test_equal_starts_out_of_order(opa):
    """The level lists' equal-start fix-up (the enclosure redone on fully
    sorted ranges), through the enclosure alone and through the join, whose
    enclosure status is read at the matching's wait: the oracle's results."""
    t = _equal_starts_trace()
    t.ncu_name = t.k_name.copy()
    o = oracle.run(t, enclose_mode="indexed")
    assert o["enclose_status"] == 0
    ctx = opa.Context(0)
    try:
        tr = opa.to_device(t)
        st, rk, nop = ctx.enclose(tr)
        np.testing.assert_array_equal(rk.cpu().numpy(), o["range_of_kernel"])
        np.testing.assert_array_equal(nop.cpu().numpy(), o["n_op_enclosing"])
        st, out, ops, summ, tot = ctx.join(tr, dedup=False)
        np.testing.assert_array_equal(out["range_of_kernel"].cpu().numpy(), o["range_of_kernel"])
        np.testing.assert_array_equal(out["n_op_enclosing"].cpu().numpy(), o["n_op_enclosing"])
        np.testing.assert_array_equal(out["ncu_idx"].cpu().numpy(), o["ncu_idx"])
        for k in ("kernel_count", "total_duration_ns", "matched_count"):
            np.testing.assert_array_equal(ops[k].cpu().numpy(), o["ops"][k])
    finally:
        ctx.close()


def _shared_start_trace(longer_ranges: bool, longer_first: bool, shuffle: bool):
    """A small trace plus two ranges of one level (stream 0, depth 0) that
    start at the same instant T, after everything else: [T, T] and
    [T, T + 10] (laminar: the zero-length range touches the longer one), or
    [T, T + 10] and [T, T + 20] (overlapping); kernels at T and T + 5.  Ranges
    in array order or permuted (the level lists then come from the sort)."""
    import dataclasses
    u = tracegen.small_random(11, n_events=80, max_depth=4, shuffle=False)
    T = int(max(u.r_end.max(), u.k_start.max())) + 100
    ends = [T + 10, T + 20] if longer_ranges else [T, T + 10]
    if longer_first:
        ends = ends[::-1]
    r_start = np.append(u.r_start, [T, T]).astype(np.int64)
    r_end = np.append(u.r_end, ends).astype(np.int64)
    r_stream = np.append(u.r_stream, [0, 0]).astype(np.uint8)
    r_depth = np.append(u.r_depth, [0, 0]).astype(np.uint8)
    r_op = np.append(u.r_op, [0, 1]).astype(np.uint32)
    if shuffle:
        p = np.random.default_rng(5).permutation(len(r_start))
        r_start, r_end, r_stream, r_depth, r_op = (x[p] for x in (r_start, r_end, r_stream, r_depth, r_op))
    k_start = np.append(u.k_start, [T, T + 5]).astype(np.int64)
    return dataclasses.replace(u, k_stream=np.append(u.k_stream, [0, 0]).astype(np.uint8), k_start=k_start,
                               k_dur=np.append(u.k_dur, [3, 3]).astype(np.int64),
                               k_name=np.append(u.k_name, [0, 0]).astype(np.uint32),
                               r_stream=r_stream, r_start=r_start, r_end=r_end, r_depth=r_depth, r_op=r_op)


@pytest.mark.parametrize("longer_ranges", [False, True])
@pytest.mark.parametrize("longer_first", [False, True])
@pytest.mark.parametrize("shuffle", [False, True])
def test_shared_start_in_one_level(opa, longer_ranges, longer_first, shuffle):
    """Two ranges of one level sharing a start: beside a zero-length range the
    longer one is the level's representative at that instant (Algorithm 2's
    closed interval, one range per depth); two longer ones overlap and are
    not nested.  The oracle's status and enclosure, whatever the array order."""
    t = _shared_start_trace(longer_ranges, longer_first, shuffle)
    ost, ork, onop = oracle.enclose(t.k_stream, t.k_start, t.r_stream, t.r_start, t.r_end, t.r_depth, t.r_op,
                                    mode="brute")
    assert (ost == oracle.E_NOT_NESTED) == longer_ranges
    ctx = opa.Context(0)
    try:
        if longer_ranges:
            with pytest.raises(opa.OpattrError) as ei:
                ctx.enclose(opa.to_device(t))
            assert ei.value.status == opa.E_NOT_NESTED
        else:
            st, rk, nop = ctx.enclose(opa.to_device(t))
            assert st == ost == 0
            np.testing.assert_array_equal(rk.cpu().numpy(), ork)
            np.testing.assert_array_equal(nop.cpu().numpy(), onop)
            longer = int(np.nonzero((t.r_start == t.r_start.max()) & (t.r_end > t.r_start))[0][0])
            assert (ork[-2:] == longer).all()
    finally:
        ctx.close()


def _with_gap(t, cut, gap):
    """Every timestamp at or after `cut` moved later by `gap` ns: an idle gap
    in the trace.  The map is monotone, so order, nesting, ties and
    containment are kept and the expected outputs are the oracle's on the new
    times."""
    import dataclasses
    f = lambda x: np.where(x >= cut, x + gap, x)
    return dataclasses.replace(t, k_start=f(t.k_start), r_start=f(t.r_start), r_end=f(t.r_end))


@pytest.mark.parametrize("shuffle", [False, True])
def test_enclose_gaps_inside_tiles(opa, shuffle):
    """Idle gaps of seconds between profiled iterations put more than 2^32 ns
    inside one tile of time-ordered kernels, where times no longer fit the
    tile's 32-bit relative encoding; gaps just below that bound stay on the
    staged path.  Against the oracle on every output."""
    t = tracegen.generate("large", n_kernels=200_000, shuffle=shuffle)
    order = np.lexsort((np.arange(t.K), t.k_stream.astype(np.int64), t.k_start))
    ts = t.k_start[order]
    # cuts inside tiles of 2,048 time-ordered kernels (each a kernel's own time:
    # the gap opens just before it, with ranges open across it stretched)
    gaps = [(2048 * 3 + 700, 2**32 - 3_000_000), (2048 * 9 + 5, 2**32), (2048 * 17 + 1000, 5_000_000_000),
            (2048 * 30 + 2047, 2**32 + 1), (2048 * 41 + 1, 10**12), (2048 * 60 + 1024, 7_000_000_000)]
    for pos, gap in sorted(gaps, reverse=True):
        t = _with_gap(t, int(ts[pos]), gap)
    o = oracle.run(t, enclose_mode="indexed")
    assert_parity(gpu_run(t), o)


@pytest.mark.parametrize("nan_frac", [0.0, 0.01])
def test_aggregate_long_ops_wide_range(opa, nan_frac):
    """Operators of 200,000 to 1,000,000 kernels (an Inductor fusion operator
    can gather every unattributed launch of a name) with counters log-uniform
    over [1e-3, 1e3] and durations log-normal with sigma 2.0: Eq. (1) within
    1e-9 relative of the fp64 oracle."""
    t, rk, idx = _agg_inputs(13, 1_600_000, [200_000, 1_000_000, 4097, 70_000, 300], 30_000, nan_frac,
                             counter_dist="loguniform", dur_sigma=2.0, dur_median=3000.0)
    o = oracle.aggregate(t.k_dur, rk, t.r_op, t.counters, idx, t.n_ops)
    _check_aggregate(_gpu_aggregate(opa, t, rk, idx), o)
