"""The oracle run in host threads over independent parts of one trace.

TEST INFRASTRUCTURE ONLY, like the rest of this directory: the benchmark's
CPU-baseline leg and its reference arm time it.  It adds no arithmetic of its
own: each part goes through the unchanged single-thread oracle functions
(``oracle.enclose`` / ``match`` / ``aggregate``), which release the GIL while
they run, and the results are scattered back.  The parts are independent by
the method's own definitions, so the outputs equal the single-thread run's
exactly:

* enclosure (Algorithm 2, Sec. 3.5): a kernel's chain holds only ranges of its
  own stream, so streams are split into groups;
* matching (Algorithm 1, Sec. 3.3, no layer deduplication): ordinals, counts
  and mismatch decisions are per kernel name, so names are split by
  ``name % parts`` (each part keeps array order, so time-order ties and ncu
  launch order are unchanged);
* aggregation (Eq. (1), Sec. 3.8.1): an operator's record depends only on its
  own kernels, so op ids are split into contiguous blocks of similar kernel
  counts (each part keeps ascending kernel order, the oracle's summation
  order); unattributed kernels join the first part for the totals.
"""
from __future__ import annotations

import concurrent.futures as cf
import os

import numpy as np

from . import SUMMARY_FIELDS, aggregate, enclose, match

__all__ = ["run_threads"]


def _first_error(statuses):
    bad = [s for s in statuses if s != 0]
    return min(bad) if bad and min(bad) < 0 else (max(bad) if bad else 0)


def _enclose(ex, t, parts):
    ks = t.k_stream
    streams = np.unique(np.concatenate([np.unique(ks), np.unique(t.r_stream)]))
    load = np.bincount(ks, minlength=256)[streams]
    groups = [[] for _ in range(parts)]
    sizes = np.zeros(parts, np.int64)
    for s, n in sorted(zip(streams.tolist(), load.tolist()), key=lambda x: -x[1]):
        g = int(np.argmin(sizes))
        groups[g].append(s)
        sizes[g] += n
    rk = np.full(t.K, -1, np.int32)
    nop = np.zeros(t.K, np.uint8)

    def one(grp):
        if not grp:
            return 0
        sel = np.zeros(256, bool)
        sel[grp] = True
        kidx = np.nonzero(sel[ks])[0]
        ridx = np.nonzero(sel[t.r_stream])[0]
        st, r, n = enclose(ks[kidx], t.k_start[kidx], t.r_stream[ridx], t.r_start[ridx], t.r_end[ridx],
                           t.r_depth[ridx], t.r_op[ridx], mode="indexed")
        rk[kidx] = np.where(r >= 0, ridx[np.maximum(r, 0)], -1)
        nop[kidx] = n
        return st
    return _first_error(list(ex.map(one, groups))), rk, nop


def _match(ex, t, parts, mode):
    kp = t.k_name % parts
    np_ = t.ncu_name % parts
    idx = np.full(t.K, -1, np.int32)
    kind = np.zeros(t.K, np.uint8)

    def one(p):
        kidx = np.nonzero(kp == p)[0]
        nidx = np.nonzero(np_ == p)[0]
        st, i, k, s = match(t.k_stream[kidx], t.k_start[kidx], t.k_name[kidx], t.ncu_name[nidx], mode=mode)
        idx[kidx] = np.where(i >= 0, nidx[np.maximum(i, 0)], -1)
        kind[kidx] = k
        return st, s
    res = list(ex.map(one, range(parts)))
    summ = {f: sum(s[f] for _, s in res) for f in SUMMARY_FIELDS}
    return _first_error([st for st, _ in res]), idx, kind, summ


def _aggregate(ex, t, rk, idx, parts):
    n_ops = int(t.n_ops)
    op = np.where(rk >= 0, t.r_op[np.maximum(rk, 0)].astype(np.int64), -1)
    cnt = np.bincount(op[op >= 0], minlength=n_ops) if n_ops else np.zeros(0, np.int64)
    cum = np.cumsum(cnt)
    total = int(cum[-1]) if n_ops else 0
    cuts = [0] + [int(np.searchsorted(cum, total * (p + 1) / parts)) + 1 for p in range(parts - 1)] + [n_ops]
    cuts = np.minimum.accumulate(np.array(cuts)[::-1])[::-1].clip(0, n_ops)
    cuts = np.maximum.accumulate(cuts)
    kc = np.zeros(n_ops, np.int64)
    td = np.zeros(n_ops, np.int64)
    mc = np.zeros(n_ops, np.int64)
    agg = np.zeros((20, n_ops), np.float64)

    def one(p):
        lo, hi = int(cuts[p]), int(cuts[p + 1])
        m = (op >= lo) & (op < hi)
        if p == 0:
            m |= op < 0
        kidx = np.nonzero(m)[0]
        r_op_local = (t.r_op.astype(np.int64) - lo).astype(np.uint32)
        st, o, tot = aggregate(t.k_dur[kidx], rk[kidx], r_op_local, t.counters, idx[kidx], hi - lo)
        kc[lo:hi], td[lo:hi], mc[lo:hi] = o["kernel_count"], o["total_duration_ns"], o["matched_count"]
        agg[:, lo:hi] = o["agg"]
        return st, tot
    res = list(ex.map(one, range(parts)))
    keys = ("total_ns", "attributed_ns", "unattributed_ns", "kernels", "attributed_kernels", "matched_kernels")
    tot = {k: sum(r[1][k] for r in res) for k in keys}
    T = tot["total_ns"]
    tot["attributed_frac"] = tot["attributed_ns"] / T if T > 0 else float("nan")
    tot["unattributed_frac"] = tot["unattributed_ns"] / T if T > 0 else float("nan")
    ops = dict(kernel_count=kc, total_duration_ns=td, matched_count=mc, agg=agg)
    return _first_error([r[0] for r in res]), ops, tot


def run_threads(trace, threads: int | None = None, mode: str = "skip_name"):
    """The join (enclose, match, aggregate) of a trace in `threads` host
    threads (default: all cores).  The matching is split by name; with layer
    deduplication (a duplicate takes a row of another name's run) or per-stream
    rows it runs whole in one thread, as ``oracle.match``.  Returns the same
    dict as ``oracle.run``."""
    threads = threads or os.cpu_count() or 1
    whole_match = (trace.k_layer is not None and bool(trace.config.get("dedup"))) or \
        getattr(trace, "ncu_stream", None) is not None
    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        st_e, rk, nop = _enclose(ex, trace, threads)
        if whole_match:
            st_m, idx, kind, summ = match(trace.k_stream, trace.k_start, trace.k_name, trace.ncu_name,
                                          trace.k_layer, trace.class_of_layer, trace.rep_of_class, mode=mode,
                                          dedup=trace.k_layer is not None and bool(trace.config.get("dedup")),
                                          ncu_stream=getattr(trace, "ncu_stream", None))
        else:
            st_m, idx, kind, summ = _match(ex, trace, threads, mode)
        st_a, ops, totals = _aggregate(ex, trace, rk, idx, threads)
    return dict(enclose_status=st_e, range_of_kernel=rk, n_op_enclosing=nop, match_status=st_m, ncu_idx=idx,
                match_kind=kind, summary=summ, aggregate_status=st_a, ops=ops, totals=totals)
