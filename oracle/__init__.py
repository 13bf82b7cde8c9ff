"""CPU oracle for the attribution join.

TEST INFRASTRUCTURE ONLY: the test-suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg are the only callers.  The CUDA library never
imports, links or runs anything in this directory, and this directory uses
nothing of the library's.

The arithmetic lives in ``oracle.c`` (plain C, fp64, Neumaier-compensated
sums); this module compiles it and marshals numpy arrays in and out.
Functions and what they follow in the paper:

* ``validate_ranges`` / ``enclose`` -- Algorithm 2 (NVTX enclosure, Sec. 3.5);
* ``match`` -- Algorithm 1 (invocation-order matching, Sec. 3.3) with layer
  deduplication (Sec. 3.7);
* ``aggregate`` -- Eq. (1) and the SUM / MAX rules of Sec. 3.8.1, per counter
  as Table 8 assigns.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_SO = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib_handle = None

OK, W_COUNT_MISMATCH, W_DEDUP_MISMATCH = 0, 1, 2
E_INVALID_ARG, E_NOT_NESTED, E_DEPTH, E_COUNT_MISMATCH, E_OOM = -1, -2, -3, -4, -6
STRUCTURAL = 0xFFFFFFFF
NONOP = 0xFFFFFFFE
N_COUNTERS = 20
MODES = {"skip_name": 0, "prefix": 1, "error": 2}
SUM, DW, MAX = 0, 1, 2
SUMMARY_FIELDS = ("kernels", "replayed", "direct", "broadcast", "unmatched",
                  "names_mismatched", "count_unmatched", "dedup_mismatch")


def build() -> str:
    """Compile oracle.c (plain C) into liboracle.so beside it."""
    if os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(_SRC):
        return _SO
    subprocess.run(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", _SRC, "-o", _SO + ".tmp", "-lm"],
                   check=True, capture_output=True)
    os.replace(_SO + ".tmp", _SO)
    return _SO


def _lib():
    global _lib_handle
    with _lock:
        if _lib_handle is None:
            lib = ctypes.CDLL(build())
            vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
            lib.orc_validate_ranges_brute.argtypes = [i64, vp, vp, vp, vp]
            lib.orc_validate_ranges_indexed.argtypes = [i64, vp, vp, vp, vp]
            lib.orc_enclose.argtypes = [ctypes.c_int, i64, vp, vp, i64, vp, vp, vp, vp, vp, vp, vp]
            lib.orc_match.argtypes = [ctypes.c_int, i64, vp, vp, vp, vp, vp, i64, vp, ctypes.c_int, i32, vp,
                                      i32, vp, ctypes.c_int, vp, vp, vp]
            lib.orc_aggregate.argtypes = [i64, vp, vp, i64, vp, i64, vp, vp, i64, vp, vp, vp, vp, vp, vp]
            lib.orc_agg_rule.argtypes = [ctypes.c_int]
            lib.orc_attribute.argtypes = [ctypes.c_int, i64, vp, vp, vp, vp, vp, i64, vp, ctypes.c_uint32, i64, vp,
                                          vp, vp, i64, vp, vp, vp, vp, vp, vp, vp]
            _lib_handle = lib
        return _lib_handle


class use_library:
    """Context manager: run the oracle functions against another build of
    oracle.c (the pin tests compile deliberately broken copies with it)."""

    def __init__(self, path: str):
        self.path = path

    def __enter__(self):
        global _lib_handle
        _lib()
        self._saved = _lib_handle
        lib = ctypes.CDLL(self.path)
        for name in ("orc_validate_ranges_brute", "orc_validate_ranges_indexed", "orc_enclose", "orc_match",
                     "orc_aggregate", "orc_agg_rule", "orc_attribute"):
            getattr(lib, name).argtypes = getattr(self._saved, name).argtypes
        _lib_handle = lib
        return self

    def __exit__(self, *exc):
        global _lib_handle
        _lib_handle = self._saved
        return False


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


def agg_rules() -> list[int]:
    """Per-counter rule (SUM / DW / MAX) as the oracle applies it."""
    lib = _lib()
    return [lib.orc_agg_rule(c) for c in range(N_COUNTERS)]


def validate_ranges(r_stream, r_start, r_end, r_depth, mode: str = "indexed") -> int:
    lib = _lib()
    a = [_c(r_stream, np.uint8), _c(r_start, np.int64), _c(r_end, np.int64), _c(r_depth, np.uint8)]
    fn = lib.orc_validate_ranges_brute if mode == "brute" else lib.orc_validate_ranges_indexed
    return fn(len(a[1]), *(_p(x) for x in a))


def enclose(k_stream, k_start, r_stream, r_start, r_end, r_depth, r_op, mode: str = "indexed"):
    """Returns (status, range_of_kernel i32[K], n_op_enclosing u8[K]).

    mode: "brute" (every range of the kernel's stream tested; all-pairs
    laminar check), "indexed" (level lists and binary search), or
    "brute_chain" (the brute per-kernel scan after the indexed laminar check,
    for kernel samples of traces with millions of ranges)."""
    lib = _lib()
    ks, kt = _c(k_stream, np.uint8), _c(k_start, np.int64)
    rs, rt, re, rd, ro = (_c(r_stream, np.uint8), _c(r_start, np.int64), _c(r_end, np.int64),
                          _c(r_depth, np.uint8), _c(r_op, np.uint32))
    K, R = len(kt), len(rt)
    out_r = np.full(K, -1, np.int32)
    out_n = np.zeros(K, np.uint8)
    st = lib.orc_enclose({"brute": 0, "indexed": 1, "brute_chain": 2}[mode], K, _p(ks), _p(kt), R, _p(rs), _p(rt), _p(re), _p(rd),
                         _p(ro), _p(out_r), _p(out_n))
    return st, out_r, out_n


def match(k_stream, k_start, k_name, ncu_name, k_layer=None, class_of_layer=None, rep_of_class=None,
          mode: str = "skip_name", dedup: bool = False, brute: bool = False, ncu_stream=None):
    """Returns (status, ncu_idx i32[K], match_kind u8[K], summary dict).

    With ncu_stream (the stream of each ncu row, from per-stream replay runs),
    Algorithm 1's key is the pair (name, stream) rather than the name: kernels
    and rows are keyed name * 256 + stream (names below 2^24), and everything
    the algorithm does with names it does with those keys.  The dedup
    broadcast (Sec. 3.7) still compares plain names: a layer and its class's
    representative may run on different streams."""
    lib = _lib()
    ks, kt, kn = _c(k_stream, np.uint8), _c(k_start, np.int64), _c(k_name, np.uint32)
    kname_plain = kn
    kl = _c(k_layer, np.int32)
    nn = _c(ncu_name, np.uint32)
    if ncu_stream is not None and len(nn) > 0:
        if (kn >= (1 << 24)).any() or (nn >= (1 << 24)).any():
            return E_INVALID_ARG, np.full(len(kt), -1, np.int32), np.zeros(len(kt), np.uint8), \
                dict(zip(SUMMARY_FIELDS, [0] * len(SUMMARY_FIELDS)))
        kn = (kn.astype(np.uint32) << np.uint32(8)) | ks.astype(np.uint32)
        nn = (nn.astype(np.uint32) << np.uint32(8)) | _c(ncu_stream, np.uint8).astype(np.uint32)
    col = _c(class_of_layer, np.int32) if class_of_layer is not None else np.zeros(1, np.int32)
    roc = _c(rep_of_class, np.int32) if rep_of_class is not None else np.zeros(1, np.int32)
    n_layers = 0 if class_of_layer is None else len(col)
    n_classes = 0 if rep_of_class is None else len(roc)
    K, M = len(kt), len(nn)
    out_i = np.full(K, -1, np.int32)
    out_k = np.zeros(K, np.uint8)
    summ = np.zeros(len(SUMMARY_FIELDS), np.int64)
    st = lib.orc_match(int(brute), K, _p(ks), _p(kt), _p(kn), _p(kname_plain), _p(kl), M, _p(nn), int(bool(dedup)),
                       n_layers, _p(col), n_classes, _p(roc), MODES[mode], _p(out_i), _p(out_k), _p(summ))
    return st, out_i, out_k, dict(zip(SUMMARY_FIELDS, (int(x) for x in summ)))


def aggregate(k_dur, range_of_kernel, r_op, counters, ncu_idx, n_ops: int):
    """Returns (status, ops dict, totals dict).

    ops: kernel_count / total_duration_ns / matched_count (i64[n_ops]) and
    agg (f64[20, n_ops], one row per counter)."""
    lib = _lib()
    kd, rk, ro = _c(k_dur, np.int64), _c(range_of_kernel, np.int32), _c(r_op, np.uint32)
    cn = _c(counters, np.float32).reshape(-1, N_COUNTERS) if counters is not None else np.zeros((0, N_COUNTERS), np.float32)
    ni = _c(ncu_idx, np.int32)
    K, R, M = len(kd), len(ro), cn.shape[0]
    kc = np.zeros(n_ops, np.int64)
    td = np.zeros(n_ops, np.int64)
    mc = np.zeros(n_ops, np.int64)
    agg = np.zeros((N_COUNTERS, n_ops), np.float64)
    tot = np.zeros(6, np.int64)
    fr = np.zeros(2, np.float64)
    st = lib.orc_aggregate(K, _p(kd), _p(rk), R, _p(ro), M, _p(cn), _p(ni), n_ops, _p(kc), _p(td), _p(mc),
                           _p(agg), _p(tot), _p(fr))
    ops = dict(kernel_count=kc, total_duration_ns=td, matched_count=mc, agg=agg)
    totals = dict(total_ns=int(tot[0]), attributed_ns=int(tot[1]), unattributed_ns=int(tot[2]),
                  kernels=int(tot[3]), attributed_kernels=int(tot[4]), matched_kernels=int(tot[5]),
                  attributed_frac=float(fr[0]), unattributed_frac=float(fr[1]))
    return st, ops, totals


OP_NONE = 0xFFFFFFFF
TIER_NONE, TIER_HIGH, TIER_NVTX, TIER_INDUCTOR = 0, 1, 2, 3
ATTR_SUMMARY_FIELDS = ("kernels", "high", "nvtx", "inductor", "none", "fused", "corr_used")


def attribute(k_stream, k_start, k_name, range_of_kernel, n_op_enclosing, r_op, n_ops: int, corr=None, fusion=None,
              brute: bool = False):
    """The attribution tiers of Fig. 2.  corr = (name, invocation, op) arrays
    of the torch.profiler correlation map or None; fusion = (op_of_name,
    list_len or None) of the Inductor fusion map or None.
    Returns (status, op_of_kernel u32[K], tier u8[K], fused_with u32[K],
    is_fused u8[K], summary dict)."""
    lib = _lib()
    ks, kt, kn = _c(k_stream, np.uint8), _c(k_start, np.int64), _c(k_name, np.uint32)
    rk, ro = _c(range_of_kernel, np.int32), _c(r_op, np.uint32)
    nop = _c(n_op_enclosing, np.uint8)
    K = len(kt)
    cn = ci = co = None
    if corr is not None:
        cn, ci, co = (_c(a, np.uint32) for a in corr)
    fo = fl = None
    if fusion is not None:
        fo = _c(fusion[0], np.uint32)
        fl = _c(fusion[1], np.uint8) if fusion[1] is not None else None
    NC = 0 if cn is None else len(cn)
    NF = 0 if fo is None else len(fo)
    op = np.full(K, OP_NONE, np.uint32)
    tier = np.zeros(K, np.uint8)
    fw = np.full(K, OP_NONE, np.uint32)
    fz = np.zeros(K, np.uint8)
    summ = np.zeros(len(ATTR_SUMMARY_FIELDS), np.int64)
    st = lib.orc_attribute(int(brute), K, _p(ks), _p(kt), _p(kn), _p(rk), _p(nop), len(ro), _p(ro),
                           ctypes.c_uint32(n_ops), NC, _p(cn), _p(ci), _p(co), NF, _p(fo), _p(fl), _p(op), _p(tier),
                           _p(fw), _p(fz), _p(summ))
    return st, op, tier, fw, fz, dict(zip(ATTR_SUMMARY_FIELDS, (int(x) for x in summ)))


def aggregate_by_op(k_dur, op_of_kernel, counters, ncu_idx, n_ops: int):
    """aggregate() with each kernel's operator given directly (OP_NONE =
    unattributed): every kernel with an operator is its own one-kernel "range"."""
    op = _c(op_of_kernel, np.uint32)
    rk = np.where(op != OP_NONE, np.arange(len(op)), -1).astype(np.int32)
    return aggregate(k_dur, rk, op, counters, ncu_idx, n_ops)


def rollup(k_dur, op_of_kernel, counters, ncu_idx, class_of_op, n_classes: int):
    """aggregate() per operator class: each kernel's operator mapped through
    class_of_op (OP_NONE leaves it out)."""
    op = _c(op_of_kernel, np.uint32).astype(np.int64)
    cm = _c(class_of_op, np.uint32)
    has = op != OP_NONE
    cls = np.full(len(op), OP_NONE, np.uint32)
    cls[has] = cm[op[has]]
    return aggregate_by_op(k_dur, cls, counters, ncu_idx, n_classes)


def run_tiers(trace, mode: str = "skip_name", enclose_mode: str = "indexed", dedup: bool | None = None,
              brute: bool = False, use_corr: bool = True, use_fusion: bool = True):
    """The join with the attribution tiers: enclose, attribute, match, aggregate by operator."""
    st_e, rk, nop = enclose(trace.k_stream, trace.k_start, trace.r_stream, trace.r_start, trace.r_end,
                            trace.r_depth, trace.r_op, mode=enclose_mode)
    corr = (trace.corr_name, trace.corr_inv, trace.corr_op) if use_corr and trace.corr_name is not None else None
    fusion = (trace.fusion_op, trace.fusion_len) if use_fusion and trace.fusion_op is not None else None
    st_t, op, tier, fw, fz, tsum = attribute(trace.k_stream, trace.k_start, trace.k_name, rk, nop, trace.r_op,
                                             trace.n_ops, corr, fusion, brute=brute)
    if dedup is None:
        dedup = bool(trace.config.get("dedup")) and trace.k_layer is not None
    st_m, idx, kind, summ = match(trace.k_stream, trace.k_start, trace.k_name, trace.ncu_name, trace.k_layer,
                                  trace.class_of_layer, trace.rep_of_class, mode=mode, dedup=dedup,
                                  ncu_stream=getattr(trace, "ncu_stream", None))
    st_a, ops, totals = aggregate_by_op(trace.k_dur, op, trace.counters, idx, trace.n_ops)
    return dict(enclose_status=st_e, range_of_kernel=rk, n_op_enclosing=nop, attribute_status=st_t,
                op_of_kernel=op, tier=tier, fused_with=fw, is_fused=fz, tier_summary=tsum, match_status=st_m,
                ncu_idx=idx, match_kind=kind, summary=summ, aggregate_status=st_a, ops=ops, totals=totals)


def run(trace, mode: str = "skip_name", enclose_mode: str = "indexed", dedup: bool | None = None):
    """The whole join on a tracegen.Trace: enclose, match, aggregate."""
    st_e, rk, nop = enclose(trace.k_stream, trace.k_start, trace.r_stream, trace.r_start, trace.r_end,
                            trace.r_depth, trace.r_op, mode=enclose_mode)
    if dedup is None:
        dedup = bool(trace.config.get("dedup")) and trace.k_layer is not None
    use_dedup = dedup
    st_m, idx, kind, summ = match(trace.k_stream, trace.k_start, trace.k_name, trace.ncu_name, trace.k_layer,
                                  trace.class_of_layer, trace.rep_of_class, mode=mode, dedup=use_dedup,
                                  ncu_stream=getattr(trace, "ncu_stream", None))
    st_a, ops, totals = aggregate(trace.k_dur, rk, trace.r_op, trace.counters, idx, trace.n_ops)
    return dict(enclose_status=st_e, range_of_kernel=rk, n_op_enclosing=nop, match_status=st_m,
                ncu_idx=idx, match_kind=kind, summary=summ, aggregate_status=st_a, ops=ops, totals=totals)
