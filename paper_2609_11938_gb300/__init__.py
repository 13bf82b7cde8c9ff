"""Python binding of libopattr, the GPU trace join for hardware-attributed
operator profiling ("Hardware-Attributed Operator Profiling for PyTorch").

Argument marshalling only: every step of the join runs in the CUDA kernels of
``libopattr.so`` (``csrc/``), reached through its C ABI (``include/opattr.h``).
PyTorch supplies device memory and the stream.  There is no CPU fallback: if
the library cannot be loaded the import of the binding's functions raises.

Function names follow the C ABI: ``opattr_create``, ``opattr_enclose``,
``opattr_match``, ``opattr_aggregate``, ``opattr_destroy``; ``Context`` wraps
them for torch tensors.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass

from . import _build

__all__ = [
    "OK", "W_COUNT_MISMATCH", "W_DEDUP_MISMATCH", "E_INVALID_ARG", "E_NOT_NESTED", "E_DEPTH",
    "E_COUNT_MISMATCH", "E_CUDA", "E_OOM", "E_TIMEOUT", "E_STATE", "OP_STRUCTURAL", "OP_NONOP",
    "N_COUNTERS", "OpattrError", "Context", "library", "build",
    "opattr_create", "opattr_enclose", "opattr_match", "opattr_aggregate", "opattr_join", "opattr_destroy",
    "opattr_status_string", "opattr_match_noalloc", "MATCH_NOALLOC_MAX",
]

OK, W_COUNT_MISMATCH, W_DEDUP_MISMATCH = 0, 1, 2
E_INVALID_ARG, E_NOT_NESTED, E_DEPTH, E_COUNT_MISMATCH = -1, -2, -3, -4
E_CUDA, E_OOM, E_TIMEOUT, E_STATE = -5, -6, -7, -8
OP_STRUCTURAL = 0xFFFFFFFF
OP_NONOP = 0xFFFFFFFE
N_COUNTERS = 20
OP_NONE = 0xFFFFFFFF
TIER_NONE, TIER_HIGH, TIER_NVTX, TIER_INDUCTOR = 0, 1, 2, 3
MATCH_NOALLOC_MAX = 65536
MISMATCH = {"skip_name": 0, "prefix": 1, "error": 2}

_vp = ctypes.c_void_p


class Kernels(ctypes.Structure):
    _fields_ = [("stream", _vp), ("start_ns", _vp), ("dur_ns", _vp), ("name_id", _vp), ("layer_id", _vp),
                ("n", ctypes.c_int64)]


class Ranges(ctypes.Structure):
    _fields_ = [("stream", _vp), ("start_ns", _vp), ("end_ns", _vp), ("depth", _vp), ("op_id", _vp),
                ("n", ctypes.c_int64)]


class Ncu(ctypes.Structure):
    _fields_ = [("name_id", _vp), ("counters", _vp), ("n", ctypes.c_int64), ("stream", _vp)]


class Dedup(ctypes.Structure):
    _fields_ = [("class_of_layer", _vp), ("rep_of_class", _vp), ("n_layers", ctypes.c_int32),
                ("n_classes", ctypes.c_int32)]


class Config(ctypes.Structure):
    _fields_ = [("mismatch", ctypes.c_int), ("dedup", ctypes.c_int32), ("checked", ctypes.c_int32),
                ("spin_limit", ctypes.c_int64)]


class MatchSummary(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int64) for f in ("kernels", "replayed", "direct", "broadcast", "unmatched",
                                              "names_mismatched", "count_unmatched", "dedup_mismatch")] + \
               [("fast_path", ctypes.c_int32), ("reserved", ctypes.c_int32)]

    def as_dict(self) -> dict:
        return {f: int(getattr(self, f)) for f, _ in self._fields_ if f != "reserved"}


class Corr(ctypes.Structure):
    _fields_ = [("name_id", _vp), ("invocation", _vp), ("op_id", _vp), ("n", ctypes.c_int64)]


class Fusion(ctypes.Structure):
    _fields_ = [("op_of_name", _vp), ("list_len", _vp), ("n_names", ctypes.c_int64)]


class AttrSummary(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int64) for f in ("kernels", "high", "nvtx", "inductor", "none", "fused", "corr_used")]

    def as_dict(self) -> dict:
        return {f: int(getattr(self, f)) for f, _ in self._fields_}


class ProfileMeta(ctypes.Structure):
    _fields_ = [("model_name", ctypes.c_char_p), ("device_name", ctypes.c_char_p), ("compile_mode", ctypes.c_char_p),
                ("capture_timestamp_utc", ctypes.c_char_p), ("include_kernels", ctypes.c_int32)]


class ProfileNames(ctypes.Structure):
    _fields_ = [("kernel_name", _vp), ("n_kernel_names", ctypes.c_int64), ("op_name", _vp),
                ("op_call_index", _vp)]


class OpAggregates(ctypes.Structure):
    _fields_ = [("kernel_count", _vp), ("total_duration_ns", _vp), ("matched_count", _vp), ("agg", _vp)]


class Totals(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int64) for f in ("total_ns", "attributed_ns", "unattributed_ns", "kernels",
                                              "attributed_kernels", "matched_kernels")] + \
               [("attributed_frac", ctypes.c_double), ("unattributed_frac", ctypes.c_double)]

    def as_dict(self) -> dict:
        return {f: getattr(self, f) for f, _ in self._fields_}


_lib_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile libopattr.so for sm_103a (no-op when up to date)."""
    return _build.build(force=force)


def library():
    """Load libopattr.so (building it first if needed).  Raises on failure."""
    global _lib
    with _lib_lock:
        if _lib is None:
            path = _build.LIB
            if not os.path.exists(path) or os.environ.get("OPATTR_REBUILD"):
                path = _build.build()
            lib = ctypes.CDLL(path)
            P = ctypes.POINTER
            lib.opattr_create.argtypes = [P(_vp), ctypes.c_int, _vp, P(Config)]
            lib.opattr_enclose.argtypes = [_vp, P(Kernels), P(Ranges), _vp, _vp]
            lib.opattr_match.argtypes = [_vp, P(Kernels), P(Ncu), P(Dedup), _vp, _vp, P(MatchSummary)]
            lib.opattr_aggregate.argtypes = [_vp, P(Kernels), P(Ranges), _vp, P(Ncu), _vp, ctypes.c_uint32,
                                             P(OpAggregates), P(Totals)]
            lib.opattr_join.argtypes = [_vp, P(Kernels), P(Ranges), P(Ncu), P(Dedup), ctypes.c_uint32, _vp, _vp, _vp,
                                        _vp, P(OpAggregates), P(MatchSummary), P(Totals)]
            lib.opattr_attribute.argtypes = [_vp, P(Kernels), P(Ranges), _vp, _vp, P(Corr), P(Fusion),
                                             ctypes.c_uint32, _vp, _vp, _vp, _vp, P(AttrSummary)]
            lib.opattr_rollup.argtypes = [_vp, P(Kernels), P(Ranges), _vp, P(Ncu), _vp, ctypes.c_uint32, _vp,
                                          ctypes.c_uint32, P(OpAggregates)]
            lib.opattr_write_profile.argtypes = [ctypes.c_char_p, P(ProfileMeta), P(ProfileNames), P(Kernels), _vp,
                                                 _vp, _vp, _vp, _vp, _vp, ctypes.c_int64, ctypes.c_uint32,
                                                 P(OpAggregates), P(ctypes.c_int64)]
            lib.opattr_write_profile.restype = ctypes.c_int
            lib.opattr_destroy.argtypes = [_vp]
            lib.opattr_destroy.restype = None
            lib.opattr_status_string.argtypes = [ctypes.c_int]
            lib.opattr_status_string.restype = ctypes.c_char_p
            lib.opattr_set_timing.argtypes = [_vp, ctypes.c_int]
            lib.opattr_set_timing_only.argtypes = [_vp, ctypes.c_char_p]
            lib.opattr_set_timing_only.restype = ctypes.c_int
            lib.opattr_timing_report.argtypes = [_vp, P(ctypes.c_char_p), P(ctypes.c_double), P(ctypes.c_int64),
                                                 ctypes.c_int]
            lib.opattr_timing_reset.argtypes = [_vp]
            lib.opattr_timing_reset.restype = None
            lib.opattr_launch_count.argtypes = [_vp]
            lib.opattr_launch_count.restype = ctypes.c_int64
            lib.opattr_match_noalloc.argtypes = [P(Kernels), P(Ncu), ctypes.c_int, _vp, _vp, P(MatchSummary), _vp]
            lib.opattr_match_noalloc.restype = ctypes.c_int
            for f in ("opattr_create", "opattr_enclose", "opattr_match", "opattr_aggregate", "opattr_attribute",
                      "opattr_rollup", "opattr_set_timing", "opattr_timing_report"):
                getattr(lib, f).restype = ctypes.c_int
            _lib = lib
        return _lib


class OpattrError(RuntimeError):
    def __init__(self, status: int, call: str):
        super().__init__(f"{call}: {opattr_status_string(status)} ({status})")
        self.status = status


def opattr_status_string(status: int) -> str:
    return library().opattr_status_string(status).decode()


# ---------------------------------------------------------------- C ABI, one to one
def opattr_create(device: int = 0, stream: int | None = None, mismatch: str = "skip_name", dedup: bool = True,
                  spin_limit: int = 0):
    """Returns (status, handle)."""
    cfg = Config(MISMATCH[mismatch], int(bool(dedup)), 0, int(spin_limit))
    h = _vp()
    st = library().opattr_create(ctypes.byref(h), int(device), _vp(stream or 0), ctypes.byref(cfg))
    return st, h


def opattr_enclose(handle, kernels: Kernels, ranges: Ranges, range_of_kernel_ptr: int, n_op_ptr: int | None) -> int:
    return library().opattr_enclose(handle, ctypes.byref(kernels), ctypes.byref(ranges), _vp(range_of_kernel_ptr),
                                    _vp(n_op_ptr or 0))


def opattr_match(handle, kernels: Kernels, ncu: Ncu, dedup: Dedup | None, idx_ptr: int, kind_ptr: int | None,
                 summary: MatchSummary) -> int:
    return library().opattr_match(handle, ctypes.byref(kernels), ctypes.byref(ncu),
                                  ctypes.byref(dedup) if dedup is not None else None, _vp(idx_ptr),
                                  _vp(kind_ptr or 0), ctypes.byref(summary))


def opattr_aggregate(handle, kernels: Kernels, ranges: Ranges, rok_ptr: int, ncu: Ncu, idx_ptr: int, n_ops: int,
                     out: OpAggregates, totals: Totals) -> int:
    return library().opattr_aggregate(handle, ctypes.byref(kernels), ctypes.byref(ranges), _vp(rok_ptr),
                                      ctypes.byref(ncu), _vp(idx_ptr), ctypes.c_uint32(n_ops), ctypes.byref(out),
                                      ctypes.byref(totals))


def opattr_join(handle, kernels: Kernels, ranges: Ranges, ncu: Ncu, dedup: Dedup | None, n_ops: int, rok_ptr: int,
                nop_ptr: int | None, idx_ptr: int, kind_ptr: int | None, out: OpAggregates, summary: MatchSummary,
                totals: Totals) -> int:
    return library().opattr_join(handle, ctypes.byref(kernels), ctypes.byref(ranges), ctypes.byref(ncu),
                                 ctypes.byref(dedup) if dedup is not None else None, ctypes.c_uint32(n_ops),
                                 _vp(rok_ptr), _vp(nop_ptr or 0), _vp(idx_ptr), _vp(kind_ptr or 0), ctypes.byref(out),
                                 ctypes.byref(summary), ctypes.byref(totals))


def opattr_attribute(handle, kernels: Kernels, ranges: Ranges, rok_ptr: int, nop_ptr: int | None,
                     corr: Corr | None, fusion: Fusion | None, n_ops: int, op_ptr: int, tier_ptr: int | None,
                     fused_with_ptr: int | None, is_fused_ptr: int | None, summary: AttrSummary) -> int:
    return library().opattr_attribute(handle, ctypes.byref(kernels), ctypes.byref(ranges), _vp(rok_ptr),
                                      _vp(nop_ptr or 0), ctypes.byref(corr) if corr is not None else None,
                                      ctypes.byref(fusion) if fusion is not None else None, ctypes.c_uint32(n_ops),
                                      _vp(op_ptr), _vp(tier_ptr or 0), _vp(fused_with_ptr or 0),
                                      _vp(is_fused_ptr or 0), ctypes.byref(summary))


def opattr_rollup(handle, kernels: Kernels, ranges: Ranges, rok_ptr: int | None, ncu: Ncu, idx_ptr: int, n_ops: int,
                  class_ptr: int, n_classes: int, out: OpAggregates) -> int:
    return library().opattr_rollup(handle, ctypes.byref(kernels), ctypes.byref(ranges), _vp(rok_ptr or 0),
                                   ctypes.byref(ncu), _vp(idx_ptr), ctypes.c_uint32(n_ops), _vp(class_ptr),
                                   ctypes.c_uint32(n_classes), ctypes.byref(out))


def write_profile(path: str, k_stream, k_dur, k_name, op_of_kernel, ncu_idx, counters, ops: dict, tier=None,
                  is_fused=None, fused_with=None, kernel_names=None, op_names=None, op_call_index=None,
                  meta: dict | None = None, include_kernels: bool = True) -> int:
    """profile.json (App. A.4) from HOST (numpy) arrays: opattr_write_profile.
    Returns the number of bytes written; raises OpattrError on failure."""
    import numpy as np
    c = lambda a, dt: None if a is None else np.ascontiguousarray(a).view(dt) if np.asarray(a).dtype.itemsize == \
        np.dtype(dt).itemsize else np.ascontiguousarray(a, dtype=dt)
    ks, kd, kn = c(k_stream, np.uint8), c(k_dur, np.int64), c(k_name, np.uint32)
    op, ni = c(op_of_kernel, np.uint32), c(ncu_idx, np.int32)
    cn = np.ascontiguousarray(counters, dtype=np.float32)
    tr, fz, fw = c(tier, np.uint8), c(is_fused, np.uint8), c(fused_with, np.uint32)
    kc, td, mc = (np.ascontiguousarray(ops[k], dtype=np.int64) for k in ("kernel_count", "total_duration_ns",
                                                                         "matched_count"))
    agg = np.ascontiguousarray(ops["agg"], dtype=np.float64)
    p = lambda a: None if a is None else a.ctypes.data
    K = len(kd)
    kern = Kernels(p(ks), None, p(kd), p(kn), None, K)
    out = OpAggregates(p(kc), p(td), p(mc), p(agg))
    keep = []
    names = ProfileNames(None, 0, None, None)
    if kernel_names is not None:
        arr = (ctypes.c_char_p * len(kernel_names))(*[s.encode() for s in kernel_names])
        keep.append(arr)
        names.kernel_name, names.n_kernel_names = ctypes.cast(arr, _vp), len(kernel_names)
    if op_names is not None:
        arr = (ctypes.c_char_p * len(op_names))(*[s.encode() for s in op_names])
        keep.append(arr)
        names.op_name = ctypes.cast(arr, _vp)
    ci = c(op_call_index, np.int64)
    if ci is not None:
        names.op_call_index = p(ci)
    m = meta or {}
    pm = ProfileMeta(*[(m.get(k).encode() if m.get(k) is not None else None)
                       for k in ("model_name", "device_name", "compile_mode", "capture_timestamp_utc")],
                     int(bool(include_kernels)))
    nbytes = ctypes.c_int64(0)
    st = library().opattr_write_profile(str(path).encode(), ctypes.byref(pm), ctypes.byref(names), ctypes.byref(kern),
                                        p(op), p(tr), p(fz), p(fw), p(ni), p(cn), cn.shape[0] if cn.ndim == 2 else
                                        cn.size // N_COUNTERS, int(len(kc)), ctypes.byref(out), ctypes.byref(nbytes))
    del keep
    if st != OK:
        raise OpattrError(st, "opattr_write_profile")
    return int(nbytes.value)


def opattr_match_noalloc(kernels: Kernels, ncu: Ncu, mismatch: str, idx_ptr: int, kind_ptr: int | None,
                         summary: MatchSummary, stream: int | None) -> int:
    """opattr_match without a context and without any device allocation, for
    callers that must not allocate (see include/opattr.h); inputs of at most
    OPATTR_MATCH_NOALLOC_MAX kernels and rows."""
    return library().opattr_match_noalloc(ctypes.byref(kernels), ctypes.byref(ncu), MISMATCH[mismatch],
                                          _vp(idx_ptr), _vp(kind_ptr or 0), ctypes.byref(summary), _vp(stream or 0))


def opattr_destroy(handle) -> None:
    if handle:
        library().opattr_destroy(handle)


# ---------------------------------------------------------------- torch convenience layer
def _ptr(t, dtype, name, device):
    if t is None:
        return None
    if t.dtype is not dtype and not (dtype is _torch().uint32 and t.dtype is _torch().int32):
        raise TypeError(f"{name}: expected {dtype}, got {t.dtype}")
    if t.get_device() != device:                 # -1 for a host tensor
        raise ValueError(f"{name}: must live on cuda:{device}")
    if not t.is_contiguous():
        raise ValueError(f"{name}: must be contiguous")
    return t.data_ptr() if t.numel() else None


def _torch():
    import torch
    return torch


@dataclass
class DeviceTrace:
    """A trace's arrays as device tensors (see include/opattr.h for layouts)."""
    k_stream: object
    k_start: object
    k_dur: object
    k_name: object
    k_layer: object
    r_stream: object
    r_start: object
    r_end: object
    r_depth: object
    r_op: object
    n_ops: int
    ncu_name: object
    counters: object
    class_of_layer: object = None   # host (numpy / list) tables
    rep_of_class: object = None
    ncu_stream: object = None       # stream of each ncu row (per-stream replay runs), or None
    corr_name: object = None        # torch.profiler correlation map (HIGH tier), or None
    corr_inv: object = None
    corr_op: object = None
    fusion_op: object = None        # Inductor fusion map per name id (INDUCTOR tier), or None
    fusion_len: object = None

    @property
    def K(self):
        return int(self.k_start.shape[0])

    @property
    def R(self):
        return int(self.r_start.shape[0])

    @property
    def M(self):
        return int(self.ncu_name.shape[0])


def to_device(trace, device: int = 0, pin: bool = False) -> DeviceTrace:
    """Copy a tracegen.Trace (numpy arrays) to the GPU as torch tensors."""
    import torch

    def d(a):
        if a is None:
            return None
        t = torch.from_numpy(a)
        if pin:
            t = t.pin_memory()
        return t.to(f"cuda:{device}", non_blocking=pin)

    return DeviceTrace(d(trace.k_stream), d(trace.k_start), d(trace.k_dur), d(trace.k_name), d(trace.k_layer),
                       d(trace.r_stream), d(trace.r_start), d(trace.r_end), d(trace.r_depth), d(trace.r_op),
                       int(trace.n_ops), d(trace.ncu_name), d(trace.counters), trace.class_of_layer,
                       trace.rep_of_class, d(getattr(trace, "ncu_stream", None)), d(getattr(trace, "corr_name", None)),
                       d(getattr(trace, "corr_inv", None)), d(getattr(trace, "corr_op", None)),
                       d(getattr(trace, "fusion_op", None)), d(getattr(trace, "fusion_len", None)))


class Context:
    """An opattr context bound to one device and one CUDA stream."""

    def __init__(self, device: int = 0, stream=None, mismatch: str = "skip_name", dedup: bool = True,
                 spin_limit: int = 0):
        import torch
        self.device = device
        if stream is None:
            stream = torch.cuda.current_stream(device)
        self.stream = stream
        st, self.handle = opattr_create(device, stream.cuda_stream, mismatch, dedup, spin_limit)
        if st != OK:
            raise OpattrError(st, "opattr_create")

    def close(self):
        if getattr(self, "handle", None):
            opattr_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # -- structs
    def kernels(self, tr: DeviceTrace) -> Kernels:
        import torch
        dv = self.device
        return Kernels(_ptr(tr.k_stream, torch.uint8, "k_stream", dv), _ptr(tr.k_start, torch.int64, "k_start", dv),
                       _ptr(tr.k_dur, torch.int64, "k_dur", dv), _ptr(tr.k_name, torch.uint32, "k_name", dv),
                       _ptr(tr.k_layer, torch.int32, "k_layer", dv), tr.K)

    def ranges(self, tr: DeviceTrace) -> Ranges:
        import torch
        dv = self.device
        return Ranges(_ptr(tr.r_stream, torch.uint8, "r_stream", dv), _ptr(tr.r_start, torch.int64, "r_start", dv),
                      _ptr(tr.r_end, torch.int64, "r_end", dv), _ptr(tr.r_depth, torch.uint8, "r_depth", dv),
                      _ptr(tr.r_op, torch.uint32, "r_op", dv), tr.R)

    def ncu(self, tr: DeviceTrace) -> Ncu:
        import torch
        dv = self.device
        return Ncu(_ptr(tr.ncu_name, torch.uint32, "ncu_name", dv), _ptr(tr.counters, torch.float32, "counters", dv),
                   tr.M, _ptr(tr.ncu_stream, torch.uint8, "ncu_stream", dv))

    # -- calls
    def enclose(self, tr: DeviceTrace, out_range=None, out_nop=None, need_nop: bool = True):
        import torch
        dev = f"cuda:{self.device}"
        if out_range is None:
            out_range = torch.empty(tr.K, dtype=torch.int32, device=dev)
        if out_nop is None and need_nop:
            out_nop = torch.empty(tr.K, dtype=torch.uint8, device=dev)
        st = opattr_enclose(self.handle, self.kernels(tr), self.ranges(tr),
                            _ptr(out_range, torch.int32, "range_of_kernel", self.device),
                            _ptr(out_nop, torch.uint8, "n_op_enclosing", self.device) if out_nop is not None else None)
        if st < 0:
            raise OpattrError(st, "opattr_enclose")
        return st, out_range, out_nop

    @staticmethod
    def _dedup(tr: DeviceTrace, dedup: bool | None):
        """(Dedup struct or None, the host arrays it points into)."""
        import numpy as np
        use = (tr.class_of_layer is not None and tr.k_layer is not None) if dedup is None else dedup
        if not use:
            return None, None
        col = np.ascontiguousarray(tr.class_of_layer, dtype=np.int32)
        roc = np.ascontiguousarray(tr.rep_of_class, dtype=np.int32)
        return Dedup(col.ctypes.data if col.size else None, roc.ctypes.data if roc.size else None, len(col),
                     len(roc)), (col, roc)

    def match(self, tr: DeviceTrace, dedup: bool | None = None, out_idx=None, out_kind=None):
        import torch
        dev = f"cuda:{self.device}"
        if out_idx is None:
            out_idx = torch.empty(tr.K, dtype=torch.int32, device=dev)
        if out_kind is None:
            out_kind = torch.empty(tr.K, dtype=torch.uint8, device=dev)
        dd, keep = self._dedup(tr, dedup)
        summ = MatchSummary()
        st = opattr_match(self.handle, self.kernels(tr), self.ncu(tr), dd,
                          _ptr(out_idx, torch.int32, "ncu_idx_of_kernel", self.device),
                          _ptr(out_kind, torch.uint8, "match_kind", self.device), summ)
        del keep
        if st < 0:
            raise OpattrError(st, "opattr_match")
        return st, out_idx, out_kind, summ.as_dict()

    def join(self, tr: DeviceTrace, dedup: bool | None = None, out=None, ops=None):
        """enclose + match + aggregate in one call (opattr_join).  `out` may hold
        preallocated range_of_kernel / n_op_enclosing / ncu_idx / match_kind
        tensors; returns (status, out, ops, match summary, totals)."""
        import torch
        dev = f"cuda:{self.device}"
        dv = self.device
        out = dict(out or {})
        for k, dt in (("range_of_kernel", torch.int32), ("n_op_enclosing", torch.uint8), ("ncu_idx", torch.int32),
                      ("match_kind", torch.uint8)):
            if out.get(k) is None:
                out[k] = torch.empty(tr.K, dtype=dt, device=dev)
        if ops is None:
            ops = self.alloc_ops(tr.n_ops)
        agg = OpAggregates(_ptr(ops["kernel_count"], torch.int64, "kernel_count", dv),
                           _ptr(ops["total_duration_ns"], torch.int64, "total_duration_ns", dv),
                           _ptr(ops["matched_count"], torch.int64, "matched_count", dv),
                           _ptr(ops["agg"], torch.float64, "agg", dv))
        dd, keep = self._dedup(tr, dedup)
        summ, tot = MatchSummary(), Totals()
        st = opattr_join(self.handle, self.kernels(tr), self.ranges(tr), self.ncu(tr), dd, tr.n_ops,
                         _ptr(out["range_of_kernel"], torch.int32, "range_of_kernel", dv),
                         _ptr(out["n_op_enclosing"], torch.uint8, "n_op_enclosing", dv),
                         _ptr(out["ncu_idx"], torch.int32, "ncu_idx_of_kernel", dv),
                         _ptr(out["match_kind"], torch.uint8, "match_kind", dv), agg, summ, tot)
        del keep
        if st < 0:
            raise OpattrError(st, "opattr_join")
        return st, out, ops, summ.as_dict(), tot.as_dict()

    def alloc_ops(self, n_ops: int):
        import torch
        dev = f"cuda:{self.device}"
        return dict(kernel_count=torch.empty(n_ops, dtype=torch.int64, device=dev),
                    total_duration_ns=torch.empty(n_ops, dtype=torch.int64, device=dev),
                    matched_count=torch.empty(n_ops, dtype=torch.int64, device=dev),
                    agg=torch.empty((N_COUNTERS, n_ops), dtype=torch.float64, device=dev))

    def attribute(self, tr: DeviceTrace, range_of_kernel, n_op_enclosing=None, use_corr: bool = True,
                  use_fusion: bool = True, out=None):
        """The attribution tiers of Fig. 2: returns (status, op_of_kernel, tier, fused_with, is_fused, summary)."""
        import torch
        dv = self.device
        dev = f"cuda:{dv}"
        if out is None:
            out = dict(op=torch.empty(tr.K, dtype=torch.int32, device=dev),
                       tier=torch.empty(tr.K, dtype=torch.uint8, device=dev),
                       fused_with=torch.empty(tr.K, dtype=torch.int32, device=dev),
                       is_fused=torch.empty(tr.K, dtype=torch.uint8, device=dev))
        corr = fusion = None
        if use_corr and tr.corr_name is not None:
            corr = Corr(_ptr(tr.corr_name, torch.uint32, "corr_name", dv), _ptr(tr.corr_inv, torch.uint32, "corr_inv", dv),
                        _ptr(tr.corr_op, torch.uint32, "corr_op", dv), int(tr.corr_name.shape[0]))
        if use_fusion and tr.fusion_op is not None:
            fusion = Fusion(_ptr(tr.fusion_op, torch.uint32, "fusion_op", dv),
                            _ptr(tr.fusion_len, torch.uint8, "fusion_len", dv), int(tr.fusion_op.shape[0]))
        summ = AttrSummary()
        st = opattr_attribute(self.handle, self.kernels(tr), self.ranges(tr),
                              _ptr(range_of_kernel, torch.int32, "range_of_kernel", dv),
                              _ptr(n_op_enclosing, torch.uint8, "n_op_enclosing", dv) if n_op_enclosing is not None
                              else None, corr, fusion, tr.n_ops, _ptr(out["op"], torch.uint32, "op_of_kernel", dv),
                              _ptr(out["tier"], torch.uint8, "tier", dv),
                              _ptr(out["fused_with"], torch.uint32, "fused_with", dv),
                              _ptr(out["is_fused"], torch.uint8, "is_fused", dv), summ)
        if st < 0:
            raise OpattrError(st, "opattr_attribute")
        return st, out["op"], out["tier"], out["fused_with"], out["is_fused"], summ.as_dict()

    def aggregate(self, tr: DeviceTrace, range_of_kernel, ncu_idx, ops=None, op_of_kernel=None):
        """Eq. (1) per operator.  With op_of_kernel (opattr_attribute's output)
        in place of range_of_kernel, each kernel's operator is taken from it."""
        import torch
        if ops is None:
            ops = self.alloc_ops(tr.n_ops)
        dv = self.device
        out = OpAggregates(_ptr(ops["kernel_count"], torch.int64, "kernel_count", dv),
                           _ptr(ops["total_duration_ns"], torch.int64, "total_duration_ns", dv),
                           _ptr(ops["matched_count"], torch.int64, "matched_count", dv),
                           _ptr(ops["agg"], torch.float64, "agg", dv))
        tot = Totals()
        if op_of_kernel is not None:
            rng = Ranges(None, None, None, None, _ptr(op_of_kernel, torch.uint32, "op_of_kernel", dv), tr.K)
            rok_ptr = None
        else:
            rng = self.ranges(tr)
            rok_ptr = _ptr(range_of_kernel, torch.int32, "range_of_kernel", dv)
        st = opattr_aggregate(self.handle, self.kernels(tr), rng, rok_ptr, self.ncu(tr),
                              _ptr(ncu_idx, torch.int32, "ncu_idx_of_kernel", dv), tr.n_ops, out, tot)
        if st < 0:
            raise OpattrError(st, "opattr_aggregate")
        return st, ops, tot.as_dict()

    def rollup(self, tr: DeviceTrace, range_of_kernel, ncu_idx, class_of_op, n_classes: int, out=None,
               op_of_kernel=None):
        """Per-class records (opattr_rollup); class_of_op: int32/uint32 device tensor of n_ops entries."""
        import torch
        if out is None:
            out = self.alloc_ops(n_classes)
        dv = self.device
        o = OpAggregates(_ptr(out["kernel_count"], torch.int64, "kernel_count", dv),
                         _ptr(out["total_duration_ns"], torch.int64, "total_duration_ns", dv),
                         _ptr(out["matched_count"], torch.int64, "matched_count", dv),
                         _ptr(out["agg"], torch.float64, "agg", dv))
        if op_of_kernel is not None:
            rng = Ranges(None, None, None, None, _ptr(op_of_kernel, torch.uint32, "op_of_kernel", dv), tr.K)
            rok_ptr = None
        else:
            rng = self.ranges(tr)
            rok_ptr = _ptr(range_of_kernel, torch.int32, "range_of_kernel", dv)
        st = opattr_rollup(self.handle, self.kernels(tr), rng, rok_ptr, self.ncu(tr),
                           _ptr(ncu_idx, torch.int32, "ncu_idx_of_kernel", dv), tr.n_ops,
                           _ptr(class_of_op, torch.uint32, "class_of_op", dv), n_classes, o)
        if st < 0:
            raise OpattrError(st, "opattr_rollup")
        return st, out

    def run(self, tr: DeviceTrace, dedup: bool | None = None):
        """enclose + match + aggregate on device-resident inputs."""
        st_e, rk, nop = self.enclose(tr)
        st_m, idx, kind, summ = self.match(tr, dedup=dedup)
        st_a, ops, tot = self.aggregate(tr, rk, idx)
        return dict(enclose_status=st_e, range_of_kernel=rk, n_op_enclosing=nop, match_status=st_m, ncu_idx=idx,
                    match_kind=kind, summary=summ, aggregate_status=st_a, ops=ops, totals=tot)

    # -- accounting
    def set_timing(self, on: bool):
        library().opattr_set_timing(self.handle, int(bool(on)))

    def set_timing_only(self, kernel: str | None):
        """With timing on, bracket only the launches of `kernel` (None: all)."""
        library().opattr_set_timing_only(self.handle, kernel.encode() if kernel else None)

    def timing_report(self) -> dict:
        lib = library()
        n = lib.opattr_timing_report(self.handle, None, None, None, 0)
        names = (ctypes.c_char_p * max(n, 1))()
        ms = (ctypes.c_double * max(n, 1))()
        cnt = (ctypes.c_int64 * max(n, 1))()
        lib.opattr_timing_report(self.handle, names, ms, cnt, n)
        return {names[i].decode(): (float(ms[i]), int(cnt[i])) for i in range(n)}

    def timing_reset(self):
        library().opattr_timing_reset(self.handle)

    def launch_count(self) -> int:
        return int(library().opattr_launch_count(self.handle))
