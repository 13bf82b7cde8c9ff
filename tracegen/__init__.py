"""Seeded synthetic traces for the attribution join (input generator only).

The arrays have the shapes of an Nsight Systems export (kernel records and NVTX
ranges per stream) and an Nsight Compute export (one counter row per replayed
launch, in launch order).  The paper's own traces are not available, so these
configurations stand in for them; the recipe is in ``tracegen.c``.

Nothing here decides enclosure, matching or aggregation: the CPU oracle and
the CUDA library both take these arrays as plain inputs.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tracegen.c")
_SO = os.path.join(_HERE, "libtracegen.so")
_lock = threading.Lock()
_lib_handle = None

STRUCTURAL = 0xFFFFFFFF
NONOP = 0xFFFFFFFE
N_COUNTERS = 20


class _Cfg(ctypes.Structure):
    _fields_ = [
        ("seed", ctypes.c_uint64), ("shape", ctypes.c_int32), ("n_streams", ctypes.c_int32),
        ("n_kernels", ctypes.c_int64), ("max_depth", ctypes.c_int32), ("n_names", ctypes.c_int32),
        ("zipf_s", ctypes.c_double), ("dur_median_ns", ctypes.c_double), ("dur_sigma", ctypes.c_double),
        ("gap_mean_ns", ctypes.c_double), ("delta_mean_ns", ctypes.c_double),
        ("p_zero_delta", ctypes.c_double), ("uncovered_frac", ctypes.c_double),
        ("uncovered_by_time", ctypes.c_int32), ("bb_run_mean", ctypes.c_double),
        ("kids_mean", ctypes.c_double), ("p_kernel_child", ctypes.c_double), ("p_nonop", ctypes.c_double),
        ("p_struct_inner", ctypes.c_double), ("p_empty", ctypes.c_double), ("p_chain", ctypes.c_double),
        ("n_iters", ctypes.c_int32), ("n_slots", ctypes.c_int32), ("n_classes", ctypes.c_int32),
        ("tmpl_len", ctypes.c_int32 * 8), ("layer_per_stream", ctypes.c_int32),
        ("step_kernels", ctypes.c_int32), ("dedup", ctypes.c_int32),
        ("counter_dist", ctypes.c_int32), ("counter_lo", ctypes.c_double), ("counter_hi", ctypes.c_double),
        ("nan_frac", ctypes.c_double), ("nan_mask", ctypes.c_uint32), ("shuffle", ctypes.c_int32),
    ]


# Workload shapes.  Sizes follow the five configurations of the attribution
# benchmark; parameters not fixed there (range-tree branching, host deltas,
# gap means) are chosen so range counts and uncovered shares land near the
# stated figures.
_BASE = dict(
    seed=0, shape=0, n_streams=1, n_kernels=2000, max_depth=4, n_names=40, zipf_s=1.1,
    dur_median_ns=8000.0, dur_sigma=1.2, gap_mean_ns=2000.0, delta_mean_ns=500.0, p_zero_delta=0.1,
    uncovered_frac=0.0, uncovered_by_time=0, bb_run_mean=8.0, kids_mean=3.0, p_kernel_child=0.8,
    p_nonop=0.05, p_struct_inner=0.03, p_empty=0.08, p_chain=0.05, n_iters=0, n_slots=0, n_classes=1,
    tmpl_len=(40, 0, 0, 0, 0, 0, 0, 0), layer_per_stream=1, step_kernels=0, dedup=0,
    counter_dist=0, counter_lo=0.0, counter_hi=100.0, nan_frac=0.0, nan_mask=0, shuffle=0,
)

CONFIGS = {
    # 1 stream, 2,000 kernels, ~300 ranges nested depth <= 4, ~10 % uncovered
    "tiny": dict(seed=0, n_streams=1, n_kernels=2000, max_depth=4, n_names=40, zipf_s=1.1,
                 dur_median_ns=8000.0, dur_sigma=1.2, gap_mean_ns=2000.0, uncovered_frac=0.10,
                 kids_mean=6.0, p_kernel_child=0.9),
    # GPT-2-small-shaped: 12 identical layers x ~40 kernels x 50 iterations on 2 streams
    "gpt2": dict(seed=1, shape=1, n_streams=2, max_depth=6, n_names=120, zipf_s=1.1,
                 dur_median_ns=8000.0, dur_sigma=1.2, gap_mean_ns=2000.0, n_iters=50, n_slots=12,
                 n_classes=1, tmpl_len=(40, 0, 0, 0, 0, 0, 0, 0), layer_per_stream=1,
                 step_kernels=1, uncovered_frac=0.0, counter_dist=1, counter_lo=1e-3, counter_hi=1e3),
    # the same shape on one stream with layer deduplication: N = 12 layers, K = 1 class
    "gpt2_dedup": dict(seed=5, shape=1, n_streams=1, max_depth=6, n_names=120, zipf_s=1.1,
                       dur_median_ns=8000.0, dur_sigma=1.2, gap_mean_ns=2000.0, n_iters=50, n_slots=12,
                       n_classes=1, tmpl_len=(40, 0, 0, 0, 0, 0, 0, 0), layer_per_stream=1,
                       step_kernels=2, dedup=1, counter_dist=1, counter_lo=1e-3, counter_hi=1e3),
    # N = 48 layers in K = 3 classes (16 each) on 4 streams, 400,000 kernels
    "dedup": dict(seed=2, shape=1, n_streams=4, max_depth=6, n_names=120, zipf_s=1.1,
                  dur_median_ns=15000.0, dur_sigma=1.0, gap_mean_ns=2000.0, n_iters=200, n_slots=12,
                  n_classes=3, tmpl_len=(42, 38, 45, 0, 0, 0, 0, 0), layer_per_stream=1, dedup=1),
    # 16 streams, 20,000,000 kernels, ~5,000,000 ranges depth <= 8, 5 % uncovered
    "large": dict(seed=3, n_streams=16, n_kernels=20_000_000, max_depth=8, n_names=5000, zipf_s=1.1,
                  dur_median_ns=8000.0, dur_sigma=1.2, gap_mean_ns=2000.0, uncovered_frac=0.05,
                  kids_mean=4.2, p_kernel_child=0.86),
    # 64 streams, 50,000,000 kernels, 85 % of runtime outside every range, depth up to 32,
    # many zero-length and identical-endpoint ranges
    "adversarial": dict(seed=4, n_streams=64, n_kernels=50_000_000, max_depth=32, n_names=50000,
                        zipf_s=1.5, dur_median_ns=3000.0, dur_sigma=2.0, gap_mean_ns=1000.0,
                        uncovered_frac=0.85, uncovered_by_time=1, bb_run_mean=3.0, p_zero_delta=0.7,
                        delta_mean_ns=200.0, kids_mean=1.5, p_kernel_child=0.55, p_empty=0.3,
                        p_chain=0.45, p_nonop=0.08, p_struct_inner=0.03),
}


def _build() -> str:
    """Compile the generator (plain C) into a shared object next to it."""
    if os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(_SRC):
        return _SO
    base = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", _SRC, "-o", _SO + ".tmp", "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(_SO + ".tmp", _SO)
    return _SO


def _lib():
    global _lib_handle
    with _lock:
        if _lib_handle is None:
            lib = ctypes.CDLL(_build())
            lib.tg_generate.argtypes = [ctypes.POINTER(_Cfg), ctypes.POINTER(ctypes.c_void_p)]
            lib.tg_generate.restype = ctypes.c_int
            lib.tg_sizes.argtypes = [ctypes.c_void_p, ctypes.POINTER(ctypes.c_int64)]
            lib.tg_copy.argtypes = [ctypes.c_void_p] + [ctypes.c_void_p] * 14
            lib.tg_free.argtypes = [ctypes.c_void_p]
            _lib_handle = lib
        return _lib_handle


@dataclass
class Trace:
    """A synthetic trace as numpy arrays (structure of arrays)."""
    k_stream: np.ndarray          # u8[K]
    k_start: np.ndarray           # i64[K]  query point T of each kernel, ns
    k_dur: np.ndarray             # i64[K]  kernel duration, ns
    k_name: np.ndarray            # u32[K]  kernel-name id
    k_layer: np.ndarray | None    # i32[K]  layer tag, -1 outside layers (None: untagged)
    r_stream: np.ndarray          # u8[R]
    r_start: np.ndarray           # i64[R]
    r_end: np.ndarray             # i64[R]
    r_depth: np.ndarray           # u8[R]
    r_op: np.ndarray              # u32[R]  op id, or STRUCTURAL / NONOP
    n_ops: int
    ncu_name: np.ndarray          # u32[M]  ncu rows in launch order
    counters: np.ndarray          # f32[M, 20]
    class_of_layer: np.ndarray | None = None   # i32[n_layers]
    rep_of_class: np.ndarray | None = None     # i32[n_classes]
    config: dict = field(default_factory=dict)
    ncu_stream: np.ndarray | None = None       # u8[M] stream of each ncu row (per-stream replay runs)
    corr_name: np.ndarray | None = None        # u32[C] torch.profiler correlation map: kernel name,
    corr_inv: np.ndarray | None = None         # u32[C]   invocation index of that name,
    corr_op: np.ndarray | None = None          # u32[C]   operator (HIGH tier)
    fusion_op: np.ndarray | None = None        # u32[n_names] Inductor fusion map: operator per name or OP_NONE
    fusion_len: np.ndarray | None = None       # u8[n_names]  operators in the fused list

    @property
    def K(self) -> int:
        return int(self.k_start.shape[0])

    @property
    def R(self) -> int:
        return int(self.r_start.shape[0])

    @property
    def M(self) -> int:
        return int(self.ncu_name.shape[0])


def config(name: str, **overrides) -> dict:
    cfg = dict(_BASE)
    cfg.update(CONFIGS[name])
    cfg.update(overrides)
    return cfg


def generate(name_or_cfg, shuffle: bool = False, **overrides) -> Trace:
    """Draw one trace.  ``name_or_cfg`` is a key of CONFIGS or a full dict."""
    cfg = config(name_or_cfg, **overrides) if isinstance(name_or_cfg, str) else {**_BASE, **name_or_cfg, **overrides}
    if shuffle:
        cfg["shuffle"] = 1
    lib = _lib()
    c = _Cfg()
    for k, v in cfg.items():
        if k == "tmpl_len":
            arr = (ctypes.c_int32 * 8)(*([int(x) for x in v] + [0] * (8 - len(v))))
            c.tmpl_len = arr
        else:
            setattr(c, k, v)
    h = ctypes.c_void_p()
    rc = lib.tg_generate(ctypes.byref(c), ctypes.byref(h))
    if rc != 0:
        raise ValueError(f"tracegen rejected the configuration (rc={rc})")
    try:
        sz = (ctypes.c_int64 * 7)()
        lib.tg_sizes(h, sz)
        K, R, M, n_ops, n_layers, n_classes, has_layer = (int(x) for x in sz)
        t = Trace(
            k_stream=np.empty(K, np.uint8), k_start=np.empty(K, np.int64), k_dur=np.empty(K, np.int64),
            k_name=np.empty(K, np.uint32), k_layer=np.empty(K, np.int32) if has_layer else None,
            r_stream=np.empty(R, np.uint8), r_start=np.empty(R, np.int64), r_end=np.empty(R, np.int64),
            r_depth=np.empty(R, np.uint8), r_op=np.empty(R, np.uint32), n_ops=n_ops,
            ncu_name=np.empty(M, np.uint32), counters=np.empty((M, N_COUNTERS), np.float32),
            class_of_layer=np.empty(n_layers, np.int32) if n_layers else None,
            rep_of_class=np.empty(n_classes, np.int32) if n_classes else None,
            config=cfg,
        )

        def p(a):
            return None if a is None else a.ctypes.data_as(ctypes.c_void_p)

        lib.tg_copy(h, p(t.k_stream), p(t.k_start), p(t.k_dur), p(t.k_name), p(t.k_layer),
                    p(t.r_stream), p(t.r_start), p(t.r_end), p(t.r_depth), p(t.r_op),
                    p(t.ncu_name), p(t.counters), p(t.class_of_layer), p(t.rep_of_class))
    finally:
        lib.tg_free(h)
    return t


def build() -> None:
    _lib()


def small_random(seed: int, n_streams: int = 2, n_events: int = 40, t_max: int = 8, max_depth: int = 4,
                 p_struct: float = 0.15, p_nonop: float = 0.15, shuffle: bool = True,
                 n_names: int = 3) -> Trace:
    """A tiny trace with integer times in [0, t_max] for brute-force checks.

    Per stream, a random push / pop / launch / tick event sequence: ranges
    stay laminar, and the small time range forces zero-length ranges,
    identical endpoints, touching siblings and kernels on range boundaries.
    """
    rng = np.random.default_rng(seed)
    ks, kt, kn, rs, rt, re, rd, ro = [], [], [], [], [], [], [], []
    next_op = 0
    for s in range(n_streams):
        t, stack = 0, []
        for _ in range(n_events):
            u = rng.random()
            if u < 0.3 and len(stack) < max_depth:
                v = rng.random()
                kind = STRUCTURAL if v < p_struct else (NONOP if v < p_struct + p_nonop else -1)
                if kind == -1:
                    kind, next_op = next_op, next_op + 1
                rs.append(s); rt.append(t); re.append(-1); rd.append(len(stack)); ro.append(kind)
                stack.append(len(rt) - 1)
            elif u < 0.55 and stack:
                re[stack.pop()] = t
            elif u < 0.85:
                ks.append(s); kt.append(t); kn.append(int(rng.integers(0, n_names)))
            elif t < t_max:
                t += 1
        while stack:
            re[stack.pop()] = t
    K, R = len(kt), len(rt)
    kp = rng.permutation(K) if shuffle else np.argsort(np.array(kt, np.int64) * 256 + np.array(ks), kind="stable")
    rp = rng.permutation(R) if shuffle else np.arange(R)
    k_stream = np.array(ks, np.uint8)[kp] if K else np.zeros(0, np.uint8)
    k_start = np.array(kt, np.int64)[kp] if K else np.zeros(0, np.int64)
    k_name = np.array(kn, np.uint32)[kp] if K else np.zeros(0, np.uint32)
    k_dur = rng.integers(0, 5, K).astype(np.int64)
    order = np.lexsort((np.arange(K), k_stream, k_start))      # time order: start, stream, index
    ncu_name = k_name[order].copy()
    counters = rng.uniform(0.0, 100.0, (K, N_COUNTERS)).astype(np.float32)
    return Trace(
        k_stream=k_stream, k_start=k_start, k_dur=k_dur, k_name=k_name, k_layer=None,
        r_stream=np.array(rs, np.uint8)[rp] if R else np.zeros(0, np.uint8),
        r_start=np.array(rt, np.int64)[rp] if R else np.zeros(0, np.int64),
        r_end=np.array(re, np.int64)[rp] if R else np.zeros(0, np.int64),
        r_depth=np.array(rd, np.uint8)[rp] if R else np.zeros(0, np.uint8),
        r_op=np.array(ro, np.uint32)[rp] if R else np.zeros(0, np.uint32),
        n_ops=next_op, ncu_name=ncu_name, counters=counters,
        config=dict(seed=seed, small=True))


def per_stream_runs(trace: Trace, stream_order=None) -> Trace:
    """The same trace with its ncu rows as Nsight Compute gives them when it
    replays one stream per run: the rows of each stream in launch order, the
    runs one after another (streams ascending, or in `stream_order`), every
    row tagged with its stream.  Needs one row per replayed kernel in kernel
    time order (the generator's default): every kernel, or with layer classes
    the kernels outside layers and in each class's representative layer."""
    import dataclasses
    tk = np.lexsort((trace.k_stream.astype(np.int64), trace.k_start))        # kernels in time order
    replayed = np.ones(trace.K, bool)
    if trace.k_layer is not None and trace.class_of_layer is not None and trace.M != trace.K:
        layer = trace.k_layer[tk]
        rep = trace.rep_of_class[trace.class_of_layer[np.maximum(layer, 0)]]
        replayed = (layer < 0) | (rep == layer)
    row_stream = trace.k_stream[tk][replayed].astype(np.int64)
    if row_stream.shape[0] != trace.M:
        raise ValueError("per_stream_runs needs one ncu row per replayed kernel")
    key = row_stream
    if stream_order is not None:
        pos = np.full(256, 256, np.int64)                   # streams not listed go last
        pos[np.asarray(stream_order, np.int64)] = np.arange(len(stream_order))
        key = pos[row_stream]
    # rows are in time order, so a stable sort by stream keeps each run in launch order
    order = np.argsort(key, kind="stable")
    return dataclasses.replace(trace, ncu_name=trace.ncu_name[order].copy(), counters=trace.counters[order].copy(),
                               ncu_stream=row_stream[order].astype(np.uint8))


OP_NONE = 0xFFFFFFFF


def with_tiers(trace: Trace, seed: int = 7, p_corr: float = 0.5, p_fused: float = 0.1, p_stray: float = 0.01,
               p_unfused_list: float = 0.3, min_count: int = 0) -> Trace:
    """The same trace with a torch.profiler correlation map and an Inductor
    fusion map, as the attribution tiers of Fig. 2 read them.

    Correlation map: for a random share p_corr of every name's invocation
    indices 0 .. count-1 an entry (name, index, operator).  Op ids follow range
    order in time, and a name's launches spread over the trace, so the
    operator of index i of a name launched c times is drawn near the same
    fraction of the op ids, floor((i + U[0,1)) / c * n_ops): map operators stay
    local in time, as dispatches are (the closer the more launches a name
    has; with min_count only names launched at least that often get entries).
    Plus stray entries (a share p_stray
    each) that name no launch: indices at or past the name's count, and names
    that never ran, with uniform operators.  Entries come in random order.  Fusion map: per name id, with
    probability p_fused an operator drawn uniformly, else OP_NONE; list lengths
    1-4 (1 with probability p_unfused_list)."""
    import dataclasses
    rng = np.random.default_rng(seed)
    K, O = trace.K, max(int(trace.n_ops), 1)
    names = trace.k_name.astype(np.int64)
    n_names = int(names.max()) + 1 if K else 0
    count = np.bincount(names, minlength=n_names) if K else np.zeros(0, np.int64)
    present = np.nonzero(count)[0]
    pair_name = np.repeat(present, count[present])
    starts = np.repeat(np.cumsum(count[present]) - count[present], count[present])
    pair_inv = np.arange(len(pair_name)) - starts
    keep = (rng.random(len(pair_name)) < p_corr) & (count[pair_name] >= min_count)
    cn, ci = pair_name[keep], pair_inv[keep]
    n_stray = int(p_stray * len(cn)) + (1 if K else 0)
    if len(present):
        sn = rng.choice(present, n_stray)
        si = count[sn] + rng.integers(0, 3, n_stray)                 # past the name's launches
        un = n_names + rng.integers(0, 100, n_stray)                  # names that never ran
        ui = rng.integers(0, 3, n_stray)
        cn = np.concatenate([cn, sn, un])
        ci = np.concatenate([ci, si, ui])
    n_named = int(keep.sum())
    frac = (ci[:n_named] + rng.random(n_named)) / np.maximum(count[cn[:n_named]], 1)
    co = np.concatenate([np.minimum((frac * O).astype(np.int64), O - 1), rng.integers(0, O, len(cn) - n_named)])
    perm = rng.permutation(len(cn))
    cn, ci, co = cn[perm], ci[perm], co[perm]
    if trace.n_ops == 0:
        cn, ci, co = cn[:0], ci[:0], co[:0]
    fo = np.where(rng.random(n_names) < p_fused, rng.integers(0, O, n_names), OP_NONE) if trace.n_ops > 0 \
        else np.full(n_names, OP_NONE)
    fl = np.where(rng.random(n_names) < p_unfused_list, 1, rng.integers(2, 5, n_names))
    return dataclasses.replace(trace, corr_name=cn.astype(np.uint32), corr_inv=ci.astype(np.uint32),
                               corr_op=co.astype(np.uint32), fusion_op=fo.astype(np.uint32),
                               fusion_len=fl.astype(np.uint8))


def op_classes(trace: Trace, n_classes: int = 64, seed: int = 11, p_none: float = 0.02) -> np.ndarray:
    """An operator class per op id (the aten:: name that dispatches share), for
    class roll-ups: classes drawn Zipf(1.1)-distributed over n_classes, a share
    p_none of the ops left out (OP_NONE)."""
    rng = np.random.default_rng(seed)
    w = 1.0 / np.arange(1, n_classes + 1) ** 1.1
    cls = rng.choice(n_classes, size=int(trace.n_ops), p=w / w.sum()).astype(np.int64)
    cls[rng.random(int(trace.n_ops)) < p_none] = OP_NONE
    return cls.astype(np.uint32)
