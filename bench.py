"""Benchmark: the attribution join (enclose + match + aggregate) on the
20M-kernel synthetic trace, one pass per step, on N GPUs (one independent
trace per rank: weak scaling, no collective on the data path).

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle on a
bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "M kernel records attributed/sec (1 GB300) and % of HBM roofline"
UNIT = "M kernels/s"
NOMINAL_HBM_GBS = 8000.0
L2_BYTES = 129 * 2**20

# Algorithmic bytes per unit (the minimum each step must move):
#   per kernel: stream 1 + start 8 + dur 8 + name 4 read, range 4 + ncu_idx 4 written
#   per range: stream 1 + start 8 + end 8 + depth 1 + op 4 read
#   per ncu row: name 4 + 20 counters x 4 read;  per op: 3 x 8 + 20 x 8 written
PATH_BYTES = dict(kernel=29, range=22, ncu=84, op=184)

# Per-launch algorithmic bytes of the kernels that can dominate a step.
KERNEL_BYTES = {
    # list 4 + duration 8 + row index 4 + counter row 80 per kernel (the row
    # index is not read when every kernel's row is its own index: 92)
    "agg_ops": lambda K, R, M, O: 96 * K + 188 * O,
    "enclose": lambda K, R, M, O: 14 * K + 20 * R,
    "agg_place": lambda K, R, M, O: 16 * K,
    "agg_count": lambda K, R, M, O: 24 * K + 4 * O,
    "match_identity": lambda K, R, M, O: 13 * K,
    "check_kernel_order": lambda K, R, M, O: 9 * K,
    "check_ranges": lambda K, R, M, O: 18 * R,
    "level_gather": lambda K, R, M, O: 44 * R,
    "level_place": lambda K, R, M, O: 42 * R,
    "match_stream_pairs": lambda K, R, M, O: 18 * K,
    "validate_levels": lambda K, R, M, O: 22 * R,
    "stream_place": lambda K, R, M, O: 5 * K,
    "stream_windows": lambda K, R, M, O: 0,
}

WORKLOADS = {
    "large": "16 streams, 20,000,000 kernels, ~5,000,000 NVTX ranges depth <= 8, 5,000 names Zipf 1.1, "
             "20 fp32 counters per ncu row U[0,100], 5% of kernels uncovered (seed 3)",
    "adversarial": "64 streams, 50,000,000 kernels, 85% of runtime outside ranges, depth up to 32, "
                   "50,000 names Zipf 1.5 (seed 4)",
    "dedup": "48 layers in 3 classes on 4 streams, 400,000 kernels, 25,000 ncu rows (seed 2)",
    "gpt2": "GPT-2-small-shaped: 12 layers x 40 kernels x 50 iterations on 2 streams (seed 1)",
    "tiny": "1 stream, 2,000 kernels, ~300 ranges (seed 0)",
}


def source_digest(files):
    """Digest of the named CUDA sources (csrc/ file names), to tie recorded ncu figures to the code they came from."""
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_11938_gb300", "csrc")
    for name in sorted(files):
        h.update(name.encode())
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel, workload, kernels):
    """DRAM bytes per launch from profiles/traffic.txt, or None if absent or taken on other sources."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.txt")) as f:
            lines = [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]
    except OSError:
        return None
    for ln in lines:
        if len(ln) == 6 and ln[0] == kernel and ln[1] == workload and int(ln[2]) == kernels:
            try:
                if ln[4] == source_digest(ln[3].split(",")):
                    return int(ln[5])
            except OSError:
                return None
    return None


def recorded_tiers(trace, seed, share=0.5):
    """The trace with the maps the attribution tiers read, as a capture would
    record them (the benchmark's input; parity tests use tracegen.with_tiers).
    Correlation map: for a random half of the launches the entry (name, number
    of earlier launches of that name in time order, operator), the operator
    being the last operator range pushed on the launch's stream before it
    started (the dispatch that launched it), or a random one for launches
    outside every range; entries in random order.  Fusion map as in
    tracegen.with_tiers."""
    import dataclasses

    import numpy as np

    import tracegen
    rng = np.random.default_rng(seed)
    t = tracegen.with_tiers(trace, seed=seed, p_corr=0.0, p_stray=0.0)
    K = trace.K
    order = np.lexsort((np.arange(K), trace.k_stream.astype(np.int64), trace.k_start))
    names = trace.k_name[order].astype(np.int64)
    by_name = np.argsort(names, kind="stable")
    first = np.searchsorted(names[by_name], names[by_name], side="left")
    inv = np.empty(K, np.int64)
    inv[order[by_name]] = np.arange(K) - first
    op = rng.integers(0, max(int(trace.n_ops), 1), K)
    is_op = trace.r_op < trace.n_ops
    for s in np.unique(trace.k_stream):
        rs = np.nonzero((trace.r_stream == s) & is_op)[0]
        rs = rs[np.argsort(trace.r_start[rs], kind="stable")]
        ks = np.nonzero(trace.k_stream == s)[0]
        p = np.searchsorted(trace.r_start[rs], trace.k_start[ks], side="right") - 1
        op[ks[p >= 0]] = trace.r_op[rs[p[p >= 0]]]
    pick = rng.permutation(np.nonzero(rng.random(K) < share)[0])
    return dataclasses.replace(t, corr_name=trace.k_name[pick].astype(np.uint32),
                               corr_inv=inv[pick].astype(np.uint32), corr_op=op[pick].astype(np.uint32))


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# ---------------------------------------------------------------- rank plumbing
def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def combine_ranks(elapsed_s: float, units: int, world: int, reduce_max, reduce_sum):
    """Max elapsed over ranks and the units all ranks processed."""
    t = reduce_max(elapsed_s) if world > 1 else elapsed_s
    u = reduce_sum(units) if world > 1 else units
    return t, u


def run_timed(step, steps: int, warmup: int, sync, barrier, start_clock=None, stop_clock=None):
    """W untimed steps, then exactly K steps between barrier + sync pairs.
    Returns seconds of the timed region (device-timed by `sync` pairs)."""
    for _ in range(warmup):
        step()
    sync()
    barrier()
    sync()
    if start_clock:
        start_clock()
    t0 = time.perf_counter()
    for _ in range(steps):
        step()
    sync()
    barrier()
    sync()
    t1 = time.perf_counter()
    if stop_clock:
        stop_clock()
    return t1 - t0


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 100 ms."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device: int):
        self.device = device
        self.proc = None
        self.path = None
        self.windows = []

    def start(self):
        fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.device), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)

    def mark(self, begin: bool):
        if begin:
            self.windows.append([time.time(), None])
        else:
            self.windows[-1][1] = time.time()

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.proc or not self.path:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = [r.split(", ") for r in open(self.path).read().strip().splitlines() if r.strip()]
        os.unlink(self.path)
        sm = [float(r[1]) for r in rows if len(r) >= 9 and r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if len(r) >= 9 and r[2].replace(".", "").isdigit()]
        power = [float(r[3]) for r in rows if len(r) >= 9 and r[3].replace(".", "").isdigit()]
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = sorted({n for r in rows if len(r) >= 9 for n, v in zip(names, r[5:9]) if v.strip() == "Active"})
        loaded = sorted(sm)[len(sm) // 2:] if sm else []
        return {"sm_mhz": statistics.median(loaded) if loaded else None, "sm_max_mhz": max(mx) if mx else None,
                "samples": len(sm), "power_w_max": max(power) if power else None, "reasons": reasons,
                "window": "warm-up + timed region + 1 s soak of the same step"}


# ---------------------------------------------------------------- CPU baseline (the oracle)
def cpu_model() -> str:
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.strip().lower().startswith("model name"):
                return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for ln in f:
                if ln.lower().startswith(("model name", "cpu part")):
                    return ln.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.processor() or platform.machine()


def time_oracle_full(trace, threads: int):
    """The CPU oracle (indexed mode) on the whole trace: one thread
    (oracle.run) or `threads` host threads (oracle.parallel.run_threads, the
    same functions over streams / names / op blocks).  Returns seconds."""
    import oracle
    t0 = time.perf_counter()
    if threads == 1:
        res = oracle.run(trace, enclose_mode="indexed")
    else:
        from oracle.parallel import run_threads
        res = run_threads(trace, threads)
    dt = time.perf_counter() - t0
    assert res["aggregate_status"] == 0 and res["enclose_status"] == 0
    return dt


def reference_trace(config_name: str, n_kernels: int = 0, shuffle: bool = False):
    import tracegen
    cfg = tracegen.config(config_name)
    if n_kernels and cfg.get("shape", 0) == 0:
        cfg["n_kernels"] = n_kernels
    return tracegen.generate(cfg, shuffle=shuffle)


# ---------------------------------------------------------------- main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="large", choices=sorted(WORKLOADS))
    ap.add_argument("--shuffle", action="store_true", help="permute kernel and range arrays (general paths)")
    ap.add_argument("--e2e-steps", type=int, default=8)
    ap.add_argument("--e2e-copy-streams", type=int, default=2,
                    help="copy streams per direction in the end-to-end run")
    ap.add_argument("--no-oracle-single", dest="oracle_single", action="store_false",
                    help="skip the single-thread oracle run of the CPU baseline (it takes about 15 s on large)")
    ap.add_argument("--per-stream-ncu", action="store_true",
                    help="ncu rows as per-stream replay runs, matched per (name, stream)")
    ap.add_argument("--tiers", action="store_true",
                    help="attribution tiers of Fig. 2 in the step: a correlation map recorded for half of the "
                         "launches, fusion entries for a tenth of the names, aggregation by each kernel's operator")
    ap.add_argument("--rollup", type=int, default=0,
                    help="also roll the operator records up to this many operator classes in each step")
    ap.add_argument("--launch-lag", type=int, default=0,
                    help="enclosure queries at start - U[0, LAG) ns (host launch times)")
    ap.add_argument("--kernels", type=int, default=0,
                    help="draw this many kernels with the config's generator parameters (profiling runs)")
    args = ap.parse_args()
    world, rank, local = dist_env()
    if args.warmup < 3:
        args.warmup = 3

    if args.impl == "reference":
        # the oracle on the whole workload in all host threads, each step one
        # full join; rank 0 alone (the other ranks exit without work)
        if rank != 0:
            return
        trace = reference_trace(args.config, args.kernels, args.shuffle)
        threads = os.cpu_count() or 1
        for _ in range(args.warmup):
            time_oracle_full(trace, threads)
        times = [time_oracle_full(trace, threads) for _ in range(args.steps)]
        tot = sum(times)
        value = trace.K * len(times) / tot / 1e6
        sample = (f"the whole {args.config} trace ({trace.K} kernels, {trace.R} ranges, {trace.M} ncu rows, "
                  f"{trace.n_ops} ops) every step; indexed oracle (enclose + match + aggregate) over {threads} "
                  f"host threads ({cpu_model()})")
        line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / len(times),
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                "data": "synthetic", "config": {"workload": f"{args.config}: {WORKLOADS[args.config]}" + (
                    f" [scaled to {trace.K} kernels]" if args.kernels else ""), "kernels": trace.K,
                    "same_config": not args.kernels},
                "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                                 "sample": sample},
                "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    import numpy as np
    import torch
    import torch.distributed as dist

    import paper_2609_11938_gb300 as opa
    import tracegen

    if world > 1:
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = local
    opa.build()

    def barrier():
        if world > 1:
            dist.barrier()

    def rmax(x):
        t = torch.tensor([float(x)], device=f"cuda:{dev}")
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    def rsum(x):
        t = torch.tensor([float(x)], device=f"cuda:{dev}", dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.SUM)
        return int(t.item())

    cfg = tracegen.config(args.config)
    cfg["seed"] = cfg["seed"] + 1000 * rank          # each rank attributes its own trace
    if args.kernels and cfg.get("shape", 0) == 0:
        cfg["n_kernels"] = args.kernels
    trace = tracegen.generate(cfg, shuffle=args.shuffle)
    if args.per_stream_ncu:
        trace = tracegen.per_stream_runs(trace)
    if args.tiers:
        trace = recorded_tiers(trace, seed=cfg["seed"])
    K, R, M, O = trace.K, trace.R, trace.M, trace.n_ops
    use_dedup = bool(cfg.get("dedup")) and trace.k_layer is not None
    tr = opa.to_device(trace, dev)
    tq = tr                                           # what the enclosure queries at
    if args.launch_lag > 0:
        lag = np.random.default_rng(cfg["seed"]).integers(0, args.launch_lag, K)
        tq = dataclasses.replace(tr, k_start=torch.from_numpy(trace.k_start - lag).to(f"cuda:{dev}"))
    torch.cuda.synchronize(dev)
    stream = torch.cuda.Stream(dev)
    ctx = opa.Context(dev, stream=stream)
    rk = torch.empty(K, dtype=torch.int32, device=f"cuda:{dev}")
    nop = torch.empty(K, dtype=torch.uint8, device=f"cuda:{dev}")
    idx = torch.empty(K, dtype=torch.int32, device=f"cuda:{dev}")
    kind = torch.empty(K, dtype=torch.uint8, device=f"cuda:{dev}")
    ops = ctx.alloc_ops(O)
    tiers_out = None
    if args.tiers:
        tiers_out = dict(op=torch.empty(K, dtype=torch.int32, device=f"cuda:{dev}"),
                         tier=torch.empty(K, dtype=torch.uint8, device=f"cuda:{dev}"),
                         fused_with=torch.empty(K, dtype=torch.int32, device=f"cuda:{dev}"),
                         is_fused=torch.empty(K, dtype=torch.uint8, device=f"cuda:{dev}"))

    rollup_out = class_of_op = None
    if args.rollup:
        class_of_op = torch.from_numpy(tracegen.op_classes(trace, n_classes=args.rollup).view(np.int32)).to(
            f"cuda:{dev}")
        rollup_out = ctx.alloc_ops(args.rollup)

    join_out = dict(range_of_kernel=rk, n_op_enclosing=nop, ncu_idx=idx, match_kind=kind)

    def make_join(tr, tq, join_out, ops, tiers_out, rollup_out):
        rk, nop, idx, kind = (join_out[k] for k in ("range_of_kernel", "n_op_enclosing", "ncu_idx", "match_kind"))

        def join():
            if tq is tr and tiers_out is None:
                # the whole join in one call (one kernel-order check for both steps)
                ctx.join(tr, dedup=use_dedup, out=join_out, ops=ops)
                if rollup_out is not None:
                    ctx.rollup(tr, rk, idx, class_of_op, args.rollup, out=rollup_out)
                return
            ctx.enclose(tq, rk, nop)
            if tiers_out is not None:
                ctx.attribute(tr, rk, nop, out=tiers_out)
            ctx.match(tr, dedup=use_dedup, out_idx=idx, out_kind=kind)
            if tiers_out is not None:
                ctx.aggregate(tr, None, idx, ops, op_of_kernel=tiers_out["op"])
            else:
                ctx.aggregate(tr, rk, idx, ops)
            if rollup_out is not None:
                ctx.rollup(tr, rk, idx, class_of_op, args.rollup, out=rollup_out,
                           op_of_kernel=tiers_out["op"] if tiers_out is not None else None)
        return join

    join = make_join(tr, tq, join_out, ops, tiers_out, rollup_out)
    in_bytes = sum(x.numel() * x.element_size() for x in (tr.k_stream, tr.k_start, tr.k_dur, tr.k_name,
                                                           tr.r_stream, tr.r_start, tr.r_end, tr.r_depth, tr.r_op,
                                                           tr.ncu_name, tr.counters))
    flush = None
    if in_bytes < 2 * L2_BYTES:
        flush = torch.empty(2 * L2_BYTES // 4, dtype=torch.float32, device=f"cuda:{dev}")

    def step():
        if flush is not None:
            with torch.cuda.stream(stream):
                flush.fill_(1.0)
        join()

    def sync():
        stream.synchronize()

    clocks = ClockSampler(dev)
    clocks.start()
    for _ in range(args.warmup):
        step()
    sync()
    # rows matched one for one (the ops pass then skips the row-index gather;
    # in a join whose matching was that identity pairing, the count pass too)
    if K > 0 and bool((idx == torch.arange(K, dtype=torch.int32, device=idx.device)).all()):
        KERNEL_BYTES["agg_ops"] = lambda K, R, M, O: 92 * K + 188 * O
        if (tq is tr and tiers_out is None and not use_dedup and not args.per_stream_ncu and M == K
                and not args.shuffle):
            KERNEL_BYTES["agg_count"] = lambda K, R, M, O: 20 * K + 4 * O
    # per-kernel breakdown: a few steps with every launch bracketed by events
    n_brk = max(1, min(args.steps, 10))
    ctx.set_timing(True)
    ctx.timing_reset()
    for _ in range(n_brk):
        step()
    sync()
    breakdown = ctx.timing_report()
    # the dominant kernel among those with algorithmic bytes (a search-bound
    # helper such as the window table has none, so no memory roofline)
    known = {k: v for k, v in breakdown.items() if k in KERNEL_BYTES and KERNEL_BYTES[k](K, R, M, O) > 0}
    dname = max((known or breakdown).items(), key=lambda kv: kv[1][0])[0]
    # the timed region brackets only the dominant kernel's launches
    ctx.set_timing_only(dname)
    ctx.timing_reset()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(); sync()
    ev0.record(stream)
    wall0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    ev1.record(stream)
    sync(); barrier(); sync()
    wall = time.perf_counter() - wall0
    elapsed = ev0.elapsed_time(ev1) / 1e3
    launches = ctx.launch_count()
    report = ctx.timing_report()
    ctx.set_timing(False)
    ctx.set_timing_only(None)
    # keep the GPU busy with the same step for ~1 s so the clock sampler sees it
    soak_end = time.perf_counter() + 1.0
    while time.perf_counter() < soak_end:
        step()
    sync()
    clocks.stop()
    t_max, units = combine_ranks(max(elapsed, 1e-9), K * args.steps, world, rmax, rsum)

    # ---- end to end through the C ABI with host buffers (pinned): every step
    # copies each input array host->device, runs the join and copies each
    # output device->host.  Steps overlap the way a caller streaming traces
    # would run them: step i+1's inputs go over on copy streams while step i's
    # join runs (two device buffer sets, used in turn), and step i's outputs
    # come back on other copy streams while step i+1 runs.
    in_names = ("k_stream", "k_start", "k_dur", "k_name", "r_stream", "r_start", "r_end", "r_depth", "r_op",
                "ncu_name", "counters")
    if args.tiers:
        in_names += ("corr_name", "corr_inv", "corr_op", "fusion_op", "fusion_len")
    if trace.k_layer is not None:
        in_names += ("k_layer",)
    if getattr(trace, "ncu_stream", None) is not None:
        in_names += ("ncu_stream",)
    host = {name: torch.from_numpy(getattr(trace, name)).pin_memory() for name in in_names}
    launch_host = tq.k_start.cpu().pin_memory() if tq is not tr else None

    def device_copy(t):
        return dataclasses.replace(t, **{f.name: getattr(t, f.name).clone() for f in dataclasses.fields(t)
                                         if torch.is_tensor(getattr(t, f.name))})

    def buffer_set(tr_b, tq_b, join_out_b, ops_b, tiers_b, rollup_b):
        return dict(tr=tr_b, tq=tq_b, rk=join_out_b["range_of_kernel"], idx=join_out_b["ncu_idx"], ops=ops_b,
                    join=make_join(tr_b, tq_b, join_out_b, ops_b, tiers_b, rollup_b))

    tr2 = device_copy(tr)
    tq2 = tr2 if tq is tr else dataclasses.replace(tr2, k_start=tq.k_start.clone())
    join_out2 = {k: torch.empty_like(v) for k, v in join_out.items()}
    ops2 = ctx.alloc_ops(O)
    tiers2 = {k: torch.empty_like(v) for k, v in tiers_out.items()} if tiers_out is not None else None
    rollup2 = ctx.alloc_ops(args.rollup) if rollup_out is not None else None
    sets = [buffer_set(tr, tq, join_out, ops, tiers_out, rollup_out),
            buffer_set(tr2, tq2, join_out2, ops2, tiers2, rollup2)]
    out_host = {"rk": torch.empty(K, dtype=torch.int32).pin_memory(),
                "idx": torch.empty(K, dtype=torch.int32).pin_memory()}
    out_host.update({k: torch.empty_like(v, device="cpu").pin_memory() for k, v in ops.items()})
    h2d = sum(v.numel() * v.element_size() for v in host.values())
    if launch_host is not None:
        h2d += launch_host.numel() * launch_host.element_size()
    d2h = sum(v.numel() * v.element_size() for v in out_host.values())
    n_cs = max(1, args.e2e_copy_streams)
    copy_in = [torch.cuda.Stream(dev) for _ in range(n_cs)]
    copy_out = [torch.cuda.Stream(dev) for _ in range(n_cs)]
    in_ev = [[torch.cuda.Event() for _ in range(n_cs)] for _ in range(2)]
    out_ev = [[torch.cuda.Event() for _ in range(n_cs)] for _ in range(2)]

    def spread(pairs, streams):
        """Copies dst <- src, arrays of 64 MB or more cut into one piece per stream."""
        j = 0
        for dst, src in pairs:
            n = dst.shape[0]
            parts = len(streams) if src.numel() * src.element_size() >= (64 << 20) else 1
            for p in range(parts):
                lo, hi = n * p // parts, n * (p + 1) // parts
                with torch.cuda.stream(streams[j % len(streams)]):
                    dst[lo:hi].copy_(src[lo:hi], non_blocking=True)
                j += 1

    def send(b):
        s = sets[b]
        pairs = [(getattr(s["tr"], name), v) for name, v in host.items()]
        if launch_host is not None:
            pairs.append((s["tq"].k_start, launch_host))
        spread(pairs, copy_in)
        for q in range(n_cs):
            in_ev[b][q].record(copy_in[q])

    def receive(b):
        s = sets[b]
        for q in range(n_cs):
            copy_out[q].wait_stream(stream)
        pairs = [(out_host["rk"], s["rk"]), (out_host["idx"], s["idx"])]
        pairs += [(out_host[k], v) for k, v in s["ops"].items()]
        spread(pairs, copy_out)
        for q in range(n_cs):
            out_ev[b][q].record(copy_out[q])

    def e2e_run(n):
        send(0)
        for i in range(n):
            b = i & 1
            if i + 1 < n:
                send(1 - b)         # set 1 - b was last read by join i - 1, which has returned
            for q in range(n_cs):
                stream.wait_event(in_ev[b][q])
                stream.wait_event(out_ev[b][q])     # step i - 2's outputs are off the device
            sets[b]["join"]()
            receive(b)

    def sync_all():
        for cs in copy_in + copy_out:
            cs.synchronize()
        stream.synchronize()

    e2e_run(2)
    sync_all()
    barrier()
    sync_all()
    t0 = time.perf_counter()
    e2e_run(args.e2e_steps)
    sync_all()
    barrier()
    sync_all()
    e2e_s = time.perf_counter() - t0
    e2e_t, e2e_units = combine_ranks(e2e_s, K * args.e2e_steps, world, rmax, rsum)

    if rank != 0:
        ctx.close()
        if world > 1:
            dist.destroy_process_group()
        return

    # ---- roofline of the dominant kernel (CUDA events around each launch)
    peak, peak_kind = load_peaks()
    dms, dcount = report.get(dname, (0.0, 0))
    dbytes = KERNEL_BYTES.get(dname, lambda *a: 0)(K, R, M, O)
    avg_s = dms / 1e3 / max(dcount, 1)
    achieved = dbytes / avg_s / 1e9 if dbytes else None
    step_s = elapsed / args.steps
    path_bytes = PATH_BYTES["kernel"] * K + PATH_BYTES["range"] * R + PATH_BYTES["ncu"] * M + PATH_BYTES["op"] * O
    path_gbs = path_bytes / step_s / 1e9
    ctx.close()

    # the oracle on the same whole trace, one thread and all host threads
    threads = os.cpu_count() or 1
    t_or1 = time_oracle_full(trace, 1) if args.oracle_single else None
    t_orn = time_oracle_full(trace, threads)
    line = {
        "metric": METRIC,
        "value": units / t_max / 1e6,
        "unit": UNIT,
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": 1e3 * t_max / args.steps,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "int64+f32x2",
        "data": "synthetic",
        "config": {"workload": f"{args.config}: {WORKLOADS[args.config]}" + (
                       f" [scaled to {K} kernels]" if args.kernels else ""), "kernels": K, "ranges": R,
                   "ncu_rows": M, "ops": O, "shuffled": bool(args.shuffle), "per_stream_ncu": bool(args.per_stream_ncu),
                   "launch_lag_ns": args.launch_lag, "tiers": bool(args.tiers), "rollup_classes": args.rollup,
                   "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2 (129 MB)" if flush is None else "L2 flushed before every step"},
        "roofline": {"bound": "hbm", "kernel": dname, "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": (achieved / peak) if achieved else None, "peak_kind": f"{peak_kind} copy bandwidth",
                     # recorded on the default options only (the variants change what the kernels move)
                     "traffic": (recorded_traffic(dname, args.config, K) if not (
                         args.shuffle or args.per_stream_ncu or args.tiers or args.rollup or args.launch_lag)
                         else None), "alg_bytes_per_launch": dbytes,
                     "avg_launch_ms": avg_s * 1e3,
                     "launches": dcount},
        "path_roofline": {"alg_bytes_per_step": path_bytes, "achieved_gbs": path_gbs,
                          "frac_of_8tbs": path_gbs / NOMINAL_HBM_GBS, "frac_of_measured": path_gbs / peak},
        "cpu_baseline": {"value": K / t_orn / 1e6, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": f"the whole trace timed on ({K} kernels), {t_orn:.2f} s; indexed oracle (enclose + "
                                   f"match + aggregate) over {threads} host threads ({cpu_model()})",
                         "single_thread": ({"value": K / t_or1 / 1e6, "unit": UNIT, "cores": 1,
                                            "seconds": round(t_or1, 3)} if t_or1 else None)},
        "e2e": {"value": e2e_units / e2e_t / 1e6, "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": launches,
        "kernel_ms_per_step": {k: round(v[0] / n_brk, 4) for k, v in sorted(breakdown.items(),
                                                                          key=lambda kv: -kv[1][0])},
        "kernel_ms_note": f"every launch bracketed by CUDA events over {n_brk} separate steps; the timed region "
                          f"brackets only {dname}",
        "wall_ms_per_step": 1e3 * wall / args.steps,
        "clocks": clocks.summary(),
    }
    print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
