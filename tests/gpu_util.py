"""Helpers for the GPU parity tests: run the CUDA path through the C ABI and
compare with the CPU oracle element by element."""
from __future__ import annotations

import numpy as np

import oracle

RTOL = 1e-9          # floating-point aggregates, relative to the fp64 oracle


def gpu_run(trace, mode: str = "skip_name", dedup: bool | None = None, ctx=None):
    import torch

    import paper_2609_11938_gb300 as opa
    own = ctx is None
    if own:
        ctx = opa.Context(0, mismatch=mode)
    try:
        tr = opa.to_device(trace)
        if dedup is None:
            dedup = bool(trace.config.get("dedup")) and trace.k_layer is not None
        st_e, rk, nop = ctx.enclose(tr)
        st_m, idx, kind, summ = ctx.match(tr, dedup=dedup)
        st_a, ops, tot = ctx.aggregate(tr, rk, idx)
        torch.cuda.synchronize()
        return dict(enclose_status=st_e, range_of_kernel=rk.cpu().numpy(), n_op_enclosing=nop.cpu().numpy(),
                    match_status=st_m, ncu_idx=idx.cpu().numpy(), match_kind=kind.cpu().numpy(), summary=summ,
                    aggregate_status=st_a, ops={k: v.cpu().numpy() for k, v in ops.items()}, totals=tot)
    finally:
        if own:
            ctx.close()


def gpu_run_tiers(trace, mode: str = "skip_name", dedup: bool | None = None, use_corr: bool = True,
                  use_fusion: bool = True, ctx=None):
    """enclose, attribute (Fig. 2 tiers), match, aggregate by operator on the GPU."""
    import torch

    import paper_2609_11938_gb300 as opa
    own = ctx is None
    if own:
        ctx = opa.Context(0, mismatch=mode)
    try:
        tr = opa.to_device(trace)
        if dedup is None:
            dedup = bool(trace.config.get("dedup")) and trace.k_layer is not None
        st_e, rk, nop = ctx.enclose(tr)
        st_t, op, tier, fw, fz, tsum = ctx.attribute(tr, rk, nop, use_corr=use_corr, use_fusion=use_fusion)
        st_m, idx, kind, summ = ctx.match(tr, dedup=dedup)
        st_a, ops, tot = ctx.aggregate(tr, None, idx, op_of_kernel=op)
        torch.cuda.synchronize()
        u32 = lambda x: x.cpu().numpy().view(np.uint32)
        return dict(enclose_status=st_e, range_of_kernel=rk.cpu().numpy(), n_op_enclosing=nop.cpu().numpy(),
                    attribute_status=st_t, op_of_kernel=u32(op), tier=tier.cpu().numpy(), fused_with=u32(fw),
                    is_fused=fz.cpu().numpy(), tier_summary=tsum, match_status=st_m, ncu_idx=idx.cpu().numpy(),
                    match_kind=kind.cpu().numpy(), summary=summ, aggregate_status=st_a,
                    ops={k: v.cpu().numpy() for k, v in ops.items()}, totals=tot)
    finally:
        if own:
            ctx.close()


def assert_parity_tiers(g, o):
    assert g["attribute_status"] == o["attribute_status"]
    for k in ("op_of_kernel", "tier", "fused_with", "is_fused"):
        np.testing.assert_array_equal(g[k], o[k], err_msg=k)
    assert g["tier_summary"] == o["tier_summary"], (g["tier_summary"], o["tier_summary"])
    assert_parity(g, o)


def assert_close(got, want, rtol=RTOL, what=""):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    assert got.shape == want.shape, what
    gn, wn = np.isnan(got), np.isnan(want)
    bad = np.nonzero(gn != wn)[0] if got.ndim == 1 else np.argwhere(gn != wn)
    assert len(bad) == 0, f"{what}: NaN pattern differs at {bad[:5]}"
    ok = ~wn
    if ok.any():
        err = np.abs(got[ok] - want[ok])
        lim = rtol * np.abs(want[ok])
        worst = np.max(err - lim)
        assert worst <= 0, f"{what}: max excess {worst}, rel err {np.max(err / np.maximum(np.abs(want[ok]), 1e-300))}"


def assert_parity(g, o, check_summary=True):
    assert g["enclose_status"] == o["enclose_status"]
    np.testing.assert_array_equal(g["range_of_kernel"], o["range_of_kernel"])
    np.testing.assert_array_equal(g["n_op_enclosing"], o["n_op_enclosing"])
    assert g["match_status"] == o["match_status"]
    np.testing.assert_array_equal(g["ncu_idx"], o["ncu_idx"])
    np.testing.assert_array_equal(g["match_kind"], o["match_kind"])
    if check_summary:
        for k in oracle.SUMMARY_FIELDS:
            assert g["summary"][k] == o["summary"][k], (k, g["summary"], o["summary"])
    assert g["aggregate_status"] == o["aggregate_status"]
    for k in ("kernel_count", "total_duration_ns", "matched_count"):
        np.testing.assert_array_equal(g["ops"][k], o["ops"][k], err_msg=k)
    assert_close(g["ops"]["agg"], o["ops"]["agg"], what="agg")
    for k in ("total_ns", "attributed_ns", "unattributed_ns", "kernels", "attributed_kernels", "matched_kernels"):
        assert g["totals"][k] == o["totals"][k], k
    for k in ("attributed_frac", "unattributed_frac"):
        a, b = g["totals"][k], o["totals"][k]
        assert (np.isnan(a) and np.isnan(b)) or a == b, (k, a, b)
