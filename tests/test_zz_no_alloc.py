"""The no-allocation matching entry point.

opattr_match_noalloc serves callers that cannot allocate device memory (an
attribution pass inside the profiled application, a host whose device memory
belongs to a caching allocator).  It must give exactly what opattr_match
gives, call after call, while its scratch is one shared fixed array.  This file
is collected last so a run that stops at the first failure has run every
other test before it."""
import os
import subprocess
import sys

import numpy as np
import pytest

import oracle
import tracegen

pytestmark = pytest.mark.gpu
HERE = os.path.dirname(os.path.abspath(__file__))


def _cases():
    # a shuffled trace with a dropped row (general path, count mismatch), then
    # an ordered trace whose rows equal its kernels (identity path)
    a = tracegen.small_random(71, n_streams=3, n_events=400, max_depth=5, shuffle=True, n_names=6)
    a.ncu_name = a.ncu_name[1:].copy()
    a.counters = a.counters[1:].copy()
    b = tracegen.generate("gpt2", n_iters=20)
    return [(a, "skip_name"), (b, "prefix"), (a, "prefix")]


def _at_limit():
    """OPATTR_MATCH_NOALLOC_MAX kernels and rows, kernels shuffled (the radix
    time order runs) and one row renamed (two names mismatch: the general
    ordinal join runs)."""
    import paper_2609_11938_gb300 as opa
    t = tracegen.generate("large", n_kernels=opa.MATCH_NOALLOC_MAX, shuffle=True)
    assert t.K == opa.MATCH_NOALLOC_MAX and t.M == opa.MATCH_NOALLOC_MAX
    names = np.unique(t.ncu_name)
    t.ncu_name = t.ncu_name.copy()
    j = int(np.nonzero(t.ncu_name == names[0])[0][0])
    t.ncu_name[j] = names[1]
    return t


def _noalloc(opa, ctx, tr, K, mode):
    import torch
    idx = torch.full((K,), -7, dtype=torch.int32, device="cuda:0")
    kind = torch.full((K,), 9, dtype=torch.uint8, device="cuda:0")
    summ = opa.MatchSummary()
    st = opa.opattr_match_noalloc(ctx.kernels(tr), ctx.ncu(tr), mode, idx.data_ptr(), kind.data_ptr(), summ,
                                  ctx.stream.cuda_stream)
    torch.cuda.synchronize()
    return st, idx.cpu().numpy(), kind.cpu().numpy(), summ.as_dict()


def test_match_noalloc_equals_match():
    """Two calls in a row per case, each equal to opattr_match."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_11938_gb300 as opa
    for trace, mode in _cases():
        assert trace.K <= opa.MATCH_NOALLOC_MAX and trace.M <= opa.MATCH_NOALLOC_MAX
        ctx = opa.Context(0, mismatch=mode)
        tr = opa.to_device(trace)
        st_ref, idx_ref, kind_ref, summ_ref = ctx.match(tr, dedup=False)
        for _ in range(2):
            st, idx, kind, summ = _noalloc(opa, ctx, tr, trace.K, mode)
            assert st == st_ref
            np.testing.assert_array_equal(idx, idx_ref.cpu().numpy())
            np.testing.assert_array_equal(kind, kind_ref.cpu().numpy())
            assert summ == summ_ref
        ctx.close()


@pytest.mark.parametrize("mode", ["skip_name", "prefix"])
def test_match_noalloc_at_limit(mode):
    """The largest input the fixed array takes, on the general path, against
    the oracle and against opattr_match; device memory unchanged by calls
    after the first."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_11938_gb300 as opa
    t = _at_limit()
    st_o, idx_o, kind_o, summ_o = oracle.match(t.k_stream, t.k_start, t.k_name, t.ncu_name, mode=mode)
    assert st_o == opa.W_COUNT_MISMATCH
    ctx = opa.Context(0, mismatch=mode)
    tr = opa.to_device(t)
    st_ref, idx_ref, kind_ref, summ_ref = ctx.match(tr, dedup=False)
    _noalloc(opa, ctx, tr, t.K, mode)                      # warm-up call (may load device code)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info(0)[0]
    for _ in range(2):
        st, idx, kind, summ = _noalloc(opa, ctx, tr, t.K, mode)
        assert st == st_o == st_ref
        np.testing.assert_array_equal(idx, idx_o)
        np.testing.assert_array_equal(kind, kind_o)
        np.testing.assert_array_equal(idx, idx_ref.cpu().numpy())
        assert summ["fast_path"] == 0
        for k in oracle.SUMMARY_FIELDS:
            assert summ[k] == summ_o[k] == summ_ref[k], k
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info(0)[0] == free0
    ctx.close()


def test_match_noalloc_after_device_reset():
    """A process (without torch) calls the entry point, resets the device and
    calls it again: the array's address is looked up in the new context."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    r = subprocess.run([sys.executable, os.path.join(HERE, "noalloc_reset_child.py")], capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "noalloc reset ok" in r.stdout


def test_match_noalloc_rejects_oversize():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_11938_gb300 as opa
    k = opa.Kernels(None, None, None, None, None, opa.MATCH_NOALLOC_MAX + 1)
    n = opa.Ncu(None, None, 0)
    st = opa.opattr_match_noalloc(k, n, "skip_name", 0, None, opa.MatchSummary(), None)
    assert st == opa.E_INVALID_ARG
