"""The no-allocation matching entry point.

opattr_match_noalloc serves callers that cannot allocate device memory (an
attribution pass inside the profiled application, a host whose device memory
belongs to a caching allocator).  It must give exactly what opattr_match
gives, call after call, while its scratch is one shared fixed array.  This file
is collected last so a run that stops at the first failure has run every
other test before it."""
import numpy as np
import pytest

import tracegen

pytestmark = pytest.mark.gpu


def _cases():
    # a shuffled trace with a dropped row (general path, count mismatch), then
    # an ordered trace whose rows equal its kernels (identity path)
    a = tracegen.small_random(71, n_streams=3, n_events=400, max_depth=5, shuffle=True, n_names=6)
    a.ncu_name = a.ncu_name[1:].copy()
    a.counters = a.counters[1:].copy()
    b = tracegen.generate("gpt2", n_iters=20)
    return [(a, "skip_name"), (b, "prefix"), (a, "prefix")]


def test_match_noalloc_equals_match():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_11938_gb300 as opa
    for trace, mode in _cases():
        assert trace.K <= opa.MATCH_NOALLOC_MAX and trace.M <= opa.MATCH_NOALLOC_MAX
        ctx = opa.Context(0, mismatch=mode)
        tr = opa.to_device(trace)
        st_ref, idx_ref, kind_ref, summ_ref = ctx.match(tr, dedup=False)
        idx = torch.full((trace.K,), -7, dtype=torch.int32, device="cuda:0")
        kind = torch.full((trace.K,), 9, dtype=torch.uint8, device="cuda:0")
        summ = opa.MatchSummary()
        st = opa.opattr_match_noalloc(ctx.kernels(tr), ctx.ncu(tr), mode, idx.data_ptr(), kind.data_ptr(), summ,
                                      ctx.stream.cuda_stream)
        torch.cuda.synchronize()
        assert st == st_ref
        np.testing.assert_array_equal(idx.cpu().numpy(), idx_ref.cpu().numpy())
        np.testing.assert_array_equal(kind.cpu().numpy(), kind_ref.cpu().numpy())
        assert summ.as_dict() == summ_ref
        ctx.close()


def test_match_noalloc_rejects_oversize():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_11938_gb300 as opa
    k = opa.Kernels(None, None, None, None, None, opa.MATCH_NOALLOC_MAX + 1)
    n = opa.Ncu(None, None, 0)
    st = opa.opattr_match_noalloc(k, n, "skip_name", 0, None, opa.MatchSummary(), None)
    assert st == opa.E_INVALID_ARG
