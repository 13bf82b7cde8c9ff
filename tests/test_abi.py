"""The C ABI library builds, loads and exports every entry point the header
declares; the binding marshals structs of the header's layout.  CPU only: no
call here touches a GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "opattr.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(opattr_[a-z_]+)\s*\(", text)))


def test_header_declares_the_join():
    names = declared_functions()
    for f in ("opattr_create", "opattr_enclose", "opattr_match", "opattr_aggregate", "opattr_destroy",
              "opattr_join", "opattr_attribute", "opattr_rollup", "opattr_write_profile", "opattr_match_noalloc"):
        assert f in names


def test_library_exports_every_declared_symbol():
    import paper_2609_11938_gb300 as opa
    path = opa.build()
    lib = ctypes.CDLL(path)
    missing = [f for f in declared_functions() if not hasattr(lib, f)]
    assert not missing, missing


def test_struct_layouts_match_header():
    import paper_2609_11938_gb300 as opa
    # pointer-sized fields then int64 n; sizes follow the C layout on LP64
    assert ctypes.sizeof(opa.Kernels) == 6 * 8
    assert ctypes.sizeof(opa.Ranges) == 6 * 8
    assert ctypes.sizeof(opa.Ncu) == 4 * 8
    assert ctypes.sizeof(opa.Dedup) == 2 * 8 + 2 * 4
    assert ctypes.sizeof(opa.Config) == 4 + 4 + 4 + 4 + 8
    assert ctypes.sizeof(opa.MatchSummary) == 8 * 8 + 2 * 4
    assert ctypes.sizeof(opa.OpAggregates) == 4 * 8
    assert ctypes.sizeof(opa.Totals) == 6 * 8 + 2 * 8
    assert ctypes.sizeof(opa.Corr) == 4 * 8
    assert ctypes.sizeof(opa.Fusion) == 3 * 8
    assert ctypes.sizeof(opa.AttrSummary) == 7 * 8


def test_status_strings_without_gpu():
    import paper_2609_11938_gb300 as opa
    assert opa.opattr_status_string(opa.E_NOT_NESTED) == "ranges are not nested per stream"
    assert opa.opattr_status_string(123) == "unknown status"


def test_create_without_gpu_fails_cleanly():
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    import paper_2609_11938_gb300 as opa
    st, h = opa.opattr_create(0)
    assert st in (opa.E_CUDA, opa.E_INVALID_ARG) and not h


def test_calls_without_a_context_are_rejected():
    """Every call checks its context and record structs before touching a
    device: a NULL context gives OPATTR_E_INVALID_ARG (no GPU needed)."""
    import paper_2609_11938_gb300 as opa
    lib = opa.library()
    k, r, n = opa.Kernels(), opa.Ranges(), opa.Ncu()
    agg, tot, summ = opa.OpAggregates(), opa.Totals(), opa.MatchSummary()
    by = ctypes.byref
    assert lib.opattr_enclose(None, by(k), by(r), None, None) == opa.E_INVALID_ARG
    assert lib.opattr_match(None, by(k), by(n), None, None, None, by(summ)) == opa.E_INVALID_ARG
    assert lib.opattr_aggregate(None, by(k), by(r), None, by(n), None, 0, by(agg), by(tot)) == opa.E_INVALID_ARG
    assert lib.opattr_join(None, by(k), by(r), by(n), None, 0, None, None, None, None, by(agg), by(summ),
                           by(tot)) == opa.E_INVALID_ARG
    assert lib.opattr_rollup(None, by(k), by(r), None, by(n), None, 0, None, 0, by(agg)) == opa.E_INVALID_ARG


def test_binding_checks_each_array():
    """The binding refuses an array of the wrong type, one on the host or on
    another device, and a strided view, before any call; it passes the data
    pointer of a valid array and NULL for an absent or empty one."""
    import torch

    import paper_2609_11938_gb300 as opa
    host = torch.zeros(8, dtype=torch.int64)
    with pytest.raises(TypeError):
        opa._ptr(host, torch.int32, "k_start", 0)
    with pytest.raises(ValueError):
        opa._ptr(host, torch.int64, "k_start", 0)            # on the host, not on cuda:0
    assert opa._ptr(host, torch.int64, "k_start", -1) == host.data_ptr()   # the host "device" -1 matches
    with pytest.raises(ValueError):
        opa._ptr(host[::2], torch.int64, "k_start", -1)      # not contiguous
    names = torch.zeros(4, dtype=torch.int32)
    assert opa._ptr(names, torch.uint32, "k_name", -1) == names.data_ptr()    # int32 stands in for uint32
    assert opa._ptr(None, torch.int64, "k_layer", 0) is None
    assert opa._ptr(torch.zeros(0, dtype=torch.int64), torch.int64, "k_start", -1) is None
