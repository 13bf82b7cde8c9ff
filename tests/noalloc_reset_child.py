"""Child process of test_zz_no_alloc.py: the no-allocation matching entry
point before and after a device reset, in a process that does not load torch
(device memory through the CUDA runtime, by ctypes).  Prints "noalloc reset
ok" and exits 0 when both calls equal opattr_match and the oracle."""
import ctypes
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import paper_2609_11938_gb300 as opa  # noqa: E402
import tracegen  # noqa: E402

lib = opa.library()
rt = ctypes.CDLL("libcudart.so.13")       # the runtime libopattr.so already loaded
vp = ctypes.c_void_p
rt.cudaMalloc.argtypes = [ctypes.POINTER(vp), ctypes.c_size_t]
rt.cudaFree.argtypes = [vp]
rt.cudaMemcpy.argtypes = [vp, vp, ctypes.c_size_t, ctypes.c_int]
rt.cudaSetDevice.argtypes = [ctypes.c_int]
H2D, D2H = 1, 2


def check(rc, what):
    if rc != 0:
        print(f"{what} failed: {rc}")
        sys.exit(1)


class Dev:
    """Device copies of the arrays the matching reads, and its outputs."""

    def __init__(self, t):
        self.bufs = []
        self.k_stream, self.k_start, self.k_name = (self.up(a) for a in (t.k_stream, t.k_start, t.k_name))
        self.ncu_name = self.up(t.ncu_name)
        self.idx = self.alloc(4 * t.K)
        self.kind = self.alloc(t.K)
        self.K, self.M = t.K, t.M

    def alloc(self, n):
        p = vp()
        check(rt.cudaMalloc(ctypes.byref(p), max(n, 1)), "cudaMalloc")
        self.bufs.append(p)
        return p

    def up(self, a):
        a = np.ascontiguousarray(a)
        p = self.alloc(a.nbytes)
        check(rt.cudaMemcpy(p, a.ctypes.data, a.nbytes, H2D), "cudaMemcpy H2D")
        return p

    def down(self):
        idx = np.empty(self.K, np.int32)
        kind = np.empty(self.K, np.uint8)
        check(rt.cudaMemcpy(idx.ctypes.data, self.idx, idx.nbytes, D2H), "cudaMemcpy D2H")
        check(rt.cudaMemcpy(kind.ctypes.data, self.kind, kind.nbytes, D2H), "cudaMemcpy D2H")
        return idx, kind

    def structs(self):
        return (opa.Kernels(self.k_stream.value, self.k_start.value, None, self.k_name.value, None, self.K),
                opa.Ncu(self.ncu_name.value, None, self.M, None))

    def free(self):
        for p in self.bufs:
            rt.cudaFree(p)


def noalloc(d, mode):
    k, n = d.structs()
    s = opa.MatchSummary()
    st = opa.opattr_match_noalloc(k, n, mode, d.idx.value, d.kind.value, s, None)
    return (st,) + d.down()


def main():
    mode = "skip_name"
    t = tracegen.small_random(5, n_streams=3, n_events=600, max_depth=5, shuffle=True, n_names=7)
    t.ncu_name = t.ncu_name[2:].copy()
    st_o, idx_o, kind_o, _ = oracle.match(t.k_stream, t.k_start, t.k_name, t.ncu_name, mode=mode)
    check(rt.cudaSetDevice(0), "cudaSetDevice")
    d = Dev(t)
    # the context entry point, for reference
    st_c, h = opa.opattr_create(0, None, mismatch=mode)
    check(st_c, "opattr_create")
    k, n = d.structs()
    st_ref = opa.opattr_match(h, k, n, None, d.idx.value, d.kind.value, opa.MatchSummary())
    idx_ref, kind_ref = d.down()
    opa.opattr_destroy(h)
    for _ in range(2):
        st, idx, kind = noalloc(d, mode)
        assert st == st_ref == st_o, (st, st_ref, st_o)
        assert (idx == idx_ref).all() and (idx == idx_o).all() and (kind == kind_o).all()
    d.free()
    check(rt.cudaDeviceReset(), "cudaDeviceReset")      # ends this process's own context only
    check(rt.cudaSetDevice(0), "cudaSetDevice")
    d = Dev(t)
    for _ in range(2):
        st, idx, kind = noalloc(d, mode)
        assert st == st_o, (st, st_o)
        assert (idx == idx_o).all() and (kind == kind_o).all()
    d.free()
    print("noalloc reset ok")


if __name__ == "__main__":
    main()
