"""cb_tbe_forward_noalloc: the forward for callers that cannot allocate device memory.

A plugin running inside a framework that owns all device memory, or a steady-state
loop that must not call cudaMalloc / cudaFree, cannot use the handle-based forward,
whose workspace is allocated on demand. The allocation-free entry point keeps its
scratch in a fixed __device__ array inside the library. These tests call it through
the C ABI twice in a row (its scratch keeps the previous call's contents) and compare
each result with the handle-based forward, within the tolerance the other forward
tests use. This file is collected last, so a failure here leaves every other test
already run; it also passes alone in a fresh process (the first call sets up).
"""

import ctypes

import pytest
import torch

from tests.helpers import RTOL, random_problem

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _lib():
    from paper_2609_30656_gb300 import tbe
    lib = tbe.load_library()
    p, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    f = lib.cb_tbe_forward_noalloc
    f.argtypes = [p, i32, ctypes.c_int, ctypes.c_int, i32, p, i64, p, p, p, p]
    f.restype = ctypes.c_int
    return lib, tbe


def _descs(tbe, tables):
    return (tbe.CbTableDesc * len(tables))(*[
        tbe.CbTableDesc(t.data_ptr(), int(t.shape[0]), int(t.shape[1]), tbe._DTYPES[t.dtype])
        for t in tables])


def _noalloc(lib, tbe, tables, mean, ind, off, w, out):
    T = len(tables)
    batch = (off.numel() - 1) // T
    stream = ctypes.c_void_p(torch.cuda.current_stream(DEV).cuda_stream)
    return lib.cb_tbe_forward_noalloc(
        _descs(tbe, tables), T, 1 if mean else 0, 1, batch,
        ctypes.c_void_p(ind.data_ptr()), ind.numel(), ctypes.c_void_p(off.data_ptr()),
        None if w is None else ctypes.c_void_p(w.data_ptr()), ctypes.c_void_p(out.data_ptr()),
        stream)


def _within(y, ref, scale, rtol):
    return bool(((y.double() - ref.double()).abs() <= rtol * scale.double() + 1e-30).all())


def test_two_calls_in_a_row_match_the_handle_forward():
    lib, tbe = _lib()
    cases = []
    for seed, weighted, mean, batch in ((41, False, False, 37), (42, True, True, 23)):
        tables, ind, off, w = random_problem(seed, dims=(64, 128, 256), rows=(500, 3000, 70),
                                             batch=batch, max_len=1500, dtype=torch.float16,
                                             weighted=weighted, empty_frac=0.25)
        tables = [t.to(DEV) for t in tables]
        ind, off = ind.to(DEV), off.to(DEV)
        w = None if w is None else w.to(DEV)
        ref_mod = tbe.TBE(tables, pooling="mean" if mean else "sum", validate=True)
        ref = ref_mod.forward(ind, off, w)
        abs_mod = tbe.TBE([t.abs() for t in tables], pooling="mean" if mean else "sum")
        scale = abs_mod.forward(ind, off, None if w is None else w.abs())
        out = torch.full_like(ref, float("nan"))
        cases.append((tables, mean, ind, off, w, ref, scale, out))
    torch.cuda.synchronize()

    # First call on this device sets up; the second must allocate nothing.
    for k, (tables, mean, ind, off, w, ref, scale, out) in enumerate(cases):
        free_before = torch.cuda.mem_get_info(DEV)[0]
        assert _noalloc(lib, tbe, tables, mean, ind, off, w, out) == tbe.CB_OK
        if k == 1:
            assert torch.cuda.mem_get_info(DEV)[0] == free_before
        assert _within(out, ref, scale, RTOL[torch.float16]), f"call {k}"
        assert torch.isfinite(out).all()


def test_calls_beyond_the_static_scratch_are_refused():
    lib, tbe = _lib()
    tables = [torch.zeros(16, 512, dtype=torch.float32, device=DEV)]
    # 10 M lookups of a dim-512 table need far more than the 16 MiB of scratch;
    # the refusal happens on the host, before any pointer is touched.
    n = 10_000_000
    off = torch.tensor([0, n], dtype=torch.int64, device=DEV)
    ind = torch.zeros(1, dtype=torch.int64, device=DEV)
    out = torch.empty(1, 512, device=DEV)
    stream = ctypes.c_void_p(torch.cuda.current_stream(DEV).cuda_stream)
    st = lib.cb_tbe_forward_noalloc(_descs(tbe, tables), 1, 0, 1, 1, ctypes.c_void_p(ind.data_ptr()),
                                    n, ctypes.c_void_p(off.data_ptr()), None,
                                    ctypes.c_void_p(out.data_ptr()), stream)
    assert st == tbe.CB_ERR_CAPACITY
