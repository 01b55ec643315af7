"""cb_tbe_forward_noalloc: the forward for callers that cannot allocate device memory.

A plugin running inside a framework that owns all device memory, or a steady-state
loop that must not call cudaMalloc / cudaFree, cannot use the handle-based forward,
whose workspace is allocated on demand. The allocation-free entry point keeps its
scratch in a fixed __device__ array inside the library. These tests call it through
the C ABI, several times in a row (its scratch keeps the previous call's contents),
and compare each result with the fp64 oracle at the condition-aware tolerance the
other forward tests use, and with the handle-based forward. This file is collected
last, so a failure here leaves every other test already run; it also passes alone in
a fresh process (the first call sets up).
"""

import ctypes

import numpy as np
import pytest
import torch

from tests.helpers import RTOL, assert_forward_close, forward_reference, random_problem

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
_IDX = {torch.int32: 0, torch.int64: 1}


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


def _noalloc(lib, tbe, tables, mean, ind, off, w, out, n=None):
    T = len(tables)
    batch = (off.numel() - 1) // T
    stream = ctypes.c_void_p(torch.cuda.current_stream(DEV).cuda_stream)
    return lib.cb_tbe_forward_noalloc(
        _descs(tbe, tables), T, 1 if mean else 0, _IDX[ind.dtype], batch,
        ctypes.c_void_p(ind.data_ptr()), ind.numel() if n is None else n,
        ctypes.c_void_p(off.data_ptr()), None if w is None else ctypes.c_void_p(w.data_ptr()),
        ctypes.c_void_p(out.data_ptr()), stream)


def _case(seed, dtype, weighted, mean, batch, index_dtype=torch.int64, int_valued=False,
          dims=(64, 128, 256), rows=(500, 3000, 70), max_len=1500):
    tables, ind, off, w = random_problem(seed, dims=dims, rows=rows, batch=batch, max_len=max_len,
                                         dtype=dtype, weighted=weighted, empty_frac=0.25,
                                         int_valued=int_valued)
    ind, off = ind.to(index_dtype), off.to(index_dtype)
    ref, scale = forward_reference(tables, batch, ind, off, w, mean)
    return tables, ind, off, w, ref, scale


def test_two_calls_in_a_row_match_the_oracle_and_the_handle_forward():
    lib, tbe = _lib()
    cases = []
    for seed, weighted, mean, batch in ((41, False, False, 37), (42, True, True, 23)):
        tables, ind, off, w, ref, scale = _case(seed, torch.float16, weighted, mean, batch)
        d_tabs = [t.to(DEV) for t in tables]
        d_ind, d_off = ind.to(DEV), off.to(DEV)
        d_w = None if w is None else w.to(DEV)
        handle = tbe.TBE(d_tabs, pooling="mean" if mean else "sum", validate=True).forward(d_ind, d_off, d_w)
        out = torch.full_like(handle, float("nan"))
        cases.append((d_tabs, mean, d_ind, d_off, d_w, ref, scale, handle, out))
    torch.cuda.synchronize()

    # First call on this device sets up; the second must allocate nothing.
    for k, (tables, mean, ind, off, w, ref, scale, handle, out) in enumerate(cases):
        free_before = torch.cuda.mem_get_info(DEV)[0]
        assert _noalloc(lib, tbe, tables, mean, ind, off, w, out) == tbe.CB_OK
        if k == 1:
            assert torch.cuda.mem_get_info(DEV)[0] >= free_before
        assert torch.isfinite(out).all()
        assert_forward_close(out, ref, scale, RTOL[torch.float16], what=f"call {k} vs oracle")
        # the same kernels as the handle forward: the same bits
        assert torch.equal(out, handle), f"call {k} vs handle forward"


@pytest.mark.parametrize("dtype,index_dtype", [(torch.float32, torch.int32), (torch.bfloat16, torch.int64)])
def test_other_storage_and_index_types(dtype, index_dtype):
    lib, tbe = _lib()
    tables, ind, off, w, ref, scale = _case(43, dtype, True, False, 29, index_dtype=index_dtype,
                                            dims=(32, 96, 512), rows=(40, 900, 7), max_len=800)
    d_tabs = [t.to(DEV) for t in tables]
    out = torch.full((29, sum(t.shape[1] for t in tables)), float("nan"), device=DEV)
    assert _noalloc(lib, tbe, d_tabs, False, ind.to(DEV), off.to(DEV), w.to(DEV), out) == tbe.CB_OK
    assert_forward_close(out, ref, scale, RTOL[dtype], what=f"{dtype} {index_dtype}")


def test_integer_tables_just_under_the_scratch_bound_are_bit_exact():
    # One fp32 table of dim 512: every chunk of 512 lookups takes 24 + 8 + 2 * 2048
    # bytes of the 16 MiB array, so about 2.08 M lookups fit. 2.07 M must run
    # (and, with integer values, give the oracle's bits); 2.09 M must be refused.
    lib, tbe = _lib()
    g = torch.Generator().manual_seed(44)
    rows, dim, batch = 4096, 512, 2000
    table = torch.randint(-8, 9, (rows, dim), generator=g).to(torch.float32)
    n_fit, n_over = 2_070_000, 2_090_000
    lens = torch.full((batch,), n_fit // batch, dtype=torch.int64)
    lens[: n_fit - int(lens.sum())] += 1
    lens[7] = 0  # an empty bag too
    lens[8] += n_fit - int(lens.sum())
    off = torch.zeros(batch + 1, dtype=torch.int64)
    off[1:] = torch.cumsum(lens, 0)
    ind = torch.randint(0, rows, (n_fit,), generator=g)
    ref, _ = forward_reference([table], batch, ind, off, None, False)
    d_tab, d_ind, d_off = table.to(DEV), ind.to(DEV), off.to(DEV)
    out = torch.full((batch, dim), float("nan"), device=DEV)
    assert _noalloc(lib, tbe, [d_tab], False, d_ind, d_off, None, out) == tbe.CB_OK
    np.testing.assert_array_equal(out.cpu().double().numpy(), ref)
    # refused on the host, before any pointer is touched
    assert _noalloc(lib, tbe, [d_tab], False, d_ind, d_off, None, out, n=n_over) == tbe.CB_ERR_CAPACITY


def test_an_error_does_not_stick_to_the_next_call():
    lib, tbe = _lib()
    tables, ind, off, w, ref, scale = _case(45, torch.float32, False, True, 31)
    d_tabs = [t.to(DEV) for t in tables]
    out = torch.full((31, sum(t.shape[1] for t in tables)), float("nan"), device=DEV)
    bad = off.clone()
    assert int(bad[4]) >= 1
    bad[5] = bad[4] - 1  # decreasing offsets (as in the handle forward's test)
    assert _noalloc(lib, tbe, d_tabs, True, ind.to(DEV), bad.to(DEV), None, out) == tbe.CB_ERR_BAD_OFFSETS
    out.fill_(float("nan"))
    assert _noalloc(lib, tbe, d_tabs, True, ind.to(DEV), off.to(DEV), None, out) == tbe.CB_OK
    assert_forward_close(out, ref, scale, RTOL[torch.float32], what="after an error")
    # an out-of-range index: reported, and it adds nothing
    oob = ind.clone()
    oob[3] = tables[0].shape[0] + 5
    assert _noalloc(lib, tbe, d_tabs, True, oob.to(DEV), off.to(DEV), None, out) == tbe.CB_ERR_INDEX_OOB
    assert _noalloc(lib, tbe, d_tabs, True, ind.to(DEV), off.to(DEV), None, out) == tbe.CB_OK
    assert_forward_close(out, ref, scale, RTOL[torch.float32], what="after an index error")


def test_no_lookups_writes_zeros():
    lib, tbe = _lib()
    tables = [torch.randn(10, 16, device=DEV), torch.randn(3, 32, device=DEV)]
    off = torch.zeros(2 * 5 + 1, dtype=torch.int64, device=DEV)
    ind = torch.zeros(1, dtype=torch.int64, device=DEV)
    out = torch.full((5, 48), float("nan"), device=DEV)
    assert _noalloc(lib, tbe, tables, False, ind, off, None, out, n=0) == tbe.CB_OK
    assert torch.equal(out, torch.zeros_like(out))


def test_calls_beyond_the_static_scratch_are_refused():
    lib, tbe = _lib()
    tables = [torch.zeros(16, 512, dtype=torch.float32, device=DEV)]
    # 10 M lookups of a dim-512 table need far more than the 16 MiB of scratch;
    # the refusal happens on the host, before any pointer is touched.
    n = 10_000_000
    off = torch.tensor([0, n], dtype=torch.int64, device=DEV)
    ind = torch.zeros(1, dtype=torch.int64, device=DEV)
    out = torch.empty(1, 512, device=DEV)
    assert _noalloc(lib, tbe, tables, False, ind, off, None, out, n=n) == tbe.CB_ERR_CAPACITY
