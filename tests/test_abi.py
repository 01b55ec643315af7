"""The C-ABI library builds, loads and exports every entry point of include/cb_tbe.h (CPU)."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    with open(os.path.join(ROOT, "include", "cb_tbe.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(cb_(?:tbe|fm|kjt|gather)_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_30656_gb300 import build, tbe
    build.build()
    return tbe.load_library()


def test_header_declares_the_expected_entry_points():
    from paper_2609_30656_gb300 import tbe
    assert _declared_functions() == sorted(tbe.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in _declared_functions():
        assert hasattr(lib, name), name


def test_status_strings_and_component_names(lib):
    from paper_2609_30656_gb300 import tbe
    assert lib.cb_tbe_status_string(0) == b"ok"
    assert lib.cb_tbe_status_string(7) == b"bounded device wait timed out"
    assert tbe.component_names() == ["fwd.prep", "fwd.gather", "fwd.fixup", "bwd.keygen",
                                     "bwd.sort", "bwd.rle", "bwd.reduce"]


def test_host_side_argument_errors_return_before_any_gpu_work(lib):
    from paper_2609_30656_gb300 import tbe
    h = ctypes.c_void_p()
    # null descriptor array / zero tables / null out pointer
    assert lib.cb_tbe_create(None, 1, 0, 1, 0, ctypes.byref(h)) == tbe.CB_ERR_INVALID_ARG
    descs = (tbe.CbTableDesc * 1)(tbe.CbTableDesc(None, 0, 16, 0))
    assert lib.cb_tbe_create(descs, 0, 0, 1, 0, ctypes.byref(h)) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_tbe_create(descs, 1, 0, 1, 0, None) == tbe.CB_ERR_INVALID_ARG
    # bad pooling / index dtype / storage dtype / row size not a multiple of 16 bytes
    assert lib.cb_tbe_create(descs, 1, 5, 1, 0, ctypes.byref(h)) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_tbe_create(descs, 1, 0, 7, 0, ctypes.byref(h)) == tbe.CB_ERR_INVALID_ARG
    bad = (tbe.CbTableDesc * 1)(tbe.CbTableDesc(None, 0, 16, 9))
    assert lib.cb_tbe_create(bad, 1, 0, 1, 0, ctypes.byref(h)) == tbe.CB_ERR_INVALID_ARG
    odd = (tbe.CbTableDesc * 1)(tbe.CbTableDesc(None, 0, 6, 1))  # 12-byte fp16 rows
    assert lib.cb_tbe_create(odd, 1, 0, 1, 0, ctypes.byref(h)) == tbe.CB_ERR_INVALID_ARG
    wide = (tbe.CbTableDesc * 1)(tbe.CbTableDesc(None, 0, 1024, 1))  # dim > 512
    assert lib.cb_tbe_create(wide, 1, 0, 1, 0, ctypes.byref(h)) == tbe.CB_ERR_INVALID_ARG
    unaligned = (tbe.CbTableDesc * 1)(tbe.CbTableDesc(8, 10, 16, 0))
    assert lib.cb_tbe_create(unaligned, 1, 0, 1, 0, ctypes.byref(h)) == tbe.CB_ERR_INVALID_ARG
    # calls on a null handle
    assert lib.cb_tbe_forward(None, 1, None, 0, None, None, None, None) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_tbe_backward(None, 1, None, 0, None, None, None, None, None) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_tbe_get_error(None) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_tbe_reserve(None, 1, 1) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_tbe_launch_count(None) == 0
    lib.cb_tbe_destroy(None)
    # the FM cross term: null buffers, a dim that is not a multiple of 4, no fields
    assert lib.cb_fm_forward(None, 1, 2, 8, 16, None, None) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_fm_forward(None, 0, 2, 6, 12, None, None) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_fm_backward(None, None, 0, 0, 8, 0, None, None) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_fm_backward(None, None, 4, 2, 8, 12, None, None) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_fm_forward(None, 0, 2, 8, 16, None, None) == tbe.CB_OK  # nothing to do
    # batch replication: factor < 1, null offsets
    assert lib.cb_kjt_replicate(None, None, None, 1, 2, 4, 0, 2, None, None, None, None) == tbe.CB_ERR_INVALID_ARG
    # weight gradient and the fused optimizer step on a null handle
    assert lib.cb_tbe_weight_grad(None, 1, None, 0, None, None, None, None) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_tbe_backward_apply(None, 1, None, 0, None, None, None, 0, 0.1, 0.0, None,
                                     None) == tbe.CB_ERR_INVALID_ARG
    assert lib.cb_tbe_apply_sparse(None, None, 0, 0.1, 0.0, None, None) == tbe.CB_ERR_INVALID_ARG


def test_product_path_fails_loudly_without_the_library(monkeypatch, tmp_path):
    from paper_2609_30656_gb300 import tbe
    monkeypatch.setattr(tbe, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(tbe, "_lib", None)
    with pytest.raises(RuntimeError, match="missing"):
        tbe.load_library()


def test_noalloc_refuses_sizes_that_would_wrap_the_scratch_layout(lib):
    # num_indices near 2^63: the chunk count alone exceeds the static scratch, so the
    # call is refused on the host before any size product can wrap around (and
    # before any pointer is touched: these are fake, aligned addresses).
    from paper_2609_30656_gb300 import tbe
    f = lib.cb_tbe_forward_noalloc
    p, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    f.argtypes = [p, i32, ctypes.c_int, ctypes.c_int, i32, p, i64, p, p, p, p]
    f.restype = ctypes.c_int
    descs = (tbe.CbTableDesc * 1)(tbe.CbTableDesc(4096, 10, 512, 0))
    for n in (2**63 - 1, 2**62, 2**40):
        assert f(descs, 1, 0, 1, 1, p(4096), n, p(8192), None, p(12288), None) == tbe.CB_ERR_CAPACITY


def test_create_refuses_a_key_space_beyond_32_bits(lib):
    # Every table's rows plus one spare key per table must stay below 2^32.
    from paper_2609_30656_gb300 import tbe
    h = ctypes.c_void_p()
    descs = (tbe.CbTableDesc * 2)(tbe.CbTableDesc(4096, 2**31, 4, 0), tbe.CbTableDesc(4096, 2**31 - 2, 4, 0))
    assert lib.cb_tbe_create(descs, 2, 0, 1, 0, ctypes.byref(h)) == tbe.CB_ERR_INVALID_ARG


@pytest.mark.parametrize("name", ["cb_gather_ceiling", "cb_gather_ceiling_f16"])
def test_gather_ceiling_rejects_bad_sizes_on_the_host(lib, name):
    from paper_2609_30656_gb300 import tbe
    p = ctypes.c_void_p
    f = getattr(lib, name)
    assert f(p(4096), 100, 96, p(8192), 64, p(12288), None) == tbe.CB_ERR_INVALID_ARG  # row size
    assert f(p(4100), 100, 512, p(8192), 64, p(12288), None) == tbe.CB_ERR_INVALID_ARG  # alignment
    assert f(p(4096), 0, 512, p(8192), 64, p(12288), None) == tbe.CB_ERR_INVALID_ARG  # no rows
    assert f(p(4096), 100, 512, None, 64, p(12288), None) == tbe.CB_ERR_INVALID_ARG  # no indices
    assert f(p(4096), 100, 512, None, 0, None, None) == tbe.CB_OK  # nothing to do


def test_tma_gather_ceiling_rejects_bad_sizes_on_the_host(lib):
    from paper_2609_30656_gb300 import tbe
    p = ctypes.c_void_p
    f = lib.cb_gather_ceiling_tma
    assert f(p(4096), 100, 128, p(8192), 64, p(12288), p(16384), None) == tbe.CB_ERR_INVALID_ARG  # row size
    assert f(p(4096), 2**31, 512, p(8192), 64, p(12288), p(16384), None) == tbe.CB_ERR_INVALID_ARG  # rows
    assert f(p(4096), 100, 512, p(8192), 64, p(12288), None, None) == tbe.CB_ERR_INVALID_ARG  # no error word
    assert f(p(4096), 100, 512, None, 0, None, p(16384), None) == tbe.CB_OK  # nothing to do
