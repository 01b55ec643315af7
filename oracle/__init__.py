"""fp64 CPU oracle for the pooled embedding-bag lookup -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py`` (its
``cpu_baseline`` leg and ``--impl reference`` arm) may import this package.
The CUDA library never calls it, and it shares no code with that library.

The arithmetic lives in ``tbe_oracle.cpp`` (plain loops in fp64, a comparison
sort for the adjoint). This module only compiles it with g++ and marshals
numpy / torch CPU arrays through ctypes.

What it computes is the standard pooled embedding bag over key-major jagged
offsets (the paper's sparse_arch lookups, Sec. IV.A.2; jagged categorical
features, Abstract) and its de-duplicated adjoint; the C++ file states the
definitions and the readings taken where the paper is silent.
"""

from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRCS = [os.path.join(_HERE, "tbe_oracle.cpp"), os.path.join(_HERE, "fm_oracle.cpp"),
         os.path.join(_HERE, "opt_oracle.cpp")]
_LIB = os.path.join(_HERE, "libtbe_oracle.so")

# Storage codes understood by the C++ file.
F32, F16, BF16 = 0, 1, 2

# Status codes returned by the C++ file.
OK, BAD_ARG, INDEX_OOB, BAD_OFFSETS = 0, 1, 2, 3
_STATUS_NAMES = {BAD_ARG: "invalid argument", INDEX_OOB: "index out of range",
                 BAD_OFFSETS: "malformed offsets"}


class OracleError(RuntimeError):
    def __init__(self, code: int):
        super().__init__(f"oracle rejected the input: {_STATUS_NAMES.get(code, code)}")
        self.code = code


def build(force: bool = False) -> str:
    """Compile the oracle with g++ (OpenMP, no FMA contraction) if it is stale."""
    if (not force and os.path.exists(_LIB)
            and all(os.path.getmtime(_LIB) >= os.path.getmtime(s) for s in _SRCS)):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["g++", "-std=c++17", "-O2", "-ffp-contract=off", "-fopenmp", "-shared", "-fPIC",
           *_SRCS, "-o", tmp]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        p, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        lib.tbe_oracle_half_to_double.argtypes = [ctypes.c_uint16]
        lib.tbe_oracle_half_to_double.restype = ctypes.c_double
        lib.tbe_oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
        lib.tbe_oracle_bf16_to_double.restype = ctypes.c_double
        lib.tbe_oracle_forward.argtypes = [i32, p, p, p, p, i32, p, i32, i64, p, p, i32, i32, p]
        lib.tbe_oracle_forward.restype = ctypes.c_int
        lib.tbe_oracle_backward_run.argtypes = [i32, p, p, i32, p, i32, i64, p, p, i32, p, i32,
                                                ctypes.POINTER(ctypes.c_int32)]
        lib.tbe_oracle_backward_run.restype = p
        lib.tbe_oracle_backward_num_unique.argtypes = [p]
        lib.tbe_oracle_backward_num_unique.restype = i64
        lib.tbe_oracle_backward_num_floats.argtypes = [p]
        lib.tbe_oracle_backward_num_floats.restype = i64
        lib.tbe_oracle_backward_fetch.argtypes = [p, p, p, p, p, p, p]
        lib.tbe_oracle_backward_fetch.restype = None
        lib.tbe_oracle_backward_free.argtypes = [p]
        lib.tbe_oracle_backward_free.restype = None
        lib.tbe_oracle_backward_dense.argtypes = [i32, p, p, i32, p, i32, i64, p, p, i32, p, p]
        lib.tbe_oracle_backward_dense.restype = ctypes.c_int
        lib.tbe_oracle_weight_grad.argtypes = [i32, p, p, p, p, i32, p, i32, i64, p, i32, p, i32, p]
        lib.tbe_oracle_weight_grad.restype = ctypes.c_int
        lib.opt_oracle_double_to_half.argtypes = [ctypes.c_double]
        lib.opt_oracle_double_to_half.restype = ctypes.c_uint16
        lib.opt_oracle_double_to_bf16.argtypes = [ctypes.c_double]
        lib.opt_oracle_double_to_bf16.restype = ctypes.c_uint16
        lib.opt_oracle_apply.argtypes = [i32, p, p, p, p, i64, p, p, p, i32, ctypes.c_double,
                                         ctypes.c_double, p]
        lib.opt_oracle_apply.restype = ctypes.c_int
        lib.fm_oracle_forward.argtypes = [i32, i32, i32, i64, p, p]
        lib.fm_oracle_forward.restype = ctypes.c_int
        lib.fm_oracle_backward.argtypes = [i32, i32, i32, i64, p, p, p]
        lib.fm_oracle_backward.restype = ctypes.c_int
        _lib = lib
    return _lib


def half_to_double(bits: int) -> float:
    return _load().tbe_oracle_half_to_double(bits)


def bf16_to_double(bits: int) -> float:
    return _load().tbe_oracle_bf16_to_double(bits)


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _table_array(x):
    """Returns (contiguous 2-D numpy array holding the stored bits, storage code)."""
    try:
        import torch
    except ImportError:  # pragma: no cover
        torch = None
    if torch is not None and isinstance(x, torch.Tensor):
        x = x.detach().cpu().contiguous()
        if x.dtype == torch.float32:
            return x.numpy(), F32
        if x.dtype == torch.float16:
            return x.numpy(), F16
        if x.dtype == torch.bfloat16:
            return x.view(torch.int16).numpy().view(np.uint16), BF16
        raise TypeError(f"unsupported table dtype {x.dtype}")
    x = np.ascontiguousarray(x)
    if x.dtype == np.float32:
        return x, F32
    if x.dtype == np.float16:
        return x, F16
    raise TypeError(f"unsupported table dtype {x.dtype}; pass bf16 tables as torch tensors")


def _np(x, dtype=None):
    if x is None:
        return None
    try:
        import torch
        if isinstance(x, torch.Tensor):
            x = x.detach().cpu().numpy()
    except ImportError:  # pragma: no cover
        pass
    x = np.ascontiguousarray(x)
    if dtype is not None and x.dtype != dtype:
        raise TypeError(f"expected {dtype}, got {x.dtype}")
    return x


def _index_arrays(indices, offsets):
    ind = _np(indices)
    off = _np(offsets)
    if ind.dtype != off.dtype or ind.dtype not in (np.int32, np.int64):
        raise TypeError("indices and offsets must both be int32 or both int64")
    return ind, off, int(ind.dtype == np.int32)


def forward(tables, batch: int, indices, offsets, weights=None, mean: bool = False,
            threads: int = 0) -> np.ndarray:
    """Pooled output [batch, sum D] in float64 (see tbe_oracle.cpp for the definition)."""
    arrs = [_table_array(t) for t in tables]
    T = len(arrs)
    rows = np.array([a.shape[0] for a, _ in arrs], dtype=np.int64)
    dims = np.array([a.shape[1] for a, _ in arrs], dtype=np.int32)
    codes = np.array([c for _, c in arrs], dtype=np.int32)
    ptrs = (ctypes.c_void_p * T)(*[a.ctypes.data for a, _ in arrs])
    ind, off, is32 = _index_arrays(indices, offsets)
    w = _np(weights, np.float32)
    out = np.zeros((batch, int(dims.sum())), dtype=np.float64)
    st = _load().tbe_oracle_forward(T, _ptr(rows), _ptr(dims), _ptr(codes),
                                    ctypes.cast(ptrs, ctypes.c_void_p), batch, _ptr(ind), is32,
                                    ind.shape[0], _ptr(off), _ptr(w), int(mean), threads, _ptr(out))
    if st != OK:
        raise OracleError(st)
    return out


def weight_grad(tables, batch: int, indices, offsets, grad_out, mean: bool = False,
                threads: int = 0) -> np.ndarray:
    """d<grad_out, y>/d w_i = s_b * <grad_out[b, Doff_t:], E_t[idx_i]>, float64 [n]."""
    arrs = [_table_array(t) for t in tables]
    T = len(arrs)
    rows = np.array([a.shape[0] for a, _ in arrs], dtype=np.int64)
    dims = np.array([a.shape[1] for a, _ in arrs], dtype=np.int32)
    codes = np.array([c for _, c in arrs], dtype=np.int32)
    ptrs = (ctypes.c_void_p * T)(*[a.ctypes.data for a, _ in arrs])
    ind, off, is32 = _index_arrays(indices, offsets)
    go = _np(grad_out, np.float32)
    out = np.zeros(ind.shape[0], dtype=np.float64)
    st = _load().tbe_oracle_weight_grad(T, _ptr(rows), _ptr(dims), _ptr(codes),
                                        ctypes.cast(ptrs, ctypes.c_void_p), batch, _ptr(ind), is32,
                                        ind.shape[0], _ptr(off), int(mean), _ptr(go), threads,
                                        _ptr(out))
    if st != OK:
        raise OracleError(st)
    return out


@dataclass
class BackwardResult:
    uniq: np.ndarray           # [U] ascending global ids row_base_t + row
    seg_start: np.ndarray      # [U + 1] run starts in the sorted order
    perm: np.ndarray           # [n] lookup positions in sorted order (stable)
    table_offsets: np.ndarray  # [T + 1]
    grad_offsets: np.ndarray   # [U + 1]
    grads: np.ndarray          # [num_floats] float64, packed D_t values per unique row

    @property
    def num_unique(self) -> int:
        return int(self.uniq.shape[0])


def backward(rows, dims, batch: int, indices, offsets, grad_out, weights=None,
             mean: bool = False, threads: int = 0) -> BackwardResult:
    """De-duplicated adjoint: one fp64 gradient row per distinct (table, row) touched."""
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    dims = np.ascontiguousarray(dims, dtype=np.int32)
    T = rows.shape[0]
    ind, off, is32 = _index_arrays(indices, offsets)
    n = ind.shape[0]
    w = _np(weights, np.float32)
    go = _np(grad_out, np.float32)
    lib = _load()
    st = ctypes.c_int32(0)
    res = lib.tbe_oracle_backward_run(T, _ptr(rows), _ptr(dims), batch, _ptr(ind), is32, n,
                                      _ptr(off), _ptr(w), int(mean), _ptr(go), threads,
                                      ctypes.byref(st))
    if not res:
        raise OracleError(st.value)
    try:
        U = lib.tbe_oracle_backward_num_unique(res)
        F = lib.tbe_oracle_backward_num_floats(res)
        out = BackwardResult(np.empty(U, np.int64), np.empty(U + 1, np.int64),
                             np.empty(n, np.int64), np.empty(T + 1, np.int64),
                             np.empty(U + 1, np.int64), np.empty(F, np.float64))
        lib.tbe_oracle_backward_fetch(res, _ptr(out.uniq), _ptr(out.seg_start), _ptr(out.perm),
                                      _ptr(out.table_offsets), _ptr(out.grad_offsets),
                                      _ptr(out.grads))
    finally:
        lib.tbe_oracle_backward_free(res)
    return out


def backward_dense(rows, dims, batch: int, indices, offsets, grad_out, weights=None,
                   mean: bool = False) -> list[np.ndarray]:
    """Dense adjoint dE_t [rows_t, D_t] in float64, by direct scatter-add (no sort)."""
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    dims = np.ascontiguousarray(dims, dtype=np.int32)
    T = rows.shape[0]
    ind, off, is32 = _index_arrays(indices, offsets)
    w = _np(weights, np.float32)
    go = _np(grad_out, np.float32)
    dense = [np.zeros((int(r), int(d)), dtype=np.float64) for r, d in zip(rows, dims)]
    ptrs = (ctypes.c_void_p * T)(*[a.ctypes.data for a in dense])
    st = _load().tbe_oracle_backward_dense(T, _ptr(rows), _ptr(dims), batch, _ptr(ind), is32,
                                           ind.shape[0], _ptr(off), _ptr(w), int(mean), _ptr(go),
                                           ctypes.cast(ptrs, ctypes.c_void_p))
    if st != OK:
        raise OracleError(st)
    return dense


# ----------------------------------------------------------------------------- FM cross term

def _fm_input(y, num_fields: int):
    y = _np(y, np.float32)
    if y.ndim != 2 or num_fields <= 0 or y.shape[1] % num_fields:
        raise ValueError("y must be [B, T * D] with T = num_fields")
    return y, y.shape[0], y.shape[1] // num_fields


def fm_forward(y, num_fields: int, threads: int = 0) -> np.ndarray:
    """fm[b] = sum over field pairs t < u of <v_bt, v_bu> in float64 (fm_oracle.cpp)."""
    y, B, D = _fm_input(y, num_fields)
    out = np.zeros(B, dtype=np.float64)
    st = _load().fm_oracle_forward(B, num_fields, D, y.shape[1], _ptr(y), _ptr(out))
    if st != OK:
        raise OracleError(st)
    return out


def fm_backward(y, grad_fm, num_fields: int) -> np.ndarray:
    """grad_y[b, t*D + j] = g[b] * sum over u != t of y[b, u*D + j], float64 [B, T*D]."""
    y, B, D = _fm_input(y, num_fields)
    g = _np(grad_fm, np.float32)
    if g.shape != (B,):
        raise ValueError("grad_fm must be [B]")
    out = np.zeros((B, num_fields * D), dtype=np.float64)
    st = _load().fm_oracle_backward(B, num_fields, D, y.shape[1], _ptr(y), _ptr(g), _ptr(out))
    if st != OK:
        raise OracleError(st)
    return out


# ----------------------------------------------------------------------------- optimizer step

OPTIMIZERS = {"sgd": 0, "adagrad": 1}


def double_to_half_bits(x: float) -> int:
    return int(_load().opt_oracle_double_to_half(float(x)))


def double_to_bf16_bits(x: float) -> int:
    return int(_load().opt_oracle_double_to_bf16(float(x)))


def apply_step(tables, batch: int, indices, offsets, grad_out, weights=None, mean: bool = False,
               kind: str = "sgd", lr: float = 0.01, eps: float = 1e-8, state=None):
    """One optimizer step on the rows the batch touches (opt_oracle.cpp).

    Returns (new tables as torch CPU tensors of the input dtypes, new state as
    a list of float32 numpy arrays or None). The inputs are not modified.
    """
    import torch
    arrs = [_table_array(t) for t in tables]
    work = [a.copy() for a, _ in arrs]
    T = len(work)
    rows = np.array([a.shape[0] for a in work], dtype=np.int64)
    dims = np.array([a.shape[1] for a in work], dtype=np.int32)
    codes = np.array([c for _, c in arrs], dtype=np.int32)
    res = backward(rows, dims, batch, indices, offsets, grad_out, weights=weights, mean=mean)
    uniq = np.ascontiguousarray(res.uniq, dtype=np.int64)
    goff = np.ascontiguousarray(res.grad_offsets, dtype=np.int64)
    grads = np.ascontiguousarray(res.grads, dtype=np.float64)
    st = None
    st_ptrs = None
    if kind == "adagrad":
        st = [np.ascontiguousarray(_np(s_, np.float32)).copy() for s_ in state]
        st_ptrs = (ctypes.c_void_p * T)(*[a.ctypes.data for a in st])
    tab_ptrs = (ctypes.c_void_p * T)(*[a.ctypes.data for a in work])
    rc = _load().opt_oracle_apply(T, ctypes.cast(tab_ptrs, ctypes.c_void_p), _ptr(codes), _ptr(dims),
                                  _ptr(rows), uniq.shape[0], _ptr(uniq), _ptr(goff), _ptr(grads),
                                  OPTIMIZERS[kind], float(lr), float(eps),
                                  None if st_ptrs is None else ctypes.cast(st_ptrs, ctypes.c_void_p))
    if rc != 0:
        raise OracleError(BAD_ARG)
    out = []
    for a, (_, code) in zip(work, arrs):
        if code == BF16:
            out.append(torch.from_numpy(a.view(np.int16)).view(torch.bfloat16))
        else:
            out.append(torch.from_numpy(a))
    return out, st


# ----------------------------------------------------------------------------- batch replication

def replicate_kjt(indices, offsets, weights, num_tables: int, factor: int):
    """The batch-size preprocessor (Sec. III): a captured batch of B bags per table,
    replicated to factor * B bags per table in the same key-major layout. Bag
    r * B + b of table t (r < factor) is bag b of table t. Plain loops over bags.
    Returns (indices, offsets, weights or None) as numpy arrays."""
    ind = _np(indices)
    off = _np(offsets)
    w = None if weights is None else _np(weights, np.float32)
    T = num_tables
    B = (off.shape[0] - 1) // T
    out_ind, out_w, out_off = [], [], [0]
    for t in range(T):
        for r in range(factor):
            for b in range(B):
                s, e = int(off[t * B + b]), int(off[t * B + b + 1])
                out_ind.extend(ind[s:e].tolist())
                if w is not None:
                    out_w.extend(w[s:e].tolist())
                out_off.append(out_off[-1] + (e - s))
    return (np.array(out_ind, dtype=ind.dtype), np.array(out_off, dtype=off.dtype),
            None if w is None else np.array(out_w, dtype=np.float32))
