"""Python binding of the C ABI in include/cb_tbe.h (ctypes; argument marshalling only).

Every step of the lookup and its backward runs in the CUDA kernels of
libcb_tbe.so. PyTorch supplies device memory and the current stream. Host
(CPU) tensors passed to ``forward`` / ``backward`` are copied to the device on
the current stream first, which is how an end-to-end caller feeds a batch from
pinned host memory.
"""

from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libcb_tbe.so")

CB_OK, CB_ERR_INVALID_ARG, CB_ERR_INDEX_OOB, CB_ERR_BAD_OFFSETS = 0, 1, 2, 3
CB_ERR_CAPACITY, CB_ERR_OOM, CB_ERR_CUDA, CB_ERR_TIMEOUT = 4, 5, 6, 7
CB_VALIDATE, CB_TIMING, CB_DEBUG_FORCE_LOOKBACK_TIMEOUT, CB_SORT_LOOKBACK = 0x1, 0x2, 0x100, 0x200
CB_OUT_F16, CB_OUT_BF16 = 0x4, 0x8
_OUT_FLAGS = {torch.float32: 0, torch.float16: CB_OUT_F16, torch.bfloat16: CB_OUT_BF16}
_DTYPES = {torch.float32: 0, torch.float16: 1, torch.bfloat16: 2}
_POOL = {"sum": 0, "mean": 1}
_IDX = {torch.int32: 0, torch.int64: 1}

# Every entry point declared in include/cb_tbe.h.
EXPORTS = ("cb_tbe_create", "cb_tbe_reserve", "cb_tbe_forward", "cb_tbe_backward",
           "cb_tbe_get_error", "cb_tbe_last_timings", "cb_tbe_component_name",
           "cb_tbe_launch_count", "cb_tbe_status_string", "cb_tbe_destroy",
           "cb_tbe_forward_noalloc", "cb_fm_forward", "cb_fm_backward", "cb_tbe_weight_grad",
           "cb_tbe_backward_apply", "cb_tbe_apply_sparse", "cb_kjt_replicate",
           "cb_tbe_sorted_payloads", "cb_gather_ceiling", "cb_gather_ceiling_f16", "cb_gather_ceiling_tma")


class CbTableDesc(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("rows", ctypes.c_int64), ("dim", ctypes.c_int32),
                ("dtype", ctypes.c_int)]


class CbSparseGrad(ctypes.Structure):
    _fields_ = [("unique_ids", ctypes.c_void_p), ("table_offsets", ctypes.c_void_p),
                ("grad_offsets", ctypes.c_void_p), ("grads", ctypes.c_void_p),
                ("cap_rows", ctypes.c_int64), ("cap_floats", ctypes.c_int64),
                ("num_unique", ctypes.c_void_p), ("num_floats", ctypes.c_void_p)]


class CbTbeError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        msg = _lib_status_string(status)
        super().__init__(f"{what}: {msg} (status {status})" if what else f"{msg} (status {status})")
        self.status = status


_lib = None


def load_library() -> ctypes.CDLL:
    """Loads libcb_tbe.so; fails loudly when it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"CUDA library {LIB_PATH} is missing; build it with "
                           "`python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(LIB_PATH)
    p, i32, i64, u32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32
    lib.cb_tbe_create.argtypes = [p, i32, ctypes.c_int, ctypes.c_int, u32, ctypes.POINTER(p)]
    lib.cb_tbe_reserve.argtypes = [p, i32, i64]
    lib.cb_tbe_forward.argtypes = [p, i32, p, i64, p, p, p, p]
    lib.cb_tbe_backward.argtypes = [p, i32, p, i64, p, p, p, ctypes.POINTER(CbSparseGrad), p]
    lib.cb_tbe_get_error.argtypes = [p]
    lib.cb_tbe_last_timings.argtypes = [p, ctypes.POINTER(ctypes.c_float), i32]
    lib.cb_tbe_component_name.argtypes = [i32]
    lib.cb_tbe_component_name.restype = ctypes.c_char_p
    lib.cb_tbe_launch_count.argtypes = [p]
    lib.cb_tbe_launch_count.restype = ctypes.c_uint64
    lib.cb_tbe_status_string.argtypes = [ctypes.c_int]
    lib.cb_tbe_status_string.restype = ctypes.c_char_p
    lib.cb_tbe_destroy.argtypes = [p]
    lib.cb_tbe_destroy.restype = None
    lib.cb_tbe_weight_grad.argtypes = [p, i32, p, i64, p, p, p, p]
    lib.cb_tbe_backward_apply.argtypes = [p, i32, p, i64, p, p, p, ctypes.c_int, ctypes.c_float,
                                          ctypes.c_float, p, p]
    lib.cb_tbe_apply_sparse.argtypes = [p, ctypes.POINTER(CbSparseGrad), ctypes.c_int, ctypes.c_float,
                                        ctypes.c_float, p, p]
    lib.cb_kjt_replicate.argtypes = [p, p, p, ctypes.c_int, i32, i32, i64, i32, p, p, p, p]
    lib.cb_tbe_sorted_payloads.argtypes = [p, p, i64, p]
    lib.cb_gather_ceiling.argtypes = [p, i64, i32, p, i64, p, p]
    lib.cb_gather_ceiling_f16.argtypes = [p, i64, i32, p, i64, p, p]
    lib.cb_gather_ceiling_tma.argtypes = [p, i64, i32, p, i64, p, p, p]
    lib.cb_fm_forward.argtypes = [p, i32, i32, i32, i64, p, p]
    lib.cb_fm_backward.argtypes = [p, p, i32, i32, i32, i64, p, p]
    for name in ("cb_tbe_create", "cb_tbe_reserve", "cb_tbe_forward", "cb_tbe_backward",
                 "cb_tbe_get_error", "cb_tbe_last_timings", "cb_fm_forward", "cb_fm_backward",
                 "cb_tbe_weight_grad", "cb_tbe_backward_apply", "cb_kjt_replicate",
                 "cb_tbe_sorted_payloads", "cb_gather_ceiling", "cb_gather_ceiling_f16", "cb_gather_ceiling_tma"):
        getattr(lib, name).restype = ctypes.c_int
    _lib = lib
    return lib


def _lib_status_string(status: int) -> str:
    try:
        return load_library().cb_tbe_status_string(status).decode()
    except Exception:  # pragma: no cover - library missing
        return f"status {status}"


def component_names() -> list[str]:
    lib = load_library()
    names, i = [], 0
    while True:
        s = lib.cb_tbe_component_name(i)
        if s is None:
            return names
        names.append(s.decode())
        i += 1


def _check(status: int, what: str):
    if status != CB_OK:
        raise CbTbeError(status, what)


def _ptr(t: torch.Tensor | None):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


@dataclass
class SparseGrad:
    """Row-sparse gradient: rows `unique_ids[:U]` with values `grads[:F]`."""
    unique_ids: torch.Tensor     # int64 [cap_rows]
    table_offsets: torch.Tensor  # int64 [T + 1]
    grad_offsets: torch.Tensor   # int64 [cap_rows + 1]
    grads: torch.Tensor | None   # fp32 [cap_floats]
    num_unique_dev: torch.Tensor  # int64 [1]
    num_floats_dev: torch.Tensor  # int64 [1]

    @property
    def num_unique(self) -> int:
        return int(self.num_unique_dev.item())

    @property
    def num_floats(self) -> int:
        return int(self.num_floats_dev.item())


class TBE:
    """Table-batched pooled embedding bag over caller-owned device tables."""

    def __init__(self, tables: list[torch.Tensor], pooling: str = "sum",
                 index_dtype: torch.dtype = torch.int64, validate: bool = False,
                 timing: bool = False, extra_flags: int = 0,
                 out_dtype: torch.dtype = torch.float32):
        lib = load_library()
        if not tables:
            raise ValueError("at least one table is needed")
        self.device = tables[0].device
        if self.device.type != "cuda":
            raise ValueError("tables must be CUDA tensors")
        for t in tables:
            if t.device != self.device or t.dim() != 2 or not t.is_contiguous():
                raise ValueError("tables must be contiguous 2-D tensors on one CUDA device")
            if t.dtype not in _DTYPES:
                raise ValueError(f"unsupported table dtype {t.dtype}")
        self.tables = list(tables)  # the ABI borrows the memory: keep it alive
        self.dims = [int(t.shape[1]) for t in tables]
        self.rows = [int(t.shape[0]) for t in tables]
        self.sum_dims = sum(self.dims)
        self.pooling = pooling
        self.index_dtype = index_dtype
        if out_dtype not in _OUT_FLAGS:
            raise ValueError(f"unsupported output dtype {out_dtype}")
        self.out_dtype = out_dtype  # pooled output and grad_out (mixed precision)
        descs = (CbTableDesc * len(tables))(*[
            CbTableDesc(t.data_ptr(), int(t.shape[0]), int(t.shape[1]), _DTYPES[t.dtype])
            for t in tables])
        flags = ((CB_VALIDATE if validate else 0) | (CB_TIMING if timing else 0) | extra_flags
                 | _OUT_FLAGS[out_dtype])
        handle = ctypes.c_void_p()
        with torch.cuda.device(self.device):
            _check(lib.cb_tbe_create(descs, len(tables), _POOL[pooling], _IDX[index_dtype], flags,
                                     ctypes.byref(handle)), "cb_tbe_create")
        self._h = handle
        self._lib = lib

    # ------------------------------------------------------------------ helpers
    def _stream(self):
        return ctypes.c_void_p(torch.cuda.current_stream(self.device).cuda_stream)

    def _dev(self, t: torch.Tensor | None, dtype: torch.dtype | None = None):
        if t is None:
            return None
        if dtype is not None and t.dtype != dtype:
            raise TypeError(f"expected {dtype}, got {t.dtype}")
        if t.device != self.device:
            t = t.to(self.device, non_blocking=True)
        return t.contiguous()

    def close(self):
        if getattr(self, "_h", None):
            self._lib.cb_tbe_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ------------------------------------------------------------------ API
    def reserve(self, batch: int, num_indices: int):
        with torch.cuda.device(self.device):
            _check(self._lib.cb_tbe_reserve(self._h, batch, num_indices), "cb_tbe_reserve")

    def forward(self, indices: torch.Tensor, offsets: torch.Tensor,
                per_sample_weights: torch.Tensor | None = None,
                out: torch.Tensor | None = None) -> torch.Tensor:
        T = len(self.dims)
        batch = (offsets.numel() - 1) // T
        ind = self._dev(indices, self.index_dtype)
        off = self._dev(offsets, self.index_dtype)
        w = self._dev(per_sample_weights, torch.float32)
        if out is None:
            out = torch.empty(batch, self.sum_dims, dtype=self.out_dtype, device=self.device)
        elif out.dtype != self.out_dtype:
            raise TypeError(f"out must be {self.out_dtype}")
        with torch.cuda.device(self.device):
            _check(self._lib.cb_tbe_forward(self._h, batch, _ptr(ind), ind.numel(), _ptr(off),
                                            _ptr(w), _ptr(out), self._stream()), "cb_tbe_forward")
        return out

    def alloc_grad(self, cap_rows: int, cap_floats: int, size_only: bool = False) -> SparseGrad:
        dev = self.device
        T = len(self.dims)
        return SparseGrad(
            unique_ids=torch.empty(max(cap_rows, 1), dtype=torch.int64, device=dev),
            table_offsets=torch.empty(T + 1, dtype=torch.int64, device=dev),
            grad_offsets=torch.empty(max(cap_rows, 0) + 1, dtype=torch.int64, device=dev),
            grads=None if size_only else torch.empty(max(cap_floats, 4), dtype=torch.float32,
                                                     device=dev),
            num_unique_dev=torch.zeros(1, dtype=torch.int64, device=dev),
            num_floats_dev=torch.zeros(1, dtype=torch.int64, device=dev))

    def backward_into(self, g: SparseGrad, indices, offsets, grad_out,
                      per_sample_weights=None, cap_rows: int | None = None,
                      cap_floats: int | None = None) -> SparseGrad:
        T = len(self.dims)
        batch = (offsets.numel() - 1) // T
        ind = self._dev(indices, self.index_dtype)
        off = self._dev(offsets, self.index_dtype)
        w = self._dev(per_sample_weights, torch.float32)
        go = self._dev(grad_out, self.out_dtype)
        cs = CbSparseGrad(
            g.unique_ids.data_ptr(), g.table_offsets.data_ptr(), g.grad_offsets.data_ptr(),
            None if g.grads is None else g.grads.data_ptr(),
            g.unique_ids.numel() if cap_rows is None else cap_rows,
            0 if g.grads is None else (g.grads.numel() if cap_floats is None else cap_floats),
            g.num_unique_dev.data_ptr(), g.num_floats_dev.data_ptr())
        with torch.cuda.device(self.device):
            _check(self._lib.cb_tbe_backward(self._h, batch, _ptr(ind), ind.numel(), _ptr(off),
                                             _ptr(w), _ptr(go), ctypes.byref(cs), self._stream()),
                   "cb_tbe_backward")
        return g

    def backward(self, indices, offsets, grad_out, per_sample_weights=None) -> SparseGrad:
        """Sizes the output with a counting call, then computes the gradient."""
        probe = self.alloc_grad(0, 0, size_only=True)
        self.backward_into(probe, indices, offsets, grad_out, per_sample_weights)
        U, F = probe.num_unique, probe.num_floats
        g = self.alloc_grad(U, F)
        return self.backward_into(g, indices, offsets, grad_out, per_sample_weights)

    def backward_apply(self, indices, offsets, grad_out, per_sample_weights=None,
                       optimizer: str = "sgd", lr: float = 0.01, eps: float = 1e-8,
                       state: list[torch.Tensor] | None = None) -> None:
        """Backward with the optimizer step fused (cb_tbe_backward_apply): updates the
        tables this handle was created with (and, for "adagrad", the fp32 [rows_t]
        state tensors) in place."""
        kind, ptrs = self._optimizer_args(optimizer, state)
        T = len(self.dims)
        batch = (offsets.numel() - 1) // T
        ind = self._dev(indices, self.index_dtype)
        off = self._dev(offsets, self.index_dtype)
        w = self._dev(per_sample_weights, torch.float32)
        go = self._dev(grad_out, self.out_dtype)
        with torch.cuda.device(self.device):
            _check(self._lib.cb_tbe_backward_apply(self._h, batch, _ptr(ind), ind.numel(), _ptr(off),
                                                   _ptr(w), _ptr(go), kind, lr, eps,
                                                   _ptr(ptrs), self._stream()),
                   "cb_tbe_backward_apply")
        self._keep = ptrs  # the pointer array must outlive the enqueued work

    def apply_sparse(self, g: SparseGrad, optimizer: str = "sgd", lr: float = 0.01,
                     eps: float = 1e-8, state: list[torch.Tensor] | None = None) -> None:
        """The optimizer step of backward_apply from a gradient that backward /
        backward_into wrote (cb_tbe_apply_sparse): same update, bit for bit."""
        if g.grads is None:
            raise ValueError("a size-only gradient holds no values")
        kind, ptrs = self._optimizer_args(optimizer, state)
        cs = CbSparseGrad(g.unique_ids.data_ptr(), g.table_offsets.data_ptr(), g.grad_offsets.data_ptr(),
                          g.grads.data_ptr(), g.unique_ids.numel(), g.grads.numel(),
                          g.num_unique_dev.data_ptr(), g.num_floats_dev.data_ptr())
        with torch.cuda.device(self.device):
            _check(self._lib.cb_tbe_apply_sparse(self._h, ctypes.byref(cs), kind, lr, eps, _ptr(ptrs),
                                                 self._stream()), "cb_tbe_apply_sparse")
        self._keep = ptrs

    def _optimizer_args(self, optimizer: str, state):
        kinds = {"sgd": 0, "adagrad": 1}
        if optimizer not in kinds:
            raise ValueError(f"unknown optimizer {optimizer!r}")
        if optimizer != "adagrad":
            return kinds[optimizer], None
        if state is None or len(state) != len(self.dims):
            raise ValueError("adagrad needs one fp32 state tensor per table")
        for s_, r in zip(state, self.rows):
            if (s_.device != self.device or s_.dtype != torch.float32 or s_.numel() != r
                    or not s_.is_contiguous()):
                raise ValueError("state[t] must be a contiguous fp32 [rows_t] tensor on the device")
        key = tuple(s_.data_ptr() for s_ in state)
        cached = getattr(self, "_state_ptrs", None)
        if cached is None or cached[0] != key:  # one small copy per new set of state tensors
            cached = (key, torch.tensor(key, dtype=torch.int64, device=self.device))
            self._state_ptrs = cached
        return kinds[optimizer], cached[1]

    def weight_grad(self, indices, offsets, grad_out,
                    out: torch.Tensor | None = None) -> torch.Tensor:
        """d<grad_out, y>/d w_i for every lookup i (cb_tbe_weight_grad), fp32 [n]."""
        T = len(self.dims)
        batch = (offsets.numel() - 1) // T
        ind = self._dev(indices, self.index_dtype)
        off = self._dev(offsets, self.index_dtype)
        go = self._dev(grad_out, self.out_dtype)
        if out is None:
            out = torch.empty(ind.numel(), dtype=torch.float32, device=self.device)
        with torch.cuda.device(self.device):
            _check(self._lib.cb_tbe_weight_grad(self._h, batch, _ptr(ind), ind.numel(), _ptr(off),
                                                _ptr(go), _ptr(out), self._stream()),
                   "cb_tbe_weight_grad")
        return out

    def sorted_payloads(self, num_indices: int) -> torch.Tensor:
        """The last backward's sorted payloads (cb_tbe_sorted_payloads) as int64 [n]:
        lookup positions (weights or mean pooling) or bags t*B + b, in sorted order."""
        buf = torch.empty(max(num_indices, 1), dtype=torch.int32, device=self.device)
        with torch.cuda.device(self.device):
            _check(self._lib.cb_tbe_sorted_payloads(self._h, _ptr(buf), num_indices, self._stream()),
                   "cb_tbe_sorted_payloads")
        return buf[:num_indices].to(torch.int64) & 0xffffffff

    def get_error(self) -> int:
        with torch.cuda.device(self.device):
            return self._lib.cb_tbe_get_error(self._h)

    def raise_on_error(self):
        st = self.get_error()
        if st != CB_OK:
            raise CbTbeError(st, "device-side check")

    def last_timings(self) -> dict[str, float]:
        names = component_names()
        buf = (ctypes.c_float * len(names))()
        with torch.cuda.device(self.device):
            _check(self._lib.cb_tbe_last_timings(self._h, buf, len(names)), "cb_tbe_last_timings")
        return {n: float(v) for n, v in zip(names, buf)}

    def launch_count(self) -> int:
        return int(self._lib.cb_tbe_launch_count(self._h))


# ----------------------------------------------------------------------------- FM cross term

def _fm_args(y: torch.Tensor, num_fields: int):
    if y.device.type != "cuda" or y.dtype != torch.float32 or y.dim() != 2:
        raise ValueError("y must be a 2-D fp32 CUDA tensor [B, T * D]")
    if y.stride(1) != 1:
        raise ValueError("y rows must be contiguous")
    if num_fields < 1 or y.shape[1] % num_fields:
        raise ValueError("the row length must be num_fields * dim")
    return y.shape[0], y.shape[1] // num_fields, y.stride(0)


def fm_forward(y: torch.Tensor, num_fields: int, out: torch.Tensor | None = None) -> torch.Tensor:
    """fm[b] = sum over field pairs t < u of <y[b, tD:(t+1)D], y[b, uD:(u+1)D]> (cb_fm_forward)."""
    lib = load_library()
    B, D, stride = _fm_args(y, num_fields)
    if out is None:
        out = torch.empty(B, dtype=torch.float32, device=y.device)
    with torch.cuda.device(y.device):
        stream = ctypes.c_void_p(torch.cuda.current_stream(y.device).cuda_stream)
        _check(lib.cb_fm_forward(_ptr(y), B, num_fields, D, stride, _ptr(out), stream),
               "cb_fm_forward")
    return out


def fm_backward(y: torch.Tensor, grad_fm: torch.Tensor, num_fields: int,
                out: torch.Tensor | None = None) -> torch.Tensor:
    """grad_y[b, tD + j] = grad_fm[b] * sum over u != t of y[b, uD + j] (cb_fm_backward)."""
    lib = load_library()
    B, D, stride = _fm_args(y, num_fields)
    if grad_fm.device != y.device or grad_fm.dtype != torch.float32 or grad_fm.numel() != B:
        raise ValueError("grad_fm must be fp32 [B] on the device of y")
    grad_fm = grad_fm.contiguous()
    if out is None:
        out = torch.empty_strided(y.shape, y.stride(), dtype=torch.float32, device=y.device)
    with torch.cuda.device(y.device):
        stream = ctypes.c_void_p(torch.cuda.current_stream(y.device).cuda_stream)
        _check(lib.cb_fm_backward(_ptr(y), _ptr(grad_fm), B, num_fields, D, stride, _ptr(out),
                                  stream), "cb_fm_backward")
    return out


# ----------------------------------------------------------------------------- measurement aid

def gather_ceiling(rows: torch.Tensor, indices: torch.Tensor, out: torch.Tensor | None = None,
                   tma: bool = False, error: torch.Tensor | None = None) -> torch.Tensor:
    """Random-row gather out of `rows` ([R, row_bytes / 4] fp32, L2-sized) at `indices`
    (int32 viewed as uint32) with the walkers' load shape (cb_gather_ceiling), or by TMA
    gather4 (tma=True, cb_gather_ceiling_tma; `error` an int32 [1] device word); returns
    the per-32-item sums. With fp16 rows ([R, row_bytes / 2]) the values are widened
    into fp32 sums as the forward does (cb_gather_ceiling_f16)."""
    lib = load_library()
    half = rows.dtype == torch.float16
    if (rows.device.type != "cuda" or rows.dtype not in (torch.float32, torch.float16) or rows.dim() != 2
            or not rows.is_contiguous() or (half and tma)):
        raise ValueError("rows must be a contiguous 2-D fp32 (or, without tma, fp16) CUDA tensor")
    if indices.device != rows.device or indices.dtype != torch.int32:
        raise ValueError("indices must be int32 on the device of rows")
    n = indices.numel()
    if out is None:
        out = torch.empty(max((n + 31) // 32, 1), dtype=torch.float32, device=rows.device)
    with torch.cuda.device(rows.device):
        stream = ctypes.c_void_p(torch.cuda.current_stream(rows.device).cuda_stream)
        if tma:
            if error is None:
                error = torch.zeros(1, dtype=torch.int32, device=rows.device)
            _check(lib.cb_gather_ceiling_tma(_ptr(rows), rows.shape[0], rows.shape[1] * 4,
                                             _ptr(indices.contiguous()), n, _ptr(out), _ptr(error), stream),
                   "cb_gather_ceiling_tma")
        elif half:
            _check(lib.cb_gather_ceiling_f16(_ptr(rows), rows.shape[0], rows.shape[1] * 2,
                                             _ptr(indices.contiguous()), n, _ptr(out), stream),
                   "cb_gather_ceiling_f16")
        else:
            _check(lib.cb_gather_ceiling(_ptr(rows), rows.shape[0], rows.shape[1] * 4, _ptr(indices.contiguous()),
                                         n, _ptr(out), stream), "cb_gather_ceiling")
    return out


# ----------------------------------------------------------------------------- batch replication

def replicate_batch(indices: torch.Tensor, offsets: torch.Tensor, weights: torch.Tensor | None,
                    num_tables: int, factor: int):
    """A captured batch replicated to factor x its bags per table (cb_kjt_replicate):
    bag r * B + b of table t is bag b of table t. Returns device tensors
    (indices, offsets, weights or None)."""
    lib = load_library()
    if indices.device.type != "cuda" or offsets.device != indices.device:
        raise ValueError("indices and offsets must be CUDA tensors on one device")
    if indices.dtype != offsets.dtype or indices.dtype not in _IDX:
        raise ValueError("indices and offsets must both be int32 or both int64")
    if num_tables < 1 or (offsets.numel() - 1) % num_tables:
        raise ValueError("offsets must have num_tables * B + 1 entries")
    B = (offsets.numel() - 1) // num_tables
    ind, off = indices.contiguous(), offsets.contiguous()
    w = None if weights is None else weights.to(indices.device, torch.float32).contiguous()
    out_ind = torch.empty(factor * ind.numel(), dtype=ind.dtype, device=ind.device)
    out_off = torch.empty(num_tables * factor * B + 1, dtype=off.dtype, device=ind.device)
    out_w = None if w is None else torch.empty(factor * ind.numel(), dtype=torch.float32, device=ind.device)
    with torch.cuda.device(ind.device):
        stream = ctypes.c_void_p(torch.cuda.current_stream(ind.device).cuda_stream)
        _check(lib.cb_kjt_replicate(_ptr(ind), _ptr(off), _ptr(w), _IDX[ind.dtype], num_tables, B,
                                    ind.numel(), factor, _ptr(out_ind), _ptr(out_off), _ptr(out_w),
                                    stream), "cb_kjt_replicate")
    return out_ind, out_off, out_w
