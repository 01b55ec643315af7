"""Shared test helpers: small random problems and torch-CPU float64 cross-checks.

The torch routines here are an independent library statement of the same
quantities (torch.nn.functional.embedding_bag and its autograd), used only to
pin the oracle; the CUDA path is never compared against them.
"""

from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as F

from paper_2609_30656_gb300 import workloads as wl


def random_problem(seed: int, dims=(8, 16, 24), rows=(7, 50, 13), batch=9, max_len=12,
                   dtype=torch.float32, int_valued=False, weighted=False, empty_frac=0.2):
    """Tables, key-major offsets and indices with ragged (and empty) bags."""
    g = torch.Generator().manual_seed(seed)
    tables = []
    for r, d in zip(rows, dims):
        if int_valued:
            x = torch.randint(-8, 9, (r, d), generator=g).to(torch.float32)
        else:
            x = torch.randn(r, d, generator=g)
        tables.append(x.to(dtype))
    lens = torch.randint(0, max_len + 1, (len(rows) * batch,), generator=g)
    lens[torch.rand(lens.shape, generator=g) < empty_frac] = 0
    offsets = torch.zeros(lens.numel() + 1, dtype=torch.int64)
    offsets[1:] = torch.cumsum(lens, 0)
    idx = []
    for t, r in enumerate(rows):
        s, e = int(offsets[t * batch]), int(offsets[(t + 1) * batch])
        idx.append(torch.randint(0, r, (e - s,), generator=g))
    indices = torch.cat(idx) if idx else torch.zeros(0, dtype=torch.int64)
    weights = None
    if weighted:
        if int_valued:
            weights = torch.randint(0, 3, (indices.numel(),), generator=g).to(torch.float32)
        else:
            weights = torch.rand(indices.numel(), generator=g)
    return tables, indices, offsets, weights


def torch_forward_f64(tables, batch, indices, offsets, weights=None, mean=False):
    """Per-table torch embedding_bag in float64 (include_last_offset)."""
    outs = []
    for t, E in enumerate(tables):
        s, e = int(offsets[t * batch]), int(offsets[(t + 1) * batch])
        off_t = (offsets[t * batch:(t + 1) * batch + 1] - s).to(torch.int64)
        ind_t = indices[s:e].to(torch.int64)
        W = E.to(torch.float64)
        if weights is None:
            y = F.embedding_bag(ind_t, W, off_t, mode="mean" if mean else "sum",
                                include_last_offset=True)
        else:
            y = F.embedding_bag(ind_t, W, off_t, mode="sum", include_last_offset=True,
                                per_sample_weights=weights[s:e].to(torch.float64))
            if mean:
                L = (off_t[1:] - off_t[:-1]).to(torch.float64)
                y = torch.where(L[:, None] > 0, y / L.clamp(min=1)[:, None], torch.zeros_like(y))
        outs.append(y)
    return torch.cat(outs, dim=1)


def torch_dense_grad_f64(tables, batch, indices, offsets, grad_out, weights=None, mean=False):
    """Dense dE_t from torch autograd through embedding_bag in float64."""
    leaves = [E.to(torch.float64).clone().requires_grad_(True) for E in tables]
    y = torch_forward_f64(leaves, batch, indices, offsets, weights, mean)
    (y * grad_out.to(torch.float64)).sum().backward()
    return [L.grad.detach().clone() for L in leaves]


def sparse_to_dense(res, rows, dims):
    """Scatter an oracle/GPU row-sparse gradient into dense per-table arrays."""
    row_base = np.concatenate([[0], np.cumsum(rows)])
    dense = [np.zeros((int(r), int(d))) for r, d in zip(rows, dims)]
    for u, key in enumerate(np.asarray(res.uniq)):
        t = int(np.searchsorted(row_base, key, side="right") - 1)
        r = int(key - row_base[t])
        go = int(res.grad_offsets[u])
        dense[t][r] = res.grads[go:go + dims[t]]
    return dense


def table_meta(tables):
    return (np.array([E.shape[0] for E in tables], dtype=np.int64),
            np.array([E.shape[1] for E in tables], dtype=np.int32))


__all__ = ["random_problem", "torch_forward_f64", "torch_dense_grad_f64", "sparse_to_dense",
           "table_meta", "wl"]
