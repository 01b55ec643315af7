"""Algorithmic byte counts of the pooled embedding bag and its backward.

"Algorithmic" bytes are what the method itself must move, with every lookup's
row counted once and nothing added for the implementation's own scratch
traffic: the embedding module's estimated bandwidth column of the paper's
result table (Sec. IV.A.1) divided by the achieved time gives the same
"bandwidth utilisation" figure. Per unit:

  forward   per lookup: D_t * e_S (stored row) + idx_bytes (+ 4 for a weight)
            per bag:    idx_bytes (offsets)    per output row: sum D * 4
  backward  per lookup: D_t * 4 (gathered grad_out slice) + idx_bytes (+ 4)
            per bag:    idx_bytes              per unique row: 8 (id) + D_t * 4
  sort      per lookup and pass: 16 (read and write a 4-byte key and payload)
  weight gradient  per lookup: D_t * e_S (stored row) + D_t * 4 (grad_out slice)
            + idx_bytes + 4 (the gradient)    per bag: idx_bytes
  FM cross term    per pooled value: 4 read (+ 4 written by the backward);
            per sample: 4 (fm written, or grad_fm read)
  fused optimizer step   the backward's reads; per touched row D_t * e_S read
            and written (+ 8 for the Adagrad state word) instead of the gradient
"""

from __future__ import annotations

from dataclasses import dataclass

import torch


@dataclass
class BatchCounts:
    """Host-side sizes of one batch; lookups_per_table from the table boundaries."""
    num_tables: int
    batch: int
    dims: tuple[int, ...]
    elem_bytes: int
    idx_bytes: int
    weighted: bool
    lookups_per_table: tuple[int, ...]
    nonempty_per_table: tuple[int, ...] = ()  # bags with at least one lookup

    @property
    def n(self) -> int:
        return int(sum(self.lookups_per_table))

    @property
    def sum_dims(self) -> int:
        return int(sum(self.dims))


def batch_counts(dims, elem_bytes: int, batch: int, offsets: torch.Tensor, weighted: bool,
                 idx_bytes: int = 8) -> BatchCounts:
    T = len(dims)
    starts = offsets[::batch][:T + 1].to("cpu").tolist() if batch > 0 else [0] * (T + 1)
    per = tuple(int(starts[t + 1] - starts[t]) for t in range(T))
    if batch > 0:
        lens = (offsets[1:T * batch + 1] - offsets[:T * batch]).view(T, batch)
        nonempty = tuple(int(x) for x in (lens > 0).sum(1).to("cpu").tolist())
    else:
        nonempty = (0,) * T
    return BatchCounts(T, batch, tuple(int(d) for d in dims), elem_bytes, idx_bytes, weighted, per,
                       nonempty)


def forward_bytes(c: BatchCounts) -> dict[str, int]:
    rows = sum(L * d * c.elem_bytes for L, d in zip(c.lookups_per_table, c.dims))
    parts = {
        "rows": rows,
        "indices": c.n * c.idx_bytes,
        "offsets": (c.num_tables * c.batch + 1) * c.idx_bytes,
        "weights": c.n * 4 if c.weighted else 0,
        "output": c.batch * c.sum_dims * 4,
    }
    parts["total"] = sum(parts.values())
    return parts


def forward_unique_bytes(c: BatchCounts, unique_per_table) -> int:
    """Compulsory forward traffic: each distinct row read once (L2-perfect reuse)."""
    f = forward_bytes(c)
    rows = sum(int(u) * d * c.elem_bytes for u, d in zip(unique_per_table, c.dims))
    return f["total"] - f["rows"] + rows


def backward_bytes(c: BatchCounts, unique_per_table) -> dict[str, int]:
    U = int(sum(int(u) for u in unique_per_table))
    parts = {
        "grad_gather": sum(L * d * 4 for L, d in zip(c.lookups_per_table, c.dims)),
        "indices": c.n * c.idx_bytes,
        "offsets": (c.num_tables * c.batch + 1) * c.idx_bytes,
        "weights": c.n * 4 if c.weighted else 0,
        "unique_ids": U * 8,
        "grads": sum(int(u) * d * 4 for u, d in zip(unique_per_table, c.dims)),
    }
    parts["total"] = sum(parts.values())
    return parts


def weight_grad_bytes(c: BatchCounts) -> int:
    """Algorithmic bytes of d<grad_out, y>/d w: each lookup's row and grad_out slice."""
    rows = sum(L * d * c.elem_bytes for L, d in zip(c.lookups_per_table, c.dims))
    slices = sum(L * d * 4 for L, d in zip(c.lookups_per_table, c.dims))
    return rows + slices + c.n * (c.idx_bytes + 4) + (c.num_tables * c.batch + 1) * c.idx_bytes


def apply_step_bytes(c: BatchCounts, unique_per_table, adagrad: bool) -> int:
    """Algorithmic bytes of the backward with the optimizer step fused: the
    backward's reads, and each touched row read and written in its storage
    type (plus its fp32 state word for row-wise Adagrad) instead of the
    gradient rows and ids."""
    b = backward_bytes(c, unique_per_table)
    rows = sum(int(u) * d * c.elem_bytes for u, d in zip(unique_per_table, c.dims))
    U = int(sum(int(u) for u in unique_per_table))
    return (b["total"] - b["grads"] - b["unique_ids"] + 2 * rows + (8 * U if adagrad else 0))


def sparse_apply_bytes(c: BatchCounts, unique_per_table, adagrad: bool) -> int:
    """Algorithmic bytes of the optimizer step as a second pass over a written
    row-sparse gradient: per touched row its id and offset (8 + 8 bytes), its
    fp32 gradient row, the table row read and written in its storage type, and
    for row-wise Adagrad its fp32 state word read and written."""
    U = int(sum(int(u) for u in unique_per_table))
    grads = sum(int(u) * d * 4 for u, d in zip(unique_per_table, c.dims))
    rows = sum(int(u) * d * c.elem_bytes for u, d in zip(unique_per_table, c.dims))
    return 16 * U + grads + 2 * rows + (8 * U if adagrad else 0)


def sort_bytes(n: int, passes: int) -> int:
    return 16 * n * passes


def radix_passes(rows) -> int:
    """8-bit passes over the row number of the largest table (ranges sorted per table)."""
    largest = max(1, int(max(rows)))
    bits = 1
    while bits < 32 and (1 << bits) <= largest:  # keys 0 .. rows_t (rows_t: out of range)
        bits += 1
    return (bits + 7) // 8


def component_bytes(c: BatchCounts, unique_per_table, rows, packed: bool) -> dict[str, int]:
    """Algorithmic bytes of each timed component (the kernels inside it)."""
    f = forward_bytes(c)
    b = backward_bytes(c, unique_per_table)
    U = int(sum(int(u) for u in unique_per_table))
    n = c.n
    return {
        "fwd.gather": f["total"],
        "bwd.keygen": n * c.idx_bytes + (c.num_tables * c.batch + 1) * c.idx_bytes + 8 * n
        + (12 * n if packed else 0),
        "bwd.sort": sort_bytes(n, radix_passes(rows)),
        "bwd.rle": 8 * n + 8 * U,
        "bwd.reduce": b["grad_gather"] + 4 * n + (8 * n if packed else 0) + 4 * U + b["grads"]
        + 16 * U,
    }


def component_compulsory_bytes(c: BatchCounts, unique_per_table, packed: bool) -> dict[str, int]:
    """Compulsory bytes of the two gather kernels: what they must move even when
    every repeated row comes from cache, i.e. each distinct table row (forward)
    or each non-empty bag's grad_out slice (backward reduce) once, plus their
    per-lookup and per-row streams and outputs. With the L2 flushed before a
    step this is the least DRAM traffic of the launch."""
    U = int(sum(int(u) for u in unique_per_table))
    n = c.n
    slices = sum(int(k) * d * 4 for k, d in zip(c.nonempty_per_table, c.dims))
    grads = sum(int(u) * d * 4 for u, d in zip(unique_per_table, c.dims))
    return {
        "fwd.gather": forward_unique_bytes(c, unique_per_table),
        "bwd.reduce": slices + 4 * n + (8 * n if packed else 0) + 4 * U + grads + 16 * U,
    }


def fm_bytes(batch: int, num_fields: int, dim: int, backward: bool) -> int:
    """Algorithmic bytes of the FM cross term: the pooled rows read once (fp32),
    plus fm [B] written (forward), or grad_fm [B] read and grad_y written (backward)."""
    y = 4 * batch * num_fields * dim
    return y + 4 * batch + (y if backward else 0)


def component_flops(c: BatchCounts, unique_per_table, mean: bool) -> dict[str, int]:
    """Algorithmic floating-point operations of each timed component: one add (or
    a multiply-add, 2, with weights or mean coefficients) per gathered value, a
    division per pooled value for mean pooling; the integer stages do none."""
    per_value = 2 if (c.weighted or mean) else 1
    gathered = sum(L * d for L, d in zip(c.lookups_per_table, c.dims))
    return {
        "fwd.prep": 0, "fwd.fixup": 0, "bwd.keygen": 0, "bwd.sort": 0, "bwd.rle": 0,
        "fwd.gather": per_value * gathered + (c.batch * c.sum_dims if mean else 0),
        "bwd.reduce": per_value * gathered,
    }
