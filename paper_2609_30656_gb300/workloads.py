"""Seeded synthetic inputs for the pooled embedding-bag lookup.

This module only draws random inputs: table contents, jagged bag lengths,
indices, per-sample weights and output gradients. It holds none of the
lookup's arithmetic, so the CUDA path and the CPU oracle can both be fed from
it. The paper's own data (a DeepFM-based DLRM on real datasets, Sec. IV) is not
available; these shapes stand in for it: jagged categorical features (Abstract),
embedding tables shrunk to fit one GPU (Sec. III.B.1), bandwidth-bound sparse
lookups (Sec. IV.A.2).

Workloads (every table initialised N(0, 0.01), then rounded to its storage type):

  cfg1   1 x 1000 x 64 fp32, batch 128, every bag 4 long, uniform indices, sum
  cfg2   8 x 100k x 128 fp32, batch 2048, Poisson(20) lengths clipped to
         [0, 100], Zipf(1.05) indices, sum
  cfg3   26 tables, rows log-uniform in [10, 1e7], dim 128 fp16, batch 4096,
         one-hot bags, Zipf(1.1) indices, sum
  cfg4   64 x 1M, dims 64/128/256 cycling, bf16, batch 8192, lognormal
         lengths (mean 50, clipped to [0, 500]), uniform indices, weights
         U(0, 1), weighted mean
  cfg5   100 x 5M x 128 fp16 (128 GB), batch 65536, 5 % empty bags, other
         lengths power law L^-2 on [7, 1000], Zipf(1.2) indices, sum
  cfg5u  cfg5 with uniform indices (no cache reuse; the bandwidth control)

Bounded Zipf: rank k in 1..N has probability proportional to k^-alpha; a rank
is drawn by inverse CDF and mapped to a row through a seeded permutation of the
table, since hashed ids scatter the hot rows.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import torch

DTYPES = {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}


@dataclass(frozen=True)
class LengthDist:
    kind: str                 # "fixed" | "poisson" | "lognormal" | "powerlaw"
    mean: float = 0.0         # fixed length, Poisson mean, or lognormal mean
    sigma: float = 1.0        # lognormal shape
    lo: int = 0               # clip / support lower bound
    hi: int = 0               # clip / support upper bound
    alpha: float = 2.0        # power-law exponent
    empty_frac: float = 0.0   # share of bags forced empty (power law)


@dataclass(frozen=True)
class Workload:
    name: str
    rows: tuple[int, ...]
    dims: tuple[int, ...]
    dtype: str
    batch: int
    lengths: LengthDist
    zipf_alpha: float | None  # None = uniform indices
    weighted: bool
    mean: bool
    backward: bool
    permute_rows: bool = True
    note: str = field(default="", compare=False)

    @property
    def num_tables(self) -> int:
        return len(self.rows)

    @property
    def sum_dims(self) -> int:
        return int(sum(self.dims))

    @property
    def torch_dtype(self) -> torch.dtype:
        return DTYPES[self.dtype]

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2


_CFG_IDS = {"cfg1": 1, "cfg2": 2, "cfg3": 3, "cfg4": 4, "cfg5": 5, "cfg5u": 6}


def _mix(*parts: int) -> int:
    """Deterministic seed mixing (splitmix64 steps over the parts)."""
    x = 0x9E3779B97F4A7C15
    for p in parts:
        x = (x ^ (int(p) & 0xFFFFFFFFFFFFFFFF)) & 0xFFFFFFFFFFFFFFFF
        x = (x + 0x9E3779B97F4A7C15) & 0xFFFFFFFFFFFFFFFF
        z = x
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & 0xFFFFFFFFFFFFFFFF
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & 0xFFFFFFFFFFFFFFFF
        x = z ^ (z >> 31)
    return x & 0x7FFFFFFFFFFFFFFF


def _gen(device, *parts: int) -> torch.Generator:
    g = torch.Generator(device=torch.device(device))
    g.manual_seed(_mix(*parts))
    return g


def get_workload(name: str, seed: int = 0) -> Workload:
    """The five workloads (plus the uniform control cfg5u), rows drawn from `seed`."""
    if name == "cfg1":
        return Workload(name, (1000,), (64,), "f32", 128, LengthDist("fixed", mean=4),
                        None, False, False, False)
    if name == "cfg2":
        return Workload(name, (100_000,) * 8, (128,) * 8, "f32", 2048,
                        LengthDist("poisson", mean=20.0, lo=0, hi=100), 1.05, False, False, True)
    if name == "cfg3":
        g = _gen("cpu", seed, 3, 0xC3)
        u = torch.rand(26, generator=g, dtype=torch.float64)
        rows = tuple(int(round(math.exp(math.log(10.0) + float(x) * (math.log(1e7) - math.log(10.0)))))
                     for x in u)
        return Workload(name, rows, (128,) * 26, "f16", 4096, LengthDist("fixed", mean=1),
                        1.1, False, False, True)
    if name == "cfg4":
        return Workload(name, (1_000_000,) * 64, tuple([64, 128, 256][t % 3] for t in range(64)),
                        "bf16", 8192,
                        LengthDist("lognormal", mean=50.0, sigma=1.0, lo=0, hi=500),
                        None, True, True, True)
    if name in ("cfg5", "cfg5u"):
        return Workload(name, (5_000_000,) * 100, (128,) * 100, "f16", 65536,
                        LengthDist("powerlaw", alpha=2.0, lo=7, hi=1000, empty_frac=0.05),
                        None if name == "cfg5u" else 1.2, False, False, True)
    raise KeyError(name)


def scaled(w: Workload, *, num_tables: int | None = None, batch: int | None = None,
           rows: int | None = None, name: str | None = None) -> Workload:
    """The same distributions on fewer tables, a smaller batch or fewer rows."""
    T = w.num_tables if num_tables is None else num_tables
    r = tuple((w.rows[t % w.num_tables] if rows is None else min(rows, w.rows[t % w.num_tables]))
              for t in range(T))
    d = tuple(w.dims[t % w.num_tables] for t in range(T))
    return replace(w, name=name or f"{w.name}-scaled", rows=r, dims=d,
                   batch=w.batch if batch is None else batch)


# ----------------------------------------------------------------------------- draws

def bag_lengths(w: Workload, gen: torch.Generator, count: int, device) -> torch.Tensor:
    """`count` bag lengths (int64) from the workload's length distribution."""
    L = w.lengths
    dev = torch.device(device)
    if L.kind == "fixed":
        return torch.full((count,), int(L.mean), dtype=torch.int64, device=dev)
    if L.kind == "poisson":
        rate = torch.full((count,), float(L.mean), dtype=torch.float64, device=dev)
        x = torch.poisson(rate, generator=gen)
        return x.clamp_(L.lo, L.hi).to(torch.int64)
    if L.kind == "lognormal":
        mu = math.log(L.mean) - 0.5 * L.sigma * L.sigma
        z = torch.randn(count, generator=gen, dtype=torch.float64, device=dev)
        x = torch.exp(mu + L.sigma * z)
        return torch.round(x).clamp_(L.lo, L.hi).to(torch.int64)
    if L.kind == "powerlaw":
        support = torch.arange(L.lo, L.hi + 1, dtype=torch.float64, device=dev)
        cdf = torch.cumsum(support.pow(-L.alpha), 0)
        cdf = cdf / cdf[-1]
        cdf[-1] = 1.0
        u = torch.rand(count, generator=gen, dtype=torch.float64, device=dev)
        k = torch.searchsorted(cdf, u).clamp_(max=support.numel() - 1)
        lens = (k + L.lo).to(torch.int64)
        if L.empty_frac > 0:
            e = torch.rand(count, generator=gen, dtype=torch.float64, device=dev) < L.empty_frac
            lens = torch.where(e, torch.zeros_like(lens), lens)
        return lens
    raise ValueError(L.kind)


_ZIPF_CDF_CACHE: dict = {}


def zipf_cdf(N: int, alpha: float, device) -> torch.Tensor:
    key = (N, alpha, str(torch.device(device)))
    c = _ZIPF_CDF_CACHE.get(key)
    if c is None:
        k = torch.arange(1, N + 1, dtype=torch.float64, device=torch.device(device))
        c = torch.cumsum(k.pow(-alpha), 0)
        c = c / c[-1]
        c[-1] = 1.0
        if len(_ZIPF_CDF_CACHE) > 8:
            _ZIPF_CDF_CACHE.clear()
        _ZIPF_CDF_CACHE[key] = c
    return c


def zipf_ranks(N: int, alpha: float, count: int, gen: torch.Generator, device) -> torch.Tensor:
    """0-based ranks of a bounded Zipf(alpha) on N items, by inverse CDF."""
    u = torch.rand(count, generator=gen, dtype=torch.float64, device=torch.device(device))
    return torch.searchsorted(zipf_cdf(N, alpha, device), u).clamp_(max=N - 1)


@dataclass
class Batch:
    indices: torch.Tensor         # int64 [n]
    offsets: torch.Tensor         # int64 [T * B + 1], key-major
    weights: torch.Tensor | None  # fp32 [n] or None

    @property
    def num_indices(self) -> int:
        return int(self.indices.numel())


def make_tables(w: Workload, seed: int, device, int_valued: bool = False,
                only=None) -> list[torch.Tensor]:
    """Row-major [rows_t, D_t] tables in the workload's storage type (`only`: a subset)."""
    out = []
    for t, (r, d) in enumerate(zip(w.rows, w.dims)):
        if only is not None and t not in only:
            continue
        g = _gen(device, seed, _CFG_IDS.get(w.name.split("-")[0], 0), t, 0x7AB)
        if int_valued:
            x = torch.randint(-8, 9, (r, d), generator=g, device=torch.device(device),
                              dtype=torch.int32).to(torch.float32)
        else:
            x = torch.randn(r, d, generator=g, device=torch.device(device), dtype=torch.float32)
            x.mul_(0.01)
        out.append(x.to(w.torch_dtype))
        del x
    return out


def make_batch(w: Workload, seed: int, device, batch_index: int = 0,
               int_valued: bool = False) -> Batch:
    """One jagged batch: key-major offsets, per-table indices, optional weights."""
    cid = _CFG_IDS.get(w.name.split("-")[0], 0)
    dev = torch.device(device)
    T, B = w.num_tables, w.batch
    g = _gen(device, seed, cid, batch_index, 0x1E9)
    lengths = bag_lengths(w, g, T * B, device)
    offsets = torch.zeros(T * B + 1, dtype=torch.int64, device=dev)
    torch.cumsum(lengths, 0, out=offsets[1:])
    n = int(offsets[-1].item())
    indices = torch.empty(n, dtype=torch.int64, device=dev)
    table_starts = offsets[:: B].tolist()  # offsets[t * B] for t = 0..T
    for t in range(T):
        s, e = table_starts[t], table_starts[t + 1]
        if e == s:
            continue
        gt = _gen(device, seed, cid, batch_index, t, 0x1D)
        if w.zipf_alpha is None:
            indices[s:e] = torch.randint(0, w.rows[t], (e - s,), generator=gt, device=dev)
        else:
            ranks = zipf_ranks(w.rows[t], w.zipf_alpha, e - s, gt, device)
            if w.permute_rows:
                # The rank -> row map is fixed per table (not per batch).
                gp = _gen(device, seed, cid, t, 0x9E)
                perm = torch.randperm(w.rows[t], generator=gp, device=dev)
                indices[s:e] = perm[ranks]
            else:
                indices[s:e] = ranks
    weights = None
    if w.weighted:
        gw = _gen(device, seed, cid, batch_index, 0x3E)
        if int_valued:
            weights = torch.randint(0, 3, (n,), generator=gw, device=dev).to(torch.float32)
        else:
            weights = torch.rand(n, generator=gw, device=dev, dtype=torch.float32)
    return Batch(indices, offsets, weights)


def make_grad_out(w: Workload, seed: int, device, batch_index: int = 0,
                  int_valued: bool = False) -> torch.Tensor:
    """Upstream gradient [B, sum D] fp32, N(0, 1) (or integers in [-8, 8])."""
    g = _gen(device, seed, _CFG_IDS.get(w.name.split("-")[0], 0), batch_index, 0x60)
    shape = (w.batch, w.sum_dims)
    if int_valued:
        return torch.randint(-8, 9, shape, generator=g, device=torch.device(device),
                             dtype=torch.int32).to(torch.float32)
    return torch.randn(shape, generator=g, device=torch.device(device), dtype=torch.float32)


def explicit_batch(lengths_per_table: list[list[int]], indices: list[int],
                   weights: list[float] | None = None, device="cpu") -> Batch:
    """A batch written out by hand: bag lengths per table and the flat indices."""
    lens = [L for per_t in lengths_per_table for L in per_t]
    off = [0]
    for L in lens:
        off.append(off[-1] + L)
    if off[-1] != len(indices):
        raise ValueError("lengths do not add up to the number of indices")
    dev = torch.device(device)
    return Batch(torch.tensor(indices, dtype=torch.int64, device=dev),
                 torch.tensor(off, dtype=torch.int64, device=dev),
                 None if weights is None else torch.tensor(weights, dtype=torch.float32, device=dev))
