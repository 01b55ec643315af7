"""cb_gather_ceiling, the L2 random-gather rate probe the bench reports, computes
what it loads: each 32-item sum against torch on the host."""

import pytest
import torch

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


@pytest.mark.parametrize("row_bytes", [64, 128, 256, 512])
def test_sums_of_gathered_rows(row_bytes):
    from paper_2609_30656_gb300 import tbe
    g = torch.Generator().manual_seed(row_bytes)
    rows = torch.randint(-8, 9, (1000, row_bytes // 4), generator=g).to(torch.float32)
    n = 32 * 77 + 5  # a ragged last batch
    idx = torch.randint(0, 1000, (n,), generator=g, dtype=torch.int64)
    got = tbe.gather_ceiling(rows.to(DEV), idx.to(torch.int32).to(DEV)).cpu()
    pad = torch.zeros(32 * ((n + 31) // 32), dtype=torch.float64)
    pad[:n] = rows.double()[idx].sum(1)
    want = pad.view(-1, 32).sum(1)
    assert torch.equal(got.double(), want)  # integers: exact in any order


@pytest.mark.parametrize("row_bytes", [256, 512])
def test_tma_gather4_sums_of_gathered_rows(row_bytes):
    from paper_2609_30656_gb300 import tbe
    g = torch.Generator().manual_seed(row_bytes + 1)
    rows = torch.randint(-8, 9, (3000, row_bytes // 4), generator=g).to(torch.float32)
    n = 32 * 301 + 7  # several batches per warp and a ragged last batch
    idx = torch.randint(0, 3000, (n,), generator=g, dtype=torch.int64)
    err = torch.zeros(1, dtype=torch.int32, device=DEV)
    got = tbe.gather_ceiling(rows.to(DEV), idx.to(torch.int32).to(DEV), tma=True, error=err).cpu()
    assert int(err.item()) == 0
    pad = torch.zeros(32 * ((n + 31) // 32), dtype=torch.float64)
    pad[:n] = rows.double()[idx].sum(1)
    want = pad.view(-1, 32).sum(1)
    assert torch.equal(got.double(), want)


@pytest.mark.parametrize("row_bytes", [128, 256, 512])
def test_half_rows_widened_into_fp32_sums(row_bytes):
    from paper_2609_30656_gb300 import tbe
    g = torch.Generator().manual_seed(row_bytes + 2)
    rows = torch.randint(-8, 9, (1500, row_bytes // 2), generator=g).to(torch.float16)
    n = 32 * 123 + 9  # a ragged last batch
    idx = torch.randint(0, 1500, (n,), generator=g, dtype=torch.int64)
    got = tbe.gather_ceiling(rows.to(DEV), idx.to(torch.int32).to(DEV)).cpu()
    pad = torch.zeros(32 * ((n + 31) // 32), dtype=torch.float64)
    pad[:n] = rows.double()[idx].sum(1)
    want = pad.view(-1, 32).sum(1)
    assert torch.equal(got.double(), want)  # integers: exact in any order


@pytest.mark.parametrize("n", [1, 31, 32, 64 * 32])
@pytest.mark.parametrize("half", [False, True])
def test_only_full_batches_or_only_a_partial_one(n, half):
    # the full batches and the partial last batch are summed by different kernels
    from paper_2609_30656_gb300 import tbe
    g = torch.Generator().manual_seed(n + 7 * half)
    dtype, width = (torch.float16, 128) if half else (torch.float32, 64)
    rows = torch.randint(-8, 9, (700, width), generator=g).to(dtype)
    idx = torch.randint(0, 700, (n,), generator=g, dtype=torch.int64)
    got = tbe.gather_ceiling(rows.to(DEV), idx.to(torch.int32).to(DEV)).cpu()
    pad = torch.zeros(32 * ((n + 31) // 32), dtype=torch.float64)
    pad[:n] = rows.double()[idx].sum(1)
    assert torch.equal(got.double(), pad.view(-1, 32).sum(1))


def test_indices_past_the_row_set_read_row_zero():
    from paper_2609_30656_gb300 import tbe
    rows = torch.arange(10 * 64, dtype=torch.float32).view(10, 64)
    idx = torch.tensor([0, 9, 10, 2**31 - 1] * 8 + [3, 11], dtype=torch.int64)  # a full batch and a tail
    got = tbe.gather_ceiling(rows.to(DEV), idx.to(torch.int32).to(DEV)).cpu().double()
    eff = torch.where(idx < 10, idx, torch.zeros_like(idx))
    want = torch.zeros(64, dtype=torch.float64)
    want[:idx.numel()] = rows.double()[eff].sum(1)
    assert torch.equal(got, want.view(-1, 32).sum(1))
