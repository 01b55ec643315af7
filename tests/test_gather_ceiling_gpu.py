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
