"""Input variants of Component Benchmark's preprocessors on the GPU: batch
replication (cb_kjt_replicate) against the oracle, and one handle driven by
batches of changing shape (dynamic jagged shapes)."""

import numpy as np
import pytest
import torch

import oracle
from tests.helpers import (assert_backward_matches, backward_reference, forward_reference,
                           random_problem, table_meta)
from paper_2609_30656_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


@pytest.mark.parametrize("factor", [1, 3, 7])
@pytest.mark.parametrize("idx_dtype,weighted", [(torch.int64, True), (torch.int32, False)])
def test_replicate_matches_the_oracle(factor, idx_dtype, weighted):
    from paper_2609_30656_gb300 import tbe
    tables, ind, off, w = random_problem(101, weighted=weighted, max_len=40, empty_frac=0.3)
    # an empty table in the middle
    B = 9
    lens = (off[1:] - off[:-1]).clone()
    lens[B:2 * B] = 0
    keep = torch.cat([torch.arange(int(off[t * B]), int(off[(t + 1) * B])) for t in (0, 2)])
    ind = ind[keep]
    w = None if w is None else w[keep]
    off = torch.zeros(3 * B + 1, dtype=torch.int64)
    off[1:] = torch.cumsum(lens, 0)
    ind, off = ind.to(idx_dtype), off.to(idx_dtype)
    gi, go, gw = tbe.replicate_batch(ind.to(DEV), off.to(DEV), None if w is None else w.to(DEV), 3, factor)
    torch.cuda.synchronize()
    ri, ro, rw = oracle.replicate_kjt(ind, off, w, 3, factor)
    np.testing.assert_array_equal(gi.cpu().numpy(), ri)
    np.testing.assert_array_equal(go.cpu().numpy(), ro)
    if weighted:
        np.testing.assert_array_equal(gw.cpu().numpy(), rw)
    else:
        assert gw is None


def test_replicated_lookup_repeats_the_small_batch_output():
    # Integer tables make every sum exact, so the replicated batch's pooled rows
    # equal the small batch's bit for bit, whatever the chunking.
    from paper_2609_30656_gb300 import tbe
    tables, ind, off, w = random_problem(102, dims=(16, 64, 128), rows=(30, 300, 3000),
                                         int_valued=True, weighted=True, max_len=700,
                                         dtype=torch.float16)
    m = tbe.TBE([t.to(DEV) for t in tables], pooling="sum", validate=True)
    y = m.forward(ind.to(DEV), off.to(DEV), w.to(DEV))
    F = 5
    ri, ro, rw = tbe.replicate_batch(ind.to(DEV), off.to(DEV), w.to(DEV), 3, F)
    y2 = m.forward(ri, ro, rw)
    torch.cuda.synchronize()
    for r in range(F):
        assert torch.equal(y2[r * 9:(r + 1) * 9], y)


def test_full_size_capture_replicated_to_the_cfg5_batch():
    # cfg5's distributions captured at batch 4096 and replicated 16x to 65536.
    from paper_2609_30656_gb300 import tbe
    w = wl.scaled(wl.get_workload("cfg5"), batch=4096)
    b = wl.make_batch(w, 0, DEV)
    ri, ro, _ = tbe.replicate_batch(b.indices, b.offsets, None, w.num_tables, 16)
    torch.cuda.synchronize()
    T, B = w.num_tables, 4096
    assert ri.numel() == 16 * b.indices.numel() and ro.numel() == T * 16 * B + 1
    off = b.offsets.cpu()
    ro_c, ri_c = ro.cpu(), ri.cpu()
    g = torch.Generator().manual_seed(3)
    for _ in range(64):
        t = int(torch.randint(0, T, (1,), generator=g))
        r = int(torch.randint(0, 16, (1,), generator=g))
        bb = int(torch.randint(0, B, (1,), generator=g))
        s, e = int(off[t * B + bb]), int(off[t * B + bb + 1])
        k = t * 16 * B + r * B + bb
        s2, e2 = int(ro_c[k]), int(ro_c[k + 1])
        assert e2 - s2 == e - s
        assert torch.equal(ri_c[s2:e2], b.indices.cpu()[s:e])


def test_one_handle_through_batches_of_changing_shape():
    # Growing, shrinking and empty batches on one handle (the workspace grows on
    # demand and is reused), forward and backward against the oracle each time.
    from paper_2609_30656_gb300 import tbe
    tables, _, _, _ = random_problem(103, dims=(8, 64, 128), rows=(20, 500, 4000),
                                     dtype=torch.bfloat16)
    m = tbe.TBE([t.to(DEV) for t in tables], pooling="mean", validate=True)
    rows, dims = table_meta(tables)
    for k, (batch, max_len) in enumerate([(5, 3), (300, 200), (1, 1), (0, 0), (77, 1500), (9, 30)]):
        g = torch.Generator().manual_seed(200 + k)
        lens = torch.randint(0, max_len + 1, (3 * batch,), generator=g)
        off = torch.zeros(3 * batch + 1, dtype=torch.int64)
        off[1:] = torch.cumsum(lens, 0)
        ind = torch.cat([torch.randint(0, int(r), (int(off[(t + 1) * batch] - off[t * batch]),), generator=g)
                         for t, r in enumerate(rows)]) if batch else torch.zeros(0, dtype=torch.int64)
        wts = torch.rand(ind.numel(), generator=g)
        y = m.forward(ind.to(DEV), off.to(DEV), wts.to(DEV))
        torch.cuda.synchronize()
        assert y.shape == (batch, int(dims.sum()))
        if batch == 0:
            continue
        ref, scale = forward_reference(tables, batch, ind, off, wts, True)
        err = np.abs(y.cpu().double().numpy() - ref)
        assert (err <= 2e-3 * scale + 1e-30).all(), k
        go = torch.randn(batch, int(dims.sum()), generator=g)
        gr = m.backward(ind.to(DEV), off.to(DEV), go.to(DEV), wts.to(DEV))
        torch.cuda.synchronize()
        res, sc = backward_reference(rows, dims, batch, ind, off, go, wts, True)
        assert_backward_matches(gr, res, sc, what=f"shape {k}")
