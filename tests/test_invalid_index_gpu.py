"""Out-of-range indices through every backward entry point, against the fp64 oracle.

The boundary's contract: a lookup whose index is negative or >= rows_t contributes
nothing and sets CB_ERR_INDEX_OOB (returned at once under CB_VALIDATE, else by
cb_tbe_get_error). For the backward that means no gradient for it, no gradient row
for its (clamped or any other) row unless a valid lookup touches that row, and no
optimizer step from it. The expected values are the oracle's on the same batch with
those lookups removed; mean pooling keeps the forward's bag length L (the removed
lookups still count in it), so the oracle's batch is then sum-pooled with weights
w_i / L.
"""

import numpy as np
import pytest
import torch

import oracle
from tests.helpers import (assert_backward_matches, backward_reference, bag_of_positions,
                           inject_out_of_range,
                           random_problem, storage_ulp, table_meta, without_lookups)

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")

# Small tables whose rows 0 and rows_t - 1 valid lookups also touch, and a large
# one where they are almost surely untouched: a clamp onto either row would show
# as a wrong value in the first and as an extra gradient row in the second.
ROWS = (5, 300, 100_000)
DIMS = (8, 64, 128)
B = 40


def _problem(seed, int_valued, weighted):
    tables, ind, off, w = random_problem(seed, dims=DIMS, rows=ROWS, batch=B, max_len=200,
                                         int_valued=int_valued, weighted=weighted, empty_frac=0.15)
    bad_ind, bad = inject_out_of_range(tables, ind, off, B, seed + 1, frac=0.06)
    assert bad.sum() > 20
    g = torch.Generator().manual_seed(seed + 2)
    sd = int(sum(DIMS))
    go = (torch.randint(-8, 9, (B, sd), generator=g).to(torch.float32) if int_valued
          else torch.randn(B, sd, generator=g))
    return tables, bad_ind, off, w, go, bad


def _module(tables, mean, validate):
    from paper_2609_30656_gb300.tbe import TBE
    return TBE([t.to(DEV).contiguous().clone() for t in tables], pooling="mean" if mean else "sum",
               validate=validate)


CASES = [  # (int_valued, weighted, mean)
    (True, False, False),
    (True, True, False),
    (False, False, True),
    (False, True, True),
]


@pytest.mark.parametrize("validate", [False, True])
@pytest.mark.parametrize("int_valued,weighted,mean", CASES)
def test_backward_drops_out_of_range_lookups(int_valued, weighted, mean, validate):
    from paper_2609_30656_gb300.tbe import CB_ERR_INDEX_OOB, CbTbeError
    tables, ind, off, w, go, bad = _problem(51, int_valued, weighted)
    m = _module(tables, mean, validate)
    args = (ind.to(DEV), off.to(DEV), go.to(DEV), None if w is None else w.to(DEV))
    if validate:
        g = m.alloc_grad(ind.numel(), ind.numel() * max(DIMS))
        with pytest.raises(CbTbeError) as e:
            m.backward_into(g, *args)
        assert e.value.status == CB_ERR_INDEX_OOB
    else:
        g = m.backward(*args)
        assert m.get_error() == CB_ERR_INDEX_OOB
    torch.cuda.synchronize()
    rows, dims = table_meta(tables)
    k_ind, k_off, k_w = without_lookups(ind, off, w, bad, mean)
    res, scale = backward_reference(rows, dims, B, k_ind, k_off, go, k_w, False)
    # integer data, sum pooling: every partial sum is exact, so every bit agrees
    assert_backward_matches(g, res, scale, rtol=0.0 if int_valued else 1e-5,
                            what=f"int={int_valued} w={weighted} mean={mean} validate={validate}")
    # the rows a clamp would have hit: 0 and rows_t - 1 of the large table are
    # not in the gradient unless a valid lookup touched them
    t = 2
    row_base = int(sum(ROWS[:t]))
    ids = g.unique_ids[:g.num_unique].cpu().numpy()
    for r in (0, ROWS[t] - 1):
        touched = bool(((k_ind[int(k_off[t * B]):int(k_off[(t + 1) * B])]) == r).any())
        assert (row_base + r in set(ids.tolist())) == touched


def _apply_expected(tables, ind, off, w, go, bad, mean, optimizer, lr, eps, state):
    k_ind, k_off, k_w = without_lookups(ind, off, w, bad, mean)
    want, want_state = oracle.apply_step(tables, B, k_ind, k_off, go, weights=k_w, mean=False,
                                         kind=optimizer, lr=lr, eps=eps, state=state)
    rows, dims = table_meta(tables)
    res = oracle.backward(rows, dims, B, k_ind, k_off, go, weights=k_w)
    _, sg = backward_reference(rows, dims, B, k_ind, k_off, go, k_w, False)
    return want, want_state, res, sg


def _compare_tables(got, want, want_state, res, sg, tables, optimizer, lr, eps, exact):
    rows, _ = table_meta(tables)
    row_base = np.concatenate([[0], np.cumsum(rows)])
    for t in range(len(tables)):
        g0, g1, e0 = got[t].double().numpy(), want[t].double().numpy(), tables[t].double().numpy()
        touched = np.zeros(g0.shape[0], bool)
        u0, u1 = int(res.table_offsets[t]), int(res.table_offsets[t + 1])
        touched[(res.uniq[u0:u1] - row_base[t]).astype(np.int64)] = True
        # rows no valid lookup touches are not written at all, clamp targets included
        np.testing.assert_array_equal(g0[~touched], e0[~touched])
        if exact:
            np.testing.assert_array_equal(g0, g1)
            continue
        tol = np.zeros_like(g0)
        for u in range(u0, u1):
            r = int(res.uniq[u] - row_base[t])
            a, b = int(res.grad_offsets[u]), int(res.grad_offsets[u + 1])
            scale = lr if optimizer == "sgd" else lr / (np.sqrt(want_state[t][r]) + eps)
            tol[r] = 2e-5 * abs(scale) * sg[a:b] + 2e-6 * abs(scale) * np.abs(res.grads[a:b]).max()
        tol += storage_ulp(g1, tables[t].dtype)
        bad = np.abs(g0 - g1) > tol
        assert not bad.any(), (t, np.argwhere(bad)[:3], g0[bad][:3], g1[bad][:3])


@pytest.mark.parametrize("validate", [False, True])
@pytest.mark.parametrize("two_pass", [False, True])
@pytest.mark.parametrize("optimizer,int_valued,mean", [("sgd", True, False), ("sgd", False, True),
                                                       ("adagrad", False, False),
                                                       ("adagrad", False, True)])
def test_optimizer_step_ignores_out_of_range_lookups(optimizer, int_valued, mean, two_pass, validate):
    from paper_2609_30656_gb300.tbe import CB_ERR_INDEX_OOB, CbTbeError
    tables, ind, off, w, go, bad = _problem(52, int_valued, weighted=True)
    lr = 2.0 ** -3 if int_valued else 0.05
    eps = 1e-8
    state = None
    if optimizer == "adagrad":
        g = torch.Generator().manual_seed(53)
        state = [torch.rand(r, generator=g).numpy().astype(np.float32) for r in ROWS]
    m = _module(tables, mean, validate)
    dev_state = None if state is None else [torch.from_numpy(s).to(DEV) for s in state]
    args = (ind.to(DEV), off.to(DEV), go.to(DEV), w.to(DEV))
    if two_pass:
        sg_buf = m.alloc_grad(ind.numel(), ind.numel() * max(DIMS))
        if validate:
            with pytest.raises(CbTbeError) as e:
                m.backward_into(sg_buf, *args)
            assert e.value.status == CB_ERR_INDEX_OOB
        else:
            m.backward_into(sg_buf, *args)
        m.apply_sparse(sg_buf, optimizer=optimizer, lr=lr, eps=eps, state=dev_state)
    elif validate:
        with pytest.raises(CbTbeError) as e:
            m.backward_apply(*args, optimizer=optimizer, lr=lr, eps=eps, state=dev_state)
        assert e.value.status == CB_ERR_INDEX_OOB
    else:
        m.backward_apply(*args, optimizer=optimizer, lr=lr, eps=eps, state=dev_state)
    if not validate:
        assert m.get_error() == CB_ERR_INDEX_OOB
    torch.cuda.synchronize()
    got = [t.cpu() for t in m.tables]
    got_state = None if dev_state is None else [s.cpu().numpy() for s in dev_state]
    want, want_state, res, sg = _apply_expected(tables, ind, off, w, go, bad, mean, optimizer, lr, eps,
                                                state)
    _compare_tables(got, want, want_state, res, sg, tables, optimizer, lr, eps,
                    exact=int_valued and optimizer == "sgd")
    if optimizer == "adagrad":
        for s0, s1 in zip(got_state, want_state):
            np.testing.assert_allclose(s0, s1, rtol=2e-5, atol=0)


def test_only_out_of_range_lookups_in_a_table():
    # Table 1 has no valid lookup at all: its spare-key run is the only run of the
    # table; table 0's gradient and table 2's must be untouched by it.
    from paper_2609_30656_gb300.tbe import CB_ERR_INDEX_OOB
    tables, ind, off, w, go, _ = _problem(54, True, False)
    s, e = int(off[1 * B]), int(off[2 * B])
    ind = ind.clone()
    ind[s:e] = torch.where(torch.arange(e - s) % 2 == 0, -1, ROWS[1])
    table_of = bag_of_positions(off) // B
    bad = (ind < 0) | (ind >= torch.tensor(ROWS)[table_of])
    m = _module(tables, False, False)
    g = m.backward(ind.to(DEV), off.to(DEV), go.to(DEV))
    assert m.get_error() == CB_ERR_INDEX_OOB
    rows, dims = table_meta(tables)
    k_ind, k_off, _ = without_lookups(ind, off, None, bad, False)
    res, scale = backward_reference(rows, dims, B, k_ind, k_off, go, None, False)
    assert res.table_offsets[2] == res.table_offsets[1]  # no row of table 1
    assert_backward_matches(g, res, scale, rtol=0.0)
