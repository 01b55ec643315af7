"""The optimizer step through the C ABI against the fp64 oracle: fused into the
backward (cb_tbe_backward_apply), and as a second pass over the gradient the
backward wrote (cb_tbe_apply_sparse), which must give the same bits."""

import numpy as np
import pytest
import torch

import oracle
from tests.conftest import parse_value
from tests.helpers import backward_reference, random_problem, storage_ulp, table_meta
from paper_2609_30656_gb300 import workloads as wl

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")
U32 = 2.0 ** -24


_ulp = storage_ulp


def _run(tables, batch, ind, off, go, w, mean, optimizer, lr, eps=1e-8, state=None, two_pass=False):
    from paper_2609_30656_gb300.tbe import TBE
    dev_tabs = [t.to(DEV).contiguous().clone() for t in tables]
    m = TBE(dev_tabs, pooling="mean" if mean else "sum", validate=True)
    dev_state = None if state is None else [torch.from_numpy(s).to(DEV) for s in state]
    args = (ind.to(DEV), off.to(DEV), go.to(DEV), None if w is None else w.to(DEV))
    if two_pass:
        m.apply_sparse(m.backward(*args), optimizer=optimizer, lr=lr, eps=eps, state=dev_state)
    else:
        m.backward_apply(*args, optimizer=optimizer, lr=lr, eps=eps, state=dev_state)
    torch.cuda.synchronize()
    return [t.cpu() for t in dev_tabs], (None if dev_state is None else [s.cpu().numpy() for s in dev_state])


def _check(tables, batch, ind, off, go, w, mean, optimizer, lr, eps=1e-8, state=None, exact=False,
           two_pass=False):
    got, got_state = _run(tables, batch, ind, off, go, w, mean, optimizer, lr, eps, state, two_pass)
    want, want_state = oracle.apply_step(tables, batch, ind, off, go, weights=w, mean=mean,
                                         kind=optimizer, lr=lr, eps=eps, state=state)
    rows, dims = table_meta(tables)
    _, sg = backward_reference(rows, dims, batch, ind, off, go, w, mean)
    res = oracle.backward(rows, dims, batch, ind, off, go, weights=w, mean=mean)
    row_base = np.concatenate([[0], np.cumsum(rows)])
    for t in range(len(tables)):
        g0, g1, e0 = got[t].double().numpy(), want[t].double().numpy(), tables[t].double().numpy()
        if exact:
            np.testing.assert_array_equal(g0, g1)
            continue
        # allowance: the fp32 gradient's error (1e-5 of its condition scale)
        # times the step's scale, plus one rounding of the storage type
        tol = np.zeros_like(g0)
        for u in range(int(res.table_offsets[t]), int(res.table_offsets[t + 1])):
            r = int(res.uniq[u] - row_base[t])
            s_g = sg[res.grad_offsets[u]:res.grad_offsets[u + 1]]
            scale = lr if optimizer == "sgd" else lr / (np.sqrt(want_state[t][r]) + eps)
            tol[r] = 2e-5 * abs(scale) * s_g + 2e-6 * abs(scale) * np.abs(
                res.grads[res.grad_offsets[u]:res.grad_offsets[u + 1]]).max()
        tol += _ulp(g1, tables[t].dtype)
        bad = np.abs(g0 - g1) > tol
        assert not bad.any(), (t, np.argwhere(bad)[:3], g0[bad][:3], g1[bad][:3])
        # rows the batch does not touch are not written at all
        touched = np.zeros(g0.shape[0], bool)
        touched[(res.uniq[res.table_offsets[t]:res.table_offsets[t + 1]] - row_base[t]).astype(np.int64)] = True
        np.testing.assert_array_equal(g0[~touched], e0[~touched])
    if optimizer == "adagrad":
        for s0, s1 in zip(got_state, want_state):
            np.testing.assert_allclose(s0, s1, rtol=2e-5, atol=0)


@pytest.mark.parametrize("two_pass", [False, True])
@pytest.mark.parametrize("case", ["sgd", "adagrad_state0", "adagrad_state53"])
def test_hand_worked(golden, case, two_pass):
    g = golden("optimizer_hand.json")
    table = torch.tensor(g["table"], dtype=torch.float32)
    args = (g["batch"], torch.tensor(g["indices"]), torch.tensor(g["offsets"]),
            torch.tensor(g["grad_out"], dtype=torch.float32), None, False)
    if case == "sgd":
        (new,), _ = _run([table], *args, "sgd", 0.5, two_pass=two_pass)
        assert new.tolist() == g["sgd_lr_0.5"]
        return
    c = g[case]
    (new,), (st,) = _run([table], *args, "adagrad", 1.0, eps=0.0,
                         state=[np.array(c["state"], np.float32)], two_pass=two_pass)
    want = np.array([[parse_value(v) for v in row] for row in c["table"]], dtype=np.float64)
    # The fp32 step rounds lr / (sqrt(m) + eps) and then E - scale * G: two
    # roundings, so a value like 1 - 2/3 may land one fp32 spacing away.
    np.testing.assert_allclose(new.double().numpy(), want, rtol=0, atol=2 * 2.0 ** -23 * 4)
    if case == "adagrad_state0":
        np.testing.assert_array_equal(new.numpy(), want.astype(np.float32))  # scale 1/2 is exact
    assert st.tolist() == c["new_state"]


@pytest.mark.parametrize("dtype", [torch.float32, torch.float16, torch.bfloat16])
@pytest.mark.parametrize("optimizer", ["sgd", "adagrad"])
@pytest.mark.parametrize("weighted,mean", [(False, False), (True, True)])
def test_random_within_tolerance(dtype, optimizer, weighted, mean):
    dims = (8, 64, 128, 256, 512)
    tables, ind, off, w = random_problem(81, dims=dims, rows=(5, 100, 1000, 64, 7), batch=37,
                                         max_len=900, dtype=dtype, weighted=weighted, empty_frac=0.3)
    go = torch.randn(37, sum(dims), generator=torch.Generator().manual_seed(11))
    state = None
    if optimizer == "adagrad":
        rng = np.random.default_rng(12)
        state = [rng.uniform(0, 2, t.shape[0]).astype(np.float32) for t in tables]
    _check(tables, 37, ind, off, go, w, mean, optimizer, lr=0.05, state=state)


@pytest.mark.parametrize("two_pass", [False, True])
@pytest.mark.parametrize("dtype", [torch.float32, torch.float16])
def test_sgd_integer_data_bit_exact_with_split_runs(dtype, two_pass):
    # Few rows, long bags: runs cross many chunks (fix-up and block-wide
    # combine); integers and a power-of-two step make every value exact
    # before the one rounding to storage.
    tables, ind, off, _ = random_problem(82, dims=(64, 128, 8), rows=(3, 40, 2000), batch=50,
                                         max_len=600, int_valued=True, dtype=dtype)
    go = torch.randint(-8, 9, (50, 200), generator=torch.Generator().manual_seed(13)).float()
    _check(tables, 50, ind, off, go, None, False, "sgd", lr=2.0 ** -7, exact=True, two_pass=two_pass)


@pytest.mark.parametrize("two_pass", [False, True])
def test_adagrad_split_runs_within_tolerance(two_pass):
    tables, ind, off, w = random_problem(83, dims=(64, 128, 8), rows=(3, 40, 2000), batch=50,
                                         max_len=600, weighted=True)
    go = torch.randn(50, 200, generator=torch.Generator().manual_seed(14))
    state = [np.zeros(t.shape[0], np.float32) for t in tables]
    _check(tables, 50, ind, off, go, w, False, "adagrad", lr=0.1, eps=1e-6, state=state, two_pass=two_pass)


def test_bad_arguments_are_rejected():
    from paper_2609_30656_gb300.tbe import CbTbeError, TBE
    tables, ind, off, _ = random_problem(84)
    m = TBE([t.to(DEV) for t in tables])
    go = torch.zeros(9, 48, device=DEV)
    with pytest.raises(ValueError):
        m.backward_apply(ind.to(DEV), off.to(DEV), go, optimizer="adagrad")  # no state
    lib = m._lib
    assert lib.cb_tbe_backward_apply(m._h, 9, 0, 0, 0, None, None, 7, 0.1, 0.0, None, None) != 0


def test_cfg2_full_size_sgd():
    # 8 x 100k x 128 fp32, batch 2048, Poisson(20) bags, Zipf(1.05): hot rows
    # repeat across many chunks.
    w = wl.get_workload("cfg2")
    tables = [t.cpu() for t in wl.make_tables(w, 0, "cpu")]
    b = wl.make_batch(w, 0, "cpu")
    go = wl.make_grad_out(w, 0, "cpu")
    _check(tables, w.batch, b.indices, b.offsets, go, None, False, "sgd", lr=0.02)


# ---------------------------------------------------------------- two-pass step

@pytest.mark.parametrize("dtype", [torch.float32, torch.float16, torch.bfloat16])
@pytest.mark.parametrize("optimizer", ["sgd", "adagrad"])
@pytest.mark.parametrize("dims,rows", [((8, 64, 128), (5, 300, 3000)),          # one column slot per lane
                                       ((8, 256, 64), (40, 200, 7)),            # two
                                       ((512, 128, 16), (64, 1000, 3))])        # four; runs split across chunks
def test_two_pass_equals_fused_bit_for_bit(dtype, optimizer, dims, rows):
    tables, ind, off, w = random_problem(85, dims=dims, rows=rows, batch=41, max_len=1200, dtype=dtype,
                                         weighted=True, empty_frac=0.2)
    go = torch.randn(41, sum(dims), generator=torch.Generator().manual_seed(15))
    state = None
    if optimizer == "adagrad":
        rng = np.random.default_rng(16)
        state = [rng.uniform(0, 2, t.shape[0]).astype(np.float32) for t in tables]
    a, sa = _run(tables, 41, ind, off, go, w, True, optimizer, 0.05, 1e-7, state)
    b, sb = _run(tables, 41, ind, off, go, w, True, optimizer, 0.05, 1e-7, state, two_pass=True)
    for x, y in zip(a, b):
        assert torch.equal(x.view(torch.int16 if x.element_size() == 2 else torch.int32),
                           y.view(torch.int16 if y.element_size() == 2 else torch.int32))
    if state is not None:
        for x, y in zip(sa, sb):
            np.testing.assert_array_equal(x.view(np.int32), y.view(np.int32))


@pytest.mark.parametrize("optimizer", ["sgd", "adagrad"])
def test_two_pass_random_within_tolerance(optimizer):
    dims = (8, 64, 128, 256, 512)
    tables, ind, off, w = random_problem(86, dims=dims, rows=(5, 100, 1000, 64, 7), batch=37,
                                         max_len=900, dtype=torch.bfloat16, weighted=True, empty_frac=0.3)
    go = torch.randn(37, sum(dims), generator=torch.Generator().manual_seed(17))
    state = None
    if optimizer == "adagrad":
        state = [np.random.default_rng(18).uniform(0, 2, t.shape[0]).astype(np.float32) for t in tables]
    _check(tables, 37, ind, off, go, w, True, optimizer, lr=0.05, state=state, two_pass=True)


def test_two_pass_after_a_capacity_error_writes_nothing():
    from paper_2609_30656_gb300.tbe import CB_ERR_CAPACITY, TBE
    tables, ind, off, _ = random_problem(87, dims=(16, 64), rows=(50, 400), batch=20, max_len=30)
    dev_tabs = [t.to(DEV).clone() for t in tables]
    m = TBE(dev_tabs)
    go = torch.randn(20, 80, device=DEV)
    g = m.alloc_grad(4, 4 * 64)  # far fewer rows than the batch touches
    m.backward_into(g, ind.to(DEV), off.to(DEV), go)
    m.apply_sparse(g, optimizer="sgd", lr=1.0)
    assert m.get_error() == CB_ERR_CAPACITY
    for t0, t1 in zip(dev_tabs, tables):
        assert torch.equal(t0.cpu(), t1)


def test_two_pass_bad_arguments_are_rejected():
    from paper_2609_30656_gb300.tbe import CbSparseGrad, TBE
    tables, ind, off, _ = random_problem(88)
    m = TBE([t.to(DEV) for t in tables])
    g = m.backward(ind.to(DEV), off.to(DEV), torch.zeros(9, 48, device=DEV))
    with pytest.raises(ValueError):
        m.apply_sparse(g, optimizer="adagrad")  # no state
    with pytest.raises(ValueError):
        m.apply_sparse(m.alloc_grad(0, 0, size_only=True))
    lib = m._lib
    cs = CbSparseGrad(g.unique_ids.data_ptr(), g.table_offsets.data_ptr(), g.grad_offsets.data_ptr(),
                      g.grads.data_ptr() + 4, 10, 100, g.num_unique_dev.data_ptr(), g.num_floats_dev.data_ptr())
    import ctypes
    assert lib.cb_tbe_apply_sparse(m._h, ctypes.byref(cs), 0, 0.1, 0.0, None, None) != 0  # misaligned grads
    cs.grads = g.grads.data_ptr()
    assert lib.cb_tbe_apply_sparse(m._h, ctypes.byref(cs), 5, 0.1, 0.0, None, None) != 0  # unknown kind
    assert lib.cb_tbe_apply_sparse(m._h, ctypes.byref(cs), 1, 0.1, 0.0, None, None) != 0  # adagrad, no state
    assert lib.cb_tbe_apply_sparse(m._h, None, 0, 0.1, 0.0, None, None) != 0


def test_cfg2_full_size_two_pass_equals_fused():
    w = wl.get_workload("cfg2")
    tables = [t.cpu() for t in wl.make_tables(w, 0, "cpu")]
    b = wl.make_batch(w, 0, "cpu")
    go = wl.make_grad_out(w, 0, "cpu")
    state = [np.zeros(t.shape[0], np.float32) for t in tables]
    a, sa = _run(tables, w.batch, b.indices, b.offsets, go, None, False, "adagrad", 0.02, 1e-8, state)
    c, sc = _run(tables, w.batch, b.indices, b.offsets, go, None, False, "adagrad", 0.02, 1e-8, state,
                 two_pass=True)
    for x, y in zip(a, c):
        assert torch.equal(x, y)
    for x, y in zip(sa, sc):
        np.testing.assert_array_equal(x, y)


def test_two_pass_skips_rows_that_are_not_this_handles():
    # A gradient written by a handle over a 1000-row table, applied through a
    # handle over a 10-row table: ids >= 10 are skipped and reported, ids < 10
    # are stepped as usual; nothing outside the small table is touched.
    from paper_2609_30656_gb300.tbe import CB_ERR_INDEX_OOB, TBE
    g_ = torch.Generator().manual_seed(19)
    big = (torch.randn(1000, 16, generator=g_) * 0.01).to(DEV)
    small_host = (torch.randn(10, 16, generator=g_) * 0.01)
    small = small_host.to(DEV)
    off = torch.tensor([0, 3, 7, 12], dtype=torch.int64)
    ind = torch.tensor([1, 5, 900, 2, 2, 999, 7, 10, 3, 4, 500, 9], dtype=torch.int64)
    go = torch.randn(3, 16, generator=g_)
    m_big, m_small = TBE([big]), TBE([small])
    g = m_big.backward(ind.to(DEV), off.to(DEV), go.to(DEV))
    m_small.apply_sparse(g, optimizer="sgd", lr=1.0)
    assert m_small.get_error() == CB_ERR_INDEX_OOB
    ids = g.unique_ids[:g.num_unique].cpu()
    offs = g.grad_offsets[:g.num_unique].cpu()
    grads = g.grads[:g.num_floats].cpu()
    want = small_host.clone()
    for k, r in enumerate(ids.tolist()):
        if r < 10:
            want[r] -= grads[int(offs[k]):int(offs[k]) + 16]
    assert torch.equal(small.cpu(), want)
