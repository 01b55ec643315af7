"""Pins of the fp64 oracle of the row-wise optimizer step (CPU).

The storage roundings are checked on every bit pattern against the formats
(and numpy's correctly rounded float64 -> float16 conversion); the step itself
against hand-worked values and, for SGD, against the dense gradient of torch's
autograd through embedding_bag.
"""

import numpy as np
import pytest
import torch

import oracle
from tests.conftest import parse_value
from tests.helpers import random_problem, torch_dense_grad_f64


def test_half_rounding_on_every_pattern_and_midpoint():
    bits = np.arange(0x7c00, dtype=np.uint16)  # every finite non-negative half
    vals = bits.view(np.float16).astype(np.float64)
    conv = np.vectorize(oracle.double_to_half_bits)
    assert (conv(vals) == bits).all()
    assert (conv(-vals[1:]) == (bits[1:] | 0x8000)).all()
    mids = (vals[:-1] + vals[1:]) / 2  # exact in float64: ties go to the even pattern
    want = np.where(bits[:-1] % 2 == 0, bits[:-1], bits[1:])
    assert (conv(mids) == want).all()
    # just off the ties, and numpy's own correctly rounded conversion
    off = np.concatenate([np.nextafter(mids, 0), np.nextafter(mids, np.inf)])
    assert (conv(off) == off.astype(np.float16).view(np.uint16)).all()
    assert oracle.double_to_half_bits(65520.0) == 0x7c00 and oracle.double_to_half_bits(1e9) == 0x7c00


def test_bf16_rounding_on_every_pattern_and_midpoint():
    bits = np.arange(0x7f80, dtype=np.uint32)  # every finite non-negative bfloat16
    vals = (bits << 16).astype(np.uint32).view(np.float32).astype(np.float64)
    conv = np.vectorize(oracle.double_to_bf16_bits)
    assert (conv(vals) == bits).all()
    mids = (vals[:-1] + vals[1:]) / 2  # 9 significant bits: exact in float32 too
    want = np.where(bits[:-1] % 2 == 0, bits[:-1], bits[1:])
    assert (conv(mids) == want).all()
    # off the ties by one float32 ulp: torch's float32 -> bfloat16 rounding
    for direction in (0.0, np.inf):
        off = np.nextafter(mids.astype(np.float32), np.float32(direction))
        want = torch.from_numpy(off).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
        assert (conv(off.astype(np.float64)) == want).all()


def _hand(golden):
    g = golden("optimizer_hand.json")
    table = torch.tensor(g["table"], dtype=torch.float32)
    args = (g["batch"], torch.tensor(g["indices"]), torch.tensor(g["offsets"]),
            torch.tensor(g["grad_out"], dtype=torch.float32))
    return g, table, args


def test_sgd_hand_worked(golden):
    g, table, args = _hand(golden)
    (new,), _ = oracle.apply_step([table], *args, kind="sgd", lr=0.5)
    assert new.tolist() == g["sgd_lr_0.5"]


@pytest.mark.parametrize("case", ["adagrad_state0", "adagrad_state53"])
def test_adagrad_hand_worked(golden, case):
    g, table, args = _hand(golden)
    c = g[case]
    (new,), (st,) = oracle.apply_step([table], *args, kind="adagrad", lr=1.0, eps=0.0,
                                      state=[np.array(c["state"], np.float32)])
    want = np.array([[parse_value(v) for v in row] for row in c["table"]], dtype=np.float64)
    np.testing.assert_array_equal(new.numpy(), want.astype(np.float32))
    assert st.tolist() == c["new_state"]


@pytest.mark.parametrize("weighted,mean", [(False, False), (True, True)])
def test_sgd_equals_the_dense_autograd_gradient(weighted, mean):
    # lr = 1 on integer fp32 data: E - G is exact for sum pooling (and within
    # one fp64 rounding for mean), so the step must equal E minus torch's dense
    # gradient once rounded to the fp32 storage.
    tables, ind, off, w = random_problem(71, int_valued=True, weighted=weighted, max_len=8)
    go = torch.randint(-8, 9, (9, 48), generator=torch.Generator().manual_seed(8)).float()
    new, _ = oracle.apply_step(tables, 9, ind, off, go, weights=w, mean=mean, kind="sgd", lr=1.0)
    dense = torch_dense_grad_f64(tables, 9, ind, off, go, w, mean)
    for t0, t1, d in zip(tables, new, dense):
        want = (t0.double() - d).float()
        assert torch.equal(t1, want)


def test_sgd_half_storage_rounds_once():
    tables, ind, off, _ = random_problem(72, dims=(8, 16), rows=(20, 30), int_valued=True,
                                         dtype=torch.float16, max_len=6)
    go = torch.randint(-8, 9, (9, 24), generator=torch.Generator().manual_seed(9)).float()
    lr = 2.0 ** -7
    new, _ = oracle.apply_step(tables, 9, ind, off, go, kind="sgd", lr=lr)
    dense = torch_dense_grad_f64(tables, 9, ind, off, go)
    for t0, t1, d in zip(tables, new, dense):
        exact = t0.double().numpy() - lr * d.numpy()  # exact in float64
        np.testing.assert_array_equal(t1.numpy(), exact.astype(np.float16))


def test_untouched_rows_and_state_are_unchanged():
    tables, ind, off, _ = random_problem(73, rows=(50, 60, 70), max_len=3)
    go = torch.randn(9, 48, generator=torch.Generator().manual_seed(10))
    state = [np.full(r, 0.5, np.float32) for r in (50, 60, 70)]
    new, st = oracle.apply_step(tables, 9, ind, off, go, kind="adagrad", lr=0.1, state=state)
    for t in range(3):
        s_, e_ = int(off[t * 9]), int(off[(t + 1) * 9])
        touched = np.zeros(tables[t].shape[0], bool)
        touched[ind[s_:e_].numpy()] = True
        assert torch.equal(new[t][~torch.from_numpy(touched)], tables[t][~torch.from_numpy(touched)])
        assert (st[t][~touched] == 0.5).all() and (st[t][touched] > 0.5).all()
