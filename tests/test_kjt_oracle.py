"""Pins of the batch-replication oracle (CPU): identity at factor 1, sizes, and
the pooled output of a replicated batch equal to the small batch's output
repeated along the batch (the preprocessor must keep what the lookup sees)."""

import numpy as np
import torch

import oracle
from tests.helpers import random_problem


def test_factor_one_is_the_identity():
    tables, ind, off, w = random_problem(91, weighted=True)
    i2, o2, w2 = oracle.replicate_kjt(ind, off, w, 3, 1)
    np.testing.assert_array_equal(i2, ind.numpy())
    np.testing.assert_array_equal(o2, off.numpy())
    np.testing.assert_array_equal(w2, w.numpy())


def test_hand_worked_layout():
    # 2 tables, B = 2: t0 bags [5] [], t1 bags [1, 2] [3]
    ind = np.array([5, 1, 2, 3], np.int64)
    off = np.array([0, 1, 1, 3, 4], np.int64)
    i2, o2, _ = oracle.replicate_kjt(ind, off, None, 2, 2)
    assert i2.tolist() == [5, 5, 1, 2, 3, 1, 2, 3]
    assert o2.tolist() == [0, 1, 1, 2, 2, 4, 5, 7, 8]


def test_sizes_and_the_pooled_output_repeat():
    tables, ind, off, w = random_problem(92, weighted=True, max_len=20)
    F = 3
    i2, o2, w2 = oracle.replicate_kjt(ind, off, w, 3, F)
    assert i2.shape[0] == F * ind.numel() and o2.shape[0] == 3 * 9 * F + 1
    y = oracle.forward(tables, 9, ind, off, weights=w, mean=True)
    y2 = oracle.forward(tables, 9 * F, torch.from_numpy(i2), torch.from_numpy(o2),
                        weights=torch.from_numpy(w2), mean=True)
    for r in range(F):
        np.testing.assert_array_equal(y2[r * 9:(r + 1) * 9], y)
