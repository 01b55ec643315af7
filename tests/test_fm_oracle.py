"""Pins of the fp64 oracle of the factorization-machine cross term (CPU).

The oracle writes the pairwise definition fm[b] = sum_{t<u} <v_bt, v_bu> and
its gradient sum_{u != t} v_bu directly. These tests tie it to things fixed
independently of that code: a case worked by hand, the closed form
1/2 [(sum_t v)^2 - sum_t v^2] (a different formula), one- and two-field special
cases, exact finite differences (fm is linear in every single coordinate),
Euler's identity for a function homogeneous of degree 2, and the row stride.
"""

import numpy as np
import pytest

import oracle


def _closed_form(y, T):
    B = y.shape[0]
    v = y[:, :y.shape[1] // T * T].astype(np.float64).reshape(B, T, -1)
    return 0.5 * ((v.sum(1) ** 2) - (v ** 2).sum(1)).sum(-1)


def test_hand_worked_three_fields():
    # v0 = (1, 2), v1 = (3, 4), v2 = (5, 6):
    # <v0,v1> + <v0,v2> + <v1,v2> = 11 + 17 + 39 = 67.
    y = np.array([[1, 2, 3, 4, 5, 6]], dtype=np.float32)
    assert oracle.fm_forward(y, 3).tolist() == [67.0]
    # gradient, upstream g = 2: 2 * (v1 + v2), 2 * (v0 + v2), 2 * (v0 + v1)
    g = oracle.fm_backward(y, np.array([2.0], dtype=np.float32), 3)
    assert g.tolist() == [[16.0, 20.0, 12.0, 16.0, 8.0, 12.0]]


def test_one_field_is_zero_and_two_fields_is_a_dot_product():
    rng = np.random.default_rng(1)
    y1 = rng.standard_normal((5, 16)).astype(np.float32)
    assert (oracle.fm_forward(y1, 1) == 0).all()
    assert (oracle.fm_backward(y1, np.ones(5, np.float32), 1) == 0).all()
    y2 = rng.standard_normal((5, 32)).astype(np.float32)
    want = (y2[:, :16].astype(np.float64) * y2[:, 16:].astype(np.float64)).sum(1)
    np.testing.assert_allclose(oracle.fm_forward(y2, 2), want, rtol=1e-13, atol=0)


@pytest.mark.parametrize("T,D", [(3, 4), (26, 8), (100, 16), (7, 128)])
def test_matches_the_closed_form(T, D):
    rng = np.random.default_rng(T * 1000 + D)
    y = rng.standard_normal((9, T * D)).astype(np.float32)
    got = oracle.fm_forward(y, T)
    scale = 0.5 * ((np.abs(y.astype(np.float64)).reshape(9, T, D).sum(1) ** 2)).sum(-1)
    assert (np.abs(got - _closed_form(y, T)) <= 1e-13 * scale).all()


def test_integer_inputs_are_exact():
    rng = np.random.default_rng(3)
    y = rng.integers(-8, 9, (11, 20 * 8)).astype(np.float32)
    np.testing.assert_array_equal(oracle.fm_forward(y, 20), _closed_form(y, 20))


def test_gradient_equals_exact_finite_differences():
    # fm has no square of a single coordinate, so it is linear in each one:
    # fm(y + e_k) - fm(y) is exactly d fm / d y_k (integers keep it exact).
    rng = np.random.default_rng(4)
    T, D = 6, 4
    y = rng.integers(-8, 9, (3, T * D)).astype(np.float32)
    g = np.ones(3, dtype=np.float32)
    grad = oracle.fm_backward(y, g, T)
    base = oracle.fm_forward(y, T)
    for k in range(T * D):
        yp = y.copy()
        yp[:, k] += 1.0
        np.testing.assert_array_equal(oracle.fm_forward(yp, T) - base, grad[:, k])


def test_euler_identity_and_upstream_scaling():
    # fm is homogeneous of degree 2: sum_k y_k * d fm / d y_k = 2 fm.
    rng = np.random.default_rng(5)
    T, D = 10, 8
    y = rng.standard_normal((4, T * D)).astype(np.float32)
    g = rng.standard_normal(4).astype(np.float32)
    grad = oracle.fm_backward(y, g, T)
    lhs = (y.astype(np.float64) * grad).sum(1)
    rhs = 2.0 * g.astype(np.float64) * oracle.fm_forward(y, T)
    np.testing.assert_allclose(lhs, rhs, rtol=1e-12, atol=1e-12)


def test_row_stride_ignores_trailing_columns():
    rng = np.random.default_rng(6)
    y = rng.standard_normal((4, 5 * 8)).astype(np.float32)
    wide = np.concatenate([y, rng.standard_normal((4, 24)).astype(np.float32)], axis=1)
    lib = oracle._load()
    out = np.zeros(4)
    assert lib.fm_oracle_forward(4, 5, 8, wide.shape[1], oracle._ptr(np.ascontiguousarray(wide)),
                                 oracle._ptr(out)) == 0
    np.testing.assert_array_equal(out, oracle.fm_forward(y, 5))


def test_bad_shapes_are_rejected():
    with pytest.raises(ValueError):
        oracle.fm_forward(np.zeros((2, 10), np.float32), 3)
    with pytest.raises(ValueError):
        oracle.fm_backward(np.zeros((2, 12), np.float32), np.zeros(3, np.float32), 3)
