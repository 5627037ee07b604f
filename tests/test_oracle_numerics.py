"""Pins for the oracle's scalar arithmetic: exp, the margin (dot product) and
the loss derivatives.  Each check compares against mathematics (fp64 values,
exact integer sums, closed forms), never against a retyped copy of the
oracle's own formula."""
import math

import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _ulp_err(got, ref64):
    ulp = np.spacing(np.abs(ref64).astype(np.float32)).astype(np.float64)
    return np.abs(got.astype(np.float64) - ref64) / ulp


def test_expf_within_2ulp_dense_grid():
    x = np.linspace(-87.0, 88.5, 2_000_001, dtype=np.float64).astype(np.float32)
    err = _ulp_err(oracle.expf(x), np.exp(x.astype(np.float64)))
    assert err.max() <= 2.0, err.max()


def test_expf_within_2ulp_random_and_small():
    rng = np.random.default_rng(5)
    x = np.concatenate([rng.uniform(-87, 88.5, 500_000), rng.normal(0, 1e-3, 100_000),
                        rng.normal(0, 1e-20, 1000)]).astype(np.float32)
    err = _ulp_err(oracle.expf(x), np.exp(x.astype(np.float64)))
    assert err.max() <= 2.0, err.max()


def test_expf_special_values():
    e = oracle.expf(np.array([0.0, -0.0, 1.0, 89.0, 100.0, 1e30, -104.0, -200.0, -1e30, np.nan], np.float32))
    assert e[0] == 1.0 and e[1] == 1.0                  # e^0 = 1 exactly
    assert abs(float(e[2]) - math.e) <= np.spacing(np.float32(math.e))
    assert np.isinf(e[3]) and np.isinf(e[4]) and np.isinf(e[5]) and e[3] > 0
    assert e[6] == 0.0 and e[7] == 0.0 and e[8] == 0.0  # below the subnormal range
    assert np.isnan(e[9])


def test_expf_subnormal_results_correctly_scaled():
    x = np.linspace(-103.0, -87.5, 20001).astype(np.float32)
    got = oracle.expf(x).astype(np.float64)
    ref = np.exp(x.astype(np.float64))
    # subnormals have an absolute spacing of 2^-149; allow 2 of them
    assert np.max(np.abs(got - ref)) <= 2 * 2.0 ** -149


def test_expf_monotone():
    x = np.linspace(-30, 30, 400_001).astype(np.float32)
    e = oracle.expf(x)
    assert np.all(np.diff(e) >= 0)


def test_dot_exact_on_small_integers():
    rng = np.random.default_rng(0)
    for k in [0, 1, 5, 31, 32, 33, 64, 100, 200, 257]:
        w = rng.integers(-50, 50, 400).astype(np.float32)
        col = rng.permutation(400)[:k].astype(np.int32)
        val = rng.integers(-50, 50, k).astype(np.float32)
        exact = int(np.sum(w[col].astype(np.int64) * val.astype(np.int64)))
        assert oracle.dot(w, col, val) == exact


def test_dot_none_values_means_ones():
    w = np.arange(10, dtype=np.float32)
    assert oracle.dot(w, np.array([1, 3, 9], np.int32), None) == 13.0


def test_dot_uses_32_partial_sums():
    # elements 0 and 32 share a partial sum and cancel exactly there; a plain
    # left-to-right sum in fp32 would absorb the 31 ones into 1e8 and give 0.
    k = 33
    w = np.ones(k, np.float32)
    col = np.arange(k, dtype=np.int32)
    val = np.ones(k, np.float32)
    val[0], val[32] = 1e8, -1e8
    assert oracle.dot(w, col, val) == 31.0


def test_dot_error_bound_random():
    rng = np.random.default_rng(1)
    for k in [3, 17, 40, 100, 200, 700]:
        w = rng.normal(size=1000).astype(np.float32)
        col = rng.permutation(1000)[:k].astype(np.int32)
        val = rng.normal(size=k).astype(np.float32)
        prods = [float(a) * float(b) for a, b in zip(w[col], val)]
        exact = math.fsum(prods)
        bound = (math.ceil(k / 32) + 5 + 1) * 2.0 ** -24 * math.fsum(abs(q) for q in prods)
        assert abs(float(oracle.dot(w, col, val)) - exact) <= bound


def test_grad_logistic_closed_forms():
    for y in (1.0, -1.0):
        assert oracle.grad(oracle.LOGISTIC, 0.0, y) == -y / 2      # sigma(0) = 1/2 exactly
        assert oracle.grad(oracle.LOGISTIC, 200.0 * y, y) == 0.0   # saturated: e^{200} = inf
        assert oracle.grad(oracle.LOGISTIC, -200.0 * y, y) == -y   # e^{-200} = 0


def test_grad_logistic_is_the_derivative_of_the_logistic_loss():
    # pinned to the loss itself, not to the oracle's formula: a central
    # difference of L(m) = log(1 + exp(-y m)) in fp64 (log1p/exp, step h with
    # truncation error ~ h^2 |L'''| / 6 and rounding ~ 1e-16 / h)
    rng = np.random.default_rng(2)
    h = 1e-5
    for m in rng.uniform(-20, 20, 2000).astype(np.float32):
        for y in (1.0, -1.0):
            def loss(t):
                z = -y * t
                return z + math.log1p(math.exp(-z)) if z > 0 else math.log1p(math.exp(z))
            fd = (loss(float(m) + h) - loss(float(m) - h)) / (2 * h)
            got = float(oracle.grad(oracle.LOGISTIC, m, y))
            assert abs(got - fd) <= 1e-9 + 4 * np.spacing(np.float32(abs(fd))), (m, y, got, fd)


def test_grad_squared_and_hinge():
    assert oracle.grad(oracle.SQUARED, 3.5, 1.25) == 2.25
    assert oracle.grad(oracle.SQUARED, -1.0, 2.0) == -3.0
    assert oracle.grad(oracle.HINGE, 1.0, 1.0) == 0.0        # tie at y*m = 1: subgradient 0
    assert oracle.grad(oracle.HINGE, -1.0, -1.0) == 0.0
    assert oracle.grad(oracle.HINGE, 0.5, 1.0) == -1.0
    assert oracle.grad(oracle.HINGE, 0.5, -1.0) == 1.0
    assert oracle.grad(oracle.HINGE, 2.0, 1.0) == 0.0
    assert oracle.grad(oracle.HINGE, -3.0, 1.0) == -1.0
