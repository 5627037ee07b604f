"""Pins for the oracle's sequential SGD (Algorithm 1) and BSP (Algorithm 2a):
Theorem 2's order invariance over every linear extension of the conflict
DAG, Theorem 1's BSP(B=1) = sequential, closed forms, full-batch gradient
descent in fp64, and the fp64 drift of the fp32 run."""
import itertools

import numpy as np
import pytest

import oracle
import synthdata

LOSSES = [oracle.LOGISTIC, oracle.SQUARED, oracle.HINGE]


def _problem(seed, n, f, k, loss, k_lo=None, ids="uniform"):
    labels = "linear" if loss == oracle.SQUARED else "sign"
    p = synthdata.generate("tiny", seed=seed, n_rows=n, n_cols=f, k=k, k_lo=k if k_lo is None else k_lo,
                           ids=ids, zipf_s=1.2, labels=labels, noise_std=0.1)
    p.loss = loss
    p.eta = 0.3
    return p


def _conflicts(p):
    sets = [set(p.col[p.row_ptr[t]:p.row_ptr[t + 1]].tolist()) for t in range(p.n_rows)]
    return [(u, t) for t in range(p.n_rows) for u in range(t) if sets[u] & sets[t]]


def _is_extension(order, edges):
    pos = {t: i for i, t in enumerate(order)}
    return all(pos[u] < pos[t] for u, t in edges)


@pytest.mark.parametrize("loss", LOSSES)
@pytest.mark.parametrize("seed", [0, 1])
def test_all_linear_extensions_give_identical_model(loss, seed):
    p = _problem(seed, n=7, f=9, k=3, loss=loss, k_lo=1)
    edges = _conflicts(p)
    w0 = np.random.default_rng(seed).normal(0, 0.3, p.n_cols).astype(np.float32)
    ref = oracle.sgd(p, w0=w0, epochs=2)
    n_ext = n_bad_diff = 0
    for perm in itertools.permutations(range(p.n_rows)):
        w = oracle.sgd(p, w0=w0, epochs=1, order=perm)
        w = oracle.sgd(p, w0=w, epochs=1, order=perm)
        if _is_extension(perm, edges):
            n_ext += 1
            assert np.array_equal(w, ref)
        elif not np.array_equal(w, ref):
            n_bad_diff += 1
    assert n_ext >= 2
    assert n_bad_diff > 0          # the check has power: some conflicting swaps change the model


def _random_topological_order(p, rng):
    sets = [p.col[p.row_ptr[t]:p.row_ptr[t + 1]] for t in range(p.n_rows)]
    last, preds = {}, [set() for _ in range(p.n_rows)]
    for t, s in enumerate(sets):
        for j in s.tolist():
            if j in last:
                preds[t].add(last[j])
            last[j] = t
    succ = [[] for _ in range(p.n_rows)]
    indeg = [len(x) for x in preds]
    for t, ps in enumerate(preds):
        for u in ps:
            succ[u].append(t)
    ready = [t for t in range(p.n_rows) if indeg[t] == 0]
    order = []
    while ready:
        t = ready.pop(rng.integers(len(ready)))
        order.append(t)
        for v in succ[t]:
            indeg[v] -= 1
            if indeg[v] == 0:
                ready.append(v)
    return np.array(order, np.int32)


@pytest.mark.parametrize("loss", LOSSES)
def test_random_linear_extensions_medium(loss):
    p = _problem(7, n=2000, f=400, k=8, loss=loss, ids="zipf")
    ref = oracle.sgd(p, epochs=1)
    rng = np.random.default_rng(11)
    for _ in range(25):
        order = _random_topological_order(p, rng)
        assert not np.array_equal(order, np.arange(p.n_rows))
        assert np.array_equal(oracle.sgd(p, epochs=1, order=order), ref)


def test_level_order_execution_equals_data_order():
    p = synthdata.generate("tiny")
    lv, L = oracle.levels(p)
    order, _ = oracle.level_order(lv, L)
    assert np.array_equal(oracle.sgd(p, order=order), oracle.sgd(p))


def test_one_logistic_step_from_zero():
    # m = 0 so g = -y/2 and w_j = eta * y * x_j / 2 (one rounding)
    rng = np.random.default_rng(3)
    val = rng.normal(size=12).astype(np.float32)
    for y in (1.0, -1.0):
        p = synthdata.from_arrays([0, 12], np.arange(12), val, [y], n_cols=20, loss="logistic", eta=0.01)
        w = oracle.sgd(p)
        ref = 0.01 * y * val.astype(np.float64) / 2
        assert np.all(np.abs(w[:12] - ref) <= np.spacing(np.abs(ref).astype(np.float32)))
        assert np.all(w[12:] == 0)


def test_squared_loss_geometric_closed_form():
    # the same example (one feature, x = 1) n times: w_{t+1} = (1-eta) w_t + eta y
    n, eta, y = 300, 0.05, 2.5
    p = synthdata.from_arrays(np.arange(n + 1), np.zeros(n), None, np.full(n, y), n_cols=1, loss="squared", eta=eta)
    w = oracle.sgd(p)
    exact = y * (1 - (1 - eta) ** n)
    assert abs(w[0] - exact) <= 1e-6 * abs(exact)


def test_hinge_with_margin_at_least_one_is_a_no_op():
    rng = np.random.default_rng(4)
    val = rng.normal(size=6).astype(np.float32)
    w0 = np.zeros(10, np.float32)
    w0[:6] = 3.0 * np.sign(val)          # y * m = 3 * sum|x| >= 1
    p = synthdata.from_arrays([0, 6], np.arange(6), val, [1.0], n_cols=10, loss="hinge", eta=0.5)
    assert np.array_equal(oracle.sgd(p, w0=w0), w0)


@pytest.mark.parametrize("name,rows", [("tiny", None), ("zipf-1m", 20000), ("deep-chain", 2000)])
def test_fp32_close_to_fp64(name, rows):
    kw = {} if rows is None else dict(n_rows=rows)
    p = synthdata.generate(name, **kw)
    w32, w64 = oracle.sgd(p), oracle.sgd_f64(p)
    if p.loss != oracle.HINGE:
        assert np.max(np.abs(w32 - w64)) <= 1e-4 * np.max(np.abs(w64))
    else:
        # hinge decisions may flip on rounding; the bulk still agrees
        assert np.median(np.abs(w32 - w64)) <= 1e-3 * np.max(np.abs(w64))


@pytest.mark.parametrize("loss", LOSSES)
def test_bsp_batch_one_is_sequential(loss):
    p = _problem(5, n=3000, f=500, k=7, loss=loss, k_lo=0, ids="zipf")
    assert np.array_equal(oracle.bsp(p, 1, epochs=2), oracle.sgd(p, epochs=2))


@pytest.mark.parametrize("loss", [oracle.LOGISTIC, oracle.SQUARED])
def test_bsp_full_batch_is_gradient_descent(loss):
    p = _problem(6, n=400, f=50, k=6, loss=loss)
    p.eta = 0.01
    w = np.zeros(p.n_cols)
    X = np.zeros((p.n_rows, p.n_cols))
    for t in range(p.n_rows):
        X[t, p.col[p.row_ptr[t]:p.row_ptr[t + 1]]] = p.val[p.row_ptr[t]:p.row_ptr[t + 1]]
    y = p.y.astype(np.float64)
    for _ in range(3):
        m = X @ w
        g = -y / (1 + np.exp(y * m)) if loss == oracle.LOGISTIC else m - y
        w = w - p.eta * (X.T @ g)
    got = oracle.bsp(p, p.n_rows, epochs=3)
    assert np.max(np.abs(got - w)) <= 1e-5 * np.max(np.abs(w))


def test_bsp_on_disjoint_examples_equals_sgd():
    n, k = 300, 4
    col = np.random.default_rng(8).permutation(n * k).astype(np.int32)
    val = np.random.default_rng(9).normal(size=n * k).astype(np.float32)
    y = np.where(np.random.default_rng(10).random(n) < 0.5, -1.0, 1.0)
    p = synthdata.from_arrays(np.arange(0, n * k + 1, k), col, val, y, n_cols=n * k, eta=0.2)
    for b in (2, 7, 64, n):
        assert np.array_equal(oracle.bsp(p, b), oracle.sgd(p))


def test_bsp_short_last_batch():
    p = _problem(12, n=10, f=6, k=3, loss=oracle.LOGISTIC)
    whole = oracle.bsp(p, 4)
    first = synthdata.from_arrays(p.row_ptr[:9], p.col[:p.row_ptr[8]], p.val[:p.row_ptr[8]], p.y[:8],
                                  n_cols=p.n_cols, loss=p.loss, eta=p.eta)
    w = oracle.bsp(first, 4)
    rest = synthdata.from_arrays(p.row_ptr[8:] - p.row_ptr[8], p.col[p.row_ptr[8]:], p.val[p.row_ptr[8]:],
                                 p.y[8:], n_cols=p.n_cols, loss=p.loss, eta=p.eta)
    w = oracle.bsp(rest, 100, w0=w)
    assert np.array_equal(whole, w)
    assert not np.array_equal(whole, oracle.bsp(p, 5))
