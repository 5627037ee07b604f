"""The seeded input generator: known-answer Philox block, shapes and
invariants of the drawn CSR, reproducibility across thread counts."""
import numpy as np
import pytest

import synthdata


def test_philox_known_answer():
    # Philox4x32-10 with zero counter and key (Salmon et al., SC'11 test vector)
    out = synthdata.philox4x32_10([0, 0, 0, 0], [0, 0])
    assert [hex(int(x)) for x in out] == ["0x6627e8d5", "0xe169c58d", "0xbc57ac4c", "0x9b00dbd8"]


@pytest.mark.parametrize("name,kw", [
    ("tiny", {}),
    ("zipf-1m", dict(n_rows=20000)),
    ("ctr", dict(n_rows=20000, n_cols=200000)),
    ("low-conflict", dict(n_rows=20000, n_cols=1_000_000)),
    ("deep-chain", dict(n_rows=2000)),
    ("dense-lr", {}),
])
def test_workload_shape(name, kw):
    p = synthdata.generate(name, **kw)
    spec = dict(synthdata.WORKLOADS[name], **kw)
    k = spec["k"]
    assert p.n_rows == spec["n_rows"] and p.nnz == p.n_rows * k
    assert np.array_equal(p.row_ptr, np.arange(p.n_rows + 1) * k)
    rows = p.col.reshape(p.n_rows, k)
    assert np.all(np.diff(rows, axis=1) > 0)            # distinct and ascending in every row
    assert p.col.min() >= 0 and p.col.max() < p.n_cols
    if spec["vals"] == "ones":
        assert p.val is None
    elif spec["vals"] == "uniform":
        assert p.val.min() >= -1 and p.val.max() < 1
    if spec["labels"] in ("sign", "bernoulli"):
        assert set(np.unique(p.y).tolist()) <= {-1.0, 1.0}
    assert p.y.dtype == np.float32 and np.all(np.isfinite(p.y))


def test_deterministic_across_threads():
    a = synthdata.generate("zipf-1m", n_rows=5000, nthreads=1)
    b = synthdata.generate("zipf-1m", n_rows=5000, nthreads=7)
    assert np.array_equal(a.col, b.col) and np.array_equal(a.val, b.val) and np.array_equal(a.y, b.y)
    c = synthdata.generate("zipf-1m", n_rows=5000, seed=99)
    assert not np.array_equal(a.col, c.col)


def test_zipf_head_frequency():
    # P(top id in a row) for k draws-without-repeats is close to 1-(1-p1)^k for small p1
    p = synthdata.generate("zipf-1m", n_rows=20000)
    s, F, k = 1.0, p.n_cols, 20
    p1 = 1.0 / np.sum(np.arange(1, F + 1, dtype=np.float64) ** -s)
    top = np.bincount(p.col, minlength=F).argmax()
    frac = np.mean([(p.col[p.row_ptr[t]:p.row_ptr[t + 1]] == top).any() for t in range(p.n_rows)])
    assert abs(frac - (1 - (1 - p1) ** k)) < 0.03


def test_ragged_rows():
    p = synthdata.generate("tiny", n_rows=2000, k_lo=0, k=12)
    lens = np.diff(p.row_ptr)
    assert lens.min() == 0 and lens.max() == 12
    assert abs(lens.mean() - 6) < 0.5


def test_dense_rows_and_linear_labels():
    # every example holds every feature; the labels are w*.x plus N(0, 0.1^2)
    # noise, so a least-squares fit recovers w* and leaves residuals of
    # standard deviation ~0.1
    p = synthdata.generate("dense-lr", n_rows=3000, n_cols=200, k=200)
    X = p.val.reshape(p.n_rows, 200).astype(np.float64)
    assert np.array_equal(p.col.reshape(p.n_rows, 200), np.tile(np.arange(200), (p.n_rows, 1)))
    coef, *_ = np.linalg.lstsq(X, p.y.astype(np.float64), rcond=None)
    resid = p.y - X @ coef
    assert 0.09 < np.std(resid) < 0.11
    assert 0.8 < np.std(coef) < 1.2          # w* ~ N(0, 1)


def test_value_distributions():
    # N(0, 1) values (tiny) and U(-1, 1) values (low-conflict): first moments
    p = synthdata.generate("tiny")
    assert abs(float(p.val.mean())) < 0.02 and abs(float(p.val.std()) - 1.0) < 0.02
    q = synthdata.generate("low-conflict", n_rows=20000, n_cols=1_000_000)
    assert abs(float(q.val.mean())) < 0.01 and abs(float(q.val.var()) - 1.0 / 3.0) < 0.005
    # sign labels of a planted w* split about evenly
    assert abs(float((p.y > 0).mean()) - 0.5) < 0.03


def test_uniform_ids_are_flat():
    # 100 distinct uniform ids per example over 10^6 features: per-feature
    # counts are Poisson-like (variance / mean = 1)
    q = synthdata.generate("low-conflict", n_rows=20000, n_cols=1_000_000)
    c = np.bincount(q.col, minlength=q.n_cols).astype(np.float64)
    assert 0.97 < c.var() / c.mean() < 1.03


@pytest.mark.parametrize("name,kw,s", [
    ("zipf-1m", dict(n_rows=100000), 1.0),
    ("ctr", dict(n_rows=50000, n_cols=1_000_000), 1.1),
    ("deep-chain", dict(n_rows=10000), 1.3),
])
def test_zipf_exponent(name, kw, s):
    # rank-frequency slope on log-log axes over ranks 1000..10000, where a
    # feature is rare enough per example that rejecting repeats inside an
    # example does not bend the curve
    p = synthdata.generate(name, **kw)
    cnt = np.sort(np.bincount(p.col, minlength=p.n_cols))[::-1].astype(np.float64)
    r = np.arange(1000, 10000)
    slope = np.polyfit(np.log(r + 1.0), np.log(cnt[r]), 1)[0]
    assert abs(-slope - s) < 0.05, -slope
