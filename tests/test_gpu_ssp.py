"""Admissible delay (Section 7) on the GPU: pdb_ssp_epoch.

delay = 0 must give the sequential result bit for bit (the asynchronous
constraints reduce to the read and write constraints).  For delay > 0 the
result depends on timing, so parity with the oracle is not defined; what
holds for every admissible interleaving is checked instead: every example's
step is applied exactly once (the final weights equal w0 minus the sum of the
recorded steps times the example values, up to fp32 summation order), and
training still converges (the loss stays close to exact SGD's)."""
import numpy as np
import pytest

from tests import _cases as C

torch = pytest.importorskip("torch")
pdb = pytest.importorskip("paper_1508_00703_gb300")

pytestmark = pytest.mark.gpu

TOL = 1e-5


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pdb.load()


def _run(name, delay, epochs=None, opts=None):
    p = C.problem(name)
    E = p.epochs if epochs is None else epochs
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    coef = torch.zeros(E * p.n_rows, dtype=torch.float32, device="cuda")
    pdb.pdb_ssp_epoch(X, y, c, s, w, p.loss, p.eta, E, delay, coef=coef, opts=opts)
    pdb.check_status(c)
    return p, w.cpu().numpy(), coef.cpu().numpy().reshape(E, p.n_rows)


def _applied_gap(p, coef, got):
    """|got - (w0 - sum of step * x over epochs and examples)| per feature, in
    fp64 (w0 = 0), and the fp32 rounding allowance of a sum of n_j terms in
    any order: n_j * 2^-23 * (sum of the terms' magnitudes)."""
    x = np.ones(p.nnz) if p.val is None else p.val.astype(np.float64)
    rows = np.repeat(np.arange(p.n_rows), np.diff(p.row_ptr))
    w = np.zeros(p.n_cols)
    mag = np.zeros(p.n_cols)
    for e in range(coef.shape[0]):
        term = coef[e][rows].astype(np.float64) * x
        np.subtract.at(w, p.col, term)
        np.add.at(mag, p.col, np.abs(term))
    cnt = np.bincount(p.col, minlength=p.n_cols) * coef.shape[0]
    return np.abs(got.astype(np.float64) - w), (cnt + 1) * 2.0 ** -23 * mag + 1e-30


def _loss(p, w):
    x = np.ones(p.nnz) if p.val is None else p.val.astype(np.float64)
    rows = np.repeat(np.arange(p.n_rows), np.diff(p.row_ptr))
    m = np.zeros(p.n_rows)
    np.add.at(m, rows, w.astype(np.float64)[p.col] * x)
    if p.loss == pdb.PDB_LOSS_LOGISTIC:
        return float(np.mean(np.logaddexp(0.0, -p.y * m)))
    if p.loss == pdb.PDB_LOSS_SQUARED:
        return float(np.mean((m - p.y) ** 2) / 2)
    return float(np.mean(np.maximum(0.0, 1.0 - p.y * m)))


@pytest.mark.parametrize("name", ["tiny", "zipf-shape", "deepchain-shape", "lowconflict-shape", "long-rows",
                                  "ctr-shape-binary", "ragged-empty-rows", "one-feature-chain"])
def test_delay_zero_is_sequential_sgd(name):
    p, got, coef = _run(name, 0)
    ref = C.oracle_sgd(name)
    assert C.rel_err(got, ref) <= TOL
    assert np.array_equal(got, ref)
    # the recorded steps reproduce the weights
    gap, allow = _applied_gap(p, coef, got)
    assert np.all(gap <= allow)


@pytest.mark.parametrize("delay", [1, 8, 64, 1 << 40])
@pytest.mark.parametrize("name", ["tiny", "zipf-shape", "deepchain-shape", "ctr-shape-binary"])
def test_delayed_run_applies_every_step_once(name, delay):
    p, got, coef = _run(name, delay)
    assert np.all(np.isfinite(got)) and np.all(np.isfinite(coef))
    gap, allow = _applied_gap(p, coef, got)
    assert np.all(gap <= allow)


@pytest.mark.parametrize("delay", [1, 16])
@pytest.mark.parametrize("name", ["tiny", "lowconflict-shape", "zipf-shape"])
def test_delayed_run_still_trains(name, delay):
    p, got, _ = _run(name, delay)
    exact = _loss(p, C.oracle_sgd(name))
    start = _loss(p, np.zeros(p.n_cols, dtype=np.float32))
    delayed = _loss(p, got)
    assert delayed < start
    assert abs(delayed - exact) <= 0.05 * abs(start - exact) + 1e-6


def test_schedule_and_argument_checks():
    p = C.problem("tiny")
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_WINDOW)
    with pytest.raises(pdb.PdbError) as e:
        pdb.pdb_ssp_epoch(X, y, c, s, w, p.loss, p.eta, 1, 0)
    assert e.value.code == pdb.PDB_ESTATE
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY)
    with pytest.raises(pdb.PdbError) as e:
        pdb.pdb_ssp_epoch(X, y, c, s, w, p.loss, p.eta, 1, -1)
    assert e.value.code == pdb.PDB_EINVAL


def test_wait_timeout_is_reported_not_hung():
    # one position asks for more writes of its feature than will ever happen
    p = C.problem("tiny")
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY)
    pdb.check_status(c)
    gate_ptr = pdb.pdb_schedule_ready(s)["gate"]
    pos = int(p.row_ptr[5])
    poison = torch.tensor([100000], dtype=torch.int32, device="cuda")
    pdb.pdb_memcpy(gate_ptr + 4 * pos, poison.data_ptr(), 4)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    pdb.pdb_ssp_epoch(X, y, c, s, w, p.loss, p.eta, 1, 4, opts=dict(wait_timeout_s=0.2))
    assert pdb.pdb_status(c) == pdb.PDB_ETIMEOUT
    assert torch.arange(10, device="cuda").sum().item() == 45
