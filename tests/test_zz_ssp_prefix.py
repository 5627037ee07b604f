"""Admissible delay (Section 7) with prefix gates on the GPU.

pdb_ssp_epoch with opts.ssp_gates = PDB_SSP_PREFIX: rank r of a feature reads
once every rank <= r - 1 - delay has written and writes once every rank
<= r - delay has read (the Write Protocol's slowest reader), on done-bitmaps
over the CSC slots.  The protocol itself is model-checked on the CPU
(tests/test_ssp_protocol.py); here the kernel must give, as under the
counting gates: the sequential result bit for bit at delay 0; every step
applied exactly once and training that converges for delay > 0; the
asynchronous Read Constraint on an execution trace; and argument checks and
an out-of-range rank reported as errors.  The degenerate inputs (no rows,
only empty rows, one row, one feature, saturated exponentials) run here
under both gate forms.  This file is collected last."""
import numpy as np
import pytest

from oracle import history
from tests import _cases as C
from tests import test_gpu_ssp as ssp

torch = pytest.importorskip("torch")
pdb = pytest.importorskip("paper_1508_00703_gb300")

pytestmark = pytest.mark.gpu

PREFIX = dict(ssp_gates=pdb.PDB_SSP_PREFIX)


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pdb.load()


@pytest.mark.parametrize("name", ["tiny", "zipf-shape", "deepchain-shape", "lowconflict-shape", "long-rows",
                                  "ctr-shape-binary", "ragged-empty-rows", "one-feature-chain"])
def test_prefix_gates_delay_zero_is_sequential_sgd(name):
    p, got, coef = ssp._run(name, 0, opts=PREFIX)
    assert np.array_equal(got, C.oracle_sgd(name))
    gap, allow = ssp._applied_gap(p, coef, got)
    assert np.all(gap <= allow)


@pytest.mark.parametrize("delay", [1, 8, 64, 1 << 40])
@pytest.mark.parametrize("name", ["tiny", "zipf-shape", "deepchain-shape", "ctr-shape-binary", "long-rows"])
def test_prefix_gates_apply_every_step_once(name, delay):
    p, got, coef = ssp._run(name, delay, opts=PREFIX)
    assert np.all(np.isfinite(got)) and np.all(np.isfinite(coef))
    gap, allow = ssp._applied_gap(p, coef, got)
    assert np.all(gap <= allow)


@pytest.mark.parametrize("delay", [1, 16])
@pytest.mark.parametrize("name", ["tiny", "lowconflict-shape", "zipf-shape"])
def test_prefix_gates_still_train(name, delay):
    p, got, _ = ssp._run(name, delay, opts=PREFIX)
    exact = ssp._loss(p, C.oracle_sgd(name))
    start = ssp._loss(p, np.zeros(p.n_cols, dtype=np.float32))
    delayed = ssp._loss(p, got)
    assert delayed < start
    assert abs(delayed - exact) <= 0.05 * abs(start - exact) + 1e-6


@pytest.mark.parametrize("delay", [0, 3, 64, 1024])
@pytest.mark.parametrize("name", ["tiny", "zipf-shape", "long-rows"])
def test_prefix_gates_trace_keeps_the_asynchronous_read_constraint(name, delay):
    p = C.problem(name)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    trace = torch.zeros(2 * p.epochs * p.n_rows, dtype=torch.int64, device="cuda")
    pdb.pdb_ssp_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs, delay,
                      opts=dict(PREFIX, trace=trace, wait_timeout_s=20.0))
    pdb.check_status(c)
    tr = trace.cpu().numpy().reshape(-1, 2)
    d = history.trace_delay_violations(p.row_ptr, p.col, p.epochs, tr, delay)
    assert d["violations"] == 0, d
    if delay == 0:
        assert np.array_equal(w.cpu().numpy(), C.oracle_sgd(name))


def test_prefix_gates_argument_checks():
    p = C.problem("tiny")
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    for bad in (-1, pdb.PDB_SSP_PREFIX + 1):
        with pytest.raises(pdb.PdbError) as e:
            pdb.pdb_ssp_epoch(X, y, c, s, w, p.loss, p.eta, 1, 0, opts=dict(ssp_gates=bad))
        assert e.value.code == pdb.PDB_EINVAL


def test_prefix_gates_report_a_rank_past_the_feature():
    # a gate word whose rank lies past its feature's occurrences (a corrupted
    # schedule) is reported as PDB_EFAULT before any bitmap access
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
    pdb.pdb_ssp_epoch(X, y, c, s, w, p.loss, p.eta, 1, 4, opts=dict(PREFIX, wait_timeout_s=0.5))
    assert pdb.pdb_status(c) == pdb.PDB_EFAULT
    assert torch.arange(10, device="cuda").sum().item() == 45


@pytest.mark.parametrize("gates", [pdb.PDB_SSP_COUNT, pdb.PDB_SSP_PREFIX])
@pytest.mark.parametrize("name", C.EDGES)
def test_edge_inputs_under_both_gate_forms(name, gates):
    p, got, coef = ssp._run(name, 0, opts=dict(ssp_gates=gates))
    assert np.array_equal(got, C.oracle_sgd(name))
    p, got, coef = ssp._run(name, 3, opts=dict(ssp_gates=gates))
    assert np.all(np.isfinite(got))
    gap, allow = ssp._applied_gap(p, coef, got)
    assert np.all(gap <= allow)
