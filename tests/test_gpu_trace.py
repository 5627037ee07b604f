"""Execution traces of the CUDA engines checked against the paper's
synchronization constraints.

With ``pdb_opts.trace`` every engine stamps, per example, the global timer
once all of its reads are done and once its update is computed (before any
of its writes is issued).  The stamps give the execution's history of reads
and writes per feature, which must satisfy the Read and Write Constraints
of Section 4.4 for every exact schedule (Theorem 2 then makes the run
equivalent to sequential SGD), and the asynchronous Read Constraint of
Section 7 under an admissible delay.  Tracing must not change the weights.

Equal stamps (one timer tick) cannot order two events; the checkers treat
them as ordered in data order, so a break is seen only when it spans more
than a tick."""
import numpy as np
import pytest

from oracle import history
from tests import _cases as C

torch = pytest.importorskip("torch")
pdb = pytest.importorskip("paper_1508_00703_gb300")

pytestmark = pytest.mark.gpu

MODES = {"levels": pdb.PDB_SCHED_LEVELS, "ready": pdb.PDB_SCHED_READY, "chain": pdb.PDB_SCHED_CHAIN,
         "window": pdb.PDB_SCHED_WINDOW}
HISTORY_OPS = 400_000       # run the operation-level history check up to this many operations


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pdb.load()


def _setup(name, mode):
    p = C.problem(name)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, mode)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    trace = torch.zeros(2 * p.epochs * p.n_rows, dtype=torch.int64, device="cuda")
    return p, X, y, c, s, w, trace


def _check_stamped(p, tr, epochs):
    k = np.tile(np.diff(p.row_ptr), epochs)
    assert np.all(tr[k > 0] > 0), "an example with features was not stamped"
    if k.size > 1000:
        assert np.ptp(tr[tr > 0]) > 0


def _check_rc_wc(p, tr, epochs):
    v = history.trace_order_violations(p.row_ptr, p.col, epochs, tr)
    assert v["self"] == 0, v
    assert v["rc"] == 0, v
    if 2 * p.nnz * epochs <= HISTORY_OPS:
        ops = history.trace_history(p.row_ptr, p.col, epochs, tr)
        assert history.satisfies_rc_wc(ops)
        assert history.per_chunk_sequential(ops)      # Theorem 2's conditions, per feature
    return v


# (case, mode): every engine behind pdb_sgd_epoch -- LEVELS; READY in one
# block (few features) and over the grid (many features, and rows longer than
# 256 ids); WINDOW with its default near distance and with the watermark path
# forced; CHAIN forwarding (short rows) and weight-resident (long rows)
CASES = [
    ("tiny", "levels"), ("long-rows", "levels"), ("zipf-shape", "levels"),
    ("tiny", "ready"), ("ragged-empty-rows", "ready"), ("lowconflict-shape", "ready"), ("ids-18bit", "ready"),
    ("long-rows", "ready"),
    ("tiny", "window"), ("lowconflict-shape", "window"), ("long-rows", "window"),
    ("tiny", "chain"), ("deepchain-shape", "chain"), ("one-feature-chain", "chain"),
    ("dense-shape", "chain"), ("long-rows", "chain"),
]


@pytest.mark.parametrize("name,mode", CASES)
def test_exact_engines_keep_rc_wc(name, mode):
    p, X, y, c, s, w, trace = _setup(name, MODES[mode])
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs, opts=dict(trace=trace, wait_timeout_s=20.0))
    pdb.check_status(c)
    assert np.array_equal(w.cpu().numpy(), C.oracle_sgd(name))      # tracing changes nothing
    tr = trace.cpu().numpy().reshape(-1, 2)
    _check_stamped(p, tr, p.epochs)
    _check_rc_wc(p, tr, p.epochs)


@pytest.mark.parametrize("mode", list(MODES))
def test_epochs_chain_across_boundaries(mode):
    # an epoch's first occurrence of a feature reads after the previous
    # epoch's last occurrence wrote; the engines overlap epochs
    import oracle
    E = 3
    p, X, y, c, s, w, _ = _setup("ragged-empty-rows", MODES[mode])
    trace = torch.zeros(2 * E * p.n_rows, dtype=torch.int64, device="cuda")
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, E, opts=dict(trace=trace, wait_timeout_s=20.0))
    pdb.check_status(c)
    assert np.array_equal(w.cpu().numpy(), oracle.sgd(p, epochs=E))
    tr = trace.cpu().numpy().reshape(-1, 2)
    _check_stamped(p, tr, E)
    _check_rc_wc(p, tr, E)


@pytest.mark.parametrize("near_dist", [7, 300])
@pytest.mark.parametrize("name", ["tiny", "zipf-shape"])
def test_window_watermark_keeps_rc_wc(name, near_dist, monkeypatch):
    monkeypatch.setenv("PDB_NEAR", str(near_dist))
    p, X, y, c, s, w, trace = _setup(name, pdb.PDB_SCHED_WINDOW)
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs, opts=dict(trace=trace, wait_timeout_s=20.0))
    pdb.check_status(c)
    assert np.array_equal(w.cpu().numpy(), C.oracle_sgd(name))
    tr = trace.cpu().numpy().reshape(-1, 2)
    _check_stamped(p, tr, p.epochs)
    _check_rc_wc(p, tr, p.epochs)


def test_ready_runs_examples_concurrently():
    # the trace shows real overlap: on data with long independent stretches
    # some example reads before an earlier (non-conflicting) one has computed
    p, X, y, c, s, w, trace = _setup("lowconflict-shape", pdb.PDB_SCHED_READY)
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, 1, opts=dict(trace=trace))
    pdb.check_status(c)
    tr = trace.cpu().numpy().reshape(-1, 2)[: p.n_rows]
    assert np.sum(tr[1:, 0] < np.maximum.accumulate(tr[:, 1])[:-1]) > 0


@pytest.mark.parametrize("delay", [0, 4, 64, 1024])
@pytest.mark.parametrize("name", ["tiny", "zipf-shape", "long-rows"])
def test_admissible_delay_trace(name, delay):
    p, X, y, c, s, w, trace = _setup(name, pdb.PDB_SCHED_READY)
    pdb.pdb_ssp_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs, delay, opts=dict(trace=trace, wait_timeout_s=20.0))
    pdb.check_status(c)
    tr = trace.cpu().numpy().reshape(-1, 2)
    _check_stamped(p, tr, p.epochs)
    d = history.trace_delay_violations(p.row_ptr, p.col, p.epochs, tr, delay)
    assert d["violations"] == 0, d
    if delay == 0:
        # the asynchronous constraints at delay 0 are the exact ones
        _check_rc_wc(p, tr, p.epochs)
        assert np.array_equal(w.cpu().numpy(), C.oracle_sgd(name))
