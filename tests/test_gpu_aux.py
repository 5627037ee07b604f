"""Checkpoint/resume and call logging on the GPU.

Resume: the training state at an epoch boundary is the weight vector (the
schedule is a pure function of the data), so a run of E1 epochs, saved to
the host and resumed for E2 epochs from fresh handles, must give the weights
of one E1 + E2 epoch run bit for bit -- under every engine, including READY,
which pipelines epochs inside one launch, and the admissible-delay engine at
delay 0.

Logging: with PDB_LOG=1 every C-ABI call prints one line of its stats."""
import numpy as np
import pytest

import oracle
from tests import _cases as C

torch = pytest.importorskip("torch")
pdb = pytest.importorskip("paper_1508_00703_gb300")

pytestmark = pytest.mark.gpu

MODES = {"levels": pdb.PDB_SCHED_LEVELS, "ready": pdb.PDB_SCHED_READY, "chain": pdb.PDB_SCHED_CHAIN,
         "window": pdb.PDB_SCHED_WINDOW, "auto": pdb.PDB_SCHED_AUTO}


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pdb.load()


def _train(p, mode, epochs, w0=None, delay=None):
    """A fresh process's view: new device copies, handles and schedule."""
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY if delay is not None else mode)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda") if w0 is None else torch.from_numpy(w0).cuda()
    if delay is None:
        pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, epochs)
    else:
        pdb.pdb_ssp_epoch(X, y, c, s, w, p.loss, p.eta, epochs, delay)
    pdb.check_status(c)
    return w.cpu().numpy()


@pytest.mark.parametrize("mode", list(MODES))
@pytest.mark.parametrize("name", ["tiny", "deepchain-shape", "dense-narrow"])
def test_resume_is_exact(name, mode):
    p = C.problem(name)
    whole = _train(p, MODES[mode], 3)
    first = _train(p, MODES[mode], 1)
    resumed = _train(p, MODES[mode], 2, w0=first.copy())
    assert np.array_equal(resumed, whole)
    assert np.array_equal(whole, oracle.sgd(p, epochs=3))


def test_resume_admissible_delay_zero():
    p = C.problem("zipf-shape")
    whole = _train(p, None, 2, delay=0)
    resumed = _train(p, None, 1, w0=_train(p, None, 1, delay=0), delay=0)
    assert np.array_equal(resumed, whole)
    assert np.array_equal(whole, oracle.sgd(p, epochs=2))


def test_pdb_log_prints_one_line_per_call(monkeypatch, capfd):
    p = C.problem("tiny")
    monkeypatch.setenv("PDB_LOG", "1")
    _train(p, pdb.PDB_SCHED_READY, 1)
    err = capfd.readouterr().err
    lines = [ln for ln in err.splitlines() if ln.startswith("pdb ")]
    assert [ln.split(":")[0] for ln in lines] == ["pdb pdb_build_conflicts", "pdb pdb_schedule_build",
                                                  "pdb pdb_sgd_epoch"]
    assert f"nnz={p.nnz}" in lines[-1] and f"sched_mode={pdb.PDB_SCHED_READY}" in lines[-1]
    assert "status=0" in lines[-1]
    monkeypatch.setenv("PDB_LOG", "0")
    _train(p, pdb.PDB_SCHED_READY, 1)
    assert "pdb " not in capfd.readouterr().err
