"""The allocation-free READY epoch against the allocating one.

pdb_sgd_epoch_ready_noalloc serves callers that must not allocate device
memory while training (work recorded into a CUDA graph capture, where
cudaMalloc cannot be captured, or a process whose memory pool owns the whole
device): its scratch is a fixed array inside the library.  Here it must give
the same weights as pdb_sgd_epoch with a READY schedule, on two calls in a
row (the second continues from the first's weights, so the shared scratch
must be reset correctly between calls)."""
import numpy as np
import pytest

import synthdata
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


@pytest.mark.parametrize("name,kw", [
    ("tiny", {}),
    ("zipf-1m", dict(n_rows=50000, n_cols=200000)),
    ("deep-chain", dict(n_rows=3000)),
])
def test_noalloc_matches_allocating_entry_point_on_two_calls(name, kw):
    p = synthdata.generate(name, **kw)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY)
    pdb.check_status(c)
    gate = pdb.pdb_schedule_ready(s)["gate"]
    w_ref = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    w_new = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    for _ in range(2):
        pdb.pdb_sgd_epoch(X, y, c, s, w_ref, p.loss, p.eta, p.epochs)
        pdb.check_status(c)
        rc = pdb.pdb_sgd_epoch_ready_noalloc(X, y, gate, w_new, p.loss, p.eta, p.epochs)
        assert rc == pdb.PDB_OK, pdb.pdb_strerror(rc)
        got, ref = w_new.cpu().numpy(), w_ref.cpu().numpy()
        assert C.rel_err(got, ref) <= TOL
        assert np.array_equal(got, ref)


def test_noalloc_rejects_more_features_than_its_scratch():
    n_cols = pdb.NOALLOC_MAX_COLS + 1
    p = synthdata.from_arrays([0, 1], [0], [1.0], [1.0], n_cols=n_cols)
    X = pdb.Csr.from_problem(p)
    y = torch.ones(1, device="cuda")
    gate = torch.zeros(1, dtype=torch.int32, device="cuda")
    w = torch.zeros(n_cols, dtype=torch.float32, device="cuda")
    rc = pdb.pdb_sgd_epoch_ready_noalloc(X, y, gate.data_ptr(), w, pdb.PDB_LOSS_LOGISTIC, 0.1, 1)
    assert rc == pdb.PDB_ETOOBIG
    assert torch.count_nonzero(w).item() == 0
