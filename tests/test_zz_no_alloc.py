"""The allocation-free READY epoch against the allocating one and the oracle.

pdb_sgd_epoch_ready_noalloc serves callers that cannot let a library
allocate device memory while they train (a server whose own memory pool owns
the whole device, a host runtime that accounts for every device allocation):
its scratch is a fixed array inside the library.  It must give the same
weights as pdb_sgd_epoch with a READY schedule and as the oracle's
sequential SGD, on two calls in a row (the second continues from the first's
weights, so the shared scratch must be reset correctly between calls), and a
call after one that stopped on an expired wait must start clean.

Collected last (file name), so a run that stops at the first failure has run
every other test before this one."""
import numpy as np
import pytest

import oracle
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


def _setup(name, kw):
    p = synthdata.generate(name, **kw)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY)
    pdb.check_status(c)
    return p, X, y, c, s, pdb.pdb_schedule_ready(s)["gate"]


@pytest.mark.parametrize("name,kw", [
    ("tiny", {}),
    ("zipf-1m", dict(n_rows=50000, n_cols=200000)),
    ("deep-chain", dict(n_rows=3000)),
    # above 2^22 positions the READY gate is built on demand from the slot-order words
    ("low-conflict", dict(n_rows=45000, n_cols=1 << 20, epochs=1)),
])
def test_noalloc_matches_allocating_entry_point_on_two_calls(name, kw):
    p, X, y, c, s, gate = _setup(name, kw)
    if name == "low-conflict":
        assert p.nnz > 1 << 22 and p.n_cols <= pdb.NOALLOC_MAX_COLS
    w_ref = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    w_new = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    for call in range(2):
        pdb.pdb_sgd_epoch(X, y, c, s, w_ref, p.loss, p.eta, p.epochs)
        pdb.check_status(c)
        rc = pdb.pdb_sgd_epoch_ready_noalloc(X, y, gate, w_new, p.loss, p.eta, p.epochs)
        assert rc == pdb.PDB_OK, pdb.pdb_strerror(rc)
        got, ref = w_new.cpu().numpy(), w_ref.cpu().numpy()
        assert C.rel_err(got, ref) <= TOL
        assert np.array_equal(got, ref)
        # and the oracle: sequential SGD over (call + 1) * epochs passes from w = 0
        w_orc = oracle.sgd(p, epochs=(call + 1) * p.epochs)
        assert C.rel_err(got, w_orc) <= TOL
        assert np.array_equal(got, w_orc)


def test_noalloc_starts_clean_after_a_call_that_timed_out():
    # The first call reads a gate word whose rank its feature never reaches:
    # its bounded waits give up (PDB_ETIMEOUT after the default 2 s limit) and
    # leave a status word, a ticket and half-updated records in the shared
    # array.  The next call, with the real gate, must not see any of it.
    p, X, y, c, s, gate = _setup("tiny", dict(n_rows=4000))
    bad = torch.empty(p.nnz, dtype=torch.int32, device="cuda")
    pdb.pdb_memcpy(bad.data_ptr(), gate, 4 * p.nnz)
    bad[int(p.row_ptr[7])] = 12345                   # first id of example 7 waits for rank 12345
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    rc = pdb.pdb_sgd_epoch_ready_noalloc(X, y, bad.data_ptr(), w, p.loss, p.eta, p.epochs)
    assert rc == pdb.PDB_ETIMEOUT, pdb.pdb_strerror(rc)
    assert torch.arange(10, device="cuda").sum().item() == 45   # the device still works
    w.zero_()
    rc = pdb.pdb_sgd_epoch_ready_noalloc(X, y, gate, w, p.loss, p.eta, p.epochs)
    assert rc == pdb.PDB_OK, pdb.pdb_strerror(rc)
    assert np.array_equal(w.cpu().numpy(), oracle.sgd(p))


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
