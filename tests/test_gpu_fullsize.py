"""Parity at the workloads' full sizes, in the configuration bench.py times
(READY schedule, default launch options), against the CPU oracle run on the
same seeded inputs: conflict chains bit for bit (rank, prev, next derived on
the device vs the oracle's last-occurrence map), weights within max relative
error 1e-5 and bitwise."""
import numpy as np
import pytest

import oracle
import synthdata
from tests import _cases as C

torch = pytest.importorskip("torch")
pdb = pytest.importorskip("paper_1508_00703_gb300")

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

TOL = 1e-5


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pdb.load()


def _arr(ptr, n, dtype):
    return pdb.device_array(ptr, n, dtype).cpu().numpy()


@pytest.mark.parametrize("name", ["tiny", "zipf-1m", "low-conflict", "deep-chain", "ctr"])
def test_full_size_chains_and_auto_weights(name):
    # AUTO picks what bench.py runs: READY for tiny and low-conflict, CHAIN for the Zipf workloads
    p = synthdata.generate(name)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_AUTO)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs)
    pdb.check_status(c)
    got_w = w.cpu().numpy()
    arrs = pdb.pdb_conflicts_arrays(c)
    pdb.check_status(c)
    ref = oracle.chains(p)
    for key in ("rank", "prev", "next"):
        assert np.array_equal(_arr(arrs[key], p.nnz, torch.int32), ref[key]), key
    del ref
    ref_w = oracle.sgd(p)
    assert C.rel_err(got_w, ref_w) <= TOL
    assert np.array_equal(got_w, ref_w)


def test_full_size_zipf_levels():
    p = synthdata.generate("zipf-1m")
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_LEVELS)
    info = pdb.pdb_schedule_levels(s)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs)
    pdb.check_status(c)
    lv, L = oracle.levels(p)
    assert info["n_levels"] == L
    assert np.array_equal(_arr(info["level"], p.n_rows, torch.int32), lv)
    ref_w = oracle.sgd(p)
    assert np.array_equal(w.cpu().numpy(), ref_w)
