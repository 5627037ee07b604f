"""The data-parallel split of Algorithm 2a through the C ABI on the GPU.

pdb_bsp_plan_build / pdb_bsp_coef / pdb_bsp_apply, driven by
bsp_epoch_data_parallel, must give pdb_bsp_epoch's weights and the oracle's
BSP bit for bit: on one rank, and with two ranks in two processes that share
this GPU and gather their coefficient shares over gloo (host tensors; no
kernel of one process waits for the other's)."""
import os
import socket

import numpy as np
import pytest

import oracle
import synthdata

torch = pytest.importorskip("torch")
import torch.distributed as dist                     # noqa: E402
import torch.multiprocessing as mp                   # noqa: E402

import paper_1508_00703_gb300 as pdb                 # noqa: E402

pytestmark = pytest.mark.gpu

CASES = [
    ("tiny", dict(n_rows=3001), 64, 1),
    ("zipf-1m", dict(n_rows=20000, n_cols=20000), 4096, 1),
    ("deep-chain", dict(n_rows=9000), 4096, 2),
    ("low-conflict", dict(n_rows=20000, n_cols=2_000_000), 4096, 1),
    ("dense-lr", dict(n_rows=800, n_cols=320, k=320, epochs=2, bsp_batch=800), 800, 2),
    ("tiny", dict(n_rows=50, n_cols=80, k=5, k_lo=0), 1, 2),      # batch 1 (= SGD), empty rows
]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pdb.load()


@pytest.mark.parametrize("ci", range(len(CASES)))
def test_bsp_split_on_one_rank_equals_bsp_epoch_and_the_oracle(ci):
    name, kw, batch, epochs = CASES[ci]
    p = synthdata.generate(name, **kw)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    pdb.check_status(c)
    w_split = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    pdb.bsp_epoch_data_parallel(X, y, c, w_split, p.loss, p.eta, batch, epochs)
    pdb.check_status(c)
    w_whole = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    pdb.pdb_bsp_epoch(X, y, c, w_whole, p.loss, p.eta, batch, epochs)
    pdb.check_status(c)
    got = w_split.cpu().numpy()
    assert np.array_equal(got, w_whole.cpu().numpy())
    assert np.array_equal(got, oracle.bsp(p, batch, epochs=epochs))


def test_bsp_split_rejects_rows_across_batches():
    p = synthdata.generate("tiny", n_rows=300)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    plan = pdb.pdb_bsp_plan_build(c, 64)
    assert plan.n_batches == 5
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    coef = torch.zeros(64, dtype=torch.float32, device="cuda")
    with pytest.raises(pdb.PdbError) as e:
        pdb.pdb_bsp_coef(plan, X, y, w, p.loss, p.eta, 60, 70, coef)
    assert e.value.code == pdb.PDB_EINVAL
    with pytest.raises(pdb.PdbError) as e:
        pdb.pdb_bsp_apply(plan, w, 5, coef)
    assert e.value.code == pdb.PDB_EINVAL


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    torch.cuda.set_device(0)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        pdb.load()
        for ci, (name, kw, batch, epochs) in enumerate(CASES):
            p = synthdata.generate(name, **kw)
            X = pdb.Csr.from_problem(p)
            y = torch.from_numpy(p.y).cuda()
            c = pdb.pdb_build_conflicts(X)
            w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
            pdb.bsp_epoch_data_parallel(X, y, c, w, p.loss, p.eta, batch, epochs)
            pdb.check_status(c)
            np.save(os.path.join(out_dir, f"w_{ci}_{rank}.npy"), w.cpu().numpy())
    finally:
        dist.destroy_process_group()


def test_bsp_split_over_two_processes_on_this_gpu(tmp_path):
    world = 2
    mp.spawn(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    for ci, (name, kw, batch, epochs) in enumerate(CASES):
        ref = oracle.bsp(synthdata.generate(name, **kw), batch, epochs=epochs)
        for r in range(world):
            assert np.array_equal(np.load(tmp_path / f"w_{ci}_{r}.npy"), ref), (name, batch, r)
