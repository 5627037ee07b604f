"""The data-parallel split of Algorithm 2a, on the CPU with two gloo ranks.

bsp_epoch_data_parallel gives each rank a contiguous share of every batch's
rows: the rank computes those rows' coefficients at the batch-start weights,
the shares are all-gathered in rank order, and every rank applies the whole
batch to its replica of w.  Here the two library calls are replaced by plain
restatements of their definitions (the oracle's margin and loss derivative;
each feature's terms summed in ascending example order from +0), so the test
checks the partitioning itself -- the row shares, the gather order, the batch
boundaries, short last batches and more ranks than rows -- against the
oracle's BSP, bit for bit, on every rank."""
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


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _problem(name, kw):
    return synthdata.generate(name, **kw)


def _cpu_ops(p, w, batch):
    """The library calls restated on the host for problem p (w: a CPU float32 tensor)."""
    n = p.n_rows
    col = p.col
    val = np.ones(p.nnz, np.float32) if p.val is None else p.val
    wn = w.numpy()                                  # shares memory with w
    eta = np.float32(p.eta)

    def coef(r0, r1, out):
        o = out.numpy()
        for t in range(r0, r1):
            b, e = int(p.row_ptr[t]), int(p.row_ptr[t + 1])
            m = oracle.dot(wn, col[b:e], val[b:e])
            o[t - r0] = np.float32(eta * np.float32(oracle.grad(p.loss, float(m), float(p.y[t]))))

    def apply(bi, coef_t):
        c = coef_t.numpy()
        r0 = bi * batch
        b, e = int(p.row_ptr[r0]), int(p.row_ptr[min(n, r0 + batch)])
        rows = np.repeat(np.arange(r0, min(n, r0 + batch)), np.diff(p.row_ptr[r0:min(n, r0 + batch) + 1]))
        order = np.lexsort((rows, col[b:e]))          # by feature, then example
        j_s, i_s, x_s = col[b:e][order], rows[order] - r0, val[b:e][order]
        s = 0
        while s < len(order):
            j = j_s[s]
            delta = np.float32(0.0)
            while s < len(order) and j_s[s] == j:
                delta = np.float32(delta + np.float32(c[i_s[s]] * x_s[s]))
                s += 1
            wn[j] = np.float32(wn[j] - delta)

    def gather(parts, mine):
        dist.all_gather(parts, mine)

    return dict(coef=coef, apply=apply, gather=gather, n_batches=(n + batch - 1) // batch, batch=batch, n_rows=n)


def _worker(rank, world, port, cases, out_dir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        for ci, (name, kw, batch, epochs) in enumerate(cases):
            p = _problem(name, kw)
            w = torch.zeros(p.n_cols, dtype=torch.float32)
            ops = _cpu_ops(p, w, batch)
            pdb.bsp_epoch_data_parallel(None, None, None, w, p.loss, p.eta, batch, epochs, ops=ops)
            np.save(os.path.join(out_dir, f"w_{ci}_{rank}.npy"), w.numpy())
    finally:
        dist.destroy_process_group()


CASES = [
    ("tiny", dict(n_rows=700, n_cols=300), 1, 1),
    ("tiny", dict(n_rows=701, n_cols=300), 64, 2),            # short last batch
    ("deep-chain", dict(n_rows=500, n_cols=400, k=20), 4096, 1),   # one batch longer than the data
    ("zipf-1m", dict(n_rows=613, n_cols=500), 64, 1),
    ("tiny", dict(n_rows=3, n_cols=50, k=4), 1, 3),           # more ranks than rows in a batch
]


def test_bsp_split_over_two_gloo_ranks_equals_the_oracle(tmp_path):
    world = 2
    mp.spawn(_worker, args=(world, _free_port(), CASES, str(tmp_path)), nprocs=world, join=True)
    for ci, (name, kw, batch, epochs) in enumerate(CASES):
        p = _problem(name, kw)
        ref = oracle.bsp(p, batch, epochs=epochs)
        for r in range(world):
            got = np.load(tmp_path / f"w_{ci}_{r}.npy")
            assert np.array_equal(got, ref), (name, batch, r)


@pytest.mark.parametrize("n,world", [(0, 2), (1, 2), (5, 2), (7, 3), (4096, 4), (10, 16)])
def test_rank_rows_partition_the_batch_in_order(n, world):
    r0 = 123
    bounds = [pdb.rank_rows(r0, r0 + n, r, world) for r in range(world)]
    assert bounds[0][0] == r0 and bounds[-1][1] == r0 + n
    for (a, b), (c, d) in zip(bounds, bounds[1:]):
        assert b == c and a <= b
    sizes = [b - a for a, b in bounds]
    assert max(sizes) - min(sizes) <= 1
