"""Host reads of handle words beside a caller's large copies.

pdb_status, pdb_schedule_build (which needs the build's info words) and
pdb_get_stats read a few words of device memory.  A device-to-host copy of
those few bytes would queue on the copy engine behind whatever large copy
the caller has in flight on another stream -- a training loop's weights
going back to the host, say -- and return only when that copy ends.  The
library stores the words into mapped pinned memory from a kernel instead.
Here a copy of 4 GB of device memory to pinned host memory (about 20 ms on
the host link) runs on one stream while a small problem is built,
scheduled, trained and checked on another: every call must return while
the copy is still moving."""
import numpy as np
import pytest

import synthdata

torch = pytest.importorskip("torch")
pdb = pytest.importorskip("paper_1508_00703_gb300")

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def big_copy():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pdb.load()
    n = 1 << 30                                   # 4 GB of float32
    dev = torch.ones(n, dtype=torch.float32, device="cuda")
    host = torch.empty(n, dtype=torch.float32).pin_memory()
    return dev, host


def test_status_and_stats_do_not_wait_for_another_streams_copy(big_copy):
    dev, host = big_copy
    p = synthdata.generate("tiny", n_rows=2000)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    copy, work = torch.cuda.Stream(), torch.cuda.Stream()

    def run():
        c = pdb.pdb_build_conflicts(X, work)
        s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_AUTO, work)
        pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, 1, stream=work)
        assert pdb.pdb_status(c, work) == pdb.PDB_OK
        return c, s, pdb.pdb_get_stats(c, s)

    c0, s0, _ = run()                             # every kernel loaded once, the pool warm
    del c0, s0
    torch.cuda.synchronize()
    done = torch.cuda.Event()
    with torch.cuda.stream(copy):
        host.copy_(dev, non_blocking=True)
        done.record(copy)
    c, s, st = run()
    still_moving = not done.query()
    torch.cuda.synchronize()
    assert st["max_chain"] > 0
    assert still_moving, "a handle read waited for the other stream's copy"
    del c, s
    assert float(host[-1]) == 1.0
