"""WINDOW without every block of its grid resident.

The engine's watermark is built from per-chunk done flags and swept by the
first block that starts, so thread blocks the device has not started yet
hold nothing back (the deadlock-freedom argument in csrc/window.cu).  Here a
helper kernel on a second stream holds about two thirds of the SMs for
0.25 s while WINDOW runs with a 0.05 s wait limit and every occurrence pair
far (each read with a predecessor waits for the watermark): the result must
be the oracle's, bit for bit, with no expired wait.  A watermark that waited
for blocks that had not started would stall past the limit.

The same helper checks that freeing handles waits only for the work
enqueued on them: with another stream busy for 0.6 s, a build, a schedule,
an epoch and both frees on this stream return well before it."""
import ctypes
import os
import subprocess

import numpy as np
import pytest

import oracle
import synthdata

torch = pytest.importorskip("torch")
pdb = pytest.importorskip("paper_1508_00703_gb300")

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def hold(tmp_path_factory):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pdb.load()
    so = str(tmp_path_factory.mktemp("hold") / "libhold.so")
    subprocess.run(["nvcc", "-gencode=arch=compute_103a,code=sm_103a", "-O2", "-shared", "-Xcompiler", "-fPIC",
                    os.path.join(HERE, "hold_kernel.cu"), "-o", so], check=True)
    lib = ctypes.CDLL(so)
    lib.hold_sms.argtypes = [ctypes.c_int, ctypes.c_double, ctypes.c_void_p]
    return lib


@pytest.mark.parametrize("name,kw", [
    ("low-conflict", dict(n_rows=20000, n_cols=2_000_000, epochs=2)),
    ("zipf-1m", dict(n_rows=20000, n_cols=50000)),
])
def test_window_runs_while_most_sms_are_held(hold, monkeypatch, name, kw):
    monkeypatch.setenv("PDB_NEAR", "1")            # every occurrence pair far: all reads use the watermark
    p = synthdata.generate(name, **kw)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_WINDOW)
    pdb.check_status(c)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    assert hold.hold_sms(2 * sms // 3, 0.25, ctypes.c_void_p(side.cuda_stream)) == 0
    main = torch.cuda.Stream()                      # two non-blocking streams: the kernels may overlap
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs, opts=dict(wait_timeout_s=0.05), stream=main)
    torch.cuda.synchronize()
    assert pdb.pdb_status(c) == pdb.PDB_OK
    assert np.array_equal(w.cpu().numpy(), oracle.sgd(p))


def test_freeing_handles_waits_only_for_their_own_work(hold):
    # a helper kernel keeps another stream busy for 0.6 s; building, training
    # and freeing handles on this stream must not wait for it
    import time
    p = synthdata.generate("tiny", n_rows=3000)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    torch.cuda.synchronize()
    side, main = torch.cuda.Stream(), torch.cuda.Stream()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    assert hold.hold_sms(sms // 2, 0.6, ctypes.c_void_p(side.cuda_stream)) == 0
    t0 = time.perf_counter()
    c = pdb.pdb_build_conflicts(X, main)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY, main)
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs, stream=main)
    assert pdb.pdb_status(c, main) == pdb.PDB_OK
    del s, c                                          # frees both handles
    elapsed = time.perf_counter() - t0
    side_done = side.query()
    torch.cuda.synchronize()
    assert elapsed < 0.4 and not side_done, (elapsed, side_done)
    assert np.array_equal(w.cpu().numpy(), oracle.sgd(p))
