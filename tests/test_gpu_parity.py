"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Bar: the conflict chains, levels and level order are integer results and
must match bit for bit; fp32 weights must be within max relative error 1e-5
(max |w_gpu - w_oracle| / max |w_oracle|).  Because both sides follow the
same fp32 operation order, the weights are also checked for bitwise
equality."""
import numpy as np
import pytest

from tests import _cases as C

torch = pytest.importorskip("torch")
pdb = pytest.importorskip("paper_1508_00703_gb300")

pytestmark = pytest.mark.gpu

TOL = 1e-5
ALL = list(C.SMALL) + C.EDGES


def _gpu(name):
    p = C.problem(name)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    return p, X, y


def _arr(ptr, n, dtype):
    return pdb.device_array(ptr, n, dtype).cpu().numpy()


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    pdb.load()


def test_expf_matches_oracle_bitwise_and_fp64():
    import oracle
    x = np.concatenate([np.linspace(-110, 95, 3_000_001, dtype=np.float64).astype(np.float32),
                        np.random.default_rng(0).normal(0, 3, 1_000_000).astype(np.float32),
                        np.array([0.0, -0.0, np.inf, -np.inf, np.nan], np.float32)])
    xt = torch.from_numpy(x).cuda()
    out = torch.empty_like(xt)
    pdb.pdb_eval_expf(xt, out)
    got = out.cpu().numpy()
    ref = oracle.expf(x)
    assert np.array_equal(got.view(np.uint32), ref.view(np.uint32))
    m = (x > -87) & (x < 88.5)
    e64 = np.exp(x[m].astype(np.float64))
    ulp = np.spacing(e64.astype(np.float32)).astype(np.float64)
    assert np.max(np.abs(got[m] - e64) / ulp) <= 2.0


@pytest.mark.parametrize("loss", [0, 1, 2])
def test_loss_derivative_matches_oracle_bitwise(loss):
    # the device's dloss/dm against the oracle's on margins from deep saturation
    # to the far side, labels +-1 (the reciprocal path of the logistic loss,
    # up to 1 + exp(ym) = 2^126 and past it), 0.5, -3 and 0, and special values
    import oracle
    rng = np.random.default_rng(11 + loss)
    m = np.concatenate([np.linspace(-120, 120, 60_001), rng.normal(0, 4, 40_000),
                        np.linspace(86.0, 89.5, 20_001)]).astype(np.float32)
    m = np.concatenate([m, np.array([0.0, -0.0, 1.0, -1.0, np.inf, -np.inf, np.nan], np.float32)])
    ys = [1.0, -1.0, 0.5, -3.0, 0.0]
    mm = np.tile(m, len(ys))
    yy = np.repeat(np.array(ys, np.float32), m.size)
    out = torch.empty(mm.size, dtype=torch.float32, device="cuda")
    pdb.pdb_eval_grad(torch.from_numpy(mm).cuda(), torch.from_numpy(yy).cuda(), out, loss)
    got = out.cpu().numpy()
    ref = np.array([oracle.grad(loss, float(a), float(b)) for a, b in zip(mm, yy)], np.float32)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan].view(np.uint32), ref[~nan].view(np.uint32))


@pytest.mark.parametrize("name", ALL)
def test_chains_bit_exact(name):
    p, X, y = _gpu(name)
    c = pdb.pdb_build_conflicts(X)
    pdb.check_status(c)
    arrs = pdb.pdb_conflicts_arrays(c)
    ref = C.oracle_chains(name)
    for key in ("csc_pos", "prev", "next", "rank"):
        assert np.array_equal(_arr(arrs[key], p.nnz, torch.int32), ref[key]), key
    assert np.array_equal(_arr(arrs["feat_ptr"], p.n_cols + 1, torch.int64), ref["feat_ptr"])
    st = pdb.pdb_get_stats(c)
    counts = np.diff(ref["feat_ptr"])
    assert st["max_chain"] == (counts.max() if counts.size else 0)


@pytest.mark.parametrize("n_rows", [45_000, 52_429])
def test_gate_words_past_the_l2_sized_path(n_rows):
    # above 2^22 positions the gate words return to position order through a
    # position sort and per-block inversion; 52,429 x 100 ids leave a ragged
    # last block (20 of 2^14 slots)
    import oracle
    import synthdata
    p = synthdata.generate("low-conflict", n_rows=n_rows, n_cols=2_000_000)
    assert p.nnz > (1 << 22)
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    arrs = pdb.pdb_conflicts_arrays(c)
    pdb.check_status(c)
    ref = oracle.chains(p)
    for key in ("prev", "next", "rank"):
        assert np.array_equal(_arr(arrs[key], p.nnz, torch.int32), ref[key]), key
    ref_w = oracle.sgd(p, epochs=1)
    # WINDOW reads the near pairs' gate words only; READY (and the admissible-delay
    # engine on it) the full position-order gate, built on first use
    for mode in (pdb.PDB_SCHED_WINDOW, pdb.PDB_SCHED_READY):
        c = pdb.pdb_build_conflicts(X)
        s = pdb.pdb_schedule_build(c, mode)
        w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
        pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, 1)
        pdb.check_status(c)
        assert np.array_equal(w.cpu().numpy(), ref_w), mode
        if mode == pdb.PDB_SCHED_READY:
            w.zero_()
            pdb.pdb_ssp_epoch(X, y, c, s, w, p.loss, p.eta, 1, 0)
            pdb.check_status(c)
            assert np.array_equal(w.cpu().numpy(), ref_w), "admissible delay 0"


@pytest.mark.parametrize("sweep", ["flow", "kahn"])
@pytest.mark.parametrize("name", ALL)
def test_levels_bit_exact(name, sweep, monkeypatch):
    # the dataflow level builder (default) and the Kahn frontier sweep
    monkeypatch.setenv("PDB_LEVELS", sweep)
    p, X, y = _gpu(name)
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_LEVELS)
    info = pdb.pdb_schedule_levels(s)
    pdb.check_status(c)
    lv, L, order, level_ptr = C.oracle_levels(name)
    assert info["n_levels"] == L
    assert np.array_equal(_arr(info["level"], p.n_rows, torch.int32), lv)
    assert np.array_equal(_arr(info["order"], p.n_rows, torch.int32), order)
    assert np.array_equal(_arr(info["level_ptr"], L + 1, torch.int64), level_ptr)
    st = pdb.pdb_get_stats(c, s)
    assert st["n_levels"] == L
    if L:
        assert st["max_level_width"] == np.max(np.diff(level_ptr))


def _sgd(name, mode, opts=None):
    p, X, y = _gpu(name)
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, mode)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs, opts=opts)
    pdb.check_status(c)
    return w.cpu().numpy()


MODES = {"levels": pdb.PDB_SCHED_LEVELS, "ready": pdb.PDB_SCHED_READY, "chain": pdb.PDB_SCHED_CHAIN,
         "window": pdb.PDB_SCHED_WINDOW}


@pytest.fixture
def near(monkeypatch):
    # the conflict build reads PDB_NEAR at each call: small distances make most
    # occurrence pairs "far", so small inputs run the watermark path
    def set_near(v):
        monkeypatch.setenv("PDB_NEAR", str(v))
    return set_near


@pytest.mark.parametrize("mode", list(MODES))
@pytest.mark.parametrize("name", ALL)
def test_sgd_weights(name, mode):
    got = _sgd(name, MODES[mode])
    ref = C.oracle_sgd(name)
    assert C.rel_err(got, ref) <= TOL
    assert np.array_equal(got, ref)       # same fp32 operation order on both sides


@pytest.mark.parametrize("near_dist", [1, 7, 300, 5000])
@pytest.mark.parametrize("name", ["tiny", "lowconflict-shape", "ragged-empty-rows", "zipf-shape", "long-rows",
                                  "ctr-shape-binary", "one-feature-chain", "exp-saturation"])
def test_window_watermark_path(name, near_dist, near):
    # WINDOW with most pairs far (watermark) or a mix of far and near pairs
    near(near_dist)
    got = _sgd(name, pdb.PDB_SCHED_WINDOW, opts=dict(wait_timeout_s=20.0))
    ref = C.oracle_sgd(name)
    assert C.rel_err(got, ref) <= TOL
    assert np.array_equal(got, ref)


def test_window_chunk_sizes(near):
    near(50)
    name = "lowconflict-shape"
    ref = C.oracle_sgd(name)
    for chunk in (1, 3, 16):
        got = _sgd(name, pdb.PDB_SCHED_WINDOW, opts=dict(ticket_chunk=chunk, blocks_per_sm=1))
        assert np.array_equal(got, ref), chunk


def test_auto_picks_window_when_near_pairs_are_rare(near):
    near(64)
    name = "lowconflict-shape"
    p, X, y = _gpu(name)
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_AUTO)
    assert pdb.pdb_get_stats(c, s)["sched_mode"] == pdb.PDB_SCHED_WINDOW
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs)
    pdb.check_status(c)
    assert np.array_equal(w.cpu().numpy(), C.oracle_sgd(name))


@pytest.mark.parametrize("name,expect", [("tiny", "ready"), ("lowconflict-shape", "ready"),
                                         ("zipf-shape", "chain"), ("deepchain-shape", "chain"),
                                         ("ctr-shape-binary", "chain"), ("one-feature-chain", "chain")])
def test_auto_schedule_choice(name, expect):
    p, X, y = _gpu(name)
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_AUTO)
    assert pdb.pdb_get_stats(c, s)["sched_mode"] == MODES[expect]
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs)
    pdb.check_status(c)
    assert np.array_equal(w.cpu().numpy(), C.oracle_sgd(name))


def test_chain_limits():
    # CHAIN keeps the weights in shared memory when they fit (rows of any
    # length); otherwise it forwards them between examples, for rows of at
    # most 256 ids, and refuses longer ones
    import synthdata
    p = synthdata.generate("tiny", n_rows=300, n_cols=2_000_000, k=300, k_lo=260)
    X = pdb.Csr.from_problem(p)
    c = pdb.pdb_build_conflicts(X)
    with pytest.raises(pdb.PdbError) as e:
        pdb.pdb_schedule_build(c, pdb.PDB_SCHED_CHAIN)
    assert e.value.code == pdb.PDB_ETOOBIG
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_AUTO)       # AUTO falls back
    assert pdb.pdb_get_stats(c, s)["sched_mode"] != pdb.PDB_SCHED_CHAIN


@pytest.mark.parametrize("mode", ["chain", "window", "ready"])
@pytest.mark.parametrize("shift", [1, 2, 3])
def test_unaligned_input_arrays(mode, shift):
    # ids and values that do not start on a 16-byte boundary (views into
    # larger buffers): the engines that stage rows in 16-byte pieces must
    # fall back to element copies and give the same weights
    for name in ("zipf-shape", "ids-18bit"):    # resident weights, and forwarded ones
        _unaligned_case(name, mode, shift)


def _unaligned_case(name, mode, shift):
    p = C.problem(name)
    col_buf = torch.zeros(p.nnz + shift, dtype=torch.int32, device="cuda")
    val_buf = torch.zeros(p.nnz + shift, dtype=torch.float32, device="cuda")
    col_buf[shift:] = torch.from_numpy(p.col).cuda()
    val_buf[shift:] = torch.from_numpy(p.val).cuda()
    X = pdb.Csr(torch.from_numpy(p.row_ptr).cuda(), col_buf[shift:], val_buf[shift:], p.n_cols)
    y = torch.from_numpy(p.y).cuda()
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, MODES[mode])
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, p.epochs)
    pdb.check_status(c)
    assert np.array_equal(w.cpu().numpy(), C.oracle_sgd(name))


def test_sgd_small_grid_and_repeat_calls():
    # a one-block-per-SM grid, and a second call continuing from the first
    name = "zipf-shape"
    p, X, y = _gpu(name)
    c = pdb.pdb_build_conflicts(X)
    for mode in (pdb.PDB_SCHED_LEVELS, pdb.PDB_SCHED_READY, pdb.PDB_SCHED_CHAIN, pdb.PDB_SCHED_WINDOW):
        s = pdb.pdb_schedule_build(c, mode)
        w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
        pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, 1, opts=dict(blocks_per_sm=1))
        pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, 1)
        pdb.check_status(c)
        import oracle
        assert np.array_equal(w.cpu().numpy(), oracle.sgd(p, epochs=2))


@pytest.mark.parametrize("batch", [1, 7, 64, 4096, 10**9])
@pytest.mark.parametrize("name", ["tiny", "deepchain-shape", "ragged-empty-rows", "ctr-shape-binary",
                                  "dense-shape"])
def test_bsp_weights(name, batch):
    import oracle
    p, X, y = _gpu(name)
    c = pdb.pdb_build_conflicts(X)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    epochs = min(p.epochs, 2)
    pdb.pdb_bsp_epoch(X, y, c, w, p.loss, p.eta, batch, epochs)
    pdb.check_status(c)
    ref = oracle.bsp(p, batch, epochs=epochs)
    got = w.cpu().numpy()
    assert C.rel_err(got, ref) <= TOL
    assert np.array_equal(got, ref)


@pytest.mark.parametrize("row_ptr,col,code", [
    ([0, 2, 1, 3], [0, 1, 2], -1),
    ([0, 2, 3], [0, 4, 1], -2),
    ([0, 2, 3], [0, -1, 1], -2),
    ([0, 3, 4], [2, 0, 2, 1], -3),
])
def test_device_validation(row_ptr, col, code):
    import synthdata
    p = synthdata.from_arrays(row_ptr, col, None, np.ones(len(row_ptr) - 1), n_cols=4)
    X = pdb.Csr.from_problem(p)
    c = pdb.pdb_build_conflicts(X)
    assert pdb.pdb_status(c) == code
    # a poisoned handle stays poisoned and later kernels do nothing
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY)
    y = torch.ones(p.n_rows, device="cuda")
    w = torch.zeros(4, device="cuda")
    pdb.pdb_sgd_epoch(X, y, c, s, w, 0, 0.1, 1)
    assert pdb.pdb_status(c) == code
    assert torch.count_nonzero(w).item() == 0


def test_wait_timeout_is_reported_not_hung():
    # One position waits for a version its feature never reaches: every
    # bounded wait gives up after the short limit, the kernel returns, the
    # status says so, and the context stays usable.
    name = "tiny"
    p, X, y = _gpu(name)
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY)
    pdb.check_status(c)
    gate_ptr = pdb.pdb_schedule_ready(s)["gate"]
    pos = int(p.row_ptr[5])                               # first element of example 5
    poison = torch.tensor([12345], dtype=torch.int32, device="cuda")
    pdb.pdb_memcpy(gate_ptr + 4 * pos, poison.data_ptr(), 4)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, 1, opts=dict(wait_timeout_s=0.2))
    assert pdb.pdb_status(c) == pdb.PDB_ETIMEOUT
    t = torch.arange(10, device="cuda").sum().item()     # the device still works
    assert t == 45


@pytest.mark.parametrize("near_dist", [1 << 22, 1])
def test_window_wait_timeout_is_reported_not_hung(near_dist, near):
    # WINDOW: one position waits for an iteration number nobody publishes, so
    # its chunk never finishes; with all pairs far (near_dist 1) every later
    # example also waits on the stalled watermark.  The waits give up after
    # the limit, the kernel returns and the status says so.
    near(near_dist)
    name = "tiny"
    p, X, y = _gpu(name)
    c = pdb.pdb_build_conflicts(X)
    s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_WINDOW)
    pdb.check_status(c)
    gate_ptr = pdb.pdb_schedule_ready(s)["gate"]
    pos = int(p.row_ptr[5])
    poison = torch.tensor([12345 | (1 << 30)], dtype=torch.int32, device="cuda")   # rank 12345, near previous
    pdb.pdb_memcpy(gate_ptr + 4 * pos, poison.data_ptr(), 4)
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, 1, opts=dict(wait_timeout_s=0.2))
    assert pdb.pdb_status(c) == pdb.PDB_ETIMEOUT
    assert torch.arange(10, device="cuda").sum().item() == 45
