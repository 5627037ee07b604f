"""The history checker against the histories the paper prints, and against
Theorems 1-3 on randomly generated worker executions."""
import os

import numpy as np
import pytest

from oracle import history

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "histories.txt")


def _golden():
    rows = []
    for line in open(GOLDEN):
        if line.strip() and not line.startswith("#"):
            name, seq, rcwc, text = [x.strip() for x in line.split("|")]
            rows.append((name, bool(int(seq)), bool(int(rcwc)), history.parse(text)))
    return rows


@pytest.mark.parametrize("name,seq,rcwc,ops", _golden(), ids=[r[0] for r in _golden()])
def test_paper_histories(name, seq, rcwc, ops):
    assert len(ops) in (8, 12)
    assert history.is_sequential(ops) == seq
    assert history.satisfies_rc_wc(ops) == rcwc
    assert history.per_chunk_sequential(ops) == rcwc


def _bsp_history(p, iters, rng):
    """Algorithm 2a: read barrier, all reads (any order), write barrier, writes."""
    ops = []
    for a in range(1, iters + 1):
        reads = [("r", i, j, a) for i in range(1, p + 1) for j in range(1, p + 1)]
        writes = [("w", i, i, a) for i in range(1, p + 1)]
        ops += [reads[q] for q in rng.permutation(len(reads))]
        ops += [writes[q] for q in rng.permutation(len(writes))]
    return ops


def _random_interleaving(p, iters, rng):
    """Each worker i runs: for each iteration, read every chunk (random order), write pi_i."""
    progs = []
    for i in range(1, p + 1):
        prog = []
        for a in range(1, iters + 1):
            prog += [("r", i, int(j) + 1, a) for j in rng.permutation(p)]
            prog.append(("w", i, i, a))
        progs.append(prog)
    idx = [0] * p
    ops = []
    while any(idx[i] < len(progs[i]) for i in range(p)):
        i = rng.choice([i for i in range(p) if idx[i] < len(progs[i])])
        ops.append(progs[i][idx[i]])
        idx[i] += 1
    return ops


def test_theorem1_and_3_bsp_histories():
    rng = np.random.default_rng(0)
    for _ in range(200):
        h = _bsp_history(int(rng.integers(1, 5)), int(rng.integers(1, 4)), rng)
        assert history.is_sequential(h)              # Theorem 1
        assert history.satisfies_rc_wc(h)            # Theorem 3
        assert history.per_chunk_sequential(h)


def test_theorem2_random_executions():
    rng = np.random.default_rng(1)
    n_ok = n_bad = 0
    for _ in range(3000):
        h = _random_interleaving(int(rng.integers(2, 4)), int(rng.integers(1, 4)), rng)
        ok = history.satisfies_rc_wc(h)
        if ok:
            n_ok += 1
            assert history.per_chunk_sequential(h)   # Theorem 2
        else:
            n_bad += 1
            assert not history.per_chunk_sequential(h)
    assert n_ok > 0 and n_bad > 0


# --- execution-trace checkers ---------------------------------------------

def _small_problem(seed, n=300, f=60, k=4):
    rng = np.random.default_rng(seed)
    lens = rng.integers(0, k + 1, n)
    rp = np.r_[0, np.cumsum(lens)]
    col = np.concatenate([np.sort(rng.permutation(f)[:m]) for m in lens]).astype(np.int64)
    return rp, col


def _brute_pairs(rp, col, n_epochs, tr):
    """Consecutive-occurrence pairs and their breaks, by plain loops."""
    n = len(rp) - 1
    last = {}
    pairs = rc = 0
    for u in range(n * n_epochs):
        t = u % n
        for p in range(rp[t], rp[t + 1]):
            j = int(col[p])
            if j in last:
                pairs += 1
                rc += tr[last[j], 1] > tr[u, 0]
            last[j] = u
    return pairs, rc


def _brute_delay(rp, col, n_epochs, tr, delay):
    n = len(rp) - 1
    bad = reads = 0
    for e in range(n_epochs):
        occ = {}
        for t in range(n):
            for p in range(rp[t], rp[t + 1]):
                occ.setdefault(int(col[p]), []).append(e * n + t)
        for us in occ.values():
            for r, u in enumerate(us):
                reads += 1
                done = sum(1 for q in us if tr[q, 1] <= tr[u, 0])
                bad += done < r - delay
    return reads, bad


def test_trace_sequential_and_level_traces_pass():
    # data order (Algorithm 1) and level order (Theorem 3) both satisfy RC/WC
    import oracle
    import synthdata
    rp, col = _small_problem(0)
    n, E = len(rp) - 1, 3
    seq = np.stack([2 * np.arange(n * E), 2 * np.arange(n * E) + 1], 1)
    assert history.trace_order_violations(rp, col, E, seq)["rc"] == 0
    ops = history.trace_history(rp, col, E, seq)
    assert history.satisfies_rc_wc(ops) and history.per_chunk_sequential(ops)
    assert history.trace_delay_violations(rp, col, E, seq, 0)["violations"] == 0
    p = synthdata.from_arrays(rp, col, np.ones(col.size), np.ones(n), n_cols=60)
    lv, L = oracle.levels(p)
    u = np.arange(n * E)
    lvl = (u // n) * (L + 1) + lv[u % n]
    tr = np.stack([3 * lvl, 3 * lvl + 1], 1)       # every example of a level reads, then all write
    v = history.trace_order_violations(rp, col, E, tr)
    assert v["self"] == 0 and v["rc"] == 0 and v["pairs"] > 0
    assert history.satisfies_rc_wc(history.trace_history(rp, col, E, tr))


def test_trace_batch_with_conflicts_is_rejected():
    # a BSP step (Algorithm 2a) over a batch of conflicting examples reads the
    # old weights of a feature another example of the batch writes: RC broken
    rp, col = _small_problem(1)
    n = len(rp) - 1
    B = 16
    u = np.arange(n)
    tr = np.stack([2 * (u // B), 2 * (u // B) + 1], 1)
    v = history.trace_order_violations(rp, col, 1, tr)
    conflicts_in_batch = 0
    for b0 in range(0, n, B):
        seen = set()
        for t in range(b0, min(n, b0 + B)):
            row = set(col[rp[t]:rp[t + 1]].tolist())
            conflicts_in_batch += len(row & seen)
            seen |= row
    assert v["rc"] == conflicts_in_batch > 0
    assert not history.satisfies_rc_wc(history.trace_history(rp, col, 1, tr))


@pytest.mark.parametrize("seed", range(6))
def test_trace_checkers_match_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    rp, col = _small_problem(seed, n=120, f=25, k=5)
    n, E = len(rp) - 1, int(rng.integers(1, 4))
    base = 4 * np.arange(n * E)
    # jittered data order with coarse ticks: some traces pass, some break RC,
    # many stamps tie
    jit = rng.integers(-int(rng.integers(0, 12)), 1 + int(rng.integers(0, 12)), size=(n * E, 2))
    tr = (base[:, None] + np.array([0, 2]) + jit) // int(rng.integers(1, 5))
    v = history.trace_order_violations(rp, col, E, tr)
    assert (v["pairs"], v["rc"]) == _brute_pairs(rp, col, E, tr)
    assert v["self"] == int(np.sum(tr[:, 0] > tr[:, 1]))
    ok = v["self"] == 0 and v["rc"] == 0
    assert history.satisfies_rc_wc(history.trace_history(rp, col, E, tr)) == ok
    for delay in (0, 1, 3, 50):
        d = history.trace_delay_violations(rp, col, E, tr, delay)
        assert (d["reads"], d["violations"]) == _brute_delay(rp, col, E, tr, delay)


def test_trace_delay_fully_parallel_epoch():
    # every example reads at 0 and writes at 1 (Hogwild-like): a read of rank
    # r sees no write, so it breaks the delay-delta constraint iff r > delta
    rp, col = _small_problem(3)
    n = len(rp) - 1
    tr = np.tile([0, 1], (n, 1))
    counts = np.bincount(col, minlength=60)
    for delay in (0, 1, 2, 5, 1000):
        want = int(sum(max(0, c - 1 - delay) for c in counts))
        assert history.trace_delay_violations(rp, col, 1, tr, delay)["violations"] == want
