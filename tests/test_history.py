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
