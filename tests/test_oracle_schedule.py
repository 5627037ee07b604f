"""Pins for the oracle's validation, occurrence chains and dependency levels:
brute force on small inputs, library sorts, and the invariants the paper's
Theorems 2 and 3 fix for a level schedule."""
import numpy as np
import pytest

import oracle
import synthdata
from oracle import history


def _small(seed, n=60, f=25, k=6, k_lo=0, ids="uniform", s=1.1):
    return synthdata.generate("tiny", seed=seed, n_rows=n, n_cols=f, k=k, k_lo=k_lo, ids=ids, zipf_s=s)


def test_validate_accepts_good_and_empty_rows():
    assert oracle.validate(synthdata.generate("tiny")) == oracle.OK
    p = synthdata.from_arrays([0, 0, 2, 2, 3], [1, 4, 1], None, [1, 1, 1, 1], n_cols=5)
    assert oracle.validate(p) == oracle.OK


@pytest.mark.parametrize("row_ptr,col,n_cols,code", [
    ([1, 2, 3], [0, 1], 4, oracle.BAD_ROWPTR),       # row_ptr[0] != 0
    ([0, 2, 1, 3], [0, 1, 2], 4, oracle.BAD_ROWPTR),  # decreasing
    ([0, 1, 2], [0, 1, 2], 4, oracle.BAD_ROWPTR),     # row_ptr[N] != nnz
    ([0, 2], [0, 4], 4, oracle.BAD_COL),              # id == F
    ([0, 2], [-1, 0], 4, oracle.BAD_COL),             # negative id
    ([0, 3], [2, 0, 2], 4, oracle.DUP),               # repeated id in one row
])
def test_validate_rejects(row_ptr, col, n_cols, code):
    p = synthdata.from_arrays(row_ptr, col, None, np.ones(len(row_ptr) - 1), n_cols=n_cols)
    assert oracle.validate(p) == code


def test_validate_same_feature_in_two_rows_is_fine():
    p = synthdata.from_arrays([0, 2, 4], [0, 3, 3, 0], None, [1, 1], n_cols=4)
    assert oracle.validate(p) == oracle.OK


@pytest.mark.parametrize("seed", range(12))
def test_chains_brute_force(seed):
    p = _small(seed, ids="zipf" if seed % 2 else "uniform")
    ch = oracle.chains(p)
    col = p.col
    nnz = p.nnz
    for q in range(nnz):
        same = np.nonzero(col == col[q])[0]
        earlier, later = same[same < q], same[same > q]
        assert ch["prev"][q] == (earlier.max() if earlier.size else -1)
        assert ch["next"][q] == (later.min() if later.size else -1)
        assert ch["rank"][q] == earlier.size
    # CSC = stable sort of positions by feature, delimited by the histogram
    assert np.array_equal(ch["csc_pos"], np.argsort(col, kind="stable"))
    assert np.array_equal(ch["feat_ptr"], np.concatenate([[0], np.cumsum(np.bincount(col, minlength=p.n_cols))]))


def test_chains_on_empty_input():
    p = synthdata.from_arrays([0, 0, 0], [], None, [1, 1], n_cols=3)
    ch = oracle.chains(p)
    assert ch["csc_pos"].size == 0 and list(ch["feat_ptr"]) == [0, 0, 0, 0]
    lv, L = oracle.levels(p, ch["prev"])
    assert list(lv) == [0, 0] and L == 1


@pytest.mark.parametrize("seed", range(16))
def test_levels_equal_brute_force(seed):
    p = _small(seed, n=80 if seed < 8 else 40, f=30 if seed % 3 else 8, k=5,
               ids="zipf" if seed % 2 else "uniform")
    lv, L = oracle.levels(p)
    bf = oracle.levels_bruteforce(p)
    assert np.array_equal(lv, bf)
    assert L == (bf.max() + 1 if bf.size else 0)


def test_levels_single_predecessor_chain():
    # each example shares exactly one feature with the one before (the first
    # link is position 0): the levels count the hops, 0, 1, 2, ...; an
    # example that reuses no feature stays at level 0
    p = synthdata.from_arrays([0, 1, 3, 5, 7, 8], [0, 0, 1, 1, 2, 2, 3, 9], None, np.ones(5), n_cols=10)
    lv, L = oracle.levels(p)
    assert lv.tolist() == [0, 1, 2, 3, 0]
    assert L == 4
    assert np.array_equal(lv, oracle.levels_bruteforce(p))


def _check_level_invariants(p, lv):
    sets = [set(p.col[p.row_ptr[t]:p.row_ptr[t + 1]].tolist()) for t in range(p.n_rows)]
    by_level = {}
    for t, l in enumerate(lv):
        by_level.setdefault(int(l), []).append(t)
    # examples of one level are pairwise feature-disjoint
    for rows in by_level.values():
        seen = set()
        for t in rows:
            assert not (sets[t] & seen)
            seen |= sets[t]
    # minimal: a level-l example (l > 0) conflicts with an earlier one at l-1;
    # a level-0 example conflicts with no earlier one; levels grow along conflicts
    last = {}
    for t in range(p.n_rows):
        pred_levels = [lv[last[j]] for j in sets[t] if j in last]
        if lv[t] == 0:
            assert not pred_levels
        else:
            assert max(pred_levels) == lv[t] - 1
        for j in sets[t]:
            last[j] = t


def test_level_invariants_tiny_workload():
    p = synthdata.generate("tiny", n_rows=3000)
    lv, L = oracle.levels(p)
    _check_level_invariants(p, lv)
    assert L == lv.max() + 1


def test_level_invariants_zipf_shape():
    p = synthdata.generate("zipf-1m", n_rows=2000, n_cols=5000)
    lv, _ = oracle.levels(p)
    _check_level_invariants(p, lv)


def test_level_order_is_stable_by_level_then_id():
    p = synthdata.generate("tiny", n_rows=5000)
    lv, L = oracle.levels(p)
    order, level_ptr = oracle.level_order(lv, L)
    assert np.array_equal(order, np.lexsort((np.arange(p.n_rows), lv)))
    assert np.array_equal(np.diff(level_ptr), np.bincount(lv, minlength=L))
    assert level_ptr[0] == 0 and level_ptr[-1] == p.n_rows


@pytest.mark.parametrize("seed", range(6))
def test_level_schedule_history_satisfies_rc_wc(seed):
    # Theorem 3: running each level as one BSP step is one of the executions
    # the read and write constraints allow, hence (Theorem 2) sequential per chunk.
    p = _small(seed, n=50, f=20, k=4, ids="zipf")
    lv, L = oracle.levels(p)
    sched = [list(np.nonzero(lv == l)[0]) for l in range(L)]
    h = history.sparse_history(p.row_ptr, p.col, sched)
    assert history.satisfies_rc_wc(h) and history.per_chunk_sequential(h)


def test_merged_conflicting_levels_violate_rc_wc():
    p = _small(3, n=50, f=20, k=4, ids="zipf")
    lv, L = oracle.levels(p)
    assert L >= 2
    sched = [list(np.nonzero(lv == l)[0]) for l in range(L)]
    bad = [sched[0] + sched[1]] + sched[2:]       # a level-1 example reads with its predecessor
    h = history.sparse_history(p.row_ptr, p.col, bad)
    assert not history.satisfies_rc_wc(h)
    assert not history.per_chunk_sequential(h)
