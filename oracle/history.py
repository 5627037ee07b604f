"""Checker for read/write histories -- TEST INFRASTRUCTURE ONLY.

An operation is (kind, worker, chunk, iteration): kind 'r' or 'w', worker an
int or None (the paper drops it for a single worker), chunk the partition
index j of pi_j, iteration the alpha of the operation.  A history is the list
of operations in the order they executed.

Three predicates, each from the paper:

* ``is_sequential`` -- Definition 4: (i) the operations of one iteration are
  not interleaved with another iteration's, (ii) inside an iteration every
  read precedes every write, (iii) iteration alpha+1 starts only after all of
  alpha has completed.
* ``satisfies_rc_wc`` -- the Read Constraint (a read of chunk j in iteration
  alpha+1 comes after the write of chunk j in iteration alpha) and the Write
  Constraint (the write of chunk i in iteration alpha comes after every read
  of chunk i in iteration alpha), Section 4.4.
* ``per_chunk_sequential`` -- the three conditions of Theorem 2's proof,
  applied to the sub-history of each chunk separately.

And checkers of execution traces (per-example read and write timestamps, as
the library records them on request): ``trace_history`` turns one into a
history for the predicates above, ``trace_order_violations`` counts breaks of
the Read and Write Constraints directly at any size, and
``trace_delay_violations`` counts breaks of the asynchronous Read Constraint
of Section 7.
"""
from __future__ import annotations

import re
from collections import defaultdict

import numpy as np

_OP = re.compile(r"([rw])(?:_(\d+))?\[pi_(\d+)\]\[(\d+)\]")


def parse(text: str) -> list[tuple]:
    """Parse the paper's notation, e.g. ``r_1[pi_2][1] w[pi_1][2]``."""
    ops = []
    for m in _OP.finditer(text):
        kind, worker, chunk, it = m.groups()
        ops.append((kind, None if worker is None else int(worker), int(chunk), int(it)))
    return ops


def _sequential(ops) -> bool:
    seen_done = set()      # iterations whose block has ended
    current = None
    wrote = False
    last_iter = None
    for kind, _, _, it in ops:
        if it != current:
            if it in seen_done:
                return False                 # (i) iteration resumed after another one ran
            if last_iter is not None and it < last_iter:
                return False                 # (iii) iterations out of order
            if current is not None:
                seen_done.add(current)
            current, wrote, last_iter = it, False, it
        if kind == "w":
            wrote = True
        elif wrote:
            return False                     # (ii) read after a write in one iteration
    return True


def is_sequential(ops) -> bool:
    """Definition 4 over the whole history."""
    return _sequential(ops)


def satisfies_rc_wc(ops) -> bool:
    """Read Constraint and Write Constraint (Section 4.4) for every chunk."""
    pos_w = {}
    reads = defaultdict(list)
    for q, (kind, _, chunk, it) in enumerate(ops):
        if kind == "w":
            pos_w[(chunk, it)] = q
        else:
            reads[(chunk, it)].append(q)
    for q, (kind, _, chunk, it) in enumerate(ops):
        if kind == "r" and it > 1:
            wq = pos_w.get((chunk, it - 1))
            if wq is None or wq > q:
                return False                 # RC: w[pi_j][alpha] < r[pi_j][alpha+1]
        if kind == "w":
            if any(rq > q for rq in reads[(chunk, it)]):
                return False                 # WC: r[pi_i][alpha] < w[pi_i][alpha]
    return True


def per_chunk_sequential(ops) -> bool:
    """Theorem 2's conditions 1-3 on each chunk's own sub-history."""
    by_chunk = defaultdict(list)
    for op in ops:
        by_chunk[op[2]].append(op)
    return all(_sequential(sub) for sub in by_chunk.values())


def sparse_history(row_ptr, col, schedule) -> list[tuple]:
    """History of a sparse SGD run executed as ``schedule``.

    ``schedule`` is a list of steps; each step is a list of example ids whose
    reads all happen, then whose writes all happen (one barrier-separated BSP
    step; a single example per step is the sequential run).  Chunk = feature;
    the iteration number of a feature's operation is the occurrence index of
    that example among the examples holding the feature, counted from 1 in
    data order (the read protocol's per-chunk iteration number, Section 5).
    """
    occ = {}
    counter = defaultdict(int)
    for t in range(len(row_ptr) - 1):
        for p in range(row_ptr[t], row_ptr[t + 1]):
            j = int(col[p])
            counter[j] += 1
            occ[(t, j)] = counter[j]
    ops = []
    for step in schedule:
        for t in step:
            for p in range(row_ptr[t], row_ptr[t + 1]):
                j = int(col[p])
                ops.append(("r", int(t), j, occ[(t, j)]))
        for t in step:
            for p in range(row_ptr[t], row_ptr[t + 1]):
                j = int(col[p])
                ops.append(("w", int(t), j, occ[(t, j)]))
    return ops


# --- execution traces ------------------------------------------------------
# A trace (the library's optional per-example timestamps) is an array of
# shape (n_epochs * n_rows, 2): for example u of the epoch-major sequence
# (u = e * n_rows + t, data row t), column 0 is the time at which all of its
# reads were done and column 1 the time at which its update was computed,
# before any of its writes.  Chunk = feature, as in sparse_history.


def _occurrences(row_ptr, col, n_epochs):
    """(example u, feature j) of every occurrence over the epoch-major
    sequence, sorted by feature and then by example (data order)."""
    row_ptr = np.asarray(row_ptr, np.int64)
    n = len(row_ptr) - 1
    ex = np.repeat(np.arange(n, dtype=np.int64), np.diff(row_ptr))
    u = (ex[None, :] + n * np.arange(n_epochs, dtype=np.int64)[:, None]).ravel()
    j = np.tile(np.asarray(col, np.int64), n_epochs)
    o = np.lexsort((u, j))
    return u[o], j[o]


def trace_history(row_ptr, col, n_epochs, trace) -> list[tuple]:
    """History of a traced run: example u reads each of its features at
    trace[u, 0] and writes each at trace[u, 1]; the iteration number of an
    operation on feature j counts j's occurrences over the whole sequence
    from 1 (so an epoch's first occurrence follows the previous epoch's
    last).  Operations with equal stamps are taken in data order, an
    example's reads before its writes: a timer tick cannot order them."""
    trace = np.asarray(trace, np.int64).reshape(-1, 2)
    u, j = _occurrences(row_ptr, col, n_epochs)
    it = np.ones(u.size, np.int64)
    if u.size:
        first = np.r_[True, j[1:] != j[:-1]]
        start = np.maximum.accumulate(np.where(first, np.arange(u.size), 0))
        it = np.arange(u.size) - start + 1
    ops_of = defaultdict(list)
    for q in range(u.size):
        ops_of[int(u[q])].append((int(j[q]), int(it[q])))
    events = sorted((int(trace[x, kind]), x, kind) for x in ops_of for kind in (0, 1))
    ops = []
    for _, x, kind in events:
        for jj, a in ops_of[x]:
            ops.append(("r" if kind == 0 else "w", x, jj, a))
    return ops


def trace_order_violations(row_ptr, col, n_epochs, trace) -> dict:
    """The Read and Write Constraints (Section 4.4) on a trace, per feature:
    with one reader and one writer per iteration of a feature (the example
    holding that occurrence), they say that every example reads before it
    writes, and that the example holding occurrence alpha of a feature
    writes no later than the one holding occurrence alpha + 1 reads.
    Returns the number of examples and of occurrence pairs that break them."""
    trace = np.asarray(trace, np.int64).reshape(-1, 2)
    u, j = _occurrences(row_ptr, col, n_epochs)
    same = j[1:] == j[:-1]
    prev, nxt = u[:-1][same], u[1:][same]
    return dict(examples=int(trace.shape[0]), self=int(np.sum(trace[:, 0] > trace[:, 1])),
                pairs=int(prev.size), rc=int(np.sum(trace[prev, 1] > trace[nxt, 0])))


def trace_delay_violations(row_ptr, col, n_epochs, trace, delay: int) -> dict:
    """The asynchronous Read Constraint (Section 7) on a trace, one epoch at a
    time, in its per-feature counting form: when the occurrence of feature j
    with 0-based rank r (data order within the epoch) has read, at least
    r - delay occurrences of j have written.  A write counts from the stamp
    taken before it, so this is a necessary condition of the constraint.
    delay = 0 is the exact Read Constraint within an epoch."""
    trace = np.asarray(trace, np.int64).reshape(-1, 2)
    n = len(row_ptr) - 1
    u, j = _occurrences(row_ptr, col, n_epochs)
    if u.size == 0:
        return dict(reads=0, violations=0)
    key = (u // n) * (int(np.max(j)) + 1) + j            # (epoch, feature) group
    o = np.lexsort((u, key))
    u, key = u[o], key[o]
    first = np.r_[True, key[1:] != key[:-1]]
    start = np.maximum.accumulate(np.where(first, np.arange(u.size), 0))
    rank = np.arange(u.size) - start
    # merge every group's write stamps with its read stamps: at equal stamps
    # a write sorts first (a tick cannot order them)
    times = np.r_[trace[u, 1], trace[u, 0]]
    kind = np.r_[np.zeros(u.size, np.int64), np.ones(u.size, np.int64)]
    keys = np.r_[key, key]
    o = np.lexsort((kind, times, keys))
    is_w = kind[o] == 0
    cw = np.cumsum(is_w)
    gfirst = np.r_[True, keys[o][1:] != keys[o][:-1]]
    base = np.maximum.accumulate(np.where(gfirst, np.arange(o.size), 0))
    done = cw - (cw[base] - is_w[base])                    # writes of the group at or before each event
    rd = ~is_w
    need = rank[(o[rd] - u.size)] - delay
    return dict(reads=int(rd.sum()), violations=int(np.sum(done[rd] < need)))
