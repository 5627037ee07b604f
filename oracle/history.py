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
"""
from __future__ import annotations

import re
from collections import defaultdict

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
