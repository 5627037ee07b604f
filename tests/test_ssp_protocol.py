"""A model check of the admissible-delay protocol (Section 7), on the CPU.

Iterations are counted per feature: the occurrence of feature j with rank r
(0-based, data order within the epoch) is iteration r of j.  Two forms of
the gates are modelled.

count   (the GPU engine, k_sgd_ssp): per feature a writes counter and a
        reads counter; rank r may read w_j once writes_j >= r - delta, and
        may write (an atomic add of its step) once reads_j >= r - delta + 1.
prefix  (the paper's protocols read per feature, "the slowest reader" and
        "the last write" as prefixes of ranks): rank r may read once every
        rank <= r - 1 - delta has written, and may write once every rank
        <= r - delta has read.

Workers take examples in data order; every read and every write of every
position is a separate step of the model, interleaved at random, and with a
worker that holds an early example and runs only when nobody else can.

Checked for both forms: no deadlock; every read of rank r sees at least
r - delta writes of its feature; every step is applied exactly once; at
delta = 0 each read sees exactly the writes of ranks 0 .. r - 1 (the
sequential computation).  For the prefix form also the two-sided bound of
Section 7's Asynchronous Read and Write Constraints: a read of rank r sees
every write of rank <= r - 1 - delta and none of rank >= r + delta.  The count
form does not keep that bound once delta >= 1: a slow reader holds no writer
back (test_count_form_lets_a_slow_reader_see_far_future_writes)."""
import numpy as np
import pytest

import oracle
import synthdata


def _prefix(done):
    k = 0
    while k in done:
        k += 1
    return k


def _simulate(p, delay, n_workers, rng, slow_ticket=None, form="count", read_wait=True, write_wait=True):
    """Runs one epoch; returns the number of reads that broke the two-sided
    bound (saw a write of rank >= r + delta, or missed one of rank
    <= r - 1 - delta) and the number that missed any earlier write."""
    ch = oracle.chains(p)
    rank = ch["rank"]
    row_ptr, col = p.row_ptr, p.col
    n = p.n_rows
    read_ranks = {j: set() for j in range(p.n_cols)}
    applied = {j: [] for j in range(p.n_cols)}     # ranks whose step is in w_j, in order

    def may_read(j, r):
        done = len(applied[j]) if form == "count" else _prefix(set(applied[j]))
        return done >= r - delay

    def may_write(j, r):
        done = len(read_ranks[j]) if form == "count" else _prefix(read_ranks[j])
        return done >= r - delay + 1

    next_ticket, done, broken, stale = 0, 0, 0, 0
    workers = [None] * n_workers                   # [example, phase, pending positions]
    steps = 0
    while done < n:
        steps += 1
        assert steps < 100 * (p.nnz + n + 10), "no progress"
        enabled = []
        for wi, st in enumerate(workers):
            if st is None:
                if next_ticket < n:
                    enabled.append((wi, "take", None))
                continue
            t, phase, pending = st
            for q in pending:
                j, r = int(col[q]), int(rank[q])
                if phase == "read" and (may_read(j, r) or not read_wait):
                    enabled.append((wi, "read", q))
                if phase == "write" and (may_write(j, r) or not write_wait):
                    enabled.append((wi, "write", q))
            if not pending:
                enabled.append((wi, "next", None))
        assert enabled, "deadlock"
        if slow_ticket is not None and rng.random() < 0.99:
            slow = [wi for wi, st in enumerate(workers) if st is not None and st[0] == slow_ticket]
            enabled = [x for x in enabled if x[0] not in slow] or enabled
        wi, kind, q = enabled[rng.integers(len(enabled))]
        if kind == "take":
            t = next_ticket
            next_ticket += 1
            workers[wi] = [t, "read", list(range(int(row_ptr[t]), int(row_ptr[t + 1])))]
            continue
        t, phase, pending = workers[wi]
        if kind == "read":
            j, r = int(col[q]), int(rank[q])
            seen = set(applied[j])
            if read_wait:
                assert len(seen) >= r - delay                   # at most delay occurrences stale
            if delay == 0 and read_wait and write_wait:
                assert applied[j] == list(range(r))             # exactly the earlier occurrences
            ok = set(range(max(0, r - delay))) <= seen and not any(s >= r + delay for s in seen)
            broken += not ok
            stale += seen != set(range(r))
            if form == "prefix" and read_wait and write_wait:
                assert ok, (j, r, sorted(seen))
            read_ranks[j].add(r)
            pending.remove(q)
            if not pending:
                workers[wi] = [t, "write", list(range(int(row_ptr[t]), int(row_ptr[t + 1])))]
        elif kind == "write":
            j, r = int(col[q]), int(rank[q])
            applied[j].append(r)
            pending.remove(q)
        else:
            done += 1
            workers[wi] = None
    for j in range(p.n_cols):
        cnt = ch["feat_ptr"][j + 1] - ch["feat_ptr"][j]
        assert sorted(applied[j]) == list(range(cnt))           # every step exactly once
    return broken, stale


def _problem(seed, rng):
    return synthdata.generate("tiny", seed=seed, n_rows=int(rng.integers(20, 70)), n_cols=int(rng.integers(4, 25)),
                              k=int(rng.integers(1, 5)), k_lo=0, ids="zipf" if seed % 2 else "uniform", zipf_s=1.1)


def _one_feature(n):
    # n examples, each the single occurrence of feature 0: one chain of n hops
    return synthdata.from_arrays(np.arange(n + 1), np.zeros(n, np.int32), None, np.ones(n), n_cols=1)


@pytest.mark.parametrize("form", ["count", "prefix"])
@pytest.mark.parametrize("delay", [0, 1, 3, 16, 1000])
@pytest.mark.parametrize("seed", range(4))
def test_admissible_delay_protocol(seed, delay, form):
    rng = np.random.default_rng(300 + 10 * seed + delay)
    p = _problem(seed, rng)
    _simulate(p, delay, n_workers=int(rng.integers(1, 8)), rng=rng, form=form)
    _simulate(p, delay, n_workers=6, rng=rng, slow_ticket=0, form=form)


@pytest.mark.parametrize("form", ["count", "prefix"])
def test_delay_admits_stale_reads(form):
    # delay > 0 really lets a read run ahead of earlier writes (else the
    # protocol would be the exact one in disguise)
    rng = np.random.default_rng(9)
    p = _one_feature(40)
    stale = sum(_simulate(p, 4, n_workers=8, rng=rng, form=form)[1] for _ in range(5))
    assert stale > 0


def test_count_form_lets_a_slow_reader_see_far_future_writes():
    # the engine's counting gates, delta = 2: the worker holding example 0
    # (rank 0) is slow; the other ranks' reads and writes fill the counters,
    # so writes of rank >= 2 land before rank 0 reads.  The prefix form (the
    # slowest reader holds writers back) never lets that happen
    rng = np.random.default_rng(4)
    p = _one_feature(30)
    assert sum(_simulate(p, 2, n_workers=6, rng=rng, slow_ticket=0, form="count")[0] for _ in range(5)) > 0
    for _ in range(5):
        assert _simulate(p, 2, n_workers=6, rng=rng, slow_ticket=0, form="prefix")[0] == 0


@pytest.mark.parametrize("form", ["count", "prefix"])
def test_ssp_protocol_model_needs_the_read_wait(form):
    # planted in the model: reads skip their gate; at delta = 0 some read
    # then misses the write of the previous occurrence
    rng = np.random.default_rng(11)
    p = synthdata.generate("tiny", seed=2, n_rows=50, n_cols=5, k=3, k_lo=1)
    assert sum(_simulate(p, 0, n_workers=6, rng=rng, form=form, read_wait=False)[1] for _ in range(10)) > 0


def test_ssp_protocol_model_needs_the_write_wait():
    # planted in the model: writes skip their gate (prefix form, delta = 1);
    # a write of rank r then lands before the read of rank r - 1, which sees
    # a write of rank >= its own + delta.  (At delta = 0 the read gate alone
    # already orders everything: rank r reads only after r writes, and a
    # write follows its own read.)
    rng = np.random.default_rng(12)
    p = _one_feature(30)
    assert sum(_simulate(p, 1, n_workers=6, rng=rng, slow_ticket=0, form="prefix", write_wait=False)[0]
               for _ in range(5)) > 0
