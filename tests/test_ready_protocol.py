"""A model check of the READY schedule's protocol, on the CPU.

READY keeps per feature one record (weight, version).  The occurrence of
feature j with rank r waits until the version equals r plus the epoch's stamp
(1 + e mod 7, in the version's top bits), reads the weight with the same
load, and later publishes (new weight, r + 1 plus the stamp) -- or, for the
feature's last occurrence of the epoch, version 0 plus the next epoch's
stamp.  All epochs run in one launch: workers take tickets over the
epoch-major sequence of examples, so epoch e + 1 starts while epoch e
finishes (cross-epoch pipelining), and the stamps keep a record of one
epoch from satisfying a wait of another.

This test restates those rules as a state machine and runs it under random
interleavings of workers taking tickets in order, with every read and every
write of every position a separate step, and checks that each read observes
exactly the write of the previous occurrence of its feature in the
epoch-major data order (Section 4.4's Read Constraint across epochs, the
reading of several epochs), and that the workers never deadlock.  It also
checks that without the stamps (versions reset every epoch but no epoch in
the word) some interleaving reads a weight of the wrong epoch."""
import numpy as np
import pytest

import oracle
import synthdata


def _simulate(p, chunk, n_workers, epochs, rng, stamps=True, slow_ticket=None):
    ch = oracle.chains(p)
    prev, rank = ch["prev"], ch["rank"]
    row_ptr, col = p.row_ptr, p.col
    n = p.n_rows
    row_of = np.repeat(np.arange(n), np.diff(row_ptr))
    last_pos = np.full(p.n_cols, -1)
    for q in range(p.nnz):
        last_pos[col[q]] = q
    is_last = np.zeros(p.nnz, bool)
    is_last[last_pos[last_pos >= 0]] = True

    def stamp(e):
        return (1 + e % 7) if stamps else 0

    # record per feature: (version, stamp, (epoch, example) of the writer or None)
    rec = {j: (0, stamp(0), None) for j in range(p.n_cols)}
    total = epochs * n
    tickets = (total + chunk - 1) // chunk
    next_ticket = 0
    done = 0
    workers = [None] * n_workers          # [ticket, index in ticket, phase, pending positions]
    steps = 0
    while done < total:
        steps += 1
        assert steps < 200 * (epochs * p.nnz + total + 10), "no progress"
        enabled = []
        for wi, st in enumerate(workers):
            if st is None:
                if next_ticket < tickets:
                    enabled.append((wi, "take", None))
                continue
            tk, ti, phase, pending = st
            u = tk * chunk + ti
            e = u // n
            for q in pending:
                if phase == "read":
                    v, s, _ = rec[int(col[q])]
                    if v == int(rank[q]) and s == stamp(e):
                        enabled.append((wi, phase, q))
                else:
                    enabled.append((wi, phase, q))
            if not pending:
                enabled.append((wi, "next", None))
        assert enabled, "deadlock"
        if slow_ticket is not None and rng.random() < 0.99:
            # the worker holding this ticket runs only when nobody else can
            slow = [wi for wi, st in enumerate(workers) if st is not None and st[0] == slow_ticket]
            others = [x for x in enabled if x[0] not in slow]
            enabled = others or enabled
        wi, kind, q = enabled[rng.integers(len(enabled))]
        if kind == "take":
            tk = next_ticket
            next_ticket += 1
            u = tk * chunk
            t = u % n
            workers[wi] = [tk, 0, "read", list(range(int(row_ptr[t]), int(row_ptr[t + 1])))]
            continue
        tk, ti, phase, pending = workers[wi]
        u = tk * chunk + ti
        e, t = divmod(u, n)
        if kind == "read":
            j = int(col[q])
            seen = rec[j][2]
            if prev[q] >= 0:
                want = (e, int(row_of[prev[q]]))
            else:                                  # first occurrence of the epoch
                want = (e - 1, int(row_of[last_pos[j]])) if e > 0 else None
            assert seen == want, (e, t, q, seen, want)
            pending.remove(q)
            if not pending:
                workers[wi] = [tk, ti, "write", list(range(int(row_ptr[t]), int(row_ptr[t + 1])))]
        elif kind == "write":
            j = int(col[q])
            if is_last[q]:
                rec[j] = (0, stamp(e + 1), (e, t))
            else:
                rec[j] = (int(rank[q]) + 1, stamp(e), (e, t))
            pending.remove(q)
        else:                                      # the example is finished
            done += 1
            ti += 1
            u = tk * chunk + ti
            if ti < chunk and u < total:
                t = u % n
                workers[wi] = [tk, ti, "read", list(range(int(row_ptr[t]), int(row_ptr[t + 1])))]
            else:
                workers[wi] = None


def _problem(seed, rng):
    return synthdata.generate("tiny", seed=seed, n_rows=int(rng.integers(20, 60)), n_cols=int(rng.integers(5, 30)),
                              k=int(rng.integers(1, 5)), k_lo=0, ids="zipf" if seed % 2 else "uniform", zipf_s=1.1)


@pytest.mark.parametrize("seed", range(12))
def test_ready_protocol_reads_follow_data_order_across_epochs(seed):
    rng = np.random.default_rng(100 + seed)
    p = _problem(seed, rng)
    _simulate(p, chunk=int(rng.integers(1, 4)), n_workers=int(rng.integers(1, 8)), epochs=int(rng.integers(1, 10)),
              rng=rng)


@pytest.mark.parametrize("seed", range(4))
def test_ready_protocol_with_a_slow_worker(seed):
    # the worker holding the first example runs only when nobody else can:
    # epochs overlap as far as the dependencies allow
    rng = np.random.default_rng(200 + seed)
    p = _problem(seed, rng)
    _simulate(p, chunk=1, n_workers=6, epochs=4, rng=rng, slow_ticket=0)


def test_ready_protocol_model_needs_the_epoch_stamps():
    # planted in the model: no epoch in the version word.  Feature 0 occurs
    # once per epoch (example 0), so its occurrence of epoch 1 waits for
    # version 0 -- which the record already holds from the start while the
    # slow worker still has epoch 0's occurrence: it reads a stale weight
    n = 24
    row_ptr = np.arange(n + 1) * 2
    col = np.concatenate([[0, 1]] + [[1 + (t % 5), 6 + (t % 7)] for t in range(1, n)])
    p = synthdata.from_arrays(row_ptr, col, None, np.ones(n), n_cols=13)
    rng = np.random.default_rng(5)
    _simulate(p, chunk=1, n_workers=6, epochs=2, rng=rng, slow_ticket=0)       # with stamps: fine
    failures = 0
    for _ in range(10):
        try:
            _simulate(p, chunk=1, n_workers=6, epochs=2, rng=rng, stamps=False, slow_ticket=0)
        except AssertionError:
            failures += 1
    assert failures > 0


@pytest.mark.parametrize("seed", range(3))
def test_ready_protocol_past_the_stamp_wrap(seed):
    # stamps repeat every 7 epochs: 16 epochs with a slow worker (and with
    # chunks of several examples) must still read only the right epoch's
    # records
    rng = np.random.default_rng(400 + seed)
    p = _problem(seed, rng)
    _simulate(p, chunk=1, n_workers=5, epochs=16, rng=rng, slow_ticket=0)
    _simulate(p, chunk=3, n_workers=4, epochs=16, rng=rng, slow_ticket=1)
