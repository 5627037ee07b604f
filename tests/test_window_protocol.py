"""A model check of the WINDOW schedule's protocol, on the CPU.

The WINDOW engine lets a position read its feature's weight in one of two
ways: if the previous occurrence lies closer than `near` positions, from a
hand-off record tagged with the reader's occurrence rank (and epoch); else
(previous occurrence far, or none at all) from the plain weight array once
the completion watermark -- the first position of the oldest unfinished
chunk of examples -- has reached min(first position of the reader's chunk,
end of the reader's example - near).  A position writes into the record when
its next occurrence is near, else into the array.

This test restates those rules as a state machine, runs it under random
interleavings of workers that take chunks of examples in data order, with
every read and every write of every position a separate step, and checks
that each read observes exactly the write of the previous occurrence of its
feature in data order (the Read Constraint of Section 4.4, which with one
writer per occurrence gives the sequential result, Theorem 2), and that the
workers never deadlock.  Occurrence chains come from the oracle.  The
watermark is either the exact one (the first position of the oldest
unfinished chunk) or the engine's: a worker that has finished chunk c sets
done[c] when it has taken its next chunk, before that chunk's first read
(or when the tickets run out); a sweeper reads the flags one at a time from
its current chunk (each read a step of its own), and when it meets an unset
flag (or has read a span of them) it publishes the first position of the
first chunk it has not seen set, raising the watermark only.

Some workers may start late: they take no step until a started worker has
exited, as thread blocks the device has not made resident start only when a
running block finishes.  The engine's watermark must not wait for them.  The
rule the engine used before, a progress word per worker that starts at 0
and that the sweeper takes the minimum of, is kept as a planted variant: a
late worker's word pins the watermark and the model reports no progress."""
import numpy as np
import pytest

import oracle
import synthdata


INF = 1 << 62


SPAN = 3     # flags the model's sweeper reads before it publishes


def _simulate(p, near, chunk, n_workers, epochs, rng, watermark_wait=True, watermark="exact", sweep_ahead=0,
              n_late=0):
    ch = oracle.chains(p)
    prev, nxt, rank = ch["prev"], ch["next"], ch["rank"]
    row_ptr, col = p.row_ptr, p.col
    n = p.n_rows
    row_of = np.repeat(np.arange(n), np.diff(row_ptr))
    pos = np.arange(p.nnz)
    near_prev = (prev >= 0) & (pos - prev < near)
    near_next = (nxt >= 0) & (nxt - pos < near)
    n_chunks = (n + chunk - 1) // chunk
    w_src = {}            # feature -> (epoch, example) whose write sits in the array
    rec = {}              # feature -> (tag, epoch, example) of the last record write
    swept = watermark in ("flags", "words")
    for ep in range(epochs):
        chunk_done = np.zeros(n_chunks, bool)
        flag = np.zeros(n_chunks, bool)  # the engine's done flags (a fresh tag every epoch)
        next_ticket = 0
        # worker state: [chunk, example index in chunk, phase, positions pending]
        workers = [None] * n_workers
        owed = [None] * n_workers        # chunk a worker has finished and not flagged yet
        prog = [0] * n_workers           # the previous engine's progress words
        exited = [False] * n_workers
        started = [wi < n_workers - n_late for wi in range(n_workers)]
        wpos = 0                         # the engine's published watermark
        sweep_c, sweep_i, sweep_m = 0, 0, INF
        steps = 0
        while not chunk_done.all():
            steps += 1
            assert steps < 200 * (p.nnz + n + 10) + 50 * n_workers * (n + 10), "no progress"
            first_open = int(np.argmin(chunk_done)) if not chunk_done.all() else n_chunks
            exact = int(row_ptr[min(first_open * chunk, n)])
            if watermark == "exact":
                wm_pos = exact
            else:
                assert wpos <= exact, "watermark ahead of the finished chunks"
                wm_pos = wpos
            enabled = []
            if swept:
                enabled.append((None, "sweep", None))
            for wi, st in enumerate(workers):
                if not started[wi]:
                    if any(exited[v] for v in range(n_workers) if v != wi):
                        enabled.append((wi, "start", None))
                    continue
                if st is None:
                    if next_ticket < n_chunks:
                        enabled.append((wi, "take", None))
                    elif swept and not exited[wi]:
                        enabled.append((wi, "exit", None))
                    elif not exited[wi]:
                        enabled.append((wi, "exit", None))
                    continue
                c, ti, phase, pending = st
                if phase == "publish":
                    enabled.append((wi, "publish", None))
                    continue
                t = c * chunk + ti
                b, e = int(row_ptr[t]), int(row_ptr[t + 1])
                for q in pending:
                    if phase == "read":
                        if near_prev[q]:
                            r = rec.get(int(col[q]))
                            ok = r is not None and r[0] == (int(rank[q]), ep)
                        else:
                            need = min(int(row_ptr[c * chunk]), e - near)
                            ok = wm_pos >= need or not watermark_wait
                    else:
                        ok = True
                    if ok:
                        enabled.append((wi, phase, q))
                if not pending:
                    enabled.append((wi, "next", None))
            assert enabled, "deadlock"
            wi, kind, q = enabled[rng.integers(len(enabled))]
            if kind == "sweep":
                if watermark == "words":
                    if sweep_i < n_workers:
                        sweep_m = min(sweep_m, prog[sweep_i])
                        sweep_i += 1
                    else:
                        wm = min(sweep_m + sweep_ahead, n_chunks)
                        wpos = max(wpos, int(row_ptr[min(n, wm * chunk)]))
                        sweep_i, sweep_m = 0, INF
                    continue
                c = sweep_c + sweep_i
                if c < n_chunks and flag[c] and sweep_i < SPAN:
                    sweep_i += 1
                else:
                    sweep_c = min(sweep_c + sweep_i + sweep_ahead, n_chunks)
                    wpos = max(wpos, int(row_ptr[min(n, sweep_c * chunk)]))
                    sweep_i = 0
                continue
            if kind == "start":
                started[wi] = True
                continue
            if kind == "exit":
                prog[wi] = INF
                if owed[wi] is not None:
                    flag[owed[wi]] = True
                    owed[wi] = None
                exited[wi] = True
                continue
            if kind == "publish":
                if watermark == "words":
                    prog[wi] = workers[wi][0]
                elif owed[wi] is not None:
                    flag[owed[wi]] = True
                    owed[wi] = None
                workers[wi][2] = "read"
                continue
            if kind == "take":
                c = next_ticket
                next_ticket += 1
                t0 = c * chunk
                first = "publish" if swept else "read"
                workers[wi] = [c, 0, first, list(range(int(row_ptr[t0]), int(row_ptr[t0 + 1])))]
                continue
            c, ti, phase, pending = workers[wi]
            t = c * chunk + ti
            if kind == "read":
                j = int(col[q])
                seen = (rec[j][1], rec[j][2]) if near_prev[q] else w_src.get(j)
                if prev[q] >= 0:
                    want = (ep, int(row_of[prev[q]]))
                else:                                   # first occurrence of the epoch
                    last = ch["feat_ptr"][j + 1] - 1    # the feature's last position
                    want = (ep - 1, int(row_of[ch["csc_pos"][last]])) if ep > 0 else None
                assert seen == want, (ep, t, q, seen, want)
                pending.remove(q)
                if not pending:
                    workers[wi] = [c, ti, "write", list(range(int(row_ptr[t]), int(row_ptr[t + 1])))]
            elif kind == "write":
                j = int(col[q])
                if near_next[q]:
                    rec[j] = ((int(rank[q]) + 1, ep), ep, t)
                else:
                    w_src[j] = (ep, t)
                pending.remove(q)
            else:                                       # the example is finished
                ti += 1
                t = c * chunk + ti
                if ti < chunk and t < n:
                    workers[wi] = [c, ti, "read", list(range(int(row_ptr[t]), int(row_ptr[t + 1])))]
                else:
                    chunk_done[c] = True
                    owed[wi] = c
                    workers[wi] = None
    # after the last epoch every feature's array entry holds its last writer
    for j in range(p.n_cols):
        cnt = ch["feat_ptr"][j + 1] - ch["feat_ptr"][j]
        if cnt:
            last = ch["feat_ptr"][j + 1] - 1
            assert w_src[j] == (epochs - 1, int(row_of[ch["csc_pos"][last]]))


@pytest.mark.parametrize("watermark", ["exact", "flags"])
@pytest.mark.parametrize("seed", range(12))
def test_window_protocol_reads_follow_data_order(seed, watermark):
    rng = np.random.default_rng(seed)
    p = synthdata.generate("tiny", seed=seed, n_rows=int(rng.integers(30, 90)), n_cols=int(rng.integers(6, 40)),
                           k=int(rng.integers(1, 6)), k_lo=0, ids="zipf" if seed % 2 else "uniform", zipf_s=1.1)
    near = int(rng.choice([1, 2, 5, 20, 10 ** 6]))     # all far .. all near
    n_workers = int(rng.integers(1, 7))
    _simulate(p, near=near, chunk=int(rng.integers(1, 4)), n_workers=n_workers,
              epochs=int(rng.integers(1, 3)), rng=rng, watermark=watermark,
              n_late=int(rng.integers(0, n_workers)) if watermark == "flags" else 0)


@pytest.mark.parametrize("seed", range(6))
def test_window_protocol_with_most_workers_starting_late(seed):
    # all far (every read with a predecessor waits on the watermark), one or
    # two workers running, the rest only after one of them has exited
    rng = np.random.default_rng(100 + seed)
    p = synthdata.generate("tiny", seed=seed, n_rows=50, n_cols=12, k=3, k_lo=1)
    n_workers = 6
    _simulate(p, near=1, chunk=int(rng.integers(1, 3)), n_workers=n_workers, epochs=2, rng=rng,
              watermark="flags", n_late=n_workers - 1 - seed % 2)


def test_window_protocol_model_rejects_progress_words_with_late_workers():
    # planted: the previous rule (per-worker progress words starting at 0,
    # minimum over all workers) with workers that start late pins the
    # watermark at chunk 0, and the running workers' far reads never pass
    rng = np.random.default_rng(9)
    p = synthdata.generate("tiny", seed=5, n_rows=40, n_cols=8, k=3, k_lo=1)
    with pytest.raises(AssertionError):
        _simulate(p, near=1, chunk=1, n_workers=4, epochs=1, rng=rng, watermark="words", n_late=2)


def test_window_protocol_words_pass_when_every_worker_is_resident():
    # the same planted rule is sound when every worker runs from the start
    rng = np.random.default_rng(10)
    p = synthdata.generate("tiny", seed=5, n_rows=40, n_cols=8, k=3, k_lo=1)
    _simulate(p, near=1, chunk=1, n_workers=4, epochs=1, rng=rng, watermark="words", n_late=0)


def test_window_protocol_model_rejects_a_missing_wait():
    # planted in the model: far reads skip the watermark; some interleaving
    # then reads a weight before its previous occurrence has written it
    rng = np.random.default_rng(7)
    p = synthdata.generate("tiny", seed=3, n_rows=60, n_cols=6, k=3, k_lo=1)
    failures = 0
    for _ in range(20):
        try:
            _simulate(p, near=1, chunk=1, n_workers=6, epochs=1, rng=rng, watermark_wait=False)
        except AssertionError:
            failures += 1
    assert failures > 0


def test_window_protocol_model_rejects_a_sweeper_one_chunk_ahead():
    # planted in the model: the sweeper publishes one chunk past the first
    # unset flag; some interleaving then lets a far read run before its
    # writer finished
    rng = np.random.default_rng(8)
    p = synthdata.generate("tiny", seed=4, n_rows=60, n_cols=6, k=3, k_lo=1)
    failures = 0
    for _ in range(20):
        try:
            _simulate(p, near=1, chunk=1, n_workers=6, epochs=1, rng=rng, watermark="flags", sweep_ahead=1)
        except AssertionError:
            failures += 1
    assert failures > 0
