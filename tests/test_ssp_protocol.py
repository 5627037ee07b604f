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


# ---------------------------------------------------------------- bitmaps
# The prefix gates as a GPU can run them without a compare-and-swap loop on
# a hot feature's word: per direction a done-bitmap over the CSC slots (the
# occurrence of j with rank r is slot feat_ptr[j] + r), set by the occurrence
# once its access is done; per feature a prefix hint P_j, raised (atomic max)
# by waiters after they observed a run of set bits.  A gate "ranks 0 .. need-1
# done" loads P_j; if short, scans the bitmap words from P_j for a run of set
# bits (clamped at need), publishes what it saw, and passes or waits for the
# first zero bit to be set.  Every shared access below is one step of the
# model, interleaved at random.


def _trailing_ones(x, width):
    t = 0
    while t < width and (x >> t) & 1:
        t += 1
    return t


def _simulate_bitmap(p, delay, n_workers, rng, word_bits=32, slow_ticket=None, plant=None):
    ch = oracle.chains(p)
    rank, fptr = ch["rank"], ch["feat_ptr"]
    row_ptr, col = p.row_ptr, p.col
    n = p.n_rows
    n_words = (p.nnz + word_bits - 1) // word_bits + 1
    bits = {"r": [0] * n_words, "w": [0] * n_words}
    hint = {"r": [0] * p.n_cols, "w": [0] * p.n_cols}
    applied = {j: [] for j in range(p.n_cols)}

    def done(kind, slot):
        return (bits[kind][slot // word_bits] >> (slot % word_bits)) & 1

    def check_hints():
        # safety: a hint never runs ahead of the bits it stands for
        for kind in ("r", "w"):
            for j in range(p.n_cols):
                for r in range(hint[kind][j]):
                    assert done(kind, int(fptr[j]) + r), ("hint ahead of the bits", kind, j, r)

    # a lane: one position of the example its worker holds
    # program: gate(w, r - delay) -> load -> mark r -> [all lanes] ->
    #          gate(r, r - delay + 1) -> add -> mark w -> end
    def new_lane(q):
        return dict(q=q, pc="gate", kind="w", need=int(rank[q]) - delay, g="load", p=0, p0=0)

    workers = [None] * n_workers          # [example, lanes]
    next_ticket, finished, steps = 0, 0, 0
    while finished < n:
        steps += 1
        assert steps < 400 * (p.nnz + n + 10), "no progress"
        enabled = []
        for wi, st in enumerate(workers):
            if st is None:
                if next_ticket < n:
                    enabled.append((wi, None))
                continue
            lanes = st[1]
            if all(l["pc"] == "end" for l in lanes):
                enabled.append((wi, "finish"))
                continue
            for li, l in enumerate(lanes):
                if l["pc"] == "barrier":
                    if all(m["pc"] in ("barrier", "gate2", "end") or m.get("phase2") for m in lanes):
                        enabled.append((wi, li))
                    continue
                if l["pc"] == "end":
                    continue
                if l["pc"] in ("gate", "gate2") and l["g"] == "block":
                    j = int(col[l["q"]])
                    if not (done(l["kind"], l["zero"]) or hint[l["kind"]][j] > l["p"]):
                        continue
                enabled.append((wi, li))
        assert enabled, "deadlock"
        if slow_ticket is not None and rng.random() < 0.99:
            slow = [wi for wi, st in enumerate(workers) if st is not None and st[0] == slow_ticket]
            enabled = [x for x in enabled if x[0] not in slow] or enabled
        wi, li = enabled[rng.integers(len(enabled))]
        if li is None:
            t = next_ticket
            next_ticket += 1
            workers[wi] = [t, [new_lane(q) for q in range(int(row_ptr[t]), int(row_ptr[t + 1]))]]
            if not workers[wi][1]:
                workers[wi][1] = [dict(pc="end")]
            continue
        if li == "finish":
            finished += 1
            workers[wi] = None
            continue
        l = workers[wi][1][li]
        q = l["q"]
        j, r = int(col[q]), int(rank[q])
        slot = int(fptr[j]) + r
        if l["pc"] in ("gate", "gate2"):
            kind, need = l["kind"], l["need"]
            assert need <= int(fptr[j + 1] - fptr[j])        # scans stay inside the feature's slots
            if need <= 0:
                l["pc"] = "access"
            elif l["g"] in ("load", "block"):
                l["p"] = l["p0"] = hint[kind][j]
                l["g"] = "scan"
                if l["p"] >= need:
                    l["pc"], l["g"] = "access", "load"
            elif l["g"] == "scan":
                s = int(fptr[j]) + l["p"]
                b = s % word_bits
                word = bits[kind][s // word_bits]
                if plant == "offset-ignored":
                    t = _trailing_ones(word, word_bits - b)
                else:
                    t = _trailing_ones(word >> b, word_bits - b)
                l["p"] = min(l["p"] + t, need)
                if l["p"] >= need:
                    l["g"], l["ok"] = "pub", True
                elif t < word_bits - b:
                    l["g"], l["ok"], l["zero"] = "pub", False, int(fptr[j]) + l["p"]
            elif l["g"] == "pub":
                pub = l["p"] + 1 if plant == "publish-one-more" else l["p"]
                if pub > l["p0"]:
                    hint[kind][j] = max(hint[kind][j], pub)
                if l["ok"]:
                    l["pc"], l["g"] = "access", "load"
                else:
                    l["g"] = "block"
            if l["pc"] == "access":
                l["phase2"] = kind == "r"
        elif l["pc"] == "access":
            if not l.get("phase2"):
                seen = set(applied[j])
                assert len(seen) >= r - delay
                if delay == 0:
                    assert applied[j] == list(range(r))
                assert set(range(max(0, r - delay))) <= seen and not any(s >= r + delay for s in seen), \
                    (j, r, sorted(seen))
                l["pc"] = "mark"
            else:
                applied[j].append(r)
                l["pc"] = "mark"
        elif l["pc"] == "mark":
            kind = "w" if l.get("phase2") else "r"
            bits[kind][slot // word_bits] |= 1 << (slot % word_bits)
            l["pc"] = "end" if l.get("phase2") else "barrier"
        elif l["pc"] == "barrier":
            l.update(pc="gate2", kind="r", need=r - delay + 1, g="load", phase2=True)
        check_hints()
    for j in range(p.n_cols):
        assert sorted(applied[j]) == list(range(int(fptr[j + 1] - fptr[j])))


@pytest.mark.parametrize("word_bits", [4, 32])
@pytest.mark.parametrize("delay", [0, 1, 3, 16])
@pytest.mark.parametrize("seed", range(3))
def test_prefix_gates_on_bitmaps(seed, delay, word_bits):
    rng = np.random.default_rng(500 + 10 * seed + delay)
    p = _problem(seed, rng)
    _simulate_bitmap(p, delay, n_workers=int(rng.integers(1, 8)), rng=rng, word_bits=word_bits)
    _simulate_bitmap(p, delay, n_workers=6, rng=rng, word_bits=word_bits, slow_ticket=0)


@pytest.mark.parametrize("word_bits", [4, 32])
def test_prefix_gates_on_bitmaps_one_hot_feature(word_bits):
    rng = np.random.default_rng(77)
    p = _one_feature(40)
    for delay in (0, 2, 5):
        _simulate_bitmap(p, delay, n_workers=8, rng=rng, word_bits=word_bits, slow_ticket=0)
        _simulate_bitmap(p, delay, n_workers=8, rng=rng, word_bits=word_bits)


@pytest.mark.parametrize("plant", ["offset-ignored", "publish-one-more"])
def test_prefix_gates_on_bitmaps_model_catches_plants(plant):
    rng = np.random.default_rng(21)
    failures = 0
    for seed in range(6):
        p = _problem(seed, rng)
        try:
            _simulate_bitmap(p, 1, n_workers=6, rng=rng, word_bits=4, plant=plant)
        except AssertionError:
            failures += 1
    assert failures > 0


def _scan_step(word, b):
    # the GPU gate's scan step on one 32-bit word from bit b: x = ~(word >> b),
    # t = (lowest set bit of x) or 32 when x is 0
    x = ~(word >> b) & 0xFFFFFFFF
    return (x & -x).bit_length() - 1 if x else 32


def test_scan_step_counts_the_run_of_set_bits_from_the_offset():
    rng = np.random.default_rng(3)
    words = [0, 0xFFFFFFFF, 0x7FFFFFFF, 0xFFFFFFFE, 0x80000000, 1] + [int(v) for v in rng.integers(0, 2 ** 32, 200)]
    words += [(1 << n) - 1 for n in range(33)] + [((1 << 32) - 1) ^ ((1 << n) - 1) for n in range(33)]
    for word in words:
        for b in range(32):
            t = _scan_step(word, b)
            assert t == _trailing_ones(word >> b, 32 - b), (hex(word), b)
            assert t <= 32 - b
