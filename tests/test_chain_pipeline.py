"""A model of the CHAIN engine's pipeline schedule, on the CPU.

One thread block runs the examples in data order, G per pipeline step, and
its warps work on different steps in the same iteration of the step loop,
separated only by the __syncthreads that ends each iteration:

  W   (G / 2 warps, two examples each)  writes through the new weights of
                   step t - 1 whose next occurrence is not pushed; the first
                   also copies row bounds L = DS + BS + 1 steps ahead into a
                   ring of RP;
  A   (one warp per example of a step)  copies ids, link words and values of
                   step t + DS into the example's slot of a ring of SLOTS;
  B   (the same warps)  gathers, for step t + BS, the weights nobody pushes
                   from global w, and where each new weight will be stored;
  C   (the compute warp)  runs the examples of step t in order, each reading
                   its weights from its slot and storing each new weight
                   into the next occurrence's slot when that lies within
                   D = G * DS examples (a push), else into its own output
                   slot for W.

The asynchronous copies (row bounds, ids, link words, values, labels,
gathered weights) of one iteration land by the end of iteration + INFLIGHT:
until then the model counts their source and destination cells as touched by
the copying warp in every iteration they may still be moving.

C comes in two forms.  For rows of more than 32 ids, every example but the
first of a step fetches its weights while the example before it is still
computing, before that example's stores; a weight whose previous occurrence
is that very example is taken from it directly.  For rows of up to 32 ids,
every example -- the first of a step too, then during the last example of
the step before -- is fetched while the example before it computes, after
the stores of the example before that; the stores of an example wait for the
next example's margin to start, and the last example of a step stores before
the step's barrier.

The model replays that schedule with the link words the engine builds from
the conflict chains (including the mark of a previous occurrence in the
example just before) and checks, on problems full of near repeats: every
example uses, for every feature, exactly the weight its previous occurrence
wrote (in the epoch, or the last one of the epoch before); global w ends each
epoch holding each feature's last writer; no two warps touch one shared or
global cell in the same iteration unless both only read it; every row bound
read comes from the ring entry of that very example; every slot the compute
warp reads holds the example it reads it for.  The same checks fail when the
constants break the engine's compile-time conditions (a gather one step
earlier, a shorter forwarding window, a ring of 16 slots, copies left in
flight one step longer)."""
import numpy as np
import pytest

import oracle
import synthdata

# the engine's pipeline shapes: rows of up to 128 ids, and of up to 256
ENGINE = dict(G=8, DS=5, BS=3, SLOTS=64, RP=128, INFLIGHT=1)
ENGINE_LONG = dict(G=4, DS=5, BS=3, SLOTS=32, RP=128, INFLIGHT=1)


def _links(p, D):
    ch = oracle.chains(p)
    prev, nxt = ch["prev"], ch["next"]
    row_of = np.repeat(np.arange(p.n_rows), np.diff(p.row_ptr))
    recv = np.zeros(p.nnz, bool)
    late = np.zeros(p.nnz, bool)
    push = {}
    for q in range(p.nnz):
        t = row_of[q]
        if prev[q] >= 0 and t - row_of[prev[q]] <= D:
            recv[q] = True
        if prev[q] >= 0 and row_of[prev[q]] == t - 1:
            late[q] = True
        if nxt[q] >= 0 and row_of[nxt[q]] - t <= D:
            push[q] = (int(row_of[nxt[q]] - t), int(nxt[q] - p.row_ptr[row_of[nxt[q]]]))
    return recv, push, late


class _Iteration:
    """Cells each warp reads and writes during one iteration of the step loop."""

    def __init__(self):
        self.reads, self.writes = {}, {}

    def r(self, warp, cell):
        self.reads.setdefault(cell, set()).add(warp)

    def w(self, warp, cell):
        self.writes.setdefault(cell, set()).add(warp)

    def check(self, t):
        for cell, ws in self.writes.items():
            others = (ws | self.reads.get(cell, set()))
            assert len(others) == 1, ("two warps touch one cell in one iteration", t, cell, sorted(others))


def _simulate(p, epochs, G, DS, BS, SLOTS, RP, INFLIGHT, D=None, one_per_lane=True):
    D = G * DS if D is None else D
    L = DS + BS + 1
    N = p.n_rows
    rp = p.row_ptr
    recv, push, late = _links(p, D)
    steps = (N + G - 1) // G
    slot_of = lambda r: r & (SLOTS - 1)
    # weights are tracked as the example (epoch, id) that wrote them; None = w0
    w = {}
    last_writer = {}                      # feature -> (epoch, example) of its latest write in data order
    for ep in range(epochs):
        ring = {}                         # rp ring: index -> example whose bound it holds
        col, wp, out, pa, xa, kk, ys = {}, {}, {}, {}, {}, {}, {}
        tables = dict(rp=ring, col=col, xa=xa, y=ys, wp=wp)
        inflight = []                     # asynchronous copies: (last iteration, warp, cells, effects)

        def bounds(it, warp, r):
            if r < 0 or r >= N:
                return None
            for e in (r, r + 1):
                it.r(warp, ("rp", e & (RP - 1)))
                assert ring.get(e & (RP - 1)) == e, ("row bound not in the ring", r, e)
            return int(rp[r]), int(rp[r + 1] - rp[r])

        expect = dict(last_writer)        # the weight the next occurrence of each feature must read
        for t in range(-L, steps + 1):
            it = _Iteration()
            effects = []                  # plain stores: land at the end of this iteration
            copies = {}                   # warp -> (cells read, cells written, effects) of this iteration's copies

            def copy(warp, src, dst, key, v):
                c = copies.setdefault(warp, ([], [], []))
                if src is not None:
                    c[0].append(src)
                c[1].append(dst)
                c[2].append((key, v))

            # W: warp i writes examples 2i, 2i + 1 of step t - 1; W0 also copies row bounds
            for warp, gs in ((f"W{i}", range(2 * i, 2 * i + 2)) for i in range(G // 2)):
                for g in gs:
                    r = (t - 1) * G + g
                    bk = bounds(it, warp, r)
                    if bk is None:
                        continue
                    b, k = bk
                    s = slot_of(r)
                    for i in range(k):
                        it.r(warp, ("link", s, i))
                        if b + i not in push:
                            it.r(warp, ("col", s, i))
                            it.r(warp, ("out", s, i))
                            j = col[(s, i)]
                            it.w(warp, ("w", j))
                            effects.append(("w", j, out[(s, i)]))
            for lane in range(G):
                e = (t + L) * G + lane
                if 0 <= e <= N:
                    copy("W0", ("row_ptr", e), ("rp", e & (RP - 1)), ("rp", e & (RP - 1)), e)
            # A and B: one warp per example g of a step
            for g in range(G):
                warp = f"AB{g}"
                r = (t + DS) * G + g
                bk = bounds(it, warp, r)
                if bk is not None:
                    b, k = bk
                    s = slot_of(r)
                    for i in range(k):
                        copy(warp, None, ("col", s, i), ("col", (s, i)), int(p.col[b + i]))
                        copy(warp, None, ("link", s, i), ("link", (s, i)), None)
                        copy(warp, None, ("xa", s, i), ("xa", (s, i)), (r, i))
                    copy(warp, None, ("y", s), ("y", s), r)
                r = (t + BS) * G + g
                bk = bounds(it, warp, r)
                if bk is not None:
                    b, k = bk
                    s = slot_of(r)
                    for i in range(k):
                        it.r(warp, ("link", s, i))
                        it.r(warp, ("col", s, i))
                        if not recv[b + i]:
                            j = col.get((s, i))
                            assert j == int(p.col[b + i]), ("gather before the id landed", r, i)
                            copy(warp, ("w", j), ("wp", s, i), ("wp", (s, i)), w.get(j))
                        it.w(warp, ("pa", s, i))
                        if b + i in push:
                            dr, e = push[b + i]
                            effects.append(("pa", (s, i), ("wp", slot_of(r + dr), e)))
                        else:
                            effects.append(("pa", (s, i), ("out", s, i)))
                    it.w(warp, ("kk", s))
                    effects.append(("kk", s, r))
            for warp, (rd, wr, eff) in copies.items():
                inflight.append((t + INFLIGHT, warp, rd, wr, eff))
            # copies still moving touch their cells in every iteration until they land
            for last, warp, rd, wr, _ in inflight:
                for cell in rd:
                    it.r(warp, cell)
                for cell in wr:
                    it.w(warp, cell)
            # C: the compute warp, examples of step t in data order (its own
            # accesses are ordered; its stores are visible to its later reads)
            if 0 <= t < steps:
                local = {}

                def fetch(r):
                    # the slot's length, label, values, ids, store words and weights
                    b, k = int(rp[r]), int(rp[r + 1] - rp[r])
                    s = slot_of(r)
                    it.r("C", ("kk", s))
                    it.r("C", ("y", s))
                    assert kk.get(s) == r and ys.get(s) == r, ("slot holds another example", r, kk.get(s), ys.get(s))
                    got, targets = [], []
                    for i in range(k):
                        for arr in ("xa", "pa", "wp"):
                            it.r("C", (arr, s, i))
                        assert xa.get((s, i)) == (r, i), ("value of another example", r, i, xa.get((s, i)))
                        assert col[(s, i)] == int(p.col[b + i]), ("id of another example", r, i)
                        got.append(local.get(("wp", s, i), wp.get((s, i))))
                        targets.append(pa[(s, i)])
                    return got, targets

                def compute(r, got, from_before):
                    # the weights the margin uses: a late one from the example just before
                    b, k = int(rp[r]), int(rp[r + 1] - rp[r])
                    for i in range(k):
                        j = int(p.col[b + i])
                        v = (ep, r - 1) if from_before and late[b + i] else got[i]
                        assert v == expect.get(j), ("wrong weight read", ep, r, j, v, expect.get(j))
                    for i in range(k):
                        expect[int(p.col[b + i])] = (ep, r)

                def store(r, targets):
                    for target in targets:
                        it.w("C", target)
                        local[target] = (ep, r)

                r0, r1 = t * G, min(N, t * G + G)
                if one_per_lane:
                    if t == 0:
                        nxt = fetch(0)
                    for r in range(r0, r1):
                        cur = nxt
                        if r > r0:
                            store(r - 1, prev_targets)
                        if r + 1 < N:
                            nxt = fetch(r + 1)
                        compute(r, cur[0], True)
                        prev_targets = cur[1]
                    store(r1 - 1, prev_targets)
                else:
                    nxt = fetch(r0)
                    for g, r in enumerate(range(r0, r1)):
                        cur = nxt
                        if r + 1 < r1:
                            nxt = fetch(r + 1)        # before this example's stores
                        compute(r, cur[0], g > 0)
                        store(r, cur[1])
                effects.extend(("cstore", cell, v) for cell, v in local.items())
            it.check(t)
            # the iteration's plain stores land before the next iteration
            # (__syncthreads), and so do the copies whose last iteration it is
            landed = [e for last, _, _, _, eff in inflight if last == t for e in eff]
            inflight = [c for c in inflight if c[0] > t]
            for kind, key, v in effects + [(k, key, v) for (k, key), v in landed]:
                if kind == "w":
                    w[key] = v
                elif kind in tables:
                    tables[kind][key] = v
                elif kind == "link":
                    pass
                elif kind == "kk":
                    kk[key] = v
                elif kind == "pa":
                    pa[key] = v
                else:
                    if key[0] == "wp":
                        wp[(key[1], key[2])] = v
                    else:
                        out[(key[1], key[2])] = v
        last_writer = expect
        # the drain at the end of the epoch leaves every feature's last writer in w
        for j, v in last_writer.items():
            assert w.get(j) == v, ("w after the epoch", ep, j, w.get(j), v)


def _problem(seed, rng):
    return synthdata.generate("tiny", seed=seed, n_rows=int(rng.integers(60, 160)), n_cols=int(rng.integers(3, 30)),
                              k=int(rng.integers(1, 6)), k_lo=0, ids="zipf" if seed % 2 else "uniform", zipf_s=1.2)


FORMS = [(ENGINE, True), (ENGINE, False), (ENGINE_LONG, False)]     # (shape, one element per lane)


@pytest.mark.parametrize("cfg,one_per_lane", FORMS)
@pytest.mark.parametrize("seed", range(8))
def test_chain_pipeline_schedule(seed, cfg, one_per_lane):
    rng = np.random.default_rng(700 + seed)
    _simulate(_problem(seed, rng), epochs=2, one_per_lane=one_per_lane, **cfg)


@pytest.mark.parametrize("cfg,one_per_lane", FORMS)
def test_chain_pipeline_one_feature_and_ragged(cfg, one_per_lane):
    # every example holds feature 0: every weight is pushed; and a ragged
    # problem with empty examples and a short last step
    n = 37
    p = synthdata.from_arrays(np.arange(n + 1), np.zeros(n, np.int32), None, np.ones(n), n_cols=1)
    _simulate(p, epochs=3, one_per_lane=one_per_lane, **cfg)
    q = synthdata.generate("tiny", seed=5, n_rows=101, n_cols=7, k=4, k_lo=0)
    _simulate(q, epochs=2, one_per_lane=one_per_lane, **cfg)


@pytest.mark.parametrize("change", [dict(BS=2), dict(D=32), dict(SLOTS=32), dict(INFLIGHT=2)])
def test_chain_pipeline_model_rejects_broken_constants(change):
    cfg, change = dict(ENGINE), dict(change)
    D = change.pop("D", None)
    cfg.update(change)
    failures = 0
    for seed in range(4):
        rng = np.random.default_rng(800 + seed)
        try:
            _simulate(_problem(seed, rng), epochs=2, D=D, **cfg)
        except AssertionError:
            failures += 1
    assert failures > 0


def _handoff_program(P, N, G, epochs):
    """The operations compute warp P (0: even examples, 1: odd ones) issues,
    in the kernel's order, for rows of up to 32 ids: waits on and arrivals at
    the named barriers C (c published) and S (stores done) of each warp, and
    the block-wide barrier that ends each step."""
    steps = (N + G - 1) // G
    for ep in range(epochs):
        for t in range(steps):
            r0, r1 = t * G, min(N, t * G + G)
            for r in range(r0 + P, r1, 2):
                if r > 0:
                    yield ("wait", ("C", P ^ 1), (ep, r))
                yield ("use", "c", (ep, r))           # reads c of r - 1, computes c of r
                if r > 0:
                    yield ("wait", ("S", P ^ 1), (ep, r))
                if r + 1 < N:
                    yield ("arrive", ("C", P), (ep, r))
                yield ("use", "store", (ep, r))
                if r + 1 < N:
                    yield ("arrive", ("S", P), (ep, r))
            yield ("block", None, (ep, t))


def _run_handoffs(N, G, epochs, seed):
    rng = np.random.default_rng(seed)
    progs = [_handoff_program(P, N, G, epochs) for P in (0, 1)]
    nxt = [next(p, None) for p in progs]
    bars = {}                    # barrier -> (warp that arrived or waits, op kind, example)
    waiting = [None, None]       # a warp blocked in a wait
    block = [None, None]         # a warp at the block barrier: its (epoch, step)
    computed, stored, released = set(), set(), {}
    while nxt[0] is not None or nxt[1] is not None or any(waiting):
        ready = [P for P in (0, 1) if nxt[P] is not None and waiting[P] is None and block[P] is None]
        if not ready:
            # only the block barrier can release now: both warps (or the one with work left) must be there
            live = [P for P in (0, 1) if block[P] is not None]
            assert live and not any(waiting), ("deadlock", N, G, nxt, waiting, block, bars)
            assert all(block[P] == block[live[0]] for P in live)
            for P in live:
                block[P] = None
                nxt[P] = next(progs[P], None)
            continue
        P = int(rng.choice(ready))
        kind, bar, ex = nxt[P]
        if kind == "block":
            block[P] = ex
            other = P ^ 1
            if nxt[other] is None or block[other] is not None:
                for Q in (0, 1):
                    if block[Q] is not None:
                        block[Q] = None
                        nxt[Q] = next(progs[Q], None)
            continue
        if kind == "use":
            ep, r = ex
            if bar == "c":
                # the weights of r's late elements come from r - 1, which must have published c
                assert r == 0 or (ep, r - 1) in released.get(("C", P ^ 1), set()), ("c of r - 1 not published", ex)
                computed.add(ex)
            else:
                stored.add(ex)
        elif kind == "arrive":
            held = bars.get(bar)
            assert held is None or held[1] == "wait", ("two arrivals before a wait", bar, held, ex)
            assert bar[1] == P
            if held is None:
                bars[bar] = (P, "arrive", ex)
            else:
                # the waiting warp is released; it waited for exactly this example
                W = held[0]
                assert W == P ^ 1 and held[2][1] == ex[1] + 1, ("wrong pairing", bar, held, ex)
                released.setdefault(bar, set()).add(ex)
                del bars[bar]
                waiting[W] = None
                nxt[W] = next(progs[W], None)
            if bar[0] == "S":
                assert ex in stored, ("stores announced before they are issued", ex)
        elif kind == "wait":
            held = bars.get(bar)
            assert bar[1] == P ^ 1
            if held is None:
                bars[bar] = (P, "wait", ex)
                waiting[P] = bar
                continue
            assert held[1] == "arrive" and held[2][1] == ex[1] - 1, ("wrong pairing", bar, held, ex)
            released.setdefault(bar, set()).add(held[2])
            del bars[bar]
        nxt[P] = next(progs[P], None)
    assert not bars, ("a barrier left half used", bars)
    assert len(computed) == N * epochs and len(stored) == N * epochs


@pytest.mark.parametrize("N", [0, 1, 2, 3, 7, 8, 9, 15, 16, 17, 40, 63])
def test_compute_warp_handoffs(N):
    # the two compute warps' named-barrier protocol: every barrier completes
    # with one arrival and one wait, for the example just before, in any
    # interleaving, and nothing is left half used at the end of an epoch
    for seed in range(30):
        _run_handoffs(N, G=8, epochs=2, seed=seed)
