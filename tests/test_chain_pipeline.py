"""A model of the CHAIN engine's pipeline schedule, on the CPU.

One thread block runs the examples in data order, G per pipeline step, and
its warps work on different steps in the same iteration of the step loop,
separated only by the __syncthreads that ends each iteration:

  W   (two warps)  writes through the new weights of step t - 1 whose next
                   occurrence is not pushed; one of them also copies row
                   bounds L = DS + BS + 1 steps ahead into a ring of RP;
  A   (one warp per example of a step)  copies ids, link words and values of
                   step t + DS into the example's slot of a ring of SLOTS;
  B   (the same warps)  gathers, for step t + BS, the weights nobody pushes
                   from global w, and where each new weight will be stored;
  C   (the compute warp)  runs the examples of step t in order, each reading
                   its weights from its slot and storing each new weight
                   into the next occurrence's slot when that lies within
                   D = G * DS examples (a push), else into its own output
                   slot for W.  Every example but the first of a step
                   fetches its weights while the example before it is still
                   computing, before that example's stores; a weight whose
                   previous occurrence is that very example is taken from
                   it directly (a shuffle, or a reload after its stores).

The model replays that schedule with the link words the engine builds from
the conflict chains (including the mark of a previous occurrence in the
example just before) and checks, on problems full of near repeats: every
example reads, for every feature, exactly the weight its previous occurrence
wrote (in the epoch, or the last one of the epoch before); global w ends each
epoch holding each feature's last writer; no two warps touch one shared or
global cell in the same iteration unless both only read it; every row bound
read comes from the ring entry of that very example.  The same checks fail
when the constants break the engine's compile-time conditions (a gather one
step earlier, a shorter forwarding window, a ring of 16 slots)."""
import numpy as np
import pytest

import oracle
import synthdata

ENGINE = dict(G=4, DS=4, BS=2, SLOTS=32, RP=64)


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


def _simulate(p, epochs, G, DS, BS, SLOTS, RP, D=None):
    D = G * DS if D is None else D
    L = DS + BS + 1
    N = p.n_rows
    rp = p.row_ptr
    recv, push, late = _links(p, D)
    steps = (N + G - 1) // G
    # weights are tracked as the example (epoch, id) that wrote them; None = w0
    w = {}
    last_writer = {}                      # feature -> (epoch, example) of its latest write in data order
    for ep in range(epochs):
        ring = {}                         # rp ring: index -> example whose bound it holds
        slot_of = lambda r: r & (SLOTS - 1)
        col, wp, out, pa, xa, kk, ys = {}, {}, {}, {}, {}, {}, {}

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
            effects = []
            # W: warps 6 (examples 0, 1 of step t - 1, and the row bounds) and 7 (examples 2, 3)
            for warp, gs in (("W6", range(0, G // 2)), ("W7", range(G // 2, G))):
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
                    it.w("W6", ("rp", e & (RP - 1)))
                    effects.append(("rp", e & (RP - 1), e))
            # A and B: one warp per example g of a step
            for g in range(G):
                warp = f"AB{g}"
                r = (t + DS) * G + g
                bk = bounds(it, warp, r)
                if bk is not None:
                    b, k = bk
                    s = slot_of(r)
                    for i in range(k):
                        for arr in ("col", "link", "xa"):
                            it.w(warp, (arr, s, i))
                        effects.append(("col", (s, i), int(p.col[b + i])))
                        effects.append(("xa", (s, i), (r, i)))
                    it.w(warp, ("y", s))
                    effects.append(("y", s, r))
                r = (t + BS) * G + g
                bk = bounds(it, warp, r)
                if bk is not None:
                    b, k = bk
                    s = slot_of(r)
                    for i in range(k):
                        it.r(warp, ("link", s, i))
                        it.r(warp, ("col", s, i))
                        if not recv[b + i]:
                            j = col[(s, i)]
                            it.r(warp, ("w", j))
                            it.w(warp, ("wp", s, i))
                            effects.append(("wp", (s, i), w.get(j)))
                        it.w(warp, ("pa", s, i))
                        if b + i in push:
                            dr, e = push[b + i]
                            effects.append(("pa", (s, i), ("wp", slot_of(r + dr), e)))
                        else:
                            effects.append(("pa", (s, i), ("out", s, i)))
                    it.w(warp, ("kk", s))
                    effects.append(("kk", s, r))
            # C: the compute warp, examples of step t in data order (its own
            # accesses are ordered; pushes into a later example of the same
            # step are read after they are stored)
            if 0 <= t < steps:
                local = {}
                fetched = local                   # the stores visible when an example fetched its weights
                for g, r in enumerate(range(t * G, min(N, t * G + G))):
                    # the compute warp takes the length from the slot, not the ring
                    b, k = int(rp[r]), int(rp[r + 1] - rp[r])
                    s = slot_of(r)
                    it.r("C", ("kk", s))
                    it.r("C", ("y", s))
                    # the slot's length, label and values were written for this very example
                    assert kk.get(s) == r and ys.get(s) == r, ("slot holds another example", r, kk.get(s), ys.get(s))
                    for i in range(k):
                        for arr in ("xa", "pa", "wp"):
                            it.r("C", (arr, s, i))
                        assert xa.get((s, i)) == (r, i), ("value of another example", r, i, xa.get((s, i)))
                        assert col[(s, i)] == int(p.col[b + i]), ("id of another example", r, i)
                        j = int(p.col[b + i])
                        if g > 0 and late[b + i]:
                            got = (ep, r - 1)         # from the example just before, once it has computed
                        else:
                            got = fetched.get(("wp", s, i), wp.get((s, i)))
                        assert got == expect.get(j), ("wrong weight read", ep, r, j, got, expect.get(j))
                    fetched = dict(local)             # the next example fetches before this one stores
                    for i in range(k):
                        j = int(p.col[b + i])
                        target = pa[(s, i)]
                        it.w("C", target)
                        local[target] = (ep, r)
                        expect[j] = (ep, r)
                effects.extend(("cstore", cell, v) for cell, v in local.items())
            it.check(t)
            # the iteration's effects land before the next iteration (__syncthreads)
            for kind, key, v in effects:
                if kind == "w":
                    w[key] = v
                elif kind == "rp":
                    ring[key] = v
                elif kind == "col":
                    col[key] = v
                elif kind == "xa":
                    xa[key] = v
                elif kind == "kk":
                    kk[key] = v
                elif kind == "y":
                    ys[key] = v
                elif kind == "wp":
                    wp[key] = v
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


@pytest.mark.parametrize("seed", range(8))
def test_chain_pipeline_schedule(seed):
    rng = np.random.default_rng(700 + seed)
    _simulate(_problem(seed, rng), epochs=2, **ENGINE)


def test_chain_pipeline_one_feature_and_ragged():
    # every example holds feature 0: every weight is pushed; and a ragged
    # problem with empty examples and a short last step
    n = 37
    p = synthdata.from_arrays(np.arange(n + 1), np.zeros(n, np.int32), None, np.ones(n), n_cols=1)
    _simulate(p, epochs=3, **ENGINE)
    q = synthdata.generate("tiny", seed=5, n_rows=101, n_cols=7, k=4, k_lo=0)
    _simulate(q, epochs=2, **ENGINE)


@pytest.mark.parametrize("change", [dict(BS=3), dict(D=12), dict(SLOTS=16)])
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
