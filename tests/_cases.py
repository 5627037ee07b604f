"""Shared parity-test inputs: seeded problems of the paper's workload shapes
at sizes the oracle finishes in seconds (several 4096-pair sort tiles and a
ragged tail), plus edge cases.  Results of the oracle are cached per case."""
import functools

import numpy as np

import oracle
import synthdata

# name -> (workload, overrides)
SMALL = {
    "tiny": ("tiny", {}),
    "ragged-empty-rows": ("tiny", dict(n_rows=5001, n_cols=3000, k=24, k_lo=0)),
    "zipf-shape": ("zipf-1m", dict(n_rows=30000, n_cols=20000)),
    "ctr-shape-binary": ("ctr", dict(n_rows=20000, n_cols=50000)),
    "lowconflict-shape": ("low-conflict", dict(n_rows=20000, n_cols=2_000_000)),
    "deepchain-shape": ("deep-chain", dict(n_rows=5000)),
    "long-rows": ("tiny", dict(n_rows=1500, n_cols=5000, k=300, k_lo=200, labels="sign")),
    "wide-ids-4pass": ("low-conflict", dict(n_rows=3000, n_cols=20_000_000, k=50)),
    "ids-18bit": ("zipf-1m", dict(n_rows=20000, n_cols=200_000)),
    "ids-20bit": ("zipf-1m", dict(n_rows=20000, n_cols=1_000_000)),
    # the paper's dense linear regression (Experiments 6.1/6.2): every example
    # conflicts with every other; rows longer than CHAIN takes, and short
    # enough for it
    "dense-shape": ("dense-lr", dict(n_rows=800, n_cols=320, k=320, epochs=3, bsp_batch=800)),
    "dense-narrow": ("dense-lr", dict(n_rows=1500, n_cols=200, k=200, epochs=2, bsp_batch=1500)),
    # the full 960-feature width (rows of 513..1024 ids: 32 registers per lane)
    "dense-wide": ("dense-lr", dict(n_rows=300, epochs=2, bsp_batch=300)),
    # rows longer than 1024 ids: the resident engine's two-pass path
    "dense-xwide": ("dense-lr", dict(n_rows=120, n_cols=1500, k=1500, epochs=1, bsp_batch=120)),
}

FULL = {
    "tiny-full": ("tiny", {}),
    "zipf-1m-full": ("zipf-1m", {}),
    "low-conflict-full": ("low-conflict", {}),
}


@functools.lru_cache(maxsize=None)
def problem(name):
    spec = SMALL.get(name) or FULL.get(name)
    if spec is not None:
        return synthdata.generate(spec[0], **spec[1])
    return edge(name)


def edge(name):
    if name == "no-rows":
        return synthdata.from_arrays([0], [], [], [], n_cols=5)
    if name == "all-empty-rows":
        return synthdata.from_arrays(np.zeros(7, np.int64), [], [], np.ones(6), n_cols=5)
    if name == "one-row":
        return synthdata.from_arrays([0, 3], [4, 0, 2], [0.5, -1.0, 2.0], [1.0], n_cols=6)
    if name == "one-feature-chain":
        n = 3000
        return synthdata.from_arrays(np.arange(n + 1), np.zeros(n), np.ones(n), np.linspace(-1, 1, n),
                                     n_cols=1, loss="squared", eta=0.01)
    if name == "exp-saturation":
        # margins far beyond exp's range: logistic gradient -> 0 or -y exactly
        n, k = 400, 4
        rng = np.random.default_rng(3)
        col = np.stack([rng.permutation(50)[:k] for _ in range(n)]).astype(np.int32)
        col.sort(axis=1)
        val = rng.choice([-400.0, 400.0], size=(n, k)).astype(np.float32)
        return synthdata.from_arrays(np.arange(0, n * k + 1, k), col.ravel(), val.ravel(),
                                     np.where(rng.random(n) < 0.5, -1.0, 1.0), n_cols=50, eta=0.5)
    raise KeyError(name)


EDGES = ["no-rows", "all-empty-rows", "one-row", "one-feature-chain", "exp-saturation"]


@functools.lru_cache(maxsize=None)
def oracle_chains(name):
    return oracle.chains(problem(name))


@functools.lru_cache(maxsize=None)
def oracle_levels(name):
    p = problem(name)
    lv, L = oracle.levels(p, oracle_chains(name)["prev"])
    order, level_ptr = oracle.level_order(lv, L)
    return lv, L, order, level_ptr


@functools.lru_cache(maxsize=None)
def oracle_sgd(name):
    return oracle.sgd(problem(name))


def rel_err(got, ref):
    """max_j |got_j - ref_j| / max_j |ref_j| (0 when both are all zero)."""
    scale = float(np.max(np.abs(ref))) if ref.size else 0.0
    diff = float(np.max(np.abs(got.astype(np.float64) - ref))) if ref.size else 0.0
    return diff / scale if scale > 0 else diff
