"""CPU model of k_slots' index logic (csrc/build.cu), against the plain
definitions of rank and feat_ptr on sorted keys.

k_slots gives each warp a contiguous range of 128-slot steps (four slots per
lane).  A slot's rank is its distance to the first slot of its feature's run
(Definition 2's chunk = feature; the rank is the read protocol's iteration
number).  The warp finds that first slot without feat_ptr. The lanes take a
running maximum of the run starts inside the step. The run in progress is
carried from one step to the next. At the start of the warp's range, a
gallop back through the sorted keys finds it. feat_ptr[b] is the first slot
whose key is >= b. Each step writes it for the features from the key before
the step up to the step's last key, each by a binary search in the step's
keys. The step that holds the last slot also writes n for the features
after the last key.  The model replays exactly that
arithmetic for random key sets and warp counts (ragged tails, empty features,
long runs that cross several steps and warps) and compares with
np.searchsorted; planted mistakes in the carry, the lane scan or the search
bounds must fail it."""
import numpy as np
import pytest

SENT = 0xFFFFFFFF


def run_start(skey, q):
    """first slot of the run of skey[q]: gallop back, then binary search"""
    j = skey[q]
    hi, lo, step = q, q - 1, 1
    while lo >= 0 and skey[lo] == j:
        hi = lo
        step <<= 1
        lo = hi - step
    lo = max(lo, -1)
    while hi - lo > 1:
        mid = lo + ((hi - lo) >> 1)
        if skey[mid] == j:
            hi = mid
        else:
            lo = mid
    return hi


def model(skey, n_cols, n_warps, plant=None):
    nnz = len(skey)
    rank = np.full(nnz, -1, np.int64)
    fp = np.full(n_cols + 1, -7, np.int64)
    steps = (nnz + 127) >> 7
    per = (steps + n_warps - 1) // n_warps

    def key(i):
        return int(skey[i]) if 0 <= i < nnz else SENT

    for w in range(n_warps):
        st0, st1 = w * per, min(steps, w * per + per)
        carry = run_start(skey, (st0 << 7) - 1) if st0 < st1 and st0 > 0 else 0
        for st in range(st0, st1):
            base = st << 7
            kk = [[key(base + 4 * lane + e - 1) for e in range(6)] for lane in range(32)]
            # last run start among each lane's valid slots (offset in the step)
            ls = []
            for lane in range(32):
                v = -1
                for e in range(4):
                    if base + 4 * lane + e < nnz and kk[lane][e] != kk[lane][e + 1]:
                        v = 4 * lane + e
                ls.append(v)
            inc = list(np.maximum.accumulate(ls))
            for lane in range(32):
                exc = inc[lane - 1] if lane > 0 else -1
                if plant == "inclusive_scan":
                    exc = inc[lane]
                before = base + exc if exc >= 0 else carry
                r = 0
                for e in range(4):
                    s = base + 4 * lane + e
                    if s >= nnz:
                        break
                    first = kk[lane][e] != kk[lane][e + 1]
                    r = 0 if first else (r + 1 if e > 0 else s - before)
                    rank[s] = r
            if inc[31] >= 0 and plant != "no_carry":
                carry = base + inc[31]
            # feat_ptr for the step's feature range
            nv = min(128, nnz - base)
            sk = [int(skey[base + i]) for i in range(nv)]
            kb = kk[0][0]
            khi = sk[nv - 1]
            b0 = 0 if base == 0 else kb + 1
            if plant == "range_from_first_key":
                b0 = 0 if base == 0 else sk[0]
            for lane in range(32):
                b = b0 + lane
                while b <= min(khi, n_cols):
                    lo, hi = 0, nv
                    while lo < hi:
                        mid = (lo + hi) >> 1
                        if sk[mid] < b:
                            lo = mid + 1
                        else:
                            hi = mid
                    fp[b] = base + lo
                    b += 32
            if base + nv == nnz and plant != "no_tail":
                for lane in range(32):
                    b = khi + 1 + lane
                    while b <= n_cols:
                        fp[b] = nnz
                        b += 32
    return rank, fp


def _keys(rng, kind, nnz, n_cols):
    if kind == "uniform":
        k = rng.integers(0, n_cols, nnz)
    elif kind == "zipf":
        k = np.minimum(rng.zipf(1.3, nnz) - 1, n_cols - 1)
    elif kind == "few":                        # runs far longer than a step
        k = rng.integers(0, max(1, n_cols // 50), nnz)
    else:                                      # sparse: most features empty
        k = rng.integers(0, n_cols, nnz) * 7 % n_cols
    return np.sort(k).astype(np.int64)


def _reference(skey, n_cols):
    nnz = len(skey)
    fp = np.searchsorted(skey, np.arange(n_cols + 1), side="left")
    rank = np.arange(nnz) - np.searchsorted(skey, skey, side="left")
    return rank, fp


CASES = [(kind, seed) for kind in ("uniform", "zipf", "few", "sparse") for seed in range(6)]


@pytest.mark.parametrize("kind,seed", CASES)
def test_rank_and_feat_ptr_match_the_definitions(kind, seed):
    rng = np.random.default_rng(1000 + seed)
    nnz = int(rng.integers(1, 2500))
    n_cols = int(rng.integers(1, 3000))
    skey = _keys(rng, kind, nnz, n_cols)
    ref_rank, ref_fp = _reference(skey, n_cols)
    for n_warps in (1, 3, int(rng.integers(2, 40))):
        rank, fp = model(skey, n_cols, n_warps)
        assert np.array_equal(rank, ref_rank), n_warps
        assert np.array_equal(fp, ref_fp), n_warps


def test_one_feature_and_exact_steps():
    # every slot one feature (a run across all warps), and nnz a multiple of 128
    for nnz in (1, 127, 128, 129, 256, 1024):
        for n_cols in (1, 5):
            skey = np.zeros(nnz, np.int64) + (n_cols - 1)
            ref_rank, ref_fp = _reference(skey, n_cols)
            for n_warps in (1, 2, 7):
                rank, fp = model(skey, n_cols, n_warps)
                assert np.array_equal(rank, ref_rank) and np.array_equal(fp, ref_fp)


def test_run_start_gallop():
    rng = np.random.default_rng(7)
    skey = np.sort(rng.integers(0, 40, 5000))
    first = np.searchsorted(skey, skey, side="left")
    for q in range(len(skey)):
        assert run_start(skey, q) == first[q]


@pytest.mark.parametrize("plant", ["inclusive_scan", "no_carry", "range_from_first_key", "no_tail"])
def test_planted_mistakes_fail(plant):
    rng = np.random.default_rng(99)
    failed = False
    for kind in ("uniform", "few", "sparse"):
        nnz, n_cols = 2000, 1500
        skey = _keys(rng, kind, nnz, n_cols)
        skey = skey[skey < n_cols - 3]          # empty features after the last key
        ref_rank, ref_fp = _reference(skey, n_cols)
        rank, fp = model(skey, n_cols, 4, plant=plant)
        failed |= not (np.array_equal(rank, ref_rank) and np.array_equal(fp, ref_fp))
    assert failed, plant
