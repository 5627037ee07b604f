"""Seeded synthetic sparse workloads (inputs only).

This module draws the CSR examples, labels and sizes that both the CPU oracle
and the CUDA path consume.  It holds none of the method's arithmetic: no
conflict chains, no levels, no SGD updates.  The drawing itself is done by
``synth.c`` (Philox4x32-10 streams keyed per row, so the arrays do not depend
on the thread count).

The five named workloads restate the synthetic shapes of the paper's sparse
SGD setting (Section 6.3 trains SGD on a sparse, ~1.5e5-feature text set;
the sizes below are the scaled GPU workloads):

=============  ==========  ===========  ====  ==========  =========  ========  ======
name           rows N      features F   k     ids         values     loss      epochs
=============  ==========  ===========  ====  ==========  =========  ========  ======
tiny           20,000      10,000       10    uniform     N(0,1)     logistic  1
zipf-1m        1,000,000   1,000,000    20    Zipf 1.0    N(0,1)     logistic  1
ctr            10,000,000  10,000,000   50    Zipf 1.1    1.0        logistic  1
low-conflict   4,000,000   100,000,000  100   uniform     U(-1,1)    squared   2
deep-chain     2,000,000   50,000       200   Zipf 1.3    N(0,1)     hinge     3
=============  ==========  ===========  ====  ==========  =========  ========  ======
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.c")
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = os.path.join(_LIBDIR, "libsynth.so")
_lock = threading.Lock()
_lib = None

LOSS_LOGISTIC, LOSS_SQUARED, LOSS_HINGE = 0, 1, 2
LOSS_NAMES = {"logistic": LOSS_LOGISTIC, "squared": LOSS_SQUARED, "hinge": LOSS_HINGE}


class _Cfg(ctypes.Structure):
    _fields_ = [
        ("n_rows", ctypes.c_int64), ("n_cols", ctypes.c_int64),
        ("k", ctypes.c_int32), ("k_lo", ctypes.c_int32),
        ("id_dist", ctypes.c_int32), ("zipf_s", ctypes.c_double),
        ("val_dist", ctypes.c_int32), ("label_kind", ctypes.c_int32),
        ("wstar_std", ctypes.c_double), ("noise_std", ctypes.c_double),
        ("seed", ctypes.c_uint64), ("wseed", ctypes.c_uint64),
        ("nthreads", ctypes.c_int32),
    ]


def build() -> str:
    """Compile libsynth.so in-tree (host code only) and return its path."""
    with _lock:
        os.makedirs(_LIBDIR, exist_ok=True)
        if os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
            return _LIB
        tmp = f"{_LIB}.{os.getpid()}.tmp"
        subprocess.run(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-pthread",
                        "-ffp-contract=off", "-o", tmp, _SRC, "-lm"], check=True)
        os.replace(tmp, _LIB)
        return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        lib.synth_row_ptr.argtypes = [ctypes.POINTER(_Cfg), ctypes.c_void_p]
        lib.synth_wstar.argtypes = [ctypes.POINTER(_Cfg), ctypes.c_void_p]
        lib.synth_fill.argtypes = [ctypes.POINTER(_Cfg)] + [ctypes.c_void_p] * 5
        lib.synth_philox4x32_10.argtypes = [ctypes.c_void_p] * 3
        _lib = lib
    return _lib


@dataclasses.dataclass
class Problem:
    """One synthetic sparse workload: CSR examples (D), labels and SGD settings."""
    name: str
    row_ptr: np.ndarray          # int64[N+1]
    col: np.ndarray              # int32[nnz]
    val: np.ndarray | None       # float32[nnz], None = every value 1.0
    y: np.ndarray                # float32[N]
    n_cols: int
    loss: int
    eta: float
    epochs: int
    bsp_batch: int | None = None

    @property
    def n_rows(self) -> int:
        return int(self.row_ptr.shape[0] - 1)

    @property
    def nnz(self) -> int:
        return int(self.col.shape[0])

    def values(self) -> np.ndarray:
        """Values as an explicit float32 array (ones when ``val`` is None)."""
        return self.val if self.val is not None else np.ones(self.nnz, np.float32)


WORKLOADS = {
    "tiny": dict(n_rows=20_000, n_cols=10_000, k=10, ids="uniform", vals="normal",
                 labels="sign", wstar_std=1.0, loss="logistic", eta=0.01, epochs=1),
    "zipf-1m": dict(n_rows=1_000_000, n_cols=1_000_000, k=20, ids="zipf", zipf_s=1.0,
                    vals="normal", labels="sign", wstar_std=1.0, loss="logistic", eta=0.01, epochs=1),
    "ctr": dict(n_rows=10_000_000, n_cols=10_000_000, k=50, ids="zipf", zipf_s=1.1,
                vals="ones", labels="bernoulli", wstar_std=0.1, loss="logistic", eta=0.05, epochs=1),
    "low-conflict": dict(n_rows=4_000_000, n_cols=100_000_000, k=100, ids="uniform",
                         vals="uniform", labels="linear", wstar_std=1.0, noise_std=0.1,
                         loss="squared", eta=0.001, epochs=2),
    "deep-chain": dict(n_rows=2_000_000, n_cols=50_000, k=200, ids="zipf", zipf_s=1.3,
                       vals="normal", labels="sign", wstar_std=1.0, loss="hinge", eta=0.01,
                       epochs=3, bsp_batch=4096),
    # the dense linear-regression setting of the paper's Experiments 6.1/6.2:
    # 960 numerical features, 5000 examples, full-batch gradient descent
    # (BSP with one batch of all examples per iteration)
    "dense-lr": dict(n_rows=5_000, n_cols=960, k=960, ids="dense", vals="normal", labels="linear",
                     wstar_std=1.0, noise_std=0.1, loss="squared", eta=1e-4, epochs=20, bsp_batch=5_000),
}

_IDS = {"uniform": 0, "zipf": 1, "dense": 2}
_VALS = {"normal": 0, "uniform": 1, "ones": 2}
_LABELS = {"sign": 0, "bernoulli": 1, "linear": 2}

DATA_SEED = 1508
WSTAR_SEED = 703


def generate(name: str, seed: int = DATA_SEED, wseed: int = WSTAR_SEED, nthreads: int | None = None,
             **overrides) -> Problem:
    """Draw workload ``name`` (a key of WORKLOADS); keyword overrides change its sizes.

    ``k_lo`` (default ``k``) makes row lengths uniform in [k_lo, k], which gives
    ragged and empty rows for edge-case tests.
    """
    spec = dict(WORKLOADS[name])
    spec.update(overrides)
    lib = _load()
    cfg = _Cfg()
    cfg.n_rows = int(spec["n_rows"])
    cfg.n_cols = int(spec["n_cols"])
    cfg.k = int(spec["k"])
    cfg.k_lo = int(spec.get("k_lo", spec["k"]))
    cfg.id_dist = _IDS[spec["ids"]]
    cfg.zipf_s = float(spec.get("zipf_s", 1.0))
    cfg.val_dist = _VALS[spec["vals"]]
    cfg.label_kind = _LABELS[spec["labels"]]
    cfg.wstar_std = float(spec.get("wstar_std", 1.0))
    cfg.noise_std = float(spec.get("noise_std", 0.0))
    cfg.seed = int(seed)
    cfg.wseed = int(wseed)
    cfg.nthreads = int(nthreads or min(64, os.cpu_count() or 1))
    row_ptr = np.empty(cfg.n_rows + 1, np.int64)
    if lib.synth_row_ptr(ctypes.byref(cfg), row_ptr.ctypes.data) != 0:
        raise ValueError(f"bad synthetic configuration {spec}")
    nnz = int(row_ptr[-1])
    col = np.empty(nnz, np.int32)
    val = None if spec["vals"] == "ones" else np.empty(nnz, np.float32)
    y = np.empty(cfg.n_rows, np.float32)
    wstar = np.empty(cfg.n_cols, np.float32)
    if lib.synth_wstar(ctypes.byref(cfg), wstar.ctypes.data) != 0:
        raise RuntimeError("w* generation failed")
    st = lib.synth_fill(ctypes.byref(cfg), row_ptr.ctypes.data, wstar.ctypes.data, col.ctypes.data,
                        None if val is None else val.ctypes.data, y.ctypes.data)
    if st != 0:
        raise RuntimeError(f"synthetic row generation failed ({st})")
    return Problem(name=name, row_ptr=row_ptr, col=col, val=val, y=y, n_cols=cfg.n_cols,
                   loss=LOSS_NAMES[spec["loss"]], eta=float(spec["eta"]), epochs=int(spec["epochs"]),
                   bsp_batch=spec.get("bsp_batch"))


def philox4x32_10(ctr, key) -> np.ndarray:
    """One Philox4x32-10 block (for the generator's known-answer test)."""
    lib = _load()
    c = np.asarray(ctr, np.uint32)
    k = np.asarray(key, np.uint32)
    out = np.empty(4, np.uint32)
    lib.synth_philox4x32_10(c.ctypes.data, k.ctypes.data, out.ctypes.data)
    return out


def from_arrays(row_ptr, col, val, y, n_cols, loss="logistic", eta=0.01, epochs=1, name="custom",
                bsp_batch=None) -> Problem:
    """Wrap hand-made arrays (edge cases in tests) as a Problem."""
    return Problem(name=name, row_ptr=np.ascontiguousarray(row_ptr, np.int64),
                   col=np.ascontiguousarray(col, np.int32),
                   val=None if val is None else np.ascontiguousarray(val, np.float32),
                   y=np.ascontiguousarray(y, np.float32), n_cols=int(n_cols),
                   loss=LOSS_NAMES[loss] if isinstance(loss, str) else int(loss), eta=float(eta),
                   epochs=int(epochs), bsp_batch=bsp_batch)
