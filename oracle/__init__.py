"""CPU oracle for serially-equivalent sparse SGD -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product library never calls it and
shares no code with it.  The arithmetic lives in ``pdb_oracle.c`` (plain C,
single thread, no contraction); this module marshals numpy arrays and adds
the pure-Python brute-force levels used on tiny cases.  ``history.py`` holds
the checker of execution histories and traces.

Every routine follows one definition of the paper:
  validate      Definitions 1 and 3 (examples are sets of features)
  chains        Section 5, read protocol (per-chunk iteration number ->
                per-feature occurrence chain and rank)
  levels        Theorem 3 (a level is one barrier step over disjoint
                transactions), longest conflict path
  expf, dot,    the written numerics of the update (the paper fixes no
  grad          summation order or exponential): Cody-Waite reduction and a
                Taylor polynomial, 32 partial sums and a butterfly, the three
                losses' derivatives
  sgd           Algorithm 1 / Definition 4, one iteration per example
  bsp           Algorithm 2a with B examples between barriers
  sgd_f64       fp64 drift reference (not a parity target)
  history.*     Definition 4 and the Read and Write Constraints (Section
                4.4) on histories; the asynchronous Read Constraint
                (Section 7) on traces

Admissible delay (Section 7) has no routine here: at delay 0 its result is
``sgd``'s; for delay > 0 many results are correct (parity unpinned), and its
runs are checked by properties instead (every step applied once, the
asynchronous Read Constraint on a trace).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pdb_oracle.c")
_LIBDIR = os.path.join(_HERE, "_lib")
_LIB = os.path.join(_LIBDIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, BAD_ROWPTR, BAD_COL, DUP, NOMEM = 0, 1, 2, 3, 4
LOGISTIC, SQUARED, HINGE = 0, 1, 2

_P = ctypes.c_void_p
_I64 = ctypes.c_int64


def build() -> str:
    """Compile liboracle.so in-tree: -O2, no FMA contraction, no fast-math."""
    with _lock:
        os.makedirs(_LIBDIR, exist_ok=True)
        if os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
            return _LIB
        tmp = f"{_LIB}.{os.getpid()}.tmp"
        subprocess.run(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-ffp-contract=off",
                        "-fno-fast-math", "-o", tmp, _SRC, "-lm"], check=True)
        os.replace(tmp, _LIB)
        return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        lib.orc_validate.argtypes = [_I64, _I64, _I64, _P, _P]
        lib.orc_chains.argtypes = [_I64, _I64, _I64, _P, _P, _P, _P, _P, _P, _P]
        lib.orc_levels.argtypes = [_I64, _I64, _P, _P, _P]
        lib.orc_levels.restype = _I64
        lib.orc_level_order.argtypes = [_I64, _I64, _P, _P, _P]
        lib.orc_expf.argtypes = [ctypes.c_float]
        lib.orc_expf.restype = ctypes.c_float
        lib.orc_expf_n.argtypes = [_P, _P, _I64]
        lib.orc_dot.argtypes = [_P, _P, _P, _I64]
        lib.orc_dot.restype = ctypes.c_float
        lib.orc_grad.argtypes = [ctypes.c_int, ctypes.c_float, ctypes.c_float]
        lib.orc_grad.restype = ctypes.c_float
        lib.orc_sgd.argtypes = [_I64, _P, _P, _P, _P, _P, ctypes.c_int, ctypes.c_float, ctypes.c_int, _P]
        lib.orc_bsp.argtypes = [_I64, _I64, _P, _P, _P, _P, _P, ctypes.c_int, ctypes.c_float, _I64, ctypes.c_int]
        lib.orc_sgd_f64.argtypes = [_I64, _P, _P, _P, _P, _P, ctypes.c_int, ctypes.c_double, ctypes.c_int]
        _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data


def _csr(problem_or_arrays):
    p = problem_or_arrays
    row_ptr = np.ascontiguousarray(p.row_ptr, np.int64)
    col = np.ascontiguousarray(p.col, np.int32)
    val = None if p.val is None else np.ascontiguousarray(p.val, np.float32)
    return row_ptr, col, val


def validate(p) -> int:
    row_ptr, col, _ = _csr(p)
    n = row_ptr.shape[0] - 1
    return int(_load().orc_validate(n, p.n_cols, col.shape[0], _ptr(row_ptr), _ptr(col)))


def chains(p) -> dict:
    """csc_pos, feat_ptr, prev, next, rank of the occurrence chains."""
    row_ptr, col, _ = _csr(p)
    nnz, n_cols = col.shape[0], p.n_cols
    out = dict(csc_pos=np.empty(nnz, np.int32), feat_ptr=np.empty(n_cols + 1, np.int64),
               prev=np.empty(nnz, np.int32), next=np.empty(nnz, np.int32), rank=np.empty(nnz, np.int32))
    rc = _load().orc_chains(row_ptr.shape[0] - 1, n_cols, nnz, _ptr(row_ptr), _ptr(col), _ptr(out["csc_pos"]),
                            _ptr(out["feat_ptr"]), _ptr(out["prev"]), _ptr(out["next"]), _ptr(out["rank"]))
    if rc != OK:
        raise MemoryError("oracle chains")
    return out


def levels(p, prev=None) -> tuple[np.ndarray, int]:
    """(level[N], L) by the longest-path recurrence over the chains."""
    row_ptr, col, _ = _csr(p)
    if prev is None:
        prev = chains(p)["prev"]
    n = row_ptr.shape[0] - 1
    level = np.empty(n, np.int32)
    L = int(_load().orc_levels(n, col.shape[0], _ptr(row_ptr), _ptr(np.ascontiguousarray(prev, np.int32)),
                               _ptr(level)))
    if L < 0:
        raise MemoryError("oracle levels")
    return level, L


def level_order(level: np.ndarray, n_levels: int) -> tuple[np.ndarray, np.ndarray]:
    """(order[N], level_ptr[L+1]): examples by level, ascending id within a level."""
    level = np.ascontiguousarray(level, np.int32)
    order = np.empty(level.shape[0], np.int32)
    level_ptr = np.empty(n_levels + 1, np.int64)
    if _load().orc_level_order(level.shape[0], n_levels, _ptr(level), _ptr(order), _ptr(level_ptr)) != OK:
        raise MemoryError("oracle level order")
    return order, level_ptr


def levels_bruteforce(p) -> np.ndarray:
    """level[t] = 1 + max{level[u] : u < t, S_u and S_t share a feature}, 0 if none.

    Pure Python over all earlier examples: O(N^2 k); tiny inputs only.
    """
    sets = [set(p.col[p.row_ptr[t]:p.row_ptr[t + 1]].tolist()) for t in range(len(p.row_ptr) - 1)]
    level = []
    for t, st in enumerate(sets):
        lv = -1
        for u in range(t):
            if sets[u] & st:
                lv = max(lv, level[u])
        level.append(lv + 1)
    return np.array(level, np.int32)


def expf(x) -> np.ndarray:
    x = np.ascontiguousarray(np.asarray(x, np.float32).ravel())
    out = np.empty_like(x)
    _load().orc_expf_n(_ptr(x), _ptr(out), x.shape[0])
    return out


def dot(w, col, val) -> np.float32:
    w = np.ascontiguousarray(w, np.float32)
    col = np.ascontiguousarray(col, np.int32)
    val = None if val is None else np.ascontiguousarray(val, np.float32)
    return np.float32(_load().orc_dot(_ptr(w), _ptr(col), _ptr(val), col.shape[0]))


def grad(loss: int, m: float, y: float) -> np.float32:
    return np.float32(_load().orc_grad(int(loss), float(np.float32(m)), float(np.float32(y))))


def sgd(p, w0=None, epochs=None, eta=None, loss=None, order=None, rows=None) -> np.ndarray:
    """Sequential SGD (Algorithm 1), returns the fp32 weights.

    ``rows`` limits the run to the first ``rows`` examples (a bounded sample
    for timing); ``order`` is an explicit execution order of the examples.
    """
    row_ptr, col, val = _csr(p)
    n = row_ptr.shape[0] - 1 if rows is None else int(rows)
    w = np.zeros(p.n_cols, np.float32) if w0 is None else np.array(w0, np.float32, copy=True)
    o = None if order is None else np.ascontiguousarray(order, np.int32)
    if o is not None:
        n = o.shape[0]
    _load().orc_sgd(n, _ptr(row_ptr), _ptr(col), _ptr(val), _ptr(np.ascontiguousarray(p.y, np.float32)), _ptr(w),
                    p.loss if loss is None else int(loss), float(p.eta if eta is None else eta),
                    int(p.epochs if epochs is None else epochs), _ptr(o))
    return w


def bsp(p, batch: int, w0=None, epochs=None, eta=None, loss=None) -> np.ndarray:
    """BSP mini-batch SGD (Algorithm 2a with ``batch`` examples per barrier pair)."""
    row_ptr, col, val = _csr(p)
    n = row_ptr.shape[0] - 1
    w = np.zeros(p.n_cols, np.float32) if w0 is None else np.array(w0, np.float32, copy=True)
    rc = _load().orc_bsp(n, p.n_cols, _ptr(row_ptr), _ptr(col), _ptr(val), _ptr(np.ascontiguousarray(p.y, np.float32)),
                         _ptr(w), p.loss if loss is None else int(loss), float(p.eta if eta is None else eta),
                         int(batch), int(p.epochs if epochs is None else epochs))
    if rc != OK:
        raise ValueError("oracle bsp")
    return w


def sgd_f64(p, epochs=None) -> np.ndarray:
    row_ptr, col, val = _csr(p)
    w = np.zeros(p.n_cols, np.float64)
    _load().orc_sgd_f64(row_ptr.shape[0] - 1, _ptr(row_ptr), _ptr(col), _ptr(val),
                        _ptr(np.ascontiguousarray(p.y, np.float32)), _ptr(w), p.loss, float(p.eta),
                        int(p.epochs if epochs is None else epochs))
    return w
