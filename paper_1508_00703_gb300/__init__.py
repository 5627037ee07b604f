"""Python binding of libpdb (serially-equivalent sparse SGD on one GPU).

Argument marshalling only: every step of the method runs in the CUDA kernels
of ``csrc/`` behind the C ABI declared in ``include/pdb.h``.  The functions
below carry the C names and forward torch tensors' device pointers and the
current CUDA stream.  There is no CPU fallback: if the compiled library is
missing or cannot load, every call raises.
"""
from __future__ import annotations

import ctypes
import glob
import os
import subprocess
import threading
from concurrent.futures import ThreadPoolExecutor

_HERE = os.path.dirname(os.path.abspath(__file__))
_ROOT = os.path.dirname(_HERE)
_CSRC = os.path.join(_HERE, "csrc")
_INCLUDE = os.path.join(_ROOT, "include")
_LIBDIR = os.path.join(_HERE, "_lib")
LIB_PATH = os.path.join(_LIBDIR, "libpdb.so")
ARCH = "-gencode=arch=compute_103a,code=sm_103a"
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-fmad=false", "-Xcompiler", "-fPIC", ARCH, f"-I{_INCLUDE}"]

PDB_OK, PDB_EINVAL, PDB_ERANGE, PDB_EDUP, PDB_ENOMEM, PDB_ECUDA, PDB_ETIMEOUT, PDB_EFAULT, PDB_ESTATE = \
    0, -1, -2, -3, -4, -5, -6, -7, -8
PDB_ETOOBIG = -9
NOALLOC_MAX_COLS = 1 << 20
PDB_LOSS_LOGISTIC, PDB_LOSS_SQUARED, PDB_LOSS_HINGE = 0, 1, 2
PDB_SCHED_LEVELS, PDB_SCHED_READY, PDB_SCHED_CHAIN, PDB_SCHED_AUTO, PDB_SCHED_WINDOW = 0, 1, 2, 3, 4
PDB_SSP_COUNT, PDB_SSP_PREFIX = 1, 2

_lock = threading.Lock()
_lib = None


class PdbError(RuntimeError):
    def __init__(self, code: int, what: str = ""):
        self.code = code
        msg = _strerror(code)
        super().__init__(f"{what}: {msg} ({code})" if what else f"{msg} ({code})")


def _sources():
    return sorted(glob.glob(os.path.join(_CSRC, "*.cu")))


def _deps():
    return _sources() + glob.glob(os.path.join(_CSRC, "*.cuh")) + [os.path.join(_INCLUDE, "pdb.h")]


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile libpdb.so in-tree for sm_103a (nvcc, one object per .cu, in parallel)."""
    with _lock:
        os.makedirs(_LIBDIR, exist_ok=True)
        if (not force and os.path.exists(LIB_PATH)
                and os.path.getmtime(LIB_PATH) >= max(os.path.getmtime(p) for p in _deps())):
            return LIB_PATH
        objs = []

        def compile_one(src):
            obj = os.path.join(_LIBDIR, os.path.basename(src)[:-3] + f".{os.getpid()}.o")
            cmd = ["nvcc", *NVCC_FLAGS, "-c", src, "-o", obj]
            if verbose:
                cmd += ["-Xptxas", "-v"]
            r = subprocess.run(cmd, capture_output=True, text=True)
            if r.returncode != 0:
                raise RuntimeError(f"nvcc failed for {src}:\n{r.stderr}")
            if verbose:
                print(r.stderr)
            return obj

        with ThreadPoolExecutor(max_workers=len(_sources())) as ex:
            objs = list(ex.map(compile_one, _sources()))
        tmp = f"{LIB_PATH}.{os.getpid()}.tmp"
        r = subprocess.run(["nvcc", "-shared", ARCH, "-o", tmp, *objs], capture_output=True, text=True)
        for o in objs:
            os.remove(o)
        if r.returncode != 0:
            raise RuntimeError(f"link of libpdb.so failed:\n{r.stderr}")
        os.replace(tmp, LIB_PATH)
        return LIB_PATH


class pdb_csr(ctypes.Structure):
    _fields_ = [("n_rows", ctypes.c_int64), ("n_cols", ctypes.c_int64), ("nnz", ctypes.c_int64),
                ("row_ptr", ctypes.c_void_p), ("col", ctypes.c_void_p), ("val", ctypes.c_void_p)]


class pdb_opts(ctypes.Structure):
    """Launch and wait options (zeroed = defaults).  The calls also take a dict of
    the same fields; a torch tensor given as `trace` passes its device pointer."""
    _fields_ = [("blocks_per_sm", ctypes.c_int32), ("ticket_chunk", ctypes.c_int32),
                ("wait_timeout_s", ctypes.c_double), ("trace", ctypes.c_void_p), ("ssp_gates", ctypes.c_int32)]


class pdb_stats(ctypes.Structure):
    _fields_ = [("n_rows", ctypes.c_int64), ("n_cols", ctypes.c_int64), ("nnz", ctypes.c_int64),
                ("n_levels", ctypes.c_int64), ("max_level_width", ctypes.c_int64), ("max_chain", ctypes.c_int64),
                ("ms_build", ctypes.c_double), ("ms_schedule", ctypes.c_double), ("ms_sgd", ctypes.c_double),
                ("ms_bsp", ctypes.c_double), ("ms_sgd_kernels", ctypes.c_double), ("sched_mode", ctypes.c_int64)]

    def as_dict(self):
        return {k: getattr(self, k) for k, _ in self._fields_}


EXPORTS = ["pdb_build_conflicts", "pdb_conflicts_arrays", "pdb_schedule_build", "pdb_schedule_levels",
           "pdb_schedule_ready",
           "pdb_sgd_epoch", "pdb_bsp_epoch", "pdb_status", "pdb_get_stats", "pdb_conflicts_free",
           "pdb_schedule_free", "pdb_strerror", "pdb_memcpy", "pdb_eval_expf", "pdb_eval_grad", "pdb_launch_count",
           "pdb_sgd_epoch_ready_noalloc", "pdb_ssp_epoch", "pdb_bsp_plan_build", "pdb_bsp_plan_batches",
           "pdb_bsp_coef", "pdb_bsp_apply", "pdb_bsp_plan_free"]


def load(path: str | None = None):
    """Load libpdb.so (building it first if it is absent or stale); raises if that fails."""
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(path or build())
        P, I64, I32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
        PP = ctypes.POINTER(ctypes.c_void_p)
        lib.pdb_build_conflicts.argtypes = [ctypes.POINTER(pdb_csr), PP, P]
        lib.pdb_conflicts_arrays.argtypes = [P, PP, PP, PP, PP, PP, P]
        lib.pdb_schedule_build.argtypes = [P, I32, PP, P]
        lib.pdb_schedule_levels.argtypes = [P, PP, PP, PP, ctypes.POINTER(I64), P]
        lib.pdb_schedule_ready.argtypes = [P, PP, PP]
        lib.pdb_sgd_epoch.argtypes = [ctypes.POINTER(pdb_csr), P, P, P, P, I32, ctypes.c_float, I32,
                                      ctypes.POINTER(pdb_opts), P]
        lib.pdb_bsp_epoch.argtypes = [ctypes.POINTER(pdb_csr), P, P, P, I32, ctypes.c_float, I64, I32,
                                      ctypes.POINTER(pdb_opts), P]
        lib.pdb_status.argtypes = [P, P]
        lib.pdb_get_stats.argtypes = [P, P, ctypes.POINTER(pdb_stats)]
        lib.pdb_conflicts_free.argtypes = [P]
        lib.pdb_conflicts_free.restype = None
        lib.pdb_schedule_free.argtypes = [P]
        lib.pdb_schedule_free.restype = None
        lib.pdb_strerror.argtypes = [I32]
        lib.pdb_strerror.restype = ctypes.c_char_p
        lib.pdb_memcpy.argtypes = [P, P, ctypes.c_size_t, P]
        lib.pdb_eval_expf.argtypes = [P, P, I64, P]
        lib.pdb_eval_grad.argtypes = [P, P, P, I64, I32, P]
        lib.pdb_sgd_epoch_ready_noalloc.argtypes = [ctypes.POINTER(pdb_csr), P, P, P, I32, ctypes.c_float, I32, P]
        lib.pdb_ssp_epoch.argtypes = [ctypes.POINTER(pdb_csr), P, P, P, P, I32, ctypes.c_float, I32, I64, P,
                                      ctypes.POINTER(pdb_opts), P]
        lib.pdb_bsp_plan_build.argtypes = [P, I64, PP, P]
        lib.pdb_bsp_plan_batches.argtypes = [P]
        lib.pdb_bsp_plan_batches.restype = I64
        lib.pdb_bsp_coef.argtypes = [P, ctypes.POINTER(pdb_csr), P, P, I32, ctypes.c_float, I64, I64, P, P]
        lib.pdb_bsp_apply.argtypes = [P, P, I64, P, P]
        lib.pdb_bsp_plan_free.argtypes = [P]
        lib.pdb_bsp_plan_free.restype = None
        lib.pdb_launch_count.argtypes = []
        lib.pdb_launch_count.restype = I64
        _lib = lib
    return _lib


def _strerror(code: int) -> str:
    try:
        return load().pdb_strerror(int(code)).decode()
    except Exception:  # the library itself failed to load
        return f"error {code}"


def _check(rc: int, what: str):
    if rc != PDB_OK:
        raise PdbError(rc, what)


def _stream(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


class Csr:
    """CSR examples on the device: int64 row_ptr, int32 col, float32 val (or None)."""

    def __init__(self, row_ptr, col, val, n_cols: int):
        self.row_ptr, self.col, self.val, self.n_cols = row_ptr, col, val, int(n_cols)
        self.struct = pdb_csr(row_ptr.numel() - 1, self.n_cols, col.numel(), _ptr(row_ptr), _ptr(col), _ptr(val))

    @classmethod
    def from_problem(cls, problem, device="cuda"):
        import torch
        row_ptr = torch.from_numpy(problem.row_ptr).to(device)
        col = torch.from_numpy(problem.col).to(device)
        val = None if problem.val is None else torch.from_numpy(problem.val).to(device)
        return cls(row_ptr, col, val, problem.n_cols)


class Conflicts:
    """Owns a pdb_conflicts handle."""

    def __init__(self, handle, n_rows, n_cols, nnz):
        self.handle = handle
        self.n_rows, self.n_cols, self.nnz = n_rows, n_cols, nnz

    def __del__(self):
        if getattr(self, "handle", None) and _lib is not None:
            _lib.pdb_conflicts_free(self.handle)
            self.handle = None


class Schedule:
    """Owns a pdb_schedule handle (keeps its conflicts alive)."""

    def __init__(self, handle, conflicts, mode):
        self.handle, self.conflicts, self.mode = handle, conflicts, mode

    def __del__(self):
        if getattr(self, "handle", None) and _lib is not None:
            _lib.pdb_schedule_free(self.handle)
            self.handle = None


def pdb_build_conflicts(X: Csr, stream=None) -> Conflicts:
    """Validate X and build its per-feature occurrence chains (Definitions 1-3,
    Section 5); errors the device finds surface through pdb_status."""
    h = ctypes.c_void_p()
    _check(load().pdb_build_conflicts(ctypes.byref(X.struct), ctypes.byref(h), _stream(stream)),
           "pdb_build_conflicts")
    return Conflicts(h, X.struct.n_rows, X.struct.n_cols, X.struct.nnz)


def pdb_conflicts_arrays(c: Conflicts, stream=None) -> dict:
    """Borrowed device pointers (ints) of csc_pos, feat_ptr, prev, next, rank."""
    ptrs = [ctypes.c_void_p() for _ in range(5)]
    _check(load().pdb_conflicts_arrays(c.handle, *[ctypes.byref(p) for p in ptrs], _stream(stream)),
           "pdb_conflicts_arrays")
    return dict(zip(["csc_pos", "feat_ptr", "prev", "next", "rank"], [p.value for p in ptrs]))


def pdb_schedule_build(c: Conflicts, mode: int, stream=None) -> Schedule:
    """Schedule for pdb_sgd_epoch: PDB_SCHED_LEVELS (Theorem 3), READY, WINDOW,
    CHAIN or AUTO (include/pdb.h describes each)."""
    h = ctypes.c_void_p()
    _check(load().pdb_schedule_build(c.handle, int(mode), ctypes.byref(h), _stream(stream)), "pdb_schedule_build")
    return Schedule(h, c, mode)


def pdb_schedule_levels(s: Schedule, stream=None) -> dict:
    """Borrowed device pointers (ints) of a LEVELS schedule's level, order and
    level_ptr arrays, and its number of levels (waits for the schedule)."""
    ptrs = [ctypes.c_void_p() for _ in range(3)]
    L = ctypes.c_int64()
    _check(load().pdb_schedule_levels(s.handle, *[ctypes.byref(p) for p in ptrs], ctypes.byref(L), _stream(stream)),
           "pdb_schedule_levels")
    return dict(level=ptrs[0].value, order=ptrs[1].value, level_ptr=ptrs[2].value, n_levels=L.value)


def pdb_schedule_ready(s: Schedule) -> dict:
    """Borrowed device pointers (ints) of the READY schedule's gate and records arrays."""
    ptrs = [ctypes.c_void_p() for _ in range(2)]
    _check(load().pdb_schedule_ready(s.handle, *[ctypes.byref(p) for p in ptrs]), "pdb_schedule_ready")
    return dict(gate=ptrs[0].value, records=ptrs[1].value)


def _opts(opts):
    if opts is None:
        return None
    if isinstance(opts, pdb_opts):
        return ctypes.byref(opts)
    kw = dict(opts)
    if kw.get("trace") is not None and not isinstance(kw["trace"], int):
        kw["trace"] = kw["trace"].data_ptr()     # a torch uint64/int64 tensor on the device
    return ctypes.byref(pdb_opts(**kw))


def pdb_sgd_epoch(X: Csr, y, c: Conflicts, s: Schedule, w, loss: int, eta: float, n_epochs: int, opts=None,
                  stream=None):
    """n_epochs of SGD over X in data order, serially equivalent (Algorithm 1,
    Theorem 2): w (float32, n_cols, on the device) is updated in place."""
    _check(load().pdb_sgd_epoch(ctypes.byref(X.struct), _ptr(y), c.handle, s.handle, _ptr(w), int(loss), float(eta),
                                int(n_epochs), _opts(opts), _stream(stream)), "pdb_sgd_epoch")


def pdb_ssp_epoch(X: Csr, y, c: Conflicts, s: Schedule, w, loss: int, eta: float, n_epochs: int, delay: int,
                  coef=None, opts=None, stream=None):
    """SGD with admissible delay (Section 7) under a READY schedule; opts may set
    ssp_gates to PDB_SSP_COUNT (default) or PDB_SSP_PREFIX.  delay = 0 is
    pdb_sgd_epoch's result bit for bit."""
    _check(load().pdb_ssp_epoch(ctypes.byref(X.struct), _ptr(y), c.handle, s.handle, _ptr(w), int(loss), float(eta),
                                int(n_epochs), int(delay), _ptr(coef), _opts(opts), _stream(stream)),
           "pdb_ssp_epoch")


def pdb_bsp_epoch(X: Csr, y, c: Conflicts, w, loss: int, eta: float, batch: int, n_epochs: int, opts=None,
                  stream=None):
    """The BSP comparison (Algorithm 2a): `batch` examples between barriers,
    margins at the batch-start weights, ordered per-feature sums."""
    _check(load().pdb_bsp_epoch(ctypes.byref(X.struct), _ptr(y), c.handle, _ptr(w), int(loss), float(eta),
                                int(batch), int(n_epochs), _opts(opts), _stream(stream)), "pdb_bsp_epoch")


class BspPlan:
    """Owns a pdb_bsp_plan handle (keeps its conflicts alive)."""

    def __init__(self, handle, conflicts, batch):
        self.handle, self.conflicts, self.batch = handle, conflicts, int(batch)
        self.n_batches = int(load().pdb_bsp_plan_batches(handle))

    def __del__(self):
        if getattr(self, "handle", None) and _lib is not None:
            _lib.pdb_bsp_plan_free(self.handle)
            self.handle = None


def pdb_bsp_plan_build(c: Conflicts, batch: int, stream=None) -> BspPlan:
    """The (batch, feature, example) order of c's pairs for the data-parallel
    BSP split of Algorithm 2a (synchronizes)."""
    h = ctypes.c_void_p()
    _check(load().pdb_bsp_plan_build(c.handle, int(batch), ctypes.byref(h), _stream(stream)), "pdb_bsp_plan_build")
    return BspPlan(h, c, min(int(batch), max(1, c.n_rows)) if c.n_rows > 0 else int(batch))


def pdb_bsp_coef(plan: BspPlan, X: Csr, y, w, loss: int, eta: float, row_begin: int, row_end: int, coef,
                 stream=None):
    """coef[i - row_begin] = eta * dloss/dm of rows [row_begin, row_end) at w
    (the rows lie inside one batch)."""
    _check(load().pdb_bsp_coef(plan.handle, ctypes.byref(X.struct), _ptr(y), _ptr(w), int(loss), float(eta),
                               int(row_begin), int(row_end), _ptr(coef), _stream(stream)), "pdb_bsp_coef")


def pdb_bsp_apply(plan: BspPlan, w, batch_index: int, coef, stream=None):
    """The write half of batch `batch_index` from all of its coefficients."""
    _check(load().pdb_bsp_apply(plan.handle, _ptr(w), int(batch_index), _ptr(coef), _stream(stream)),
           "pdb_bsp_apply")


def rank_rows(r0: int, r1: int, rank: int, world: int) -> tuple[int, int]:
    """The contiguous share of rows [r0, r1) that rank `rank` of `world` computes
    (the first (r1 - r0) % world ranks take one row more)."""
    n = r1 - r0
    q, extra = divmod(n, world)
    lo = r0 + rank * q + min(rank, extra)
    return lo, lo + q + (1 if rank < extra else 0)


def bsp_epoch_data_parallel(X: Csr, y, c: Conflicts, w, loss: int, eta: float, batch: int, n_epochs: int,
                            group=None, plan: BspPlan | None = None, ops=None, stream=None):
    """Algorithm 2a over the ranks of a torch.distributed group, each holding
    the whole data and a replica of w: per batch every rank computes the
    coefficients of its share of the rows (pdb_bsp_coef), the shares are
    all-gathered in rank order (= row order), and every rank applies the
    batch (pdb_bsp_apply).  Without an initialized process group it runs on
    one rank.  The result equals pdb_bsp_epoch's bit for bit.

    `ops` replaces the three library calls (coef, apply, all_gather) with
    callables of the same meaning; the CPU tests use it to check the
    partitioning without a GPU."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group) if dist.is_available() and dist.is_initialized() else 1
    rank = dist.get_rank(group) if world > 1 else 0
    if ops is None:
        plan = plan or pdb_bsp_plan_build(c, batch, stream)
        n_batches, B = plan.n_batches, plan.batch

        def coef_fn(r0, r1, out):
            pdb_bsp_coef(plan, X, y, w, loss, eta, r0, r1, out, stream)

        def apply_fn(b, coef):
            pdb_bsp_apply(plan, w, b, coef, stream)

        def gather_fn(parts, mine):
            if world == 1:
                return
            if dist.get_backend(group) == "nccl":
                dist.all_gather(parts, mine, group=group)
            else:                              # gloo: host tensors
                host = [torch.empty(p.numel(), dtype=p.dtype) for p in parts]
                dist.all_gather(host, mine.cpu(), group=group)
                for p, h in zip(parts, host):
                    p.copy_(h)
        device = w.device
    else:
        coef_fn, apply_fn, gather_fn = ops["coef"], ops["apply"], ops["gather"]
        n_batches, B = ops["n_batches"], ops["batch"]
        device = ops.get("device", "cpu")
    n_rows = X.struct.n_rows if hasattr(X, "struct") else ops["n_rows"]
    coef = torch.empty(max(B, 1), dtype=torch.float32, device=device)
    for _ in range(n_epochs):
        for b in range(n_batches):
            r0, r1 = b * B, min(n_rows, (b + 1) * B)
            bounds = [rank_rows(r0, r1, r, world) for r in range(world)]
            # one slice per rank, padded to the longest so that every all_gather part has one size
            width = max(hi - lo for lo, hi in bounds)
            if world == 1:
                coef_fn(r0, r1, coef[: r1 - r0])
                apply_fn(b, coef[: r1 - r0])
                continue
            parts = [torch.zeros(width, dtype=torch.float32, device=device) for _ in range(world)]
            lo, hi = bounds[rank]
            coef_fn(lo, hi, parts[rank][: hi - lo])
            gather_fn(parts, parts[rank])
            for r, (l2, h2) in enumerate(bounds):
                coef[l2 - r0: h2 - r0].copy_(parts[r][: h2 - l2])
            apply_fn(b, coef[: r1 - r0])


def pdb_sgd_epoch_ready_noalloc(X: Csr, y, gate_ptr: int, w, loss: int, eta: float, n_epochs: int,
                                stream=None) -> int:
    """READY-schedule SGD epochs that allocate no device memory (scratch is a
    fixed array inside the library, up to NOALLOC_MAX_COLS features).  For
    callers that cannot let a library allocate while they train, e.g. a
    server whose own memory pool owns the whole device.  Synchronizes the
    stream and returns the status code (PDB_OK on success)."""
    return int(load().pdb_sgd_epoch_ready_noalloc(ctypes.byref(X.struct), _ptr(y), ctypes.c_void_p(gate_ptr), _ptr(w),
                                                  int(loss), float(eta), int(n_epochs), _stream(stream)))


def pdb_status(c: Conflicts, stream=None) -> int:
    """Synchronize the stream and return the first error a kernel recorded in c
    (PDB_OK when none)."""
    return int(load().pdb_status(c.handle, _stream(stream)))


def pdb_get_stats(c: Conflicts, s: Schedule | None = None) -> dict:
    """Sizes, level counts and CUDA-event timings of the last calls on c (and s)
    as a dict; synchronizes the device."""
    st = pdb_stats()
    _check(load().pdb_get_stats(c.handle, None if s is None else s.handle, ctypes.byref(st)), "pdb_get_stats")
    return st.as_dict()


def pdb_memcpy(dst_ptr: int, src_ptr: int, nbytes: int, stream=None):
    """Stream-ordered copy between device or host pointers (ints)."""
    _check(load().pdb_memcpy(ctypes.c_void_p(dst_ptr), ctypes.c_void_p(src_ptr), int(nbytes), _stream(stream)),
           "pdb_memcpy")


def pdb_eval_grad(m, y, out, loss: int, stream=None):
    """out = the library's device loss derivative at margins m and labels y
    (float32 device tensors of one length)."""
    _check(load().pdb_eval_grad(_ptr(m), _ptr(y), _ptr(out), m.numel(), int(loss), _stream(stream)), "pdb_eval_grad")


def pdb_eval_expf(x, out, stream=None):
    """out = the library's device exponential of x (float32 tensors), for tests."""
    _check(load().pdb_eval_expf(_ptr(x), _ptr(out), x.numel(), _stream(stream)), "pdb_eval_expf")


def pdb_launch_count() -> int:
    """Kernels this process has launched through the library so far."""
    return int(load().pdb_launch_count())


def pdb_strerror(code: int) -> str:
    return _strerror(code)


def device_array(ptr: int, n: int, dtype, stream=None):
    """Copy n elements of a borrowed device array into a new torch tensor."""
    import torch
    out = torch.empty(n, dtype=dtype, device="cuda")
    if n:
        pdb_memcpy(out.data_ptr(), ptr, n * out.element_size(), stream)
    return out


def check_status(c: Conflicts, stream=None):
    """Synchronize and raise PdbError if a kernel recorded an error in c."""
    rc = pdb_status(c, stream)
    if rc != PDB_OK:
        raise PdbError(rc, "device status")
