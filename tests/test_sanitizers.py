"""The oracle and the input generator under AddressSanitizer and
UndefinedBehaviorSanitizer, on the CPU.

A mistake of memory or of undefined behaviour in the C code that pins the
GPU path (an out-of-range index, a signed overflow, a misaligned access)
could pass every value test by luck on one compiler.  Here both libraries are
rebuilt with -fsanitize=address,undefined (UB aborts), loaded in a child
Python with the sanitizer runtimes preloaded, and run on problems of every
shape: the workloads at reduced sizes (ids at their full ranges), rows longer
than 256 ids, empty rows, no rows, one feature, dense rows, saturated
exponentials."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SCRIPT = r"""
import sys
import numpy as np
import oracle, synthdata
oracle.build = lambda: sys.argv[1]
synthdata.build = lambda: sys.argv[2]
from tests import _cases as C
problems = [synthdata.generate(n, **kw) for n, kw in [
    ("tiny", {}), ("zipf-1m", dict(n_rows=30000)), ("ctr", dict(n_rows=20000)),
    ("low-conflict", dict(n_rows=3000)), ("deep-chain", dict(n_rows=2000)), ("dense-lr", dict(n_rows=300)),
    ("tiny", dict(n_rows=1500, n_cols=5000, k=300, k_lo=200)), ("tiny", dict(n_rows=5001, n_cols=3000, k=24, k_lo=0))]]
problems += [C.edge(n) for n in C.EDGES]
for p in problems:
    assert oracle.validate(p) == oracle.OK
    ch = oracle.chains(p)
    lv, L = oracle.levels(p)
    oracle.level_order(lv, L)
    w = oracle.sgd(p)
    wb = oracle.bsp(p, 64)
    assert np.all(np.isfinite(w)) and np.all(np.isfinite(wb))
    if p.nnz and p.n_rows <= 400:
        assert np.array_equal(oracle.levels_bruteforce(p), lv)
x = np.linspace(-120.0, 100.0, 200001, dtype=np.float32)
oracle.expf(x)
# malformed inputs take the validation's error paths
bad = synthdata.from_arrays([0, 2, 1], [0, 1], None, [1.0, 1.0], n_cols=3)
assert oracle.validate(bad) != oracle.OK
dup = synthdata.from_arrays([0, 2], [1, 1], None, [1.0], n_cols=3)
assert oracle.validate(dup) == oracle.DUP
rng = synthdata.from_arrays([0, 1], [7], None, [1.0], n_cols=3)
assert oracle.validate(rng) == oracle.BAD_COL
print("sanitized run ok")
"""


def _runtime(name):
    path = subprocess.run(["gcc", f"-print-file-name={name}"], capture_output=True, text=True).stdout.strip()
    return path if os.path.isabs(path) and os.path.exists(path) else None


FLAGS = ["-O1", "-g", "-std=c11", "-shared", "-fPIC", "-ffp-contract=off", "-fno-fast-math",
         "-fsanitize=address,undefined", "-fno-sanitize-recover=undefined", "-fno-omit-frame-pointer"]


def _sanitized_run(tmp_path, oracle_src, script):
    asan, ubsan = _runtime("libasan.so"), _runtime("libubsan.so")
    if not (asan and ubsan):
        pytest.skip("gcc has no sanitizer runtime here")
    src = tmp_path / "pdb_oracle.c"
    src.write_text(oracle_src)
    lib_o, lib_s = tmp_path / "liboracle_san.so", tmp_path / "libsynth_san.so"
    subprocess.run(["gcc", *FLAGS, "-o", str(lib_o), str(src), "-lm"], check=True)
    subprocess.run(["gcc", *FLAGS, "-pthread", "-o", str(lib_s), os.path.join(ROOT, "synthdata", "synth.c"), "-lm"],
                   check=True)
    env = dict(os.environ, LD_PRELOAD=f"{asan}:{ubsan}", ASAN_OPTIONS="detect_leaks=0:halt_on_error=1",
               UBSAN_OPTIONS="print_stacktrace=1:halt_on_error=1", PYTHONPATH=ROOT)
    return subprocess.run([sys.executable, "-c", script, str(lib_o), str(lib_s)], capture_output=True, text=True,
                          env=env, cwd=ROOT, timeout=600)


def _oracle_source():
    return open(os.path.join(ROOT, "oracle", "pdb_oracle.c")).read()


def test_oracle_and_generator_under_asan_and_ubsan(tmp_path):
    out = _sanitized_run(tmp_path, _oracle_source(), SCRIPT)
    assert out.returncode == 0, out.stderr[-4000:]
    assert "runtime error" not in out.stderr and "AddressSanitizer" not in out.stderr, out.stderr[-4000:]
    assert "sanitized run ok" in out.stdout


def test_the_sanitized_run_catches_a_planted_overflow(tmp_path):
    # planted in a copy of the oracle: the chain builder initialises one
    # entry past its last-occurrence table
    src = _oracle_source()
    old = "for (int64_t j = 0; j < n_cols; ++j) last[j] = -1;"
    assert src.count(old) == 1
    script = ("import sys, oracle, synthdata\n"
              "oracle.build = lambda: sys.argv[1]\nsynthdata.build = lambda: sys.argv[2]\n"
              "oracle.chains(synthdata.generate('tiny', n_rows=50))\n")
    planted = src.replace(old, old.replace("j < n_cols", "j <= n_cols"))
    line = planted[:planted.index(old.replace("j < n_cols", "j <= n_cols"))].count("\n") + 1
    out = _sanitized_run(tmp_path, planted, script)
    assert out.returncode != 0, out.stderr[-2000:]
    assert "runtime error" in out.stderr or "heap-buffer-overflow" in out.stderr, out.stderr[-2000:]
    assert f"pdb_oracle.c:{line}" in out.stderr, out.stderr[-2000:]
