"""The C ABI library builds for sm_103a, loads without a GPU, and exports
every function include/pdb.h declares (no compute calls here)."""
import ctypes
import os
import re
import subprocess

import pytest

import paper_1508_00703_gb300 as pdb

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names |= set(re.findall(r"\b(pdb_\w+)\s*\(", text))
    return names


def test_library_exports_every_declared_symbol():
    path = pdb.build()
    out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True, text=True, check=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    declared = _declared()
    assert declared, "no declarations found"
    assert declared <= exported, declared - exported
    assert set(pdb.EXPORTS) == declared


def test_library_loads_and_resolves():
    lib = ctypes.CDLL(pdb.build())
    for name in _declared():
        assert getattr(lib, name) is not None


def test_strerror_without_gpu():
    lib = pdb.load()
    assert lib.pdb_strerror(pdb.PDB_EDUP).decode().startswith("feature id repeated")
    assert lib.pdb_strerror(0).decode() == "ok"


def test_host_argument_errors_need_no_gpu():
    # argument checks happen on the host before any CUDA call
    lib = pdb.load()
    h = ctypes.c_void_p()
    assert lib.pdb_build_conflicts(None, ctypes.byref(h), None) == pdb.PDB_EINVAL
    bad = pdb.pdb_csr(-1, 4, 0, None, None, None)
    assert lib.pdb_build_conflicts(ctypes.byref(bad), ctypes.byref(h), None) == pdb.PDB_EINVAL
    big = pdb.pdb_csr(1, 4, 1 << 31, ctypes.c_void_p(8), ctypes.c_void_p(8), None)
    assert lib.pdb_build_conflicts(ctypes.byref(big), ctypes.byref(h), None) == pdb.PDB_EINVAL
    assert lib.pdb_schedule_build(None, 0, ctypes.byref(h), None) == pdb.PDB_EINVAL


def test_nvcc_targets_sm_103a_only():
    assert pdb.ARCH == "-gencode=arch=compute_103a,code=sm_103a"
    assert "-fmad=false" in pdb.NVCC_FLAGS and "--use_fast_math" not in pdb.NVCC_FLAGS


def test_graft_entry_build():
    import __graft_entry__
    __graft_entry__.build()


def test_struct_layouts_match_the_header(tmp_path):
    # the binding's ctypes structs against the C compiler's view of include/pdb.h
    structs = {"pdb_csr": pdb.pdb_csr, "pdb_opts": pdb.pdb_opts, "pdb_stats": pdb.pdb_stats}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "pdb.h"', "int main(void) {"]
    for name, cls in structs.items():
        lines.append(f'printf("{name} size %zu\\n", sizeof({name}));')
        for field, _ in cls._fields_:
            lines.append(f'printf("{name} {field} %zu\\n", offsetof({name}, {field}));')
    lines += ["return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c11", f"-I{os.path.join(ROOT, 'include')}", str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split("\n")
    got = {tuple(ln.split()[:2]): int(ln.split()[2]) for ln in out if ln.strip()}
    for name, cls in structs.items():
        assert got[(name, "size")] == ctypes.sizeof(cls), name
        for field, _ in cls._fields_:
            assert got[(name, field)] == getattr(cls, field).offset, (name, field)


def test_constants_match_the_header(tmp_path):
    # every PDB_* value the header defines (error codes, enum members) as the
    # C compiler sees it, against the binding's constant of the same name
    text = open(os.path.join(ROOT, "include", "pdb.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = set(re.findall(r"#define\s+(PDB_[A-Z_]+)\s+\(?-?\d+\)?", text))
    for body in re.findall(r"typedef\s+enum\s*\{(.*?)\}", text, flags=re.S):
        names |= set(re.findall(r"\b(PDB_[A-Z_]+)\s*=", body))
    assert {"PDB_OK", "PDB_EDUP", "PDB_SCHED_WINDOW", "PDB_SSP_PREFIX", "PDB_LOSS_HINGE"} <= names
    lines = ['#include <stdio.h>', '#include "pdb.h"', "int main(void) {"]
    lines += [f'printf("{n} %lld\\n", (long long)({n}));' for n in sorted(names)]
    lines += ["return 0;", "}"]
    src = tmp_path / "consts.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "consts"
    subprocess.run(["gcc", "-std=c11", f"-I{os.path.join(ROOT, 'include')}", str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split("\n")
    got = {ln.split()[0]: int(ln.split()[1]) for ln in out if ln.strip()}
    assert set(got) == names
    for n, v in got.items():
        assert getattr(pdb, n) == v, n


def test_every_compute_call_cites_its_passage():
    # the comment above each compute call's declaration names the passage of
    # the paper that defines the operation
    text = open(os.path.join(ROOT, "include", "pdb.h")).read()
    cite = re.compile(r"Section \d|Definitions? \d|Algorithm \d|Theorem \d")
    found = {}
    for m in re.finditer(r"(/\*(?:(?!\*/).)*\*/)\s*int\s+(pdb_\w+)\s*\(", text, flags=re.S):
        found[m.group(2)] = bool(cite.search(m.group(1)))
    compute = ["pdb_build_conflicts", "pdb_conflicts_arrays", "pdb_schedule_build", "pdb_schedule_levels",
               "pdb_schedule_ready", "pdb_sgd_epoch", "pdb_ssp_epoch", "pdb_bsp_epoch", "pdb_sgd_epoch_ready_noalloc"]
    assert all(found.get(n) for n in compute), {n: found.get(n) for n in compute}
