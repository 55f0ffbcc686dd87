"""Build ``libgoldy.so`` (the C-ABI library) in-tree for sm_103a.

Plain nvcc/g++ invocations, one object per translation unit, compiled in
parallel: ``planner.cpp`` (host C++), ``runtime.cu`` (launch manager),
``noalloc.cu`` (the entry point with a compiled-in scratch array) and
``kernels.cu`` once per GO-Kernel kind (``-DGOLDY_KIND=k``).  Objects go to
``_build/`` next to this file and the library to
``paper_2409_02227_gb300/libgoldy.so``; both are git-ignored.  A rebuild is
skipped when the library is newer than every source and header.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libgoldy.so")
NUM_KINDS = 11

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def _nvcc() -> str:
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found")
    return cand


def _sources_mtime() -> float:
    files = glob.glob(os.path.join(CSRC, "*")) + glob.glob(os.path.join(INCLUDE, "*.h"))
    files.append(os.path.abspath(__file__))
    return max(os.path.getmtime(f) for f in files)


def _jobs(ptxas_verbose: bool):
    nvcc = _nvcc()
    common = ["-std=c++17", "-O3", "-Xcompiler", "-fPIC", "-I", CSRC, "-I", INCLUDE]
    cu = [nvcc] + common + ARCH + ["-lineinfo"]
    if ptxas_verbose:
        cu += ["-Xptxas", "-v"]
    jobs = []
    jobs.append(("planner", ["g++", "-std=c++17", "-O2", "-ffp-contract=off", "-fPIC", "-Wall", "-I", CSRC, "-I", INCLUDE,
                             "-c", os.path.join(CSRC, "planner.cpp")]))
    jobs.append(("runtime", cu + ["-c", os.path.join(CSRC, "runtime.cu")]))
    jobs.append(("noalloc", cu + ["-c", os.path.join(CSRC, "noalloc.cu")]))
    jobs.append(("ewise", cu + ["-c", os.path.join(CSRC, "ewise.cu")]))
    for k in range(NUM_KINDS):
        jobs.append((f"kernels_k{k}", cu + [f"-DGOLDY_KIND={k}", "-c", os.path.join(CSRC, "kernels.cu")]))
    return jobs


def build(force: bool = False, verbose: bool = False, ptxas_verbose: bool = False) -> str:
    """Compile and link; returns the library path."""
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= _sources_mtime():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    jobs = _jobs(ptxas_verbose)

    def run(job):
        name, cmd = job
        obj = os.path.join(BUILD, name + ".o")
        proc = subprocess.run(cmd + ["-o", obj], capture_output=True, text=True)
        return name, obj, proc

    workers = max(1, min(len(jobs), os.cpu_count() or 4))
    objs = []
    errors = []
    with cf.ThreadPoolExecutor(workers) as ex:
        for name, obj, proc in ex.map(run, jobs):
            if verbose or ptxas_verbose:
                sys.stderr.write(proc.stdout + proc.stderr)
            if proc.returncode != 0:
                errors.append(f"--- {name} ---\n{proc.stdout}{proc.stderr}")
            objs.append(obj)
    if errors:
        raise RuntimeError("build failed:\n" + "\n".join(errors))
    tmp = LIB + f".tmp{os.getpid()}"
    link = [_nvcc(), "-shared"] + ARCH + objs + ["-o", tmp]
    proc = subprocess.run(link, capture_output=True, text=True)
    if proc.returncode != 0:
        raise RuntimeError("link failed:\n" + proc.stdout + proc.stderr)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv,
                ptxas_verbose="--ptxas" in sys.argv))
