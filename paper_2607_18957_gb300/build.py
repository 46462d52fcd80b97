"""Builds libcfa.so in-tree: the unpack kernels and runtime for sm_103a plus the host plan builder.

    python -m paper_2607_18957_gb300.build            # or __graft_entry__.build()

Translation units compile in parallel; the result lands next to this file so the Python
binding (and the driver's loaded-library check) finds it in the tree.
"""
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libcfa.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
CU_SOURCES = ["cfa_unpack.cu", "cfa_bulk.cu", "cfa_runtime.cu", "cfa_noalloc.cu"]
C_SOURCES = ["cfa_plan.c", "cfa_files.c"]


def _nvcc():
    cand = os.environ.get("NVCC") or shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    return cand


def _sources():
    return [os.path.join(CSRC, f) for f in CU_SOURCES + C_SOURCES +
            ["cfa_internal.h", "cfa_pool.h", "cfa_device.cuh"]] + \
        [os.path.join(INCLUDE, "cfa.h")]


def up_to_date():
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(s) <= t for s in _sources())


def build(force=False, verbose=False, ptxas_info=False):
    """Compiles and links libcfa.so; returns its path."""
    if not force and up_to_date():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    nvcc = _nvcc()
    inc = ["-I", INCLUDE, "-I", CSRC]
    jobs = []
    objs = []
    for f in CU_SOURCES:
        obj = os.path.join(BUILD, f + ".o")
        cmd = [nvcc, *ARCH, "-lineinfo", "-O3", "-std=c++17", "-Xcompiler", "-fPIC",
               "-Xcompiler", "-Wall", *inc, "-c", os.path.join(CSRC, f), "-o", obj]
        if ptxas_info:
            cmd.insert(1, "-Xptxas=-v")
        jobs.append(cmd)
        objs.append(obj)
    for f in C_SOURCES:
        obj = os.path.join(BUILD, f + ".o")
        jobs.append(["gcc", "-O2", "-std=c11", "-fPIC", "-Wall", *inc, "-c",
                     os.path.join(CSRC, f), "-o", obj])
        objs.append(obj)
    procs = [(cmd, subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT,
                                    text=True)) for cmd in jobs]
    failed = []
    for cmd, pr in procs:
        out, _ = pr.communicate()
        if verbose or ptxas_info or pr.returncode:
            sys.stderr.write(out)
        if pr.returncode:
            failed.append(" ".join(cmd))
    if failed:
        raise RuntimeError("compilation failed:\n" + "\n".join(failed))
    tmp = LIB + ".tmp"
    link = [nvcc, *ARCH, "-shared", "-Xcompiler", "-fPIC", *objs, "-o", tmp, "-lpthread"]
    r = subprocess.run(link, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if r.returncode:
        sys.stderr.write(r.stdout)
        raise RuntimeError("link failed: " + " ".join(link))
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose=True, ptxas_info="--ptxas" in sys.argv)
    print(LIB)
