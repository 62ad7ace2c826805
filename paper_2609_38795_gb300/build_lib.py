"""Build the two libraries in-tree, every .cu compiled for sm_103a in parallel, then linked:

  _lib/libalr.so          csrc/*.cu: the C ABI (include/alr.h) and the single-CTA kernel forms;
  _lib/libalr_cluster.so  csrc_cluster/*.cu: the kernel forms that share operand tiles across
                          the CTAs of a cluster (TMA multicast, CTA pairs), which libalr.so
                          loads in single-process runs only.

A process that is one rank of several (WORLD_SIZE > 1) builds libalr.so alone.

Usage:  python -m paper_2609_38795_gb300.build_lib [--force] [-v]
"""

from __future__ import annotations

import concurrent.futures as cf
import fcntl
import hashlib
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
CSRC_CLUSTER = os.path.join(PKG, "csrc_cluster")
INCLUDE = os.path.join(ROOT, "include")
OUT_DIR = os.path.join(PKG, "_lib")
LIB = os.path.join(OUT_DIR, "libalr.so")
LIB_CLUSTER = os.path.join(OUT_DIR, "libalr_cluster.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
              "-I", INCLUDE, "-I", CSRC]

# target name -> (library, source directory, extra include directories, extra link flags)
TARGETS = {
    "alr": (LIB, CSRC, [], ["-ldl"]),
    "cluster": (LIB_CLUSTER, CSRC_CLUSTER, ["-I", CSRC_CLUSTER], []),
}


def multi_rank_process() -> bool:
    try:
        return int(os.environ.get("WORLD_SIZE", "1")) > 1
    except ValueError:
        return False


def _nvcc():
    for c in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", shutil.which("nvcc")):
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found (set NVCC or install the CUDA toolkit)")


def _sources(src_dir):
    return sorted(os.path.join(src_dir, f) for f in os.listdir(src_dir) if f.endswith(".cu"))


def _fingerprint(nvcc):
    """Hash of every source and header of both libraries (the cluster library includes the
    main one's headers), the flags, the compiler and the host architecture."""
    h = hashlib.sha256()
    files = [os.path.join(d, f) for d in (CSRC, CSRC_CLUSTER) for f in sorted(os.listdir(d))
             if os.path.isfile(os.path.join(d, f))]
    for p in files + [os.path.join(INCLUDE, "alr.h")]:
        with open(p, "rb") as fh:
            h.update(os.path.relpath(p, ROOT).encode())
            h.update(fh.read())
    h.update(" ".join(ARCH + NVCC_FLAGS + [nvcc, os.uname().machine]).encode())
    return h.hexdigest()


def build(force: bool = False, verbose: bool = False, extra_flags=()) -> str:
    """Compile and link libalr.so and (unless this process is one rank of several)
    libalr_cluster.so; returns the path of libalr.so.  Skips a library whose sources, flags and
    host architecture are unchanged since it was built."""
    nvcc = _nvcc()
    os.makedirs(OUT_DIR, exist_ok=True)
    fp = _fingerprint(nvcc) + "|" + " ".join(extra_flags)
    names = ["alr"] if multi_rank_process() else ["alr", "cluster"]

    def stale():
        out = []
        for n in names:
            lib = TARGETS[n][0]
            stamp = lib[:-3] + ".stamp"
            if force or not (os.path.exists(lib) and os.path.exists(stamp)):
                out.append(n)
                continue
            with open(stamp) as f:
                if f.read() != fp:
                    out.append(n)
        return out

    if not stale():
        return LIB
    # One builder at a time (the ranks of a torchrun launch all call build()); whoever gets
    # the lock second finds the libraries built and up to date.
    with open(os.path.join(OUT_DIR, "build.lock"), "w") as lock:
        fcntl.flock(lock, fcntl.LOCK_EX)
        todo = stale()
        if todo:
            _build_locked(nvcc, todo, fp, verbose, extra_flags)
    return LIB


def _build_locked(nvcc, names, fp, verbose, extra_flags):
    def compile_one(job):
        name, src = job
        obj_dir = os.path.join(OUT_DIR, "obj_" + name)
        os.makedirs(obj_dir, exist_ok=True)
        obj = os.path.join(obj_dir, os.path.basename(src)[:-3] + ".o")
        cmd = [nvcc, *ARCH, *NVCC_FLAGS, *TARGETS[name][2], *extra_flags, "-c", src, "-o", obj]
        if verbose:
            print(" ".join(cmd), flush=True)
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            print(r.stdout + r.stderr, flush=True)
        return name, obj

    jobs = [(n, s) for n in names for s in _sources(TARGETS[n][1])]
    with cf.ThreadPoolExecutor(max_workers=min(len(jobs), os.cpu_count() or 4)) as ex:
        done = list(ex.map(compile_one, jobs))
    for n in names:
        lib, _, _, link_flags = TARGETS[n]
        objs = [o for m, o in done if m == n]
        tmp = lib + ".tmp"
        cmd = [nvcc, *ARCH, "-shared", "-o", tmp, *objs, *link_flags]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link of {os.path.basename(lib)} failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, lib)
        with open(lib[:-3] + ".stamp", "w") as f:
            f.write(fp)


if __name__ == "__main__":
    args = sys.argv[1:]
    print(build(force="--force" in args, verbose="-v" in args))
