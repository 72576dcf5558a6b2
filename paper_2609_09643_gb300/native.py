"""In-tree build of libunison.so for sm_103a (nvcc, one object per source,
compiled in parallel, then linked).  Output: paper_2609_09643_gb300/_build/.

build_debug() makes a separate test library of the ranking call with the
debug hooks of include/unison_debug.h compiled in (short bounded waits that
a test can make run out); the default library never contains them."""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(PKG, "csrc")
OUT = os.path.join(PKG, "_build")
LIB = os.path.join(OUT, "libunison.so")
SOURCES = ["trace.cu", "replay.cu", "rank.cu", "profile.cu", "selftest.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2"]


def nvcc() -> str:
    p = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(p):
        raise RuntimeError("nvcc not found")
    return p


def _stale(obj: str, src: str) -> bool:
    if not os.path.exists(obj):
        return True
    deps = [src, os.path.join(CSRC, "common.cuh"), os.path.join(CSRC, "profile.cuh"),
            os.path.join(PKG, "..", "include", "unison.h")]
    return any(os.path.getmtime(d) > os.path.getmtime(obj) for d in deps if os.path.exists(d))


def build(force: bool = False, verbose: bool = False, out: str = OUT, lib: str = LIB,
          sources=SOURCES, extra=()) -> str:
    os.makedirs(out, exist_ok=True)
    cc = nvcc()
    jobs = []
    for s in sources:
        src = os.path.join(CSRC, s)
        obj = os.path.join(out, s.replace(".cu", ".o"))
        if force or _stale(obj, src):
            jobs.append([cc, *ARCH, *FLAGS, *extra, "-c", src, "-o", obj])

    def run(cmd):
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("nvcc failed:\n" + " ".join(cmd) + "\n" + r.stdout + r.stderr)
        if verbose:
            print(r.stdout + r.stderr)

    with cf.ThreadPoolExecutor(max_workers=len(sources)) as ex:
        list(ex.map(run, jobs))
    objs = [os.path.join(out, s.replace(".cu", ".o")) for s in sources]
    if force or jobs or not os.path.exists(lib):
        tmp = lib + f".tmp{os.getpid()}"
        run([cc, *ARCH, "-shared", "-o", tmp, *objs])
        os.replace(tmp, lib)
    return lib


OUT_DEBUG = os.path.join(PKG, "_build_debug")
LIB_DEBUG = os.path.join(OUT_DEBUG, "libunison_rank_debug.so")
DEBUG_SOURCES = ["trace.cu", "rank.cu", "profile.cu", "selftest.cu"]


def build_debug(force: bool = False) -> str:
    """The ranking call with the test hooks of include/unison_debug.h."""
    return build(force=force, out=OUT_DEBUG, lib=LIB_DEBUG, sources=DEBUG_SOURCES,
                 extra=("-DUNISON_DEBUG_HOOKS",))
