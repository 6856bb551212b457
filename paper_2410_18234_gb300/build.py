"""Build the verification library in-tree: paper_2410_18234_gb300/_lib/libmds.so.

nvcc compiles every translation unit for sm_103a only (GB300), in parallel,
and links one shared library with the C ABI declared in include/mds.h.
"""
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
OUT_DIR = os.path.join(HERE, "_lib")
LIB = os.path.join(OUT_DIR, "libmds.so")
BUILD_DIR = os.path.join(ROOT, "_build")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-cudart", "static", "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I" + os.path.join(ROOT, "include")]
SOURCES = ["mds_kernel.cu", "mds_flow.cu", "mds_topk.cu", "mds_api.cu", "mds_noalloc.cu"]


def nvcc():
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", "nvcc"):
        if cand and (os.path.isabs(cand) and os.path.exists(cand) or not os.path.isabs(cand)):
            return cand
    return "nvcc"


TIMERS_LIB = os.path.join(OUT_DIR, "libmds_timers.so")


def _compile(src, extra=(), tag=""):
    obj = os.path.join(BUILD_DIR, tag + os.path.splitext(src)[0] + ".o")
    cmd = [nvcc(), *ARCH, *FLAGS, *extra, "-c", os.path.join(CSRC, src), "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stderr}")
    return obj


def build(verbose=False, timers=False):
    """Build libmds.so; with timers=True the instrumented variant
    libmds_timers.so (phase counters of the slice-dataflow engine, read with
    mds_phase_timers), which the binding loads when MDS_LIBRARY names it."""
    os.makedirs(OUT_DIR, exist_ok=True)
    os.makedirs(BUILD_DIR, exist_ok=True)
    extra = ("-DMDS_PHASE_TIMERS",) if timers else ()
    tag = "timers_" if timers else ""
    lib = TIMERS_LIB if timers else LIB
    def obj(src):
        # only the dataflow engine carries the timers: the instrumented build
        # reuses the other objects of the default build when they exist
        plain = os.path.join(BUILD_DIR, os.path.splitext(src)[0] + ".o")
        if timers and src != "mds_flow.cu" and os.path.exists(plain):
            return plain
        return _compile(src, extra if src == "mds_flow.cu" else (), tag if src == "mds_flow.cu" else "")

    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(obj, SOURCES))
    cmd = [nvcc(), *ARCH, "-shared", "-cudart", "static", "-o", lib, *objs]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stderr}")
    if verbose:
        print(f"built {lib}")
    return lib


if __name__ == "__main__":
    build(verbose=True, timers="--timers" in sys.argv)
    sys.exit(0)
