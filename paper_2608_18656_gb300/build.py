"""Builds libfav.so (the C-ABI library) in-tree with nvcc for sm_103a.

Each CUDA translation unit is compiled in parallel, then linked with the static CUDA runtime
into ``paper_2608_18656_gb300/libfav.so``.  Objects go to ``paper_2608_18656_gb300/_build``.
"""
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libfav.so")
SOURCES = ["fav_api.cu", "fav_simt.cu", "fav_decode.cu", "fav_prefill.cu", "fav_prefill_pair.cu",
           "fav_v16.cu", "fav_noalloc.cu", "fav_nonflash.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc():
    home = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    path = os.path.join(home, "bin", "nvcc")
    return path if os.path.exists(path) else "nvcc"


def compile_one(src, extra=(), objdir=BUILD):
    obj = os.path.join(objdir, os.path.splitext(src)[0] + ".o")
    cmd = [nvcc(), *ARCH, "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
           "-Xcompiler", "-fvisibility=hidden", "-I", os.path.join(HERE, "..", "include"),
           *extra, "-c", os.path.join(CSRC, src), "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("nvcc failed for %s:\n%s%s" % (src, r.stdout, r.stderr))
    return obj, r.stderr


def build(verbose=False, extra=(), lib=LIB, objdir=BUILD):
    """Compiles every translation unit (with the extra nvcc flags) into objdir and links lib."""
    os.makedirs(objdir, exist_ok=True)
    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        results = list(ex.map(lambda s: compile_one(s, extra, objdir), SOURCES))
    if verbose:
        for _, log in results:
            if log:
                sys.stderr.write(log)
    tmp = lib + ".tmp.%d" % os.getpid()
    cmd = [nvcc(), *ARCH, "-shared", "-cudart", "static", "-ldl", "-o", tmp] + [o for o, _ in results]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("link failed:\n%s%s" % (r.stdout, r.stderr))
    os.replace(tmp, lib)
    return lib


# The self-checking variant (-DFAV_DEBUG_CHECKS: shared-memory bounds, TMA destination
# alignment, global indices, per-role unit and tile totals; a violation prints, sets device
# status 6 and skips the access).  Load it with FAV_LIBRARY=<DEBUG_LIB> in the environment.
DEBUG_LIB = os.path.join(HERE, "libfav_debug.so")
DEBUG_BUILD = os.path.join(HERE, "_build_debug")


def build_debug(verbose=False):
    return build(verbose, ("-DFAV_DEBUG_CHECKS",), DEBUG_LIB, DEBUG_BUILD)


if __name__ == "__main__":
    extra = sys.argv[1:]
    print(build(verbose=True, extra=extra))
