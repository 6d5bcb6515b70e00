"""Build libdkv.so (the C ABI of include/dkv.h) in-tree for sm_103a with nvcc.

Each .cu file compiles in its own nvcc process (in parallel), then nvcc links a
shared library with the CUDA runtime linked statically. Only one -gencode:
compute_103a -> sm_103a (GB300).

build_library(debug=True) builds libdkv_debug.so instead: the same sources
with -DDKV_DEBUG, whose kernels check the indices and offsets they read and set
DKV_DEV_BOUNDS in the plan's status word (the stand-in for a memory checker).
"""
import fcntl
import glob
import os
import subprocess
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIB = os.path.join(PKG, "libdkv.so")
OBJDIR = os.path.join(PKG, "_build")
LIB_DEBUG = os.path.join(PKG, "libdkv_debug.so")
OBJDIR_DEBUG = os.path.join(PKG, "_build_debug")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC,-O2", "-I" + INCLUDE, "-I" + CSRC]


def _nvcc():
    home = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    cand = os.path.join(home, "bin", "nvcc")
    return cand if os.path.exists(cand) else "nvcc"


def sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + [os.path.join(INCLUDE, "dkv.h"), __file__]


def up_to_date(lib=LIB):
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(p) <= t for p in _deps())


def build_library(force=False, verbose=False, extra_flags=(), debug=False):
    """Compile every csrc/*.cu and link libdkv.so (libdkv_debug.so with
    debug=True). Returns the library path.

    Processes that build at the same time (one per rank under torchrun, or test
    workers) serialise on a lock file; the ones that wait find the library up to
    date and return it."""
    lib, objdir = (LIB_DEBUG, OBJDIR_DEBUG) if debug else (LIB, OBJDIR)
    flags = (*extra_flags, "-DDKV_DEBUG") if debug else tuple(extra_flags)
    if not force and up_to_date(lib):
        return lib
    os.makedirs(objdir, exist_ok=True)
    with open(os.path.join(objdir, ".lock"), "w") as lock:
        fcntl.flock(lock, fcntl.LOCK_EX)
        try:
            if not force and up_to_date(lib):
                return lib
            return _build_locked(verbose, flags, lib, objdir)
        finally:
            fcntl.flock(lock, fcntl.LOCK_UN)


def _build_locked(verbose, extra_flags, lib, objdir):
    nvcc = _nvcc()

    def compile_one(src):
        obj = os.path.join(objdir, os.path.basename(src)[:-3] + ".o")
        cmd = [nvcc, *ARCH, *NVCC_FLAGS, *extra_flags, "-c", src, "-o", obj]
        if verbose:
            print(" ".join(cmd))
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        return obj

    with ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 4)) as ex:
        objs = list(ex.map(compile_one, sources()))
    tmp = lib + ".tmp"
    cmd = [nvcc, *ARCH, "-shared", "-o", tmp, *objs]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build_library(force=True, verbose=True))
