"""Build ``libspec.so`` (the C-ABI library of include/spec.h) for sm_103a.

Each ``csrc/*.cu`` translation unit is compiled in parallel with nvcc, then
linked into one shared library next to this file.  No cmake, no torch
extension machinery: the library has a plain C ABI.
"""
import concurrent.futures as cf
import glob
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIBRARY = os.path.join(HERE, "libspec.so")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")

NVCC = os.environ.get("NVCC", "nvcc")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
         "--expt-relaxed-constexpr", "-I", INCLUDE]


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return _sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(INCLUDE, "*.h"))


def up_to_date() -> bool:
    if not os.path.exists(LIBRARY):
        return False
    t = os.path.getmtime(LIBRARY)
    return all(os.path.getmtime(d) <= t for d in _deps())


# Translation units that call the device runtime (device-side cudaGraphLaunch):
# compiled as relocatable device code, device-linked with libcudadevrt.
RDC_SOURCES = {"round.cu"}


def _compile(src, extra):
    obj = os.path.join(BUILD, os.path.basename(src) + ".o")
    rdc = ["-rdc=true"] if os.path.basename(src) in RDC_SOURCES else []
    cmd = [NVCC, *ARCH, *FLAGS, *rdc, *extra, "-c", src, "-o", obj]
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{res.stdout}\n{res.stderr}")
    return obj, res.stderr


def build(force: bool = False, verbose: bool = False, extra=()) -> str:
    """Compile every CUDA source and link libspec.so; returns its path."""
    if not force and up_to_date():
        return LIBRARY
    os.makedirs(BUILD, exist_ok=True)
    with cf.ThreadPoolExecutor(max_workers=len(_sources())) as ex:
        results = list(ex.map(lambda s: _compile(s, list(extra)), _sources()))
    if verbose:
        for _, log in results:
            if log.strip():
                print(log)
    tmp = LIBRARY + ".tmp"
    cmd = [NVCC, *ARCH, "-shared", "-rdc=true", "-o", tmp, *[o for o, _ in results], "-lcudadevrt"]
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError(f"link failed:\n{res.stdout}\n{res.stderr}")
    os.replace(tmp, LIBRARY)
    return LIBRARY


if __name__ == "__main__":
    verbose = "-v" in sys.argv
    extra = ["-Xptxas", "-v"] if "--ptxas" in sys.argv else []
    print(build(force=True, verbose=verbose or bool(extra), extra=extra))
