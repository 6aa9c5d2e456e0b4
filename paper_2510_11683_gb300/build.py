"""Builds the in-tree CUDA library ``lib/libbgpo.so`` for sm_103a with nvcc.

Translation units are compiled in parallel and linked into one shared library
(static CUDA runtime). ``python -m paper_2510_11683_gb300.build`` runs it;
``--checked`` builds ``lib/libbgpo_checked.so`` instead, the same sources with
-DBGPO_CHECKED (device-side bounds checks that record BGPO_ERR_BOUNDS).
"""
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG_DIR)
CSRC = os.path.join(PKG_DIR, "csrc")
INCLUDE = os.path.join(ROOT, "include")
LIB_DIR = os.path.join(PKG_DIR, "lib")
LIB_PATH = os.path.join(LIB_DIR, "libbgpo.so")
CHECKED_LIB_PATH = os.path.join(LIB_DIR, "libbgpo_checked.so")
OBJ_DIR = os.path.join(PKG_DIR, "_build")

ARCH_FLAGS = ["-gencode", "arch=compute_103a,code=sm_103a"]
COMMON_FLAGS = ["-std=c++17", "-O3", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
                f"-I{INCLUDE}", f"-I{CSRC}"]
SOURCES = ["k_gemm.cu", "k_small.cu", "bgpo_api.cu", "bgpo_noalloc.cu"]


def nvcc():
    cand = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc")
    return cand if os.path.exists(cand) else "nvcc"


def _compile(src, extra, obj_dir, verbose):
    obj = os.path.join(obj_dir, os.path.splitext(src)[0] + ".o")
    cmd = [nvcc(), *ARCH_FLAGS, *COMMON_FLAGS, *extra, "-c", os.path.join(CSRC, src), "-o", obj]
    if verbose:
        print(" ".join(cmd), flush=True)
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    if verbose and (r.stdout or r.stderr):
        print(r.stdout + r.stderr, flush=True)
    return obj


def build(verbose=False, ptxas_verbose=False, checked=False):
    """Compiles every CUDA source and links lib/libbgpo.so (checked=True:
    lib/libbgpo_checked.so with -DBGPO_CHECKED). Returns its path."""
    obj_dir = os.path.join(OBJ_DIR, "checked") if checked else OBJ_DIR
    out = CHECKED_LIB_PATH if checked else LIB_PATH
    os.makedirs(obj_dir, exist_ok=True)
    os.makedirs(LIB_DIR, exist_ok=True)
    extra = (["-Xptxas", "-v"] if ptxas_verbose else []) + (["-DBGPO_CHECKED"] if checked else [])
    with ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(lambda s: _compile(s, extra, obj_dir, verbose or ptxas_verbose),
                           SOURCES))
    tmp = out + ".tmp"
    cmd = [nvcc(), *ARCH_FLAGS, "-shared", "-o", tmp, *objs]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build(verbose=True, ptxas_verbose="-v" in sys.argv, checked="--checked" in sys.argv))
