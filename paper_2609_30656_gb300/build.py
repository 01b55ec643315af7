"""Builds libcb_tbe.so (the CUDA library behind include/cb_tbe.h) in-tree.

Each translation unit under csrc/ is compiled for sm_103a only, in parallel,
then linked into one shared library against the shared CUDA runtime (so that
streams created by PyTorch in the same process are the same objects).
"""

from __future__ import annotations

import concurrent.futures
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libcb_tbe.so")
SOURCES = ["cb_tbe.cu", "tbe_plan.cu", "tbe_forward.cu", "tbe_forward_f32.cu", "tbe_forward_f16.cu",
           "tbe_forward_bf16.cu", "tbe_backward.cu", "tbe_sort.cu", "cb_tbe_noalloc.cu",
           "fm_interaction.cu", "tbe_weight_grad.cu", "tbe_backward_apply.cu", "kjt_replicate.cu",
           "tbe_reduce_f16.cu", "tbe_reduce_bf16.cu", "tbe_reduce_f32.cu", "gather_ceiling.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", shutil.which("nvcc")):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found; the CUDA library cannot be built")


def _deps() -> list[str]:
    files = [os.path.join(CSRC, f) for f in os.listdir(CSRC)]
    files.append(os.path.join(INCLUDE, "cb_tbe.h"))
    files.append(os.path.abspath(__file__))
    return files


def _stale() -> bool:
    if os.environ.get("CB_TBE_NVCC_FLAGS"):
        return True
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(f) > t for f in _deps())


def build(force: bool = False, verbose: bool = False, ptxas_info: bool = False) -> str:
    """Compiles and links the library if any source is newer; returns its path."""
    if not force and not _stale():
        return LIB
    os.makedirs(BUILD_DIR, exist_ok=True)
    cc = nvcc()
    flags = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-I", INCLUDE, "-I", CSRC,
             *ARCH]
    if ptxas_info:
        flags += ["-Xptxas", "-v"]
    flags += os.environ.get("CB_TBE_NVCC_FLAGS", "").split()

    def compile_one(src: str) -> tuple[str, str]:
        obj = os.path.join(BUILD_DIR, src.replace(".cu", ".o"))
        cmd = [cc, *flags, "-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        return obj, r.stdout + r.stderr

    with concurrent.futures.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        results = list(ex.map(compile_one, SOURCES))
    if verbose or ptxas_info:
        for _, log in results:
            if log.strip():
                print(log, file=sys.stderr)
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [cc, "-shared", *ARCH, "-cudart", "shared", "-o", tmp, *[o for o, _ in results]]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True, ptxas_info="--ptxas" in sys.argv))
