"""Build the KVpop CUDA library (sm_103a) in-tree: ``paper_2607_05061_gb300/libkvpop.so``.

Each translation unit is compiled in parallel with one ``-gencode`` target
(GB300 is sm_103a), then linked into a shared library with the C ABI of
``include/kvpop.h``.  Run ``python -m paper_2607_05061_gb300.build``.

``build(checked=True)`` (``-c`` on the command line) makes the device-check
variant ``libkvpop_checked.so``: the same sources with ``-DKVPOP_DEVICE_CHECKS``,
whose kernels check their indices and record a failed check in the device error
word that ``kvpop_check`` / ``kvpop_standalone_status`` report, instead of
trapping.  The binding loads it when ``KVPOP_DEVICE_CHECKS=1``.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libkvpop.so")
BUILD_CHECKED = os.path.join(HERE, "_build_checked")
LIB_CHECKED = os.path.join(HERE, "libkvpop_checked.so")
SOURCES = ["kvpop_api.cu", "kvpop_ingest.cu", "kvpop_ingest_cluster.cu", "kvpop_attend.cu", "kvpop_attend_tc.cu",
           "kvpop_prefill.cu", "kvpop_noalloc.cu", "kvpop_mlstm.cu", "kvpop_topk.cu", "kvpop_prompt.cu", "kvpop_prompt_tc5.cu", "kvpop_target.cu",
           "kvpop_score_tf32.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc_path() -> str:
    cand = [os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc"),
            shutil.which("nvcc") or ""]
    for c in cand:
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found (set CUDA_HOME)")


def cuda_home() -> str:
    return os.path.dirname(os.path.dirname(nvcc_path()))


def _compile(src: str, verbose_ptxas: bool, checked: bool = False) -> str:
    obj = os.path.join(BUILD_CHECKED if checked else BUILD, os.path.splitext(src)[0] + ".o")
    cmd = [nvcc_path(), *ARCH, "-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
           "--expt-relaxed-constexpr", "-c", os.path.join(CSRC, src), "-o", obj]
    if checked:
        cmd.insert(1, "-DKVPOP_DEVICE_CHECKS")
    # optional -D overrides of the kernels' compile-time tuning constants
    cmd[1:1] = os.environ.get("KVPOP_NVCC_DEFINES", "").split()
    if verbose_ptxas:
        cmd.insert(1, "-Xptxas=-v")
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    if verbose_ptxas:
        sys.stderr.write(r.stderr)
    return obj


def build(verbose_ptxas: bool = False, force: bool = False, checked: bool = False) -> str:
    bdir, lib = (BUILD_CHECKED, LIB_CHECKED) if checked else (BUILD, LIB)
    os.makedirs(bdir, exist_ok=True)
    srcs = ([os.path.join(CSRC, s) for s in os.listdir(CSRC)]
            + [os.path.join(HERE, "..", "include", "kvpop.h")])
    if (not force and os.path.exists(lib)
            and os.path.getmtime(lib) > max(os.path.getmtime(s) for s in srcs)):
        return lib
    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(lambda s: _compile(s, verbose_ptxas, checked), SOURCES))
    lib64 = os.path.join(cuda_home(), "lib64")
    tmp = lib + ".tmp"
    cmd = [nvcc_path(), *ARCH, "-shared", "-cudart", "shared", "-o", tmp, *objs,
           "-Xlinker", f"-rpath,{lib64}"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build(verbose_ptxas="-v" in sys.argv, force="-f" in sys.argv, checked="-c" in sys.argv))
