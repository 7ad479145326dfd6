"""Compile ``libdora.so`` (the C ABI of include/dora.h) in-tree for sm_103a.

Each translation unit is compiled in parallel with nvcc and linked into a
shared library next to this file.  The CUDA runtime is linked shared so the
library and PyTorch use the same runtime instance (same current device).
"""
from __future__ import annotations

import os
import shutil
import subprocess
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD_DIR = os.path.join(HERE, "_build")
LIB_PATH = os.path.join(HERE, "libdora.so")
# The timeout-path test library: the same objects, except that the attention
# kernels' bounded waits give up after 5 ms and their first CTA withholds its
# first K/V load, so a wait runs out (tests/test_gpu_timeout.py).
TIMEOUT_TEST_LIB_PATH = os.path.join(HERE, "libdora_timeout_test.so")
TIMEOUT_TEST_FLAGS = ["-DDORA_TEST_WITHHOLD_KV_LOAD", "-DDORA_TEST_WAIT_LIMIT_NS=5000000ull"]
SOURCES = ["token_ops.cu", "gemm_tcgen05.cu", "attn_tcgen05.cu", "attn_exchange_tcgen05.cu",
           "api.cu", "noalloc.cu", "actor.cu", "embed_head.cu", "training.cu"]
# the attention translation units, rebuilt with the test flags for the timeout-path library
ATTN_SOURCES = ("attn_tcgen05.cu", "attn_exchange_tcgen05.cu")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA 13 toolkit is required to build libdora.so")


def _cuda_lib_dir(nvcc: str) -> str:
    return os.path.join(os.path.dirname(os.path.dirname(os.path.realpath(nvcc))), "lib64")


def _deps() -> list:
    files = [os.path.join(CSRC, f) for f in os.listdir(CSRC)]
    files.append(os.path.join(INCLUDE, "dora.h"))
    files.append(os.path.abspath(__file__))
    return files


def up_to_date() -> bool:
    for lib in (LIB_PATH, TIMEOUT_TEST_LIB_PATH):
        if not os.path.exists(lib):
            return False
        t = os.path.getmtime(lib)
        if not all(os.path.getmtime(f) <= t for f in _deps()):
            return False
    return True


def build(force: bool = False, verbose: bool = False, extra_flags: list | None = None) -> str:
    """Build libdora.so if any source is newer; returns its path."""
    if not force and up_to_date():
        return LIB_PATH
    nvcc = _nvcc()
    os.makedirs(BUILD_DIR, exist_ok=True)
    common = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE,
                     "-I", CSRC, "--expt-relaxed-constexpr"] + list(extra_flags or [])

    def compile_one(job) -> str:
        src, tag, flags = job
        obj = os.path.join(BUILD_DIR, os.path.splitext(src)[0] + tag + ".o")
        cmd = [nvcc] + common + flags + ["-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            print(r.stdout, r.stderr)
        return obj

    jobs = [(src, "", []) for src in SOURCES] + [(src, "_timeout_test", TIMEOUT_TEST_FLAGS)
                                                  for src in ATTN_SOURCES]
    with ThreadPoolExecutor(len(jobs)) as ex:
        objs = list(ex.map(compile_one, jobs))
    main_objs = objs[:len(SOURCES)]
    test_attn = dict(zip(ATTN_SOURCES, objs[len(SOURCES):]))
    test_objs = [test_attn.get(s, o) for s, o in zip(SOURCES, main_objs)]

    def link(objs_, path):
        tmp = path + ".tmp"
        cmd = [nvcc] + ARCH + ["-shared", "-cudart", "shared", "-o", tmp] + objs_ + [
            "-Xlinker", "-rpath," + _cuda_lib_dir(nvcc)]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{' '.join(cmd)}\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, path)

    link(test_objs, TIMEOUT_TEST_LIB_PATH)
    link(main_objs, LIB_PATH)
    return LIB_PATH


if __name__ == "__main__":
    print(build(force=True, verbose=True))
