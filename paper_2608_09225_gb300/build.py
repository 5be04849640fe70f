"""Build libkvgov.so in-tree with nvcc for sm_103a.

Each translation unit under csrc/ is compiled in parallel, then linked into
one shared library next to this file.  `python -m paper_2608_09225_gb300.build`
does the same from the command line.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
ROOT = os.path.dirname(HERE)
INCLUDE = os.path.join(ROOT, "include")
LIB = os.path.join(HERE, "libkvgov.so")
PEAK_LIB = os.path.join(HERE, "libkvgov_peak.so")
BUILD_DIR = os.path.join(HERE, "_build")

# library -> its translation units
LIBS = {LIB: ["kvgov_chain.cu", "kvgov_chain_split.cu", "kvgov_blkoff.cu", "kvgov_salts.cu", "kvgov_table.cu", "kvgov_arrival.cu", "kvgov_boundary.cu", "kvgov_response.cu", "kvgov_origami.cu", "kvgov_pipeline.cu"], PEAK_LIB: ["int_peak.cu", "gather_peak.cu"]}
SOURCES = [s for srcs in LIBS.values() for s in srcs]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", INCLUDE]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: libkvgov needs the CUDA toolkit to build")


def _inputs():
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC)]
    deps += [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE)]
    return [d for d in deps if os.path.isfile(d)]


def up_to_date() -> bool:
    if not all(os.path.exists(lib) for lib in LIBS):
        return False
    t = min(os.path.getmtime(lib) for lib in LIBS)
    return all(os.path.getmtime(d) <= t for d in _inputs())


def build(force: bool = False, verbose: bool = False, extra: list[str] | None = None) -> str:
    """Compile every CUDA source and link libkvgov.so; returns its path."""
    if not force and not extra and up_to_date():
        return LIB
    os.makedirs(BUILD_DIR, exist_ok=True)
    cc = nvcc()
    flags = FLAGS + (extra or [])

    def compile_one(src):
        obj = os.path.join(BUILD_DIR, src.replace(".cu", ".o"))
        cmd = [cc, *ARCH, *flags, "-c", os.path.join(CSRC, src), "-o", obj]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{res.stderr}")
        return obj, res.stderr

    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        results = dict(zip(SOURCES, ex.map(compile_one, SOURCES)))
    if verbose:
        for _, log in results.values():
            sys.stderr.write(log)
    for lib, srcs in LIBS.items():
        tmp = lib + f".tmp{os.getpid()}"
        cmd = [cc, *ARCH, "-shared", "-o", tmp, *[results[s][0] for s in srcs]]
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"nvcc link failed for {os.path.basename(lib)}:\n{res.stderr}")
        os.replace(tmp, lib)
    return LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
