"""Builds libregmem.so in-tree from csrc/ with nvcc for sm_103a.

One translation unit per kernel family, compiled in parallel, linked with the
static CUDA runtime (the driver API is reached through the runtime's
entry-point query, so the library loads on machines without a GPU driver).
"""
from __future__ import annotations

import concurrent.futures
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
SRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libregmem.so")
# the same sources with the kernels' range guards compiled in
CHECKED_BUILD_DIR = os.path.join(HERE, "_build_checked")
CHECKED_LIB = os.path.join(HERE, "libregmem_checked.so")
CHECKED_FLAGS = ["-DREGMEM_DEVICE_CHECKS"]

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "--expt-relaxed-constexpr",
         "-Xcompiler", "-fPIC,-fvisibility=hidden", "-I", INCLUDE, "-I", SRC]


def nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def sources() -> list[str]:
    return sorted(os.path.join(SRC, f) for f in os.listdir(SRC) if f.endswith(".cu"))


def _deps() -> list[str]:
    deps = [os.path.join(SRC, f) for f in os.listdir(SRC)]
    deps.append(os.path.join(INCLUDE, "regmem.h"))
    return deps


def up_to_date(lib: str = LIB) -> bool:
    if not os.path.exists(lib):
        return False
    t = os.path.getmtime(lib)
    return all(os.path.getmtime(d) <= t for d in _deps())


def _compile(src: str, extra: list[str], build_dir: str = BUILD_DIR) -> str:
    obj = os.path.join(build_dir, os.path.basename(src) + ".o")
    cmd = [nvcc(), *ARCH, *FLAGS, *extra, "-c", src, "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed on {os.path.basename(src)}:\n{r.stderr}")
    return obj


def _link(objs: list[str], lib: str) -> None:
    tmp = lib + ".tmp"
    r = subprocess.run([nvcc(), *ARCH, "-shared", "-o", tmp, *objs], capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stderr}")
    os.replace(tmp, lib)


def build(force: bool = False, verbose: bool = False, extra: list[str] | None = None,
          checked: bool = True) -> str:
    """Compile csrc/*.cu and link libregmem.so next to this file (and, with
    `checked`, libregmem_checked.so with the range guards); returns the path
    of libregmem.so.  Every translation unit of both builds compiles in
    parallel."""
    targets = [(LIB, BUILD_DIR, list(extra or []))]
    if checked:
        targets.append((CHECKED_LIB, CHECKED_BUILD_DIR, list(extra or []) + CHECKED_FLAGS))
    targets = [t for t in targets if force or not up_to_date(t[0])]
    if not targets:
        return LIB
    srcs = sources()
    jobs = []
    for lib, bdir, flags in targets:
        os.makedirs(bdir, exist_ok=True)
        jobs += [(lib, src, flags, bdir) for src in srcs]
    with concurrent.futures.ThreadPoolExecutor(max_workers=len(jobs)) as ex:
        objs = list(ex.map(lambda j: (j[0], _compile(j[1], j[2], j[3])), jobs))
    for lib, _, _ in targets:
        _link([o for l, o in objs if l == lib], lib)
        if verbose:
            print(f"built {lib}", file=sys.stderr)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose=True)
