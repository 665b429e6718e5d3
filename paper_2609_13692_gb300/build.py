"""Build libmpt.so (the CUDA kernels and the C ABI of include/mpt.h) in-tree for sm_103a."""

from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
from pathlib import Path

PKG = Path(__file__).resolve().parent
ROOT = PKG.parent
CSRC = PKG / "csrc"
BUILD = PKG / "_build"
LIB = BUILD / "libmpt.so"
# the bounds-checked variant (-DMPT_BOUNDS): device checks on indices, window
# offsets and split entries that report MPT_ERR_INTERNAL instead of reading or
# writing out of range; for tests, slower
BOUNDS_BUILD = PKG / "_build_bounds"
BOUNDS_LIB = BOUNDS_BUILD / "libmpt.so"
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
SOURCES = ["k_scatter_zeta.cu", "k_dp_general.cu", "k_dp_blocked.cu", "k_walk.cu", "mpt_api.cu", "mpt_noalloc.cu", "k_batch.cu", "mpt_batch.cu", "k_greedy.cu", "k_sched.cu", "k_probe.cu", "k_tables.cu", "k_dp_wide.cu"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libmpt")


def _stale(out: Path, deps: list[Path]) -> bool:
    if not out.exists():
        return True
    t = out.stat().st_mtime
    return any(d.stat().st_mtime > t for d in deps)


def build(force: bool = False, verbose: bool = False, bounds: bool = False) -> Path:
    """Compile every CUDA translation unit (in parallel) and link libmpt.so
    (with bounds=True the bounds-checked variant, in its own directory)."""
    out_dir, lib = (BOUNDS_BUILD, BOUNDS_LIB) if bounds else (BUILD, LIB)
    out_dir.mkdir(exist_ok=True)
    headers = [CSRC / "mpt_internal.cuh", ROOT / "include" / "mpt.h"]
    flags = ["-std=c++17", "-O3", "-lineinfo", *ARCH, "-Xcompiler", "-fPIC", "-I", str(ROOT / "include")]
    if bounds:
        flags.append("-DMPT_BOUNDS")
    objs, jobs = [], []
    for src in SOURCES:
        obj = out_dir / (Path(src).stem + ".o")
        objs.append(obj)
        if force or _stale(obj, [CSRC / src, *headers]):
            tmp = out_dir / f"{obj.stem}.{os.getpid()}.o"
            jobs.append(([nvcc(), *flags, "-c", str(CSRC / src), "-o", str(tmp)], tmp, obj))
    with cf.ThreadPoolExecutor(max_workers=len(jobs) or 1) as ex:
        futs = {ex.submit(subprocess.run, cmd, capture_output=True, text=True): (cmd, tmp, obj) for cmd, tmp, obj in jobs}
        for fut in cf.as_completed(futs):
            cmd, tmp, obj = futs[fut]
            r = fut.result()
            if r.returncode != 0:
                raise RuntimeError(f"nvcc failed for {obj.name}:\n{r.stdout}\n{r.stderr}")
            if verbose and (r.stdout or r.stderr):
                print(r.stdout, r.stderr)
            os.replace(tmp, obj)
    if force or jobs or _stale(lib, objs):
        tmp = out_dir / f"libmpt.{os.getpid()}.so"
        r = subprocess.run([nvcc(), *ARCH, "-shared", "-o", str(tmp), *map(str, objs)], capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build(verbose=True))
