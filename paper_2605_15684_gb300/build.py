"""Builds libssba.so (the CUDA library behind include/ssba.h) for sm_103a, in-tree.

Each .cu file under csrc/ is compiled by nvcc in parallel and linked into one shared
object with the CUDA runtime linked statically, so the library loads on a machine
without a GPU driver (the driver is only needed once a call reaches the device).

Variants (built only on request, each in a folder and a library of its own, so that the
default libssba.so is never affected):
  timeline  -DSSBA_TIMELINE=2: the attention kernel records time stamps of its phases and of
            every tile of a few sampled pipelines (read by ssba_timeline_read; see timeline.py);
  phases    -DSSBA_TIMELINE=1: the phase stamps only, which barely perturb the launch;
  checked   -DSSBA_CHECKED: the kernels check the invariants of the index lists they read or
            write (labels in [0, Tb), ascending, count == keep) and report a violation in the
            device status word (SSBA_ERR_CHECK) instead of using the bad value.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OBJDIR = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libssba.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
VARIANTS = {"": [], "timeline": ["-DSSBA_TIMELINE=2"], "phases": ["-DSSBA_TIMELINE=1"], "checked": ["-DSSBA_CHECKED"]}


def library_file(variant: str = "") -> str:
    return LIB if not variant else os.path.join(HERE, f"libssba_{variant}.so")


def _nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def sources():
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))


def _headers():
    hs = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cuh", ".h"))]
    hs += [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE) if f.endswith(".h")]
    return hs


def _stale(target: str, deps) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, verbose: bool = False, extra_flags=(), variant: str = "") -> str:
    """Compile every csrc/*.cu for sm_103a and link libssba.so (or the variant's library);
    returns its path."""
    if variant not in VARIANTS:
        raise ValueError(f"unknown build variant {variant!r}")
    objdir = OBJDIR if not variant else OBJDIR + "_" + variant
    lib = library_file(variant)
    os.makedirs(objdir, exist_ok=True)
    nvcc = _nvcc()
    hdrs = _headers()
    flags = ARCH + ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-fvisibility=hidden",
                    "-I", INCLUDE, "-I", CSRC, "--expt-relaxed-constexpr"] + VARIANTS[variant] + list(extra_flags)
    jobs = []
    for src in sources():
        obj = os.path.join(objdir, os.path.basename(src)[:-3] + ".o")
        if force or _stale(obj, [src] + hdrs):
            jobs.append((src, obj))

    def compile_one(job):
        src, obj = job
        cmd = [nvcc, "-c", src, "-o", obj + ".tmp"] + flags
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        os.replace(obj + ".tmp", obj)
        return r.stderr

    with cf.ThreadPoolExecutor(max_workers=max(1, min(len(jobs), os.cpu_count() or 4))) as ex:
        for out in ex.map(compile_one, jobs):
            if verbose and out:
                print(out, file=sys.stderr)
    objs = [os.path.join(objdir, os.path.basename(s)[:-3] + ".o") for s in sources()]
    if force or jobs or _stale(lib, objs):
        tmp = lib + f".tmp{os.getpid()}"
        cmd = [nvcc, "-shared", "-o", tmp] + objs + ARCH + ["-cudart", "static", "-Xcompiler", "-fPIC", "-ldl"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    var = next((a.split("=", 1)[1] for a in sys.argv[1:] if a.startswith("--variant=")), "")
    print(build(force="--force" in sys.argv, verbose=True, variant=var))
