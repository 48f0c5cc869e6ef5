"""In-tree build of the ESTP CUDA library (libestp.so) for sm_103a.

Each translation unit is compiled in parallel with nvcc, then linked into one
shared library under ``_build/``.  Only out-of-date objects are rebuilt.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OUT = os.path.join(PKG, "_build")
LIB = os.path.join(OUT, "libestp.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-I", INCLUDE, "-I", CSRC,
              "--expt-relaxed-constexpr", "-Xptxas", "-warn-spills"]


def _nvcc() -> str:
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", "nvcc"):
        if cand and (os.path.sep not in cand or os.path.exists(cand)):
            return cand
    return "nvcc"


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps_mtime() -> float:
    files = glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(INCLUDE, "*.h"))
    files.append(os.path.abspath(__file__))
    return max(os.path.getmtime(f) for f in files)


def _compile(src: str, extra: list[str], out: str = OUT) -> tuple[str, str]:
    obj = os.path.join(out, os.path.basename(src).replace(".cu", ".o"))
    cmd = [_nvcc(), *ARCH, *NVCC_FLAGS, *extra, "-c", src, "-o", obj]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    return obj, r.stderr


OUT_CHECKS = os.path.join(PKG, "_build_checks")
LIB_CHECKS = os.path.join(OUT_CHECKS, "libestp_checks.so")


def build_checks(force: bool = False) -> str:
    """The debug variant: the same sources with -DESTP_CHECKS (device bounds checks that
    record ESTP_ERR_BOUNDS in the status word), linked as libestp_checks.so."""
    return build(force=force, extra=["-DESTP_CHECKS"], out=OUT_CHECKS, lib=LIB_CHECKS)


def build(force: bool = False, verbose: bool = False, extra: list[str] | None = None,
          out: str = OUT, lib: str = LIB) -> str:
    """Compile every csrc/*.cu for sm_103a into `out` and link `lib` (libestp.so by
    default); returns the library's path."""
    os.makedirs(out, exist_ok=True)
    extra = list(extra or [])
    dep = _deps_mtime()
    srcs = _sources()
    todo = []
    for s in srcs:
        obj = os.path.join(out, os.path.basename(s).replace(".cu", ".o"))
        if force or not os.path.exists(obj) or os.path.getmtime(obj) < max(dep, os.path.getmtime(s)):
            todo.append(s)
    if todo:
        with cf.ThreadPoolExecutor(max_workers=min(len(todo), os.cpu_count() or 4)) as ex:
            for obj, log in ex.map(lambda s: _compile(s, extra, out), todo):
                if verbose and log.strip():
                    print(log)
    objs = [os.path.join(out, os.path.basename(s).replace(".cu", ".o")) for s in srcs]
    if todo or not os.path.exists(lib) or os.path.getmtime(lib) < max(os.path.getmtime(o) for o in objs):
        tmp = lib + f".tmp{os.getpid()}"
        cmd = [_nvcc(), *ARCH, "-shared", "-o", tmp, *objs]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, lib)
    return lib


def build_synth(force: bool = False) -> str:
    """Compile the device side of the input generator (synth/synth.cu)."""
    src = os.path.join(ROOT, "synth", "synth.cu")
    out = os.path.join(ROOT, "synth", "_build", "libsynth.so")
    os.makedirs(os.path.dirname(out), exist_ok=True)
    if force or not os.path.exists(out) or os.path.getmtime(out) < os.path.getmtime(src):
        tmp = out + f".tmp{os.getpid()}"
        cmd = [_nvcc(), *ARCH, "-O3", "-std=c++17", "-Xcompiler", "-fPIC", "-shared", src, "-o", tmp]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for synth.cu:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, out)
    return out


if __name__ == "__main__":
    print(build(verbose=True))
    print(build_synth())
