"""Build libpifa.so in-tree from csrc/ for sm_103a (nvcc for .cu, g++ for .cpp, compiled in
parallel, one -gencode). Usage: ``python -m paper_2501_19090_gb300.build``."""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libpifa.so")
ARCH = "-gencode=arch=compute_103a,code=sm_103a"


def _cuda_home() -> str:
    home = os.environ.get("CUDA_HOME") or os.environ.get("CUDA_PATH")
    if home and os.path.isdir(home):
        return home
    nvcc = shutil.which("nvcc")
    if nvcc:
        return os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))
    return "/usr/local/cuda"


def _sources():
    out = []
    for f in sorted(os.listdir(CSRC)):
        if f.endswith((".cu", ".cpp")):
            out.append(os.path.join(CSRC, f))
    return out


def _compile_cmd(src: str, obj: str, cuda: str, extra_cu=()) -> list[str]:
    inc = ["-I", INCLUDE, "-I", CSRC, "-I", os.path.join(cuda, "include")]
    if src.endswith(".cu"):
        return [os.path.join(cuda, "bin", "nvcc"), ARCH, "-O3", "-lineinfo", "-std=c++17",
                "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr", *extra_cu, *inc, "-c", src, "-o", obj]
    return ["g++", "-O3", "-std=c++17", "-fPIC", "-fopenmp", "-Wall", *inc, "-c", src, "-o", obj]


def build(verbose: bool = False, ptxas_verbose: bool = False) -> str:
    """Compile every source under csrc/ and link libpifa.so; returns the library path."""
    cuda = _cuda_home()
    os.makedirs(BUILD, exist_ok=True)
    srcs = _sources()
    extra = ("-Xptxas", "-v") if ptxas_verbose else ()
    jobs = []
    for s in srcs:
        obj = os.path.join(BUILD, os.path.basename(s) + ".o")
        jobs.append((s, obj, _compile_cmd(s, obj, cuda, extra)))

    def run(job):
        src, obj, cmd = job
        res = subprocess.run(cmd, capture_output=True, text=True)
        return src, res

    with cf.ThreadPoolExecutor(max_workers=min(8, len(jobs))) as ex:
        results = list(ex.map(run, jobs))
    failed = False
    for src, res in results:
        if verbose or res.returncode != 0 or ptxas_verbose:
            sys.stderr.write(f"--- {os.path.basename(src)} (rc={res.returncode})\n{res.stdout}{res.stderr}")
        failed |= res.returncode != 0
    if failed:
        raise RuntimeError("libpifa build failed (see compiler output above)")
    tmp = LIB + ".tmp"
    link = [os.path.join(cuda, "bin", "nvcc"), ARCH, "-shared", "-Xcompiler", "-fPIC,-fopenmp",
            *[j[1] for j in jobs], "-o", tmp, "-lgomp"]
    res = subprocess.run(link, capture_output=True, text=True)
    if res.returncode != 0:
        sys.stderr.write(res.stdout + res.stderr)
        raise RuntimeError("libpifa link failed")
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv, ptxas_verbose="--ptxas" in sys.argv))
