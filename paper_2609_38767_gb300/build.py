"""Compile the CUDA libraries in-tree for sm_103a with nvcc.

libtda.so        -- the attribution hot path (include/tda.h)
libtda_synth.so  -- the seeded synthetic-factor generator (include/tda_synth.h)

Translation units compile in parallel into ``_build/`` and are linked with
``nvcc -shared`` next to this file. A library is rebuilt when any of its
sources or headers is newer than it.
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(ROOT, "_build")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC = os.environ.get("NVCC", "/usr/local/cuda/bin/nvcc")
FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
         "-Xptxas", "-warn-spills"]

LIBS = {
    "libtda.so": ["api.cu", "calibrate.cu", "k_project_simt.cu", "k_project_tc.cu", "k_routes.cu",
                  "k_precond.cu", "k_score.cu", "stream_host.cu", "noalloc.cu", "selftest.cu", "k_gemm_tc.cu", "k_gram_tc.cu", "k_kfac.cu", "k_tokens.cu", "k_tokens_tc.cu", "k_materialize_tc.cu"],
    "libtda_synth.so": ["synth.cu"],
}


def lib_path(name: str) -> str:
    return os.path.join(HERE, name)


def _headers() -> list[str]:
    return glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(ROOT, "include", "*.h"))


def _stale(target: str, deps: list[str]) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def _compile(src: str, extra: list[str]) -> str:
    obj = os.path.join(BUILD, os.path.basename(src).replace(".cu", ".o"))
    if _stale(obj, [src] + _headers()):
        cmd = [NVCC, *ARCH, *FLAGS, *extra, "-c", src, "-o", obj + ".tmp"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
        os.replace(obj + ".tmp", obj)
    return obj


def build_synth_cpu() -> str:
    """gcc build of the CPU side of the input generator (OpenMP, no FP contraction)."""
    src = os.path.join(CSRC, "synth_cpu.c")
    target = lib_path("libtda_synth_cpu.so")
    if _stale(target, [src]):
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
               "-o", target + ".tmp", src, "-lm"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"gcc failed for {src}:\n{r.stderr}")
        os.replace(target + ".tmp", target)
    return target


def build(verbose: bool = False, extra: list[str] | None = None) -> dict[str, str]:
    """Build every library that is out of date; returns {name: path}."""
    os.makedirs(BUILD, exist_ok=True)
    extra = extra or []
    out = {}
    with cf.ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 4)) as ex:
        futs = {name: [ex.submit(_compile, os.path.join(CSRC, s), extra) for s in srcs]
                for name, srcs in LIBS.items()}
        for name, fl in futs.items():
            objs = [f.result() for f in fl]
            target = lib_path(name)
            if _stale(target, objs):
                cmd = [NVCC, *ARCH, "-shared", "-o", target + ".tmp", *objs]
                r = subprocess.run(cmd, capture_output=True, text=True)
                if r.returncode != 0:
                    raise RuntimeError(f"link failed for {name}:\n{r.stdout}\n{r.stderr}")
                os.replace(target + ".tmp", target)
                if verbose:
                    print("built", target)
            out[name] = target
    out["libtda_synth_cpu.so"] = build_synth_cpu()
    return out


if __name__ == "__main__":
    for k, v in build(verbose=True).items():
        print(k, v)
