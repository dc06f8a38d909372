"""Build ``libvqc.so`` in-tree with nvcc for sm_103a (GB300).

The translation units (host compiler, C ABI, one kernel unit per real type and
mode) compile in parallel; the result is linked into one shared library next
to this file.  Nothing is installed outside the source tree.
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
ROOT = os.path.dirname(HERE)
OUT = os.path.join(HERE, "libvqc.so")
BUILD = os.path.join(HERE, "_build")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC,-O2,-ffp-contract=off",
              "--expt-relaxed-constexpr", "-I" + os.path.join(ROOT, "include")]
UNITS = ["compiler.cpp", "qasm.cpp", "capi.cu", "noalloc.cu", "host_eval.cu",
         "kernels_f32_fwd.cu", "kernels_f32_bwd.cu", "kernels_f64_fwd.cu", "kernels_f64_bwd.cu",
         "kernels_f32_fwd_small.cu", "kernels_f32_bwd_small.cu", "kernels_f64_fwd_small.cu",
         "kernels_f64_bwd_small.cu", "kernels_hbm.cu", "kernels_cluster.cu",
         "kernels_f32_fused.cu", "kernels_f64_fused.cu", "fma_peak.cu",
         "kernels_dd_fwd.cu", "kernels_dd_bwd.cu", "kernels_dd_fused.cu", "kernels_dd_hbm.cu",
         "tc_stage.cu", "kernels_f32_fwd_nph.cu", "kernels_f32_bwd_nph.cu", "kernels_hbm_nph.cu",
         "kernels_f32_fused_nph.cu", "kernels_cluster_bwd.cu"]


def nvcc() -> str:
    for cand in (shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libvqc.so")


def _sources_digest() -> str:
    h = hashlib.sha256()
    for name in sorted(os.listdir(CSRC)):
        with open(os.path.join(CSRC, name), "rb") as f:
            h.update(name.encode() + f.read())
    with open(os.path.join(ROOT, "include", "vqc.h"), "rb") as f:
        h.update(f.read())
    # flags without the include path, so that a checkout anywhere hashes alike
    h.update(" ".join(ARCH + [f for f in NVCC_FLAGS if not f.startswith("-I")]).encode())
    return h.hexdigest()


def build(force: bool = False, verbose: bool = False, ptxas_info: bool = False) -> str:
    """Compile and link libvqc.so if the sources changed; return its path."""
    digest = _sources_digest()
    stamp = OUT + ".sha256"
    if not force and os.path.exists(OUT) and os.path.exists(stamp):
        with open(stamp) as f:
            if f.read().strip() == digest:
                return OUT
    os.makedirs(BUILD, exist_ok=True)
    cc = nvcc()
    extra = ["-Xptxas", "-v"] if ptxas_info else []

    def compile_one(unit):
        obj = os.path.join(BUILD, unit + ".o")
        cmd = [cc] + ARCH + NVCC_FLAGS + extra + ["-c", os.path.join(CSRC, unit), "-o", obj]
        if unit.endswith(".cpp"):
            cmd = [cc, "-x", "c++"] + NVCC_FLAGS + ["-c", os.path.join(CSRC, unit), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("nvcc failed for %s:\n%s%s" % (unit, r.stdout, r.stderr))
        return obj, r.stdout + r.stderr

    with cf.ThreadPoolExecutor(max_workers=len(UNITS)) as ex:
        results = list(ex.map(compile_one, UNITS))
    if verbose or ptxas_info:
        for _, log in results:
            if log.strip():
                print(log)
    tmp = OUT + ".tmp.%d" % os.getpid()
    cmd = [cc] + ARCH + ["-shared", "-o", tmp] + [o for o, _ in results]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("link failed:\n%s%s" % (r.stdout, r.stderr))
    os.replace(tmp, OUT)
    with open(stamp, "w") as f:
        f.write(digest)
    return OUT


if __name__ == "__main__":
    import sys
    print(build(force="--force" in sys.argv, verbose=True, ptxas_info="-v" in sys.argv))
