"""Build the AGN CUDA library (libagn_gb300.so) in-tree for sm_103a.

Each translation unit is compiled by nvcc in parallel, then linked into one
shared library under `_build/`.  Objects are rebuilt when a source or header
is newer.  Host code is compiled without floating-point contraction so that
the seeded input generator gives the same bits on every host.

`build(check=True)` also builds the bounds-checked variant
(`_build_check/libagn_gb300_check.so`, compiled with -DAGN_BOUNDS_CHECK: every
wrapped kernel access is checked against the library's table of device
buffers, see csrc/bounds.cuh); both variants' units compile in one parallel
batch.  The binding loads the checked variant when AGN_LIB_VARIANT=check.
"""

from __future__ import annotations

import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")
BUILD = os.path.join(HERE, "_build")
LIB_NAME = "libagn_gb300.so"
LIB_PATH = os.path.join(BUILD, LIB_NAME)
BUILD_CHECK = os.path.join(HERE, "_build_check")
LIB_CHECK_PATH = os.path.join(BUILD_CHECK, "libagn_gb300_check.so")

SOURCES = ["agn_api.cu", "commit_pull.cu", "commit_pull_noalloc.cu", "mlp_simt.cu", "mlp_head.cu",
           "mlp_tc.cu", "mlp_tc_dw.cu", "mlp_eval.cu", "optim.cu", "host_inputs.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "--expt-relaxed-constexpr",
              "-Xcompiler", "-fPIC,-ffp-contract=off,-O3", "-I", INCLUDE]
# (output directory, library path, extra nvcc flags) of each variant
VARIANTS = {"normal": (BUILD, LIB_PATH, []),
            "check": (BUILD_CHECK, LIB_CHECK_PATH, ["-DAGN_BOUNDS_CHECK"])}


def _nvcc() -> str:
    cand = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found: the AGN library needs the CUDA toolkit to build")
    return cand


def _headers():
    out = [os.path.join(INCLUDE, f) for f in os.listdir(INCLUDE)]
    out += [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".cuh"))]
    return out


def build(verbose: bool = False, force: bool = False, check: bool = False) -> str:
    """Compile and link; returns the path of the normal library (and builds
    the bounds-checked one too when `check`)."""
    nvcc = _nvcc()
    hdr_time = max(os.path.getmtime(h) for h in _headers())
    names = ["normal", "check"] if check else ["normal"]
    procs = []
    objs = {v: [] for v in names}
    for v in names:
        out_dir, _, extra = VARIANTS[v]
        os.makedirs(out_dir, exist_ok=True)
        for src in SOURCES:
            sp = os.path.join(CSRC, src)
            op = os.path.join(out_dir, src.replace(".cu", ".o"))
            objs[v].append(op)
            if (not force and os.path.exists(op)
                    and os.path.getmtime(op) >= max(os.path.getmtime(sp), hdr_time)):
                continue
            cmd = [nvcc, *ARCH, *NVCC_FLAGS, *extra, "-c", sp, "-o", op]
            if verbose:
                print(" ".join(cmd), flush=True)
            procs.append((f"{v}:{src}",
                          subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT)))
    failed = []
    for src, p in procs:
        out, _ = p.communicate()
        if p.returncode != 0:
            failed.append((src, out.decode(errors="replace")))
        elif verbose and out:
            print(out.decode(errors="replace"))
    if failed:
        msg = "\n".join(f"--- {s}\n{o}" for s, o in failed)
        raise RuntimeError(f"nvcc failed:\n{msg}")
    for v in names:
        _, lib_path, _ = VARIANTS[v]
        relink = force or not os.path.exists(lib_path) or any(
            os.path.getmtime(o) > os.path.getmtime(lib_path) for o in objs[v])
        if relink:
            tmp = lib_path + ".tmp"
            cmd = [nvcc, *ARCH, "-shared", "-cudart", "shared", "-o", tmp, *objs[v], "-lcuda"]
            if verbose:
                print(" ".join(cmd), flush=True)
            r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT)
            if r.returncode != 0:
                raise RuntimeError("link failed:\n" + r.stdout.decode(errors="replace"))
            os.replace(tmp, lib_path)
    return LIB_PATH


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv, force="-f" in sys.argv, check="--check" in sys.argv))
