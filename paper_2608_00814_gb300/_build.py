"""Build the CUDA library in-tree: paper_2608_00814_gb300/_lib/liboos.so.

Every translation unit is compiled by nvcc for sm_103a only (GB300), in
parallel, and linked into one shared library with the C ABI of include/oos.h.
build(timeline=True) builds a second copy, _lib/liboos_timeline.so, with the
per-CTA event times of the step-timeline profile compiled in (timeline.py).
"""

import concurrent.futures as cf
import os
import subprocess
import sys

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
SRC = os.path.join(PKG, "csrc")
OUT_DIR = os.path.join(PKG, "_lib")
LIB = os.path.join(OUT_DIR, "liboos.so")
LIB_TIMELINE = os.path.join(OUT_DIR, "liboos_timeline.so")
UNITS = ["oos_api.cu", "small.cu", "gemm.cu", "attn.cu", "noalloc.cu", "hint.cu", "decode.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc():
    cand = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc")
    return cand if os.path.exists(cand) else "nvcc"


def _flags(verbose_ptxas=False, timeline=False):
    f = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", os.path.join(ROOT, "include"),
                "--expt-relaxed-constexpr"]
    if timeline:
        f += ["-DOOS_TIMELINE"]
    if verbose_ptxas:
        f += ["-Xptxas", "-v"]
    return f


def _stale(lib):
    if not os.path.exists(lib):
        return True
    t = os.path.getmtime(lib)
    deps = [os.path.join(SRC, f) for f in os.listdir(SRC)] + [os.path.join(ROOT, "include", "oos.h")]
    return any(os.path.getmtime(d) > t for d in deps)


def build(force=False, verbose_ptxas=False, timeline=False):
    lib = LIB_TIMELINE if timeline else LIB
    if not force and not _stale(lib):
        return lib
    obj_dir = os.path.join(OUT_DIR, "timeline") if timeline else OUT_DIR
    os.makedirs(obj_dir, exist_ok=True)
    objs = []

    def compile_one(u):
        obj = os.path.join(obj_dir, u.replace(".cu", ".o"))
        cmd = [nvcc()] + _flags(verbose_ptxas, timeline) + ["-c", os.path.join(SRC, u), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("nvcc failed for %s:\n%s\n%s" % (u, r.stdout, r.stderr))
        return obj, r.stderr

    with cf.ThreadPoolExecutor(len(UNITS)) as ex:
        for obj, err in ex.map(compile_one, UNITS):
            objs.append(obj)
            if verbose_ptxas and err:
                sys.stderr.write(err)
    tmp = lib + ".tmp%d" % os.getpid()
    cmd = [nvcc()] + ARCH + ["-shared", "-o", tmp] + objs
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("link failed:\n%s\n%s" % (r.stdout, r.stderr))
    os.replace(tmp, lib)
    return lib


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose_ptxas="-v" in sys.argv, timeline="--timeline" in sys.argv))
