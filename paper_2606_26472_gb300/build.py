"""In-tree build of libepikv.so (and of the synthetic-input generator's
libepikv_synth.so) for sm_103a with nvcc: one object per translation unit,
compiled in parallel, linked against the shared CUDA runtime.  The input
generator's host twin (libepikv_synth_host.so, plain C) is built with gcc."""
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
LIB = os.path.join(PKG, "libepikv.so")
SYNTH_DIR = os.path.join(ROOT, "synth")
SYNTH_LIB = os.path.join(SYNTH_DIR, "libepikv_synth.so")
SYNTH_HOST_LIB = os.path.join(SYNTH_DIR, "libepikv_synth_host.so")
# the host twin of the input generator: plain C, every float operation rounded
# on its own (no contraction), the same bytes on x86-64 and aarch64
HOST_CFLAGS = ["-O2", "-std=c99", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math"]

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVFLAGS = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
                  "--expt-relaxed-constexpr", "-Xptxas", "-warn-spills"]


def _nvcc():
    p = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(p):
        raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libepikv")
    return p


def _cuda_lib_dir():
    return os.path.join(os.path.dirname(os.path.dirname(os.path.realpath(_nvcc()))), "lib64")


def _run(cmd):
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("command failed: " + " ".join(cmd) + "\n" + r.stdout + r.stderr)
    return r.stdout + r.stderr


def _stale(target, sources):
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(s) > t for s in sources)


def _build_so(target, sources, headers, include_dirs, obj_dir, verbose=False, extra=()):
    if not _stale(target, list(sources) + list(headers)):
        return False
    os.makedirs(obj_dir, exist_ok=True)
    nvcc = _nvcc()
    incs = [f"-I{d}" for d in include_dirs]

    def compile_one(src):
        obj = os.path.join(obj_dir, os.path.basename(src) + ".o")
        out = _run([nvcc, *NVFLAGS, *extra, *incs, "-c", src, "-o", obj])
        if verbose and out.strip():
            print(out, file=sys.stderr)
        return obj

    with cf.ThreadPoolExecutor(max_workers=min(8, len(sources))) as ex:
        objs = list(ex.map(compile_one, sources))
    libdir = _cuda_lib_dir()
    _run([nvcc, *ARCH, "-shared", "-cudart", "shared", "-o", target + ".tmp", *objs,
          f"-L{libdir}", "-Xlinker", f"-rpath,{libdir}"])
    os.replace(target + ".tmp", target)
    return True


def build(verbose=False):
    """Build both shared libraries if any source is newer than the library."""
    srcs = sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))
    hdrs = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cuh", ".h"))]
    hdrs.append(os.path.join(INCLUDE, "epikv.h"))
    _build_so(LIB, srcs, hdrs, [INCLUDE, CSRC], os.path.join(ROOT, "_build", "epikv"), verbose)
    ssrc = [os.path.join(SYNTH_DIR, "synth_gen.cu")]
    _build_so(SYNTH_LIB, ssrc, [], [], os.path.join(ROOT, "_build", "synth"), verbose)
    hsrc = os.path.join(SYNTH_DIR, "synth_host.c")
    if _stale(SYNTH_HOST_LIB, [hsrc]):
        cc = shutil.which("gcc") or shutil.which("cc")
        if cc is None:
            raise RuntimeError("no C compiler found for the host input generator")
        _run([cc, *HOST_CFLAGS, "-o", SYNTH_HOST_LIB + ".tmp", hsrc])
        os.replace(SYNTH_HOST_LIB + ".tmp", SYNTH_HOST_LIB)
    return LIB


if __name__ == "__main__":
    build(verbose=True)
    print(LIB)
