"""Build step of the CUDA library: nvcc, sm_103a only, in-tree output.

``python -m paper_2310_07109_gb300.build`` (or ``build_library()``) compiles
``csrc/*.cu`` into ``libsparsecoder.so`` next to this file.  The translation
units are compiled in parallel and linked with the CUDA runtime; the TMA
descriptor encoder is reached through the runtime's driver entry point, so no
link against libcuda is needed.
"""
from __future__ import annotations

import os
import subprocess
import sys
import tempfile
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")
LIB = os.path.join(HERE, "libsparsecoder.so")
SOURCES = ["sc_kernels.cu", "sc_band.cu", "sc_tail.cu", "sc_encoder.cu", "sc_api.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    cand = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc")
    return cand if os.path.exists(cand) else "nvcc"


def _stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC)]
    deps.append(os.path.join(INCLUDE, "sparsecoder.h"))
    return any(os.path.getmtime(d) > t for d in deps if os.path.exists(d))


def build_library(force: bool = False, verbose: bool = False) -> str:
    if not force and not _stale():
        return LIB
    flags = ARCH + ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC",
                    "-I", INCLUDE, "-Xptxas", "-v" if verbose else "-O3"]
    with tempfile.TemporaryDirectory() as tmp:
        objs = [os.path.join(tmp, s.replace(".cu", ".o")) for s in SOURCES]

        def compile_one(i):
            cmd = [nvcc(), *flags, "-c", os.path.join(CSRC, SOURCES[i]), "-o", objs[i]]
            r = subprocess.run(cmd, capture_output=True, text=True)
            if r.returncode != 0:
                raise RuntimeError("nvcc failed for %s:\n%s%s" % (SOURCES[i], r.stdout, r.stderr))
            return r.stderr

        with ThreadPoolExecutor(len(SOURCES)) as ex:
            logs = list(ex.map(compile_one, range(len(SOURCES))))
        if verbose:
            sys.stderr.write("".join(logs))
        out = LIB + ".%d.tmp" % os.getpid()
        cmd = [nvcc(), *ARCH, "-shared", "-cudart", "shared", "-o", out, *objs,
               "-Xlinker", "-rpath", "-Xlinker", os.path.join(os.path.dirname(os.path.dirname(nvcc())), "lib64")]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("link failed:\n%s%s" % (r.stdout, r.stderr))
        os.replace(out, LIB)
    return LIB


if __name__ == "__main__":
    print(build_library(force="--force" in sys.argv, verbose="-v" in sys.argv))
