"""In-tree build of the CUDA library ``_build/libquasar.so`` for sm_103a.

Each translation unit is compiled by its own nvcc process (in parallel) and
the objects are linked into one shared library with the CUDA runtime linked
statically, so the library depends only on the driver.
"""
from __future__ import annotations

import os
import subprocess
from concurrent.futures import ThreadPoolExecutor

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(BUILD, "libquasar.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I" + INCLUDE, "-I" + CSRC]

# (source, extra flags, object name)
UNITS = [
    ("quasar_abi.cu", [], "quasar_abi.o"),
    ("kernels_int.cu", ["-DQUASAR_NCH=1", "-DQUASAR_SS=4"], "kernels_int_nch1_ss4.o"),
    ("kernels_int.cu", ["-DQUASAR_NCH=1", "-DQUASAR_SS=8"], "kernels_int_nch1_ss8.o"),
    ("kernels_int.cu", ["-DQUASAR_NCH=1", "-DQUASAR_SS=3"], "kernels_int_nch1_ss3.o"),
    ("kernels_int.cu", ["-DQUASAR_NCH=1", "-DQUASAR_SS=2"], "kernels_int_nch1_ss2.o"),
    ("kernels_int.cu", ["-DQUASAR_NCH=1", "-DQUASAR_SS=1"], "kernels_int_nch1_ss1.o"),
    ("kernels_int.cu", ["-DQUASAR_NCH=2", "-DQUASAR_SS=4"], "kernels_int_nch2_ss4.o"),
    ("kernels_int.cu", ["-DQUASAR_NCH=2", "-DQUASAR_SS=2"], "kernels_int_nch2_ss2.o"),
    ("kernels_int.cu", ["-DQUASAR_NCH=2", "-DQUASAR_SS=1"], "kernels_int_nch2_ss1.o"),
    ("kernels_int.cu", ["-DQUASAR_NCH=4", "-DQUASAR_SS=4"], "kernels_int_nch4_ss4.o"),
    ("kernels_int.cu", ["-DQUASAR_NCH=4", "-DQUASAR_SS=2"], "kernels_int_nch4_ss2.o"),
    ("kernels_int.cu", ["-DQUASAR_NCH=4", "-DQUASAR_SS=1"], "kernels_int_nch4_ss1.o"),
    ("kernels_nvfp4.cu", [], "kernels_nvfp4.o"),
    ("kernels_lut.cu", [], "kernels_lut.o"),
    ("kernels_sym.cu", [], "kernels_sym.o"),
]


def _nvcc() -> str:
    cuda = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    path = os.path.join(cuda, "bin", "nvcc")
    return path if os.path.exists(path) else "nvcc"


def _inputs():
    files = [os.path.join(INCLUDE, "quasar.h"), os.path.abspath(__file__)]
    for name in os.listdir(CSRC):
        files.append(os.path.join(CSRC, name))
    return files


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(f) <= t for f in _inputs())


def build(force: bool = False, verbose: bool = False, ptxas_info: bool = False) -> str:
    """Compile (if needed) and return the path of libquasar.so."""
    if not force and up_to_date():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    nvcc = _nvcc()

    def compile_one(unit):
        src, extra, obj = unit
        cmd = [nvcc, *ARCH, *NVCC_FLAGS, *extra, "-c", os.path.join(CSRC, src),
               "-o", os.path.join(BUILD, obj)]
        if ptxas_info:
            cmd.insert(1, "-Xptxas=-v")
        res = subprocess.run(cmd, capture_output=True, text=True)
        if res.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src} {extra}:\n{res.stderr}")
        return res.stderr

    with ThreadPoolExecutor(max_workers=len(UNITS)) as ex:
        logs = list(ex.map(compile_one, UNITS))
    if verbose or ptxas_info:
        for log in logs:
            print(log)
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [nvcc, *ARCH, "-shared", "-Xcompiler", "-fPIC", "-o", tmp,
           *[os.path.join(BUILD, u[2]) for u in UNITS]]
    res = subprocess.run(cmd, capture_output=True, text=True)
    if res.returncode != 0:
        raise RuntimeError(f"link failed:\n{res.stderr}")
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    import sys
    print(build(force="--force" in sys.argv, verbose=True, ptxas_info="--ptxas" in sys.argv))
