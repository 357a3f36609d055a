"""Compile the CUDA sources into the in-tree shared library (sm_103a only).

Each translation unit is compiled in parallel with nvcc, then linked into
``_lib/libwitcert.so`` next to this file.  No torch extension is involved:
the library exports a plain C ABI (``include/witcert.h``).
"""

import concurrent.futures as cf
import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
OUT_DIR = os.path.join(HERE, "_lib")
LIB = os.path.join(OUT_DIR, "libwitcert.so")
LIB_METER_OFF = os.path.join(OUT_DIR, "libwitcert_meteroff.so")
SOURCES = ["api.cu", "write_kernel.cu", "decode_kernel.cu", "gate_kernel.cu", "repair_kernel.cu",
           "decode_g32_kernel.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2"]


def _nvcc():
    for cand in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", shutil.which("nvcc")):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def build(verbose=False, extra_flags=()):
    os.makedirs(OUT_DIR, exist_ok=True)
    nvcc = _nvcc()
    objs = []

    def compile_one(src):
        obj = os.path.join(OUT_DIR, src.replace(".cu", ".o"))
        cmd = [nvcc, *ARCH, *FLAGS, *extra_flags, "-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stderr}")
        if verbose and r.stderr:
            print(r.stderr)
        return obj

    def compile_meter_off():
        obj = os.path.join(OUT_DIR, "decode_kernel_meteroff.o")
        cmd = [nvcc, *ARCH, *FLAGS, *extra_flags, "-DWC_METER_OFF", "-c", os.path.join(CSRC, "decode_kernel.cu"),
               "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on decode_kernel.cu (meter off):\n{r.stderr}")
        return obj

    with cf.ThreadPoolExecutor(max_workers=len(SOURCES) + 1) as ex:
        off = ex.submit(compile_meter_off)
        objs = list(ex.map(compile_one, SOURCES))
        off_obj = off.result()

    def link(out, objects):
        tmp = out + ".tmp"
        r = subprocess.run([nvcc, *ARCH, "-shared", "-o", tmp, *objects, "-lcudart"], capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stderr}")
        os.replace(tmp, out)

    link(LIB, objs)
    # the same library with the certificate compiled out of the warp-specialized
    # decode: the benchmark's meter-on / meter-off measurement only
    link(LIB_METER_OFF, [off_obj if o.endswith("decode_kernel.o") else o for o in objs])
    return LIB


if __name__ == "__main__":
    print(build(verbose=True))
