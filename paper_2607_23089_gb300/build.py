"""Builds librowop.so in-tree with nvcc for sm_103a (GB300).

Each translation unit under ``csrc/`` is compiled in parallel, then linked
into ``_build/librowop.so`` with the CUDA runtime linked statically, so the
library loads with nothing but the NVIDIA driver present.  A stamp of the
sources and flags skips the build when nothing changed.
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(BUILD, "librowop.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
                     "-Xcompiler", "-fvisibility=hidden", "-I", CSRC,
                     "-I", INCLUDE]
# (source, object name, extra flags): ops_instance.cu (forward) and
# bwd_instance.cu (backward) once per operator and element type
_OPS = [("kSoftmax", "softmax"), ("kLogSoftmax", "logsoftmax"), ("kLayerNorm", "layernorm"),
        ("kRmsNorm", "rmsnorm")]
_TYPES = [("float", "f32"), ("__nv_bfloat16", "bf16"), ("__half", "f16")]
UNITS = [("rowop_api.cu", "rowop_api.o", []), ("pad_moe.cu", "pad_moe.o", [])] + [
    (src, f"{pre}_{on}_{tn}.o", [f"-DROWOP_INST_OP={o}", f"-DROWOP_INST_T={t}"])
    for src, pre in (("ops_instance.cu", "ops"), ("bwd_instance.cu", "bwd"))
    for o, on in _OPS for t, tn in _TYPES]


def nvcc() -> str:
    path = shutil.which("nvcc")
    if path:
        return path
    cand = "/usr/local/cuda/bin/nvcc"
    if os.path.exists(cand):
        return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build "
                       "librowop")


def _stamp(extra_flags) -> str:
    h = hashlib.sha256()
    for d in (CSRC, INCLUDE):
        for name in sorted(os.listdir(d)):
            if name.endswith((".cu", ".cuh", ".h")):
                with open(os.path.join(d, name), "rb") as f:
                    h.update(name.encode())
                    h.update(f.read())
    h.update(" ".join(NVCC_FLAGS + list(extra_flags)).encode())
    return h.hexdigest()


def build(force: bool = False, extra_flags=(), verbose: bool = False) -> str:
    """Compile and link librowop.so; returns its path."""
    os.makedirs(BUILD, exist_ok=True)
    stamp_path = os.path.join(BUILD, "librowop.stamp")
    stamp = _stamp(extra_flags)
    if (not force and os.path.exists(LIB) and os.path.exists(stamp_path)
            and open(stamp_path).read() == stamp):
        return LIB
    cc = nvcc()

    def compile_one(unit):
        name, objname, defs = unit
        src = os.path.join(CSRC, name)
        obj = os.path.join(BUILD, objname)
        cmd = [cc] + NVCC_FLAGS + defs + list(extra_flags) + ["-c", src, "-o", obj]
        if verbose:
            print(" ".join(cmd))
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {objname}:\n{r.stderr}")
        return obj, r.stderr

    with cf.ThreadPoolExecutor(max_workers=min(len(UNITS), os.cpu_count() or 4)) as ex:
        results = list(ex.map(compile_one, UNITS))
    objs = [o for o, _ in results]
    if verbose:
        for _, err in results:
            if err.strip():
                print(err)
    tmp = LIB + f".tmp{os.getpid()}"
    cmd = [cc] + ARCH + ["-shared", "-cudart", "static", "-o", tmp] + objs
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"link failed:\n{r.stderr}")
    os.replace(tmp, LIB)
    with open(stamp_path, "w") as f:
        f.write(stamp)
    return LIB


if __name__ == "__main__":
    import sys
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
