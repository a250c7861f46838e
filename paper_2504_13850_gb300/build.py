"""Build the C-ABI shared library libfedoptima.so in-tree with nvcc for
sm_103a (GB300).  Sources compile in parallel; objects go to _build/.

Several processes may call build() at once (one per rank under torchrun):
an exclusive file lock serialises them, and every object and the library
are written under a temporary name and renamed into place, so a process
never loads a half-written library."""
from __future__ import annotations

import concurrent.futures as cf
import fcntl
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
OUT = os.path.join(HERE, "libfedoptima.so")
BUILD = os.path.join(HERE, "_build")

SOURCES = ["fo_server.cu", "k_elementwise.cu", "k_simt_conv.cu", "k_attention.cu", "k_tc_gemm.cu", "k_tc_gemm_fwd.cu", "k_tc_gemm_dgrad.cu", "k_tc_gemm_wgrad.cu", "k_head.cu", "k_vec.cu", "fo_noalloc.cu", "k_attention_tc.cu", "fo_preproc.cu", "k_mobile.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
         "-Xcompiler", "-fvisibility=hidden"]


def nvcc():
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


def _compile(src, extra):
    obj = os.path.join(BUILD, os.path.splitext(src)[0] + ".o")
    srcp = os.path.join(CSRC, src)
    deps = [srcp] + [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".h", ".hpp", ".cuh"))]
    deps.append(os.path.join(HERE, "..", "include", "fedoptima.h"))
    if os.path.exists(obj) and all(os.path.getmtime(obj) >= os.path.getmtime(d) for d in deps):
        return obj, ""
    tmp = f"{obj}.{os.getpid()}.tmp"
    cmd = [nvcc(), *ARCH, *FLAGS, *extra, "-c", srcp, "-o", tmp]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        if os.path.exists(tmp):
            os.remove(tmp)
        raise RuntimeError(f"nvcc failed for {src}:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, obj)
    return obj, r.stderr


def build(verbose=False, extra=()):
    os.makedirs(BUILD, exist_ok=True)
    with open(os.path.join(BUILD, ".lock"), "w") as lock:
        try:
            fcntl.flock(lock, fcntl.LOCK_EX)  # released when the file closes
        except OSError:                       # a filesystem without locks: build unserialised
            pass
        with cf.ThreadPoolExecutor(max_workers=min(len(SOURCES), os.cpu_count() or 4)) as ex:
            results = list(ex.map(lambda s: _compile(s, list(extra)), SOURCES))
        objs = [o for o, _ in results]
        if verbose:
            for _, log in results:
                if log:
                    sys.stderr.write(log)
        newest = max(os.path.getmtime(o) for o in objs)
        if not os.path.exists(OUT) or os.path.getmtime(OUT) < newest:
            tmp = f"{OUT}.{os.getpid()}.tmp"
            cmd = [nvcc(), *ARCH, "-shared", "-o", tmp, *objs]
            r = subprocess.run(cmd, capture_output=True, text=True)
            if r.returncode != 0:
                if os.path.exists(tmp):
                    os.remove(tmp)
                raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
            os.replace(tmp, OUT)
    return OUT


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv, extra=[a for a in sys.argv[1:] if a != "-v"]))
