"""Build step of the library: compiles csrc/*.cu for sm_103a with nvcc and links libtss.so in-tree.

Translation units compile in parallel; the object files go to _build/ (git-ignored).
"""
import concurrent.futures
import os
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
LIB = os.path.join(HERE, "libtss.so")
SOURCES = ("api.cu", "gemm.cu", "attention.cu", "attn_tc.cu", "misc.cu", "noalloc.cu", "prefill.cu", "verify_mk.cu")
HEADERS = ("common.cuh", "internal.h", "attn_body.cuh")
ARCH = ("-gencode", "arch=compute_103a,code=sm_103a")
FLAGS = ("-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr")


def nvcc() -> str:
    home = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    path = os.path.join(home, "bin", "nvcc")
    return path if os.path.exists(path) else "nvcc"


def _inputs():
    inc = os.path.join(os.path.dirname(HERE), "include", "tss.h")
    return [os.path.join(CSRC, f) for f in SOURCES + HEADERS] + [inc]


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(p) <= t for p in _inputs())


def build(force: bool = False, verbose: bool = False, extra_flags=()) -> str:
    """Compile and link libtss.so; returns its path.  Raises RuntimeError with nvcc's output."""
    if not force and not extra_flags and up_to_date():
        return LIB
    objdir = os.path.join(os.path.dirname(HERE), "_build")
    os.makedirs(objdir, exist_ok=True)
    jobs = []
    for src in SOURCES:
        obj = os.path.join(objdir, src.replace(".cu", ".o"))
        cmd = [nvcc(), *ARCH, *FLAGS, *extra_flags, "-c", os.path.join(CSRC, src), "-o", obj]
        jobs.append((cmd, obj))

    def run(cmd):
        r = subprocess.run(cmd, capture_output=True, text=True)
        return cmd, r

    objs = []
    with concurrent.futures.ThreadPoolExecutor(max_workers=len(jobs)) as ex:
        for cmd, r in ex.map(lambda j: run(j[0]), jobs):
            if verbose or r.returncode != 0:
                sys.stderr.write(" ".join(cmd) + "\n" + r.stdout + r.stderr)
            if r.returncode != 0:
                raise RuntimeError(f"nvcc failed for {cmd[-3]}:\n{r.stderr[-4000:]}")
    objs = [o for _, o in jobs]
    tmp = LIB + ".tmp"
    libdir = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "lib64")
    link = [nvcc(), *ARCH, "-shared", "-cudart", "shared", *objs, "-Xlinker", "-rpath", "-Xlinker", libdir,
            "-o", tmp]
    r = subprocess.run(link, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("link failed:\n" + r.stderr[-4000:])
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose="-v" in sys.argv,
          extra_flags=("-Xptxas", "-v") if "--ptxas-v" in sys.argv else ())
    print(LIB)
