"""Build libumim.so in-tree for sm_103a with nvcc (no cmake, no torch extension).

Every .cu file under csrc/ is compiled in parallel to an object file, then the
objects are linked into paper_2609_27233_gb300/libumim.so.  The same sources
compiled with UMIM_DEBUG defined (device-side checks at the kernels' access
sites) are linked into paper_2609_27233_gb300/libumim_debug.so; both variants
are compiled in one pool.
"""
import concurrent.futures
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
OUT = os.path.join(HERE, "libumim.so")
OUT_DEBUG = os.path.join(HERE, "libumim_debug.so")
BUILD = os.path.join(ROOT, "_build")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-O2", "--expt-relaxed-constexpr",
         "-I" + os.path.join(ROOT, "include")]


def nvcc():
    for c in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found")


def sources():
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))


VARIANTS = {
    "release": (OUT, BUILD, []),
    "debug": (OUT_DEBUG, os.path.join(BUILD, "debug"), ["-DUMIM_DEBUG"]),
}


def build(verbose: bool = False, extra=None, variants=("release", "debug")) -> str:
    """Compile and link the requested variants; returns the release library's path."""
    cc = nvcc()
    extra = list(extra or [])

    def one(job):
        src, bdir, defs = job
        obj = os.path.join(bdir, os.path.basename(src) + ".o")
        cmd = [cc, *ARCH, *FLAGS, *defs, *extra, "-c", src, "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed for {src} {' '.join(defs)}:\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            sys.stderr.write(r.stdout + r.stderr)
        return obj

    jobs = {}
    for v in variants:
        out, bdir, defs = VARIANTS[v]
        os.makedirs(bdir, exist_ok=True)
        jobs[v] = [(src, bdir, defs) for src in sources()]
    flat = [j for v in variants for j in jobs[v]]
    with concurrent.futures.ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 4)) as ex:
        objs = list(ex.map(one, flat))
    k = 0
    for v in variants:
        out = VARIANTS[v][0]
        n = len(jobs[v])
        tmp = out + ".tmp"
        cmd = [cc, *ARCH, "-shared", "-o", tmp, *objs[k:k + n]]
        k += n
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stdout}\n{r.stderr}")
        os.replace(tmp, out)
    return OUT


if __name__ == "__main__":
    v = "-v" in sys.argv
    extra = ["-Xptxas", "-v"] if "--ptxas" in sys.argv else None
    which = ("debug",) if "--debug-only" in sys.argv else (("release",) if "--release-only" in sys.argv
                                                           else ("release", "debug"))
    print(build(verbose=v or bool(extra), extra=extra, variants=which))
