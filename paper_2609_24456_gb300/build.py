"""Compile libedp.so (sm_103a) in-tree with nvcc.

Each translation unit under csrc/ is compiled in parallel, then linked into
``paper_2609_24456_gb300/libedp.so`` (CUDA runtime linked statically, so the
library depends only on the driver).  Objects go to ``_build/``.
"""
import concurrent.futures as cf
import glob
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libedp.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
              "-Xcompiler", "-ffp-contract=off", "-Xcompiler",
              "-fvisibility=hidden", "--expt-relaxed-constexpr",
              "-I", INCLUDE, "-I", CSRC]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"),
                 "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: libedp needs the CUDA toolkit")


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return (_sources() + glob.glob(os.path.join(CSRC, "*.cuh"))
            + [os.path.join(INCLUDE, "edp.h"), os.path.abspath(__file__)])


def _stale(target, deps):
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, verbose: bool = False, ptxas_v: bool = False) -> str:
    deps = _deps()
    if not force and not _stale(LIB, deps):
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    cc = nvcc()
    headers = glob.glob(os.path.join(CSRC, "*.cuh")) + [os.path.join(INCLUDE, "edp.h")]

    def compile_one(src):
        obj = os.path.join(BUILD, os.path.basename(src)[:-3] + ".o")
        if not force and not _stale(obj, [src] + headers + [os.path.abspath(__file__)]):
            return obj, ""
        cmd = [cc] + ARCH + NVCC_FLAGS + (["-Xptxas", "-v"] if ptxas_v else []) + [
            "-c", src, "-o", obj]
        p = subprocess.run(cmd, capture_output=True, text=True)
        if p.returncode != 0:
            raise RuntimeError("nvcc failed for %s:\n%s%s" % (src, p.stdout, p.stderr))
        return obj, p.stdout + p.stderr

    with cf.ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 2)) as ex:
        results = list(ex.map(compile_one, _sources()))
    if verbose or ptxas_v:
        for obj, log in results:
            if log:
                print(log)
    objs = [o for o, _ in results]
    tmp = LIB + ".tmp.%d" % os.getpid()
    cmd = [cc] + ARCH + ["-shared", "-cudart", "static", "-o", tmp] + objs + ["-ldl"]
    p = subprocess.run(cmd, capture_output=True, text=True)
    if p.returncode != 0:
        raise RuntimeError("link failed:\n%s%s" % (p.stdout, p.stderr))
    os.replace(tmp, LIB)
    return LIB


PROBE_SRC = os.path.join(ROOT, "tests", "curand_philox_probe.cu")
PROBE_LIB = os.path.join(ROOT, "tests", "_build", "curand_philox_probe.so")


def build_curand_probe(force: bool = False) -> str:
    """Compile the tests' cuRAND Philox probe (test infrastructure, not part
    of libedp) with the same nvcc and target."""
    if not force and not _stale(PROBE_LIB, [PROBE_SRC, os.path.abspath(__file__)]):
        return PROBE_LIB
    os.makedirs(os.path.dirname(PROBE_LIB), exist_ok=True)
    tmp = PROBE_LIB + ".tmp.%d" % os.getpid()
    cmd = [nvcc()] + ARCH + ["-O2", "-shared", "-Xcompiler", "-fPIC", PROBE_SRC, "-o", tmp]
    p = subprocess.run(cmd, capture_output=True, text=True)
    if p.returncode != 0:
        raise RuntimeError("nvcc failed for %s:\n%s%s" % (PROBE_SRC, p.stdout, p.stderr))
    os.replace(tmp, PROBE_LIB)
    return PROBE_LIB


WAIT_PROBE_SRC = os.path.join(ROOT, "tests", "mbar_wait_probe.cu")
WAIT_PROBE_LIB = os.path.join(ROOT, "tests", "_build", "mbar_wait_probe.so")


def build_wait_probe(force: bool = False) -> str:
    """Compile the tests' bounded-wait probe (test infrastructure, not part
    of libedp): libedp's mbarrier wait helper run on its own."""
    deps = [WAIT_PROBE_SRC, os.path.join(CSRC, "edp_internal.cuh"), os.path.abspath(__file__)]
    if not force and not _stale(WAIT_PROBE_LIB, deps):
        return WAIT_PROBE_LIB
    os.makedirs(os.path.dirname(WAIT_PROBE_LIB), exist_ok=True)
    tmp = WAIT_PROBE_LIB + ".tmp.%d" % os.getpid()
    cmd = [nvcc()] + ARCH + ["-O2", "-std=c++17", "-shared", "-Xcompiler", "-fPIC",
                             "-I", INCLUDE, "-I", CSRC, WAIT_PROBE_SRC, "-o", tmp]
    p = subprocess.run(cmd, capture_output=True, text=True)
    if p.returncode != 0:
        raise RuntimeError("nvcc failed for %s:\n%s%s" % (WAIT_PROBE_SRC, p.stdout, p.stderr))
    os.replace(tmp, WAIT_PROBE_LIB)
    return WAIT_PROBE_LIB


if __name__ == "__main__":
    print(build(force="--force" in sys.argv, verbose=True,
                ptxas_v="--ptxas-v" in sys.argv))
