"""Build libaloco.so in place (nvcc for sm_103a, g++ for host code).

The translation units compile in parallel; the result is linked with the
static CUDA runtime so the library needs only the driver at run time.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(os.path.dirname(HERE), "include")
LIB = os.path.join(HERE, "libaloco.so")
OBJ_DIR = os.path.join(HERE, "_build")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
              "-Xcompiler", "-Wall", "--expt-relaxed-constexpr"]
CXX_FLAGS = ["-O2", "-std=c++17", "-fPIC", "-Wall", "-Wextra",
             "-Wno-unused-parameter"]


def _cuda_home() -> str:
    home = os.environ.get("CUDA_HOME") or os.environ.get("CUDA_PATH")
    if home:
        return home
    nvcc = shutil.which("nvcc")
    if nvcc:
        return os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))
    return "/usr/local/cuda"


def _sources():
    srcs = sorted(os.listdir(CSRC))
    return ([os.path.join(CSRC, s) for s in srcs if s.endswith(".cu")],
            [os.path.join(CSRC, s) for s in srcs if s.endswith(".cpp")])


def _deps():
    return [os.path.join(CSRC, s) for s in os.listdir(CSRC)] + \
        [os.path.join(INCLUDE, s) for s in os.listdir(INCLUDE)]


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(d) <= t for d in _deps())


def build(force: bool = False, verbose: bool = False, ptxas_info: bool = False,
          out: str = None, defines=()) -> str:
    """Compile and link the library.  `out` and `defines` (e.g.
    ("ALOCO_UNROLL=2",)) build a variant with other tuning knobs into
    another file; the default build uses the knobs' defaults."""
    lib_path = out or LIB
    if not force and out is None and not defines and up_to_date():
        return LIB
    cuda = _cuda_home()
    nvcc = os.path.join(cuda, "bin", "nvcc")
    obj_dir = OBJ_DIR if out is None else lib_path + ".objs"
    os.makedirs(obj_dir, exist_ok=True)
    cu, cpp = _sources()
    jobs = []
    dflags = [f"-D{d}" for d in defines]
    for src in cu:
        obj = os.path.join(obj_dir, os.path.basename(src) + ".o")
        cmd = [nvcc, *ARCH, *NVCC_FLAGS, *dflags, "-I", INCLUDE, "-c", src,
               "-o", obj]
        if ptxas_info:
            cmd[1:1] = ["-Xptxas", "-v"]
        jobs.append((cmd, obj))
    for src in cpp:
        obj = os.path.join(obj_dir, os.path.basename(src) + ".o")
        cmd = ["g++", *CXX_FLAGS, *dflags, "-I", INCLUDE, "-I",
               os.path.join(cuda, "include"), "-c", src, "-o", obj]
        jobs.append((cmd, obj))

    def run(job):
        cmd, _ = job
        if verbose:
            print(" ".join(cmd), file=sys.stderr)
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("compile failed:\n" + " ".join(cmd) + "\n" +
                               r.stdout + r.stderr)
        return r.stdout + r.stderr

    with cf.ThreadPoolExecutor(max_workers=max(1, len(jobs))) as ex:
        logs = list(ex.map(run, jobs))
    if verbose or ptxas_info:
        for log in logs:
            if log:
                print(log, file=sys.stderr)
    tmp = lib_path + ".tmp%d" % os.getpid()
    link = [nvcc, *ARCH, "-shared", "-o", tmp,
            *[obj for _, obj in jobs], "-cudart", "static"]
    r = subprocess.run(link, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("link failed:\n" + " ".join(link) + "\n" +
                           r.stdout + r.stderr)
    os.replace(tmp, lib_path)
    return lib_path


if __name__ == "__main__":
    build(force="--force" in sys.argv, verbose=True,
          ptxas_info="--ptxas" in sys.argv)
    print(LIB)
