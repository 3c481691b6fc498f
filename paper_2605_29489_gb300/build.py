"""In-tree build of the native libraries (no cmake, no setuptools).

* ``_build/libmergepipe.so``  — the CUDA path behind ``include/mergepipe.h``
  (every ``csrc/*.cu`` compiled for sm_103a in parallel, then linked);
* ``_build/libmergepipe_checked.so`` — the same sources with ``-DMP_CHECKED``: every
  range a kernel streams is checked against the block table and the buffers first
  (``csrc/checked.cuh``); loaded instead of the default library when the
  environment sets ``MERGEPIPE_CHECKED=1``;
* ``_build/libmpsynth_host.so`` — the synthetic-family host fill (gcc);
* ``_build/libmpsynth_dev.so``  — the synthetic-family device fill (nvcc).

A library is rebuilt when its sources, flags or host machine change (a stamp
file beside it records them).
"""
from __future__ import annotations

import concurrent.futures as cf
import glob
import hashlib
import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
OUT = os.path.join(HERE, "_build")
INCLUDE = os.path.join(ROOT, "include")
CSRC = os.path.join(HERE, "csrc")
SYNTH = os.path.join(HERE, "synth")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-fmad=false", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
              "--expt-relaxed-constexpr", "-Xptxas", "-warn-spills"]


def nvcc() -> str:
    cand = os.environ.get("NVCC") or shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand):
        raise RuntimeError("nvcc not found: the CUDA toolkit is required to build the merge library")
    return cand


def _stamp(paths, flags) -> str:
    h = hashlib.sha256()
    for p in sorted(paths):
        h.update(p.encode())
        with open(p, "rb") as f:
            h.update(f.read())
    h.update(" ".join(flags).encode())
    h.update(os.uname().machine.encode())
    return h.hexdigest()


def _fresh(lib: str, stamp: str) -> bool:
    sp = lib + ".stamp"
    if os.path.exists(lib) and os.path.exists(sp):
        with open(sp) as f:
            return f.read() == stamp
    return False


def _write_stamp(lib: str, stamp: str):
    with open(lib + ".stamp", "w") as f:
        f.write(stamp)


def _run(cmd):
    r = subprocess.run(cmd, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
    if r.returncode != 0:
        raise RuntimeError("build step failed: " + " ".join(cmd) + "\n" + r.stdout)
    return r.stdout


def build_mergepipe(force: bool = False, verbose: bool = False, checked: bool = False) -> str:
    os.makedirs(OUT, exist_ok=True)
    lib = os.path.join(OUT, "libmergepipe_checked.so" if checked else "libmergepipe.so")
    srcs = sorted(glob.glob(os.path.join(CSRC, "*.cu")))
    deps = srcs + sorted(glob.glob(os.path.join(CSRC, "*.cuh"))) + sorted(glob.glob(os.path.join(INCLUDE, "*.h")))
    flags = ARCH + NVCC_FLAGS + (["-DMP_CHECKED"] if checked else [])
    stamp = _stamp(deps, flags)
    if not force and _fresh(lib, stamp):
        return lib
    objs = []
    cmds = []
    for s in srcs:
        o = os.path.join(OUT, os.path.basename(s)[:-3] + (".checked" if checked else "") + f".{os.getpid()}.o")
        objs.append(o)
        cmds.append([nvcc(), *flags, "-I", INCLUDE, "-I", CSRC, "-c", s, "-o", o])
    with cf.ThreadPoolExecutor(max_workers=min(len(cmds), os.cpu_count() or 4)) as ex:
        outs = list(ex.map(_run, cmds))
    if verbose:
        for o in outs:
            if o.strip():
                print(o)
    tmp = lib + f".tmp{os.getpid()}"
    _run([nvcc(), *ARCH, "-shared", "-o", tmp, *objs, "-cudart", "static"])
    os.replace(tmp, lib)
    for o in objs:
        os.remove(o)
    _write_stamp(lib, stamp)
    return lib


def build_synth_host(force: bool = False) -> str:
    os.makedirs(OUT, exist_ok=True)
    lib = os.path.join(OUT, "libmpsynth_host.so")
    srcs = [os.path.join(SYNTH, "synth_host.c")]
    deps = srcs + [os.path.join(SYNTH, "synth_core.h")]
    flags = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-pthread"]
    stamp = _stamp(deps, flags)
    if not force and _fresh(lib, stamp):
        return lib
    tmp = lib + f".tmp{os.getpid()}"
    _run(["gcc", *flags, *srcs, "-o", tmp])
    os.replace(tmp, lib)
    _write_stamp(lib, stamp)
    return lib


def build_synth_dev(force: bool = False) -> str:
    os.makedirs(OUT, exist_ok=True)
    lib = os.path.join(OUT, "libmpsynth_dev.so")
    srcs = [os.path.join(SYNTH, "synth_dev.cu")]
    deps = srcs + [os.path.join(SYNTH, "synth_core.h")]
    flags = ARCH + ["-O3", "-std=c++17", "-fmad=false", "-Xcompiler", "-fPIC", "-shared", "-cudart", "static"]
    stamp = _stamp(deps, flags)
    if not force and _fresh(lib, stamp):
        return lib
    tmp = lib + f".tmp{os.getpid()}"
    _run([nvcc(), *flags, *srcs, "-o", tmp])
    os.replace(tmp, lib)
    _write_stamp(lib, stamp)
    return lib


def build_all(force: bool = False, verbose: bool = False):
    with cf.ThreadPoolExecutor(max_workers=4) as ex:
        fs = [ex.submit(build_mergepipe, force, verbose), ex.submit(build_mergepipe, force, verbose, True),
              ex.submit(build_synth_host, force), ex.submit(build_synth_dev, force)]
        return [f.result() for f in fs]


if __name__ == "__main__":
    for p in build_all(force=True, verbose=True):
        print(p)
