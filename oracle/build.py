"""Build the CPU oracle (plain C, gcc) into oracle/_build/liboracle.so.

Test infrastructure: compiled with -ffp-contract=off so that no multiply-add is
fused unless the source calls fmaf, and without fast-math.
"""
import hashlib
import os
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
OUT_DIR = os.path.join(HERE, "_build")
SOURCES = [os.path.join(HERE, "oracle.c")]
HEADERS = [os.path.join(HERE, "oracle.h")]
CFLAGS = ["-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared", "-Wall", "-Wextra"]


def _stamp() -> str:
    h = hashlib.sha256()
    for p in SOURCES + HEADERS:
        with open(p, "rb") as f:
            h.update(f.read())
    h.update(" ".join(CFLAGS).encode())
    h.update(os.uname().machine.encode())
    return h.hexdigest()


def build(force: bool = False) -> str:
    os.makedirs(OUT_DIR, exist_ok=True)
    lib = os.path.join(OUT_DIR, "liboracle.so")
    stamp_path = lib + ".stamp"
    stamp = _stamp()
    if not force and os.path.exists(lib) and os.path.exists(stamp_path):
        with open(stamp_path) as f:
            if f.read() == stamp:
                return lib
    tmp = lib + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", *CFLAGS, *SOURCES, "-o", tmp, "-lm"])
    os.replace(tmp, lib)
    with open(stamp_path, "w") as f:
        f.write(stamp)
    return lib


if __name__ == "__main__":
    print(build(force=True))
