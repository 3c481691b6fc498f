"""The checked build (libmergepipe_checked.so, compiled with -DMP_CHECKED).

Its kernels check every range they stream (a block of the catalog pass, a chunk of the
merge, a block of the host-pool gather or of the hash pass) against the block table, the
launch's block range, the buffers' extents, the 16-byte alignment of bulk copies and the
number of experts before touching it, and the planner checks every compaction slot and unit
id it writes; a range that fails is skipped and reported through the call's error word.

CPU: the predicate itself on hand-made ranges, each case written out with the outcome it must
have; the checked library exports what the header declares.  GPU: the parity cases of the
catalog, plan, merge, host-pool, hash and touched-only tests run again through the checked
library (a child process with MERGEPIPE_CHECKED=1): every check passes on valid inputs, so
every result must still equal the oracle's and no call may report a failed check."""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2605_29489_gb300", "csrc")

# (label, b, b_begin, b_end, blk_off, blk_len, off, n, experts, K, elem_size, x_origin, span, x_span, expected)
CASES = [
    ("a whole block", 3, 0, 10, 4096, 4096, 4096, 4096, 0b101, 3, 2, 0, 1 << 20, 1 << 20, 1),
    ("a chunk inside a block", 3, 0, 10, 4096, 4096, 6144, 2048, 0b1, 3, 2, 0, 1 << 20, 1 << 20, 1),
    ("an empty range at the block's end", 3, 0, 10, 4096, 4096, 8192, 0, 0b1, 3, 2, 0, 1 << 20, 1 << 20, 1),
    ("the base alone (no experts)", 3, 0, 10, 4096, 4096, 4096, 4096, 0, 3, 2, 1 << 30, 1 << 20, 0, 1),
    ("all 32 experts", 0, 0, 1, 0, 64, 0, 64, 0xFFFFFFFF, 32, 4, 0, 64, 64, 1),
    ("a host-pool segment's staging", 7, 5, 9, 70000, 1000, 70000, 1000, 0b11, 2, 2, 69000, 1 << 20, 2000, 1),
    ("block below the launch's range", 4, 5, 9, 70000, 1000, 70000, 1000, 0b11, 2, 2, 69000, 1 << 20, 2000, 0),
    ("block at the launch's end", 9, 5, 9, 70000, 1000, 70000, 1000, 0b11, 2, 2, 69000, 1 << 20, 2000, 0),
    ("range starting before its block", 3, 0, 10, 4096, 4096, 4088, 8, 0b1, 3, 2, 0, 1 << 20, 1 << 20, 0),
    ("range running past its block", 3, 0, 10, 4096, 4096, 6144, 2056, 0b1, 3, 2, 0, 1 << 20, 1 << 20, 0),
    ("range starting past its block", 3, 0, 10, 4096, 4096, 8200, 0, 0b1, 3, 2, 0, 1 << 20, 1 << 20, 0),
    ("block past the buffers' span", 3, 0, 10, 4096, 4096, 4096, 4096, 0b1, 3, 2, 0, 8000, 1 << 20, 0),
    ("start not on a 16-byte boundary (bf16)", 3, 0, 10, 4100, 4096, 4100, 4096, 0b1, 3, 2, 0, 1 << 20, 1 << 20, 0),
    ("start not on a 16-byte boundary (fp32)", 3, 0, 10, 4098, 4096, 4098, 4096, 0b1, 3, 4, 0, 1 << 20, 1 << 20, 0),
    ("an expert bit at K", 3, 0, 10, 4096, 4096, 4096, 4096, 0b1000, 3, 2, 0, 1 << 20, 1 << 20, 0),
    ("experts before the staging's origin", 7, 5, 9, 68000, 1000, 68000, 1000, 0b1, 2, 2, 69000, 1 << 20, 2000, 0),
    ("experts past the staging's end", 7, 5, 9, 70000, 1000, 70600, 400, 0b1, 2, 2, 69000, 1 << 20, 1500, 0),
    ("the same range read from the base only", 7, 5, 9, 70000, 1000, 70600, 400, 0, 2, 2, 69000, 1 << 20, 1500, 1),
    ("an offset whose byte address wraps", 3, 0, 10, (1 << 63) + 8, 16, (1 << 63) + 8, 16, 0, 3, 2, 0, (1 << 64) - 1,
     0, 0),
]

PROGRAM = r"""
#include <stdio.h>
#include "checked.cuh"
using namespace mp;
struct Case { const char* label; unsigned long long b, b0, b1, blk_off; unsigned blk_len; unsigned long long off;
              unsigned n; unsigned long long experts; unsigned K, es; unsigned long long x_origin, span, x_span;
              int want; };
static const Case cases[] = {
%s
};
int main() {
  int fails = 0;
  for (const Case& c : cases) {
    const Extents x{c.span, c.x_span};
    const int got = chunk_in_bounds(c.b, c.b0, c.b1, c.blk_off, c.blk_len, c.off, c.n, c.experts, c.K, c.es,
                                    c.x_origin, x) ? 1 : 0;
    if (got != c.want) { printf("FAIL %%s: got %%d\n", c.label, got); ++fails; }
  }
  /* expert runs */
  if (expert_run(0, 3) != 0x7ull || expert_run(4, 4) != 0xF0ull || expert_run(0, 32) != 0xFFFFFFFFull ||
      expert_run(5, 0) != 0ull || expert_run(64, 1) != ~0ull) { printf("FAIL expert_run\n"); ++fails; }
  printf("fails=%%d\n", fails);
  return fails != 0;
}
"""


def test_chunk_check_predicate(tmp_path):
    from paper_2605_29489_gb300 import build
    lines = []
    for (label, b, b0, b1, blk_off, blk_len, off, n, ex, K, es, x0, span, x_span, want) in CASES:
        lines.append(f'  {{"{label}", {b}ull, {b0}ull, {b1}ull, {blk_off}ull, {blk_len}u, {off}ull, {n}u, {ex}ull, '
                     f'{K}u, {es}u, {x0}ull, {span}ull, {x_span}ull, {want}}},')
    src = tmp_path / "chk.cu"
    src.write_text(PROGRAM % "\n".join(lines))
    exe = tmp_path / "chk"
    subprocess.check_call([build.nvcc(), "-std=c++17", "-I", CSRC, str(src), "-o", str(exe)])
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and "fails=0" in r.stdout, r.stdout + r.stderr


def test_checked_library_exports_every_declared_symbol():
    import ctypes

    from paper_2605_29489_gb300 import build
    from test_abi_exports import declared_functions
    lib = build.build_mergepipe(checked=True)
    assert lib.endswith("libmergepipe_checked.so")
    L = ctypes.CDLL(lib)
    missing = [n for n in declared_functions() if not hasattr(L, n)]
    assert not missing, missing
    L.mp_version.restype = ctypes.c_char_p
    assert b"checked" in L.mp_version()


SUBSET = [
    ("tests/test_gpu_parity.py", "small_families or signed or tiny_config or non_anticipation or nonfinite"),
    ("tests/test_gpu_hostpool.py", "small_families"),
    ("tests/test_gpu_ties_window.py", ""),
    ("tests/test_gpu_hashes.py", ""),
    ("tests/test_gpu_touched.py", ""),
    ("tests/test_gpu_fallback.py", "ragged or host_resident"),
]


@pytest.mark.gpu
def test_parity_through_the_checked_build():
    env = dict(os.environ, MERGEPIPE_CHECKED="1")
    v = subprocess.run([sys.executable, "-c", "import paper_2605_29489_gb300 as mp; print(mp.mp_version())"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert v.returncode == 0 and "checked" in v.stdout, v.stdout + v.stderr
    for path, k in SUBSET:
        cmd = [sys.executable, "-m", "pytest", path, "-m", "gpu", "-x", "-q", "-p", "no:cacheprovider"]
        if k:
            cmd += ["-k", k]
        r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=1200)
        assert r.returncode == 0, f"{path} -k '{k}' through the checked build:\n" + (r.stdout + r.stderr)[-4000:]
        assert " passed" in r.stdout and " failed" not in r.stdout, r.stdout[-2000:]
