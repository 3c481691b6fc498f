"""Register spills of the default library (CPU: ptxas resource reports, no GPU).

Every kernel of the default build keeps its working set in registers — ptxas reports 0 bytes
of spill stores and loads — except one known case: the streaming TIES merge for bf16
(`merge_tma_kernel<true, TIES>`, launched only for TIES with more than 8 experts) spills 60
bytes of stores and 32 of loads at its register cap.  A change that makes another kernel
spill, or this one spill more (a larger unroll, another live array), slows it without changing
any result, so the parity tests would not notice; this test does.  The checked build
(-DMP_CHECKED) is not held to this."""
import concurrent.futures as cf
import glob
import os
import re
import subprocess

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2605_29489_gb300", "csrc")


def _report(src, out_dir):
    from paper_2605_29489_gb300 import build
    flags = [f for f in build.NVCC_FLAGS if f != "-lineinfo"]
    o = os.path.join(out_dir, os.path.basename(src) + ".o")
    r = subprocess.run([build.nvcc(), *build.ARCH, *flags, "-Xptxas", "-v", "-I", os.path.join(ROOT, "include"),
                        "-I", CSRC, "-c", src, "-o", o], capture_output=True, text=True)
    assert r.returncode == 0, r.stdout + r.stderr
    return r.stdout + r.stderr


# (mangled-name pattern, most spill-store bytes, most spill-load bytes) of the known case
ALLOWED = [(r"merge_tma_kernelILb1ELi1EE", 60, 32)]


def test_default_build_kernels_do_not_spill(tmp_path):
    srcs = sorted(glob.glob(os.path.join(CSRC, "*.cu")))
    with cf.ThreadPoolExecutor(max_workers=min(len(srcs), os.cpu_count() or 4)) as ex:
        reports = dict(zip(srcs, ex.map(lambda s: _report(s, str(tmp_path)), srcs)))
    n_kernels = 0
    spilling = []
    for src, rep in reports.items():
        entry = None
        for line in rep.splitlines():
            m = re.search(r"ptxas info\s*: Compiling entry function '([^']+)'", line)
            if m:
                entry = m.group(1)
                n_kernels += 1
                continue
            m = re.search(r"^\s*\d+ bytes stack frame, (\d+) bytes spill stores, (\d+) bytes spill loads", line)
            if m and entry and (int(m.group(1)) or int(m.group(2))):
                st, ld = int(m.group(1)), int(m.group(2))
                if not any(re.search(pat, entry) and st <= a and ld <= b for pat, a, b in ALLOWED):
                    spilling.append((os.path.basename(src), entry, st, ld))
    assert n_kernels >= 20, f"only {n_kernels} kernels reported"
    assert not spilling, spilling
