"""Host code under AddressSanitizer and UndefinedBehaviorSanitizer (CPU only).

The oracle (plain C) is built with -fsanitize=address,undefined together with a driver that
runs every oracle function on small random families: bf16 and fp32 checkpoints, ragged
tensors, both TIES trim scopes, TIES after masking, every operator, both planning scores and
budgets from zero to above the full read.  The library's host layer (geometry building,
argument checks, catalog import, the no-allocation planner's refusals, the trace API) is
built with the same sanitizers for its host code and driven by the C program of
test_c_abi_from_c.py.  Any out-of-bounds access, use after free, overflow of a signed type
or misaligned access ends the program with a report and a non-zero status."""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SAN = ["-fsanitize=address,undefined", "-fno-sanitize-recover=all", "-fno-omit-frame-pointer", "-g"]
ENV = dict(os.environ, ASAN_OPTIONS="detect_leaks=0:protect_shadow_gap=0", UBSAN_OPTIONS="print_stacktrace=1")

DRIVER = r"""
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>
#include "oracle.h"

static uint64_t rs = 88172645463325252ull;
static uint64_t rnd(void) { rs ^= rs << 13; rs ^= rs >> 7; rs ^= rs << 17; return rs; }
static float unif(void) { return (float)((rnd() >> 11) * (1.0 / 9007199254740992.0)) * 2.0f - 1.0f; }

static int run(int dtype) {
  enum { K = 3, NT = 3 };
  const uint64_t numel[NT] = {5000, 777, 4096};
  const uint32_t be = 1024;
  uint64_t t_off[NT], n = 0;
  for (int t = 0; t < NT; ++t) { t_off[t] = n; n += (numel[t] + 7) / 8 * 8; }
  uint64_t nb = 0;
  for (int t = 0; t < NT; ++t) nb += (numel[t] + be - 1) / be;
  uint64_t* off = malloc(nb * 8);
  uint32_t *len = malloc(nb * 4), *grp = malloc(nb * 4), *grp1 = malloc(nb * 4), *tens = malloc(nb * 4);
  uint64_t b = 0;
  for (int t = 0; t < NT; ++t)
    for (uint64_t s = 0; s < numel[t]; s += be, ++b) {
      off[b] = t_off[t] + s;
      len[b] = (uint32_t)(numel[t] - s < be ? numel[t] - s : be);
      grp[b] = (uint32_t)t;
      grp1[b] = 0;
      tens[b] = (uint32_t)t;
    }
  const size_t es = dtype == ORC_BF16 ? 2 : 4;
  void* base = calloc(n, es);
  void* ex[K];
  for (int i = 0; i < K; ++i) ex[i] = calloc(n, es);
  for (uint64_t j = 0; j < n; ++j) {
    const float x = unif();
    if (dtype == ORC_BF16) ((uint16_t*)base)[j] = orc_f32_to_bf16(x); else ((float*)base)[j] = x;
    for (int i = 0; i < K; ++i) {
      const float y = (rnd() % 4 == 0) ? x : x + 0.01f * unif();  /* some exact zeros */
      if (dtype == ORC_BF16) ((uint16_t*)ex[i])[j] = orc_f32_to_bf16(y); else ((float*)ex[i])[j] = y;
    }
  }
  orc_family f = {dtype, K, nb, off, len, grp, NT, base, (const void* const*)ex};
  orc_family f1 = f;
  f1.blk_group = grp1;
  f1.n_groups = 1;
  float* norm = malloc(K * nb * 4);
  float* mx = malloc(K * nb * 4);
  uint32_t* nnz = malloc(K * nb * 4);
  uint32_t tau[K * NT], tau1[K];
  if (orc_index(&f, norm, mx, nnz)) return 1;
  if (orc_ties_thresholds(&f, 0.2f, tau) || orc_ties_thresholds(&f1, 0.5f, tau1)) return 2;
  uint64_t* bh = malloc(nb * 8);
  uint64_t* eh = malloc(K * nb * 8);
  if (orc_index_hashes(&f, bh, eh)) return 3;
  const float alpha[K] = {0.5f, 0.3f, 0.2f};
  const int kinds[7] = {ORC_AVG, ORC_TA, ORC_TIES, ORC_DARE, ORC_AVG_RENORM, ORC_DARE_TIES, ORC_TIES_MASKED};
  uint32_t* mask = malloc(nb * 4);
  uint32_t* order = malloc(K * nb * 4);
  void* out = calloc(n, es);
  const uint64_t full = (uint64_t)K * n * es;
  const uint64_t budgets[5] = {0, full / 10, full / 2, full, full * 2};
  for (int q = 0; q < 7; ++q)
    for (int sm = 0; sm < 2; ++sm)
      for (int bi = 0; bi < 5; ++bi) {
        orc_op op;
        memset(&op, 0, sizeof(op));
        op.kind = kinds[q];
        op.K = K;
        op.alpha = alpha;
        op.lambda = 1.0f;
        op.density = 0.2f;
        op.drop_p = 0.9;
        op.seed = 1234567;
        op.score_mode = (uint32_t)sm;
        const int ties = op.kind == ORC_TIES || op.kind == ORC_TIES_MASKED;
        uint64_t chat, ns, nc, sh, dg;
        if (orc_plan(K, nb, len, grp, NT, (uint32_t)es, &op, norm, mx, nnz, op.kind == ORC_TIES ? tau : NULL,
                     budgets[bi], mask, &chat, &ns, &nc, &sh, &dg, order, tens, NT))
          return 4;
        const uint32_t* t = tau;
        uint32_t tm[K * NT];
        if (op.kind == ORC_TIES_MASKED) {
          if (orc_ties_masked_thresholds(&f, 0.2f, mask, tm)) return 5;
          t = tm;
        }
        if (orc_merge(&f, &op, ties ? t : NULL, mask, out, nnz)) return 6;
      }
  printf("checksum %llu\n", (unsigned long long)orc_block_hash(out, n * es));
  free(off); free(len); free(grp); free(grp1); free(tens); free(base);
  for (int i = 0; i < K; ++i) free(ex[i]);
  free(norm); free(mx); free(nnz); free(bh); free(eh); free(mask); free(order); free(out);
  return 0;
}

int main(void) {
  int r = run(ORC_BF16);
  if (!r) r = run(ORC_F32);
  printf("result %d\n", r);
  return r;
}
"""


def _need(tool):
    if shutil.which(tool) is None:
        pytest.skip(f"{tool} is not available")


def test_oracle_under_address_and_undefined_behaviour_sanitizers(tmp_path):
    _need("gcc")
    src = tmp_path / "drv.c"
    src.write_text(DRIVER)
    exe = tmp_path / "drv"
    subprocess.check_call(["gcc", "-std=c11", "-O1", "-ffp-contract=off", *SAN, "-I", os.path.join(ROOT, "oracle"),
                           os.path.join(ROOT, "oracle", "oracle.c"), str(src), "-lm", "-o", str(exe)])
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=600, env=ENV)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "result 0" in r.stdout


def test_library_host_layer_under_address_and_undefined_behaviour_sanitizers(tmp_path):
    _need("gcc")
    sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))
    from test_c_abi_from_c import PROGRAM
    from paper_2605_29489_gb300 import build

    nvcc = build.nvcc()
    csrc = os.path.join(ROOT, "paper_2605_29489_gb300", "csrc")
    srcs = sorted(os.path.join(csrc, f) for f in os.listdir(csrc) if f.endswith(".cu"))
    # host compiler options one by one (-Xcompiler splits its argument at commas)
    host_opts = ["-fPIC", "-fsanitize=address", "-fsanitize=undefined", "-fno-sanitize-recover=all",
                 "-fno-omit-frame-pointer"]
    xc = [a for o in host_opts for a in ("-Xcompiler", o)]
    procs = [subprocess.Popen([nvcc, *build.ARCH, "-std=c++17", "-O1", "--expt-relaxed-constexpr", *xc,
                               "-I", os.path.join(ROOT, "include"), "-I", csrc, "-c", s, "-o",
                               str(tmp_path / (os.path.basename(s)[:-3] + ".o"))],
                              stdout=subprocess.PIPE, stderr=subprocess.STDOUT) for s in srcs]
    for p in procs:
        out, _ = p.communicate(timeout=900)
        assert p.returncode == 0, out.decode()
    lib = tmp_path / "libmergepipe_san.so"
    subprocess.check_call([nvcc, *build.ARCH, "-shared", "-o", str(lib), *[str(tmp_path / (os.path.basename(s)[:-3] + ".o"))
                                                                           for s in srcs],
                           "-cudart", "static", *xc[2:]])
    src = tmp_path / "abi.c"
    src.write_text(PROGRAM)
    exe = tmp_path / "abi"
    subprocess.check_call(["gcc", "-std=c11", *SAN, "-I", os.path.join(ROOT, "include"), str(src), "-L", str(tmp_path),
                           "-lmergepipe_san", f"-Wl,-rpath,{tmp_path}", "-o", str(exe)])
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=300, env=ENV)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "fails=0" in r.stdout
