"""The boundary is a plain C ABI: a C program that includes only include/mergepipe.h (no
CUDA or torch header), built with gcc and linked against the library, calls the entry
points that need no GPU and gets the documented results (CPU; no compute call)."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

PROGRAM = r"""
#include <stdio.h>
#include <string.h>
#include "mergepipe.h"

static int fails = 0;
#define CHECK(c) do { if (!(c)) { printf("FAIL line %d: %s\n", __LINE__, #c); ++fails; } } while (0)

int main(void) {
  /* two tensors: 4096 and 300 bf16 elements, the second starting on a 16-byte boundary */
  mp_tensor ts[2] = {{0, 4096}, {4096, 300}};
  static unsigned short base[4400], e0[4400], e1[4400], e2[4400];
  const void* ex[3] = {e0, e1, e2};
  mp_family f;
  memset(&f, 0, sizeof(f));
  f.dtype = MP_BF16;
  f.n_tensors = 2;
  f.tensors = ts;
  f.block_elems = 1024;
  f.base = base;
  f.K = 3;
  f.experts = ex;
  f.experts_location = 0;

  CHECK(strstr(mp_version(), "sm_103a") != NULL);
  const unsigned long long full = 3ull * 4396ull * 2ull;
  CHECK(mp_budget_from_fraction(&f, 1.0) == full);
  CHECK(mp_budget_from_fraction(&f, 0.25) == full / 4);
  CHECK(mp_budget_from_fraction(&f, 7.0) == full);       /* clamped to f = 1 */
  CHECK(mp_budget_from_fraction(&f, -1.0) == 0);

  /* an invalid family gives a budget of 0 */
  mp_family bad = f;
  bad.block_elems = 100;
  CHECK(mp_budget_from_fraction(&bad, 1.0) == 0);

  /* argument errors come back as MP_ERR_INVALID_ARG with a message, before any CUDA call */
  mp_index* ix = (mp_index*)1;
  CHECK(mp_index_blocks(NULL, NULL, NULL, &ix) == MP_ERR_INVALID_ARG && ix == NULL);
  CHECK(strlen(mp_last_error()) > 0);
  /* 5 blocks (4 of tensor 0, 1 of tensor 1), expert-major [3][5] */
  float norm[3 * 5], maxabs[3 * 5];
  uint32_t nnz[3 * 5];
  for (int q = 0; q < 15; ++q) { norm[q] = 1.0f; maxabs[q] = 1.0f; nnz[q] = 3; }
  nnz[14] = 301;  /* expert 2's last block holds 300 elements */
  float alpha[3] = {0.5f, 0.25f, 0.25f};
  mp_op op;
  memset(&op, 0, sizeof(op));
  op.kind = MP_OP_TA;
  op.alpha = alpha;
  CHECK(mp_index_import(&f, &op, norm, maxabs, nnz, NULL, NULL, NULL, NULL, &ix) == MP_ERR_INVALID_ARG);
  CHECK(ix == NULL);
  CHECK(strstr(mp_last_error(), "catalog entry 14") != NULL);

  /* mp_plan_noalloc refuses a misaligned buffer with a literal message */
  uint32_t w[64];
  uint64_t s8[8];
  CHECK(mp_plan_noalloc(3, 6, 1, MP_BF16, w, NULL, (const float*)((char*)w + 2), (const float*)w, w, NULL, w,
                        &op, 1000, w, w, s8, NULL) == MP_ERR_INVALID_ARG);
  CHECK(strstr(mp_last_error(), "aligned") != NULL);

  /* every entry point refuses a NULL handle with MP_ERR_INVALID_ARG and a message */
  uint64_t u64 = 0, u64b = 0;
  uint32_t u32 = 0;
  mp_plan_t* pl = (mp_plan_t*)1;
  mp_manifest* man = (mp_manifest*)1;
  CHECK(mp_plan(NULL, &op, 100, NULL, &pl) == MP_ERR_INVALID_ARG && pl == NULL);
  CHECK(mp_merge(&f, NULL, NULL, base, NULL, &man) == MP_ERR_INVALID_ARG && man == NULL);
  man = (mp_manifest*)1;
  CHECK(mp_merge_touched(&f, NULL, NULL, base, NULL, &man) == MP_ERR_INVALID_ARG && man == NULL);
  CHECK(mp_index_stats(NULL, norm, maxabs, nnz, NULL) == MP_ERR_INVALID_ARG);
  CHECK(mp_index_shape(NULL, &u64, &u64b, &u32) == MP_ERR_INVALID_ARG);
  CHECK(mp_index_hashes(&f, NULL, NULL) == MP_ERR_INVALID_ARG);
  CHECK(mp_index_hash_values(NULL, &u64, &u64b) == MP_ERR_INVALID_ARG);
  CHECK(mp_plan_info(NULL, &u64, &u64b, NULL, NULL, NULL, NULL) == MP_ERR_INVALID_ARG);
  CHECK(mp_manifest_info(NULL, &u64, &u64b, NULL, NULL) == MP_ERR_INVALID_ARG);
  CHECK(mp_manifest_validate(&f, NULL, NULL, base, NULL, NULL) == MP_ERR_INVALID_ARG);
  CHECK(mp_manifest_validation(NULL, &u64, &u64b, NULL) == MP_ERR_INVALID_ARG);
  CHECK(mp_manifest_threshold_reads(NULL, &u64) == MP_ERR_INVALID_ARG);
  CHECK(mp_manifest_lineage(NULL, &u64) == MP_ERR_INVALID_ARG);
  CHECK(strstr(mp_last_error(), "handle") != NULL);
  CHECK(mp_plan_noalloc(3, 6, 1, MP_BF16, w, NULL, (const float*)w, (const float*)w, w, NULL, w, NULL, 1000, w, w, s8,
                        NULL) == MP_ERR_INVALID_ARG);

  /* the trace API checks its arguments on the host; a stop without a start holds nothing */
  CHECK(mp_trace_start(0) == MP_ERR_INVALID_ARG);
  CHECK(mp_trace_start((1u << 20) + 1u) == MP_ERR_INVALID_ARG);
  u64 = 7;
  CHECK(mp_trace_stop(&u64) == MP_OK && u64 == 0);
  CHECK(mp_trace_read(NULL, 1) == MP_ERR_INVALID_ARG);
  CHECK(mp_trace_read(NULL, 0) == MP_OK);

  /* NULL is a no-op for mp_free */
  mp_free(NULL);
  printf("fails=%d\n", fails);
  return fails != 0;
}
"""


def test_c_program_uses_the_abi():
    import paper_2605_29489_gb300 as mp  # noqa: F401  (builds the library if it is stale)
    from paper_2605_29489_gb300 import build

    if shutil.which("gcc") is None:
        pytest.skip("gcc is not available")
    lib = build.build_mergepipe()
    d = os.path.join(ROOT, "paper_2605_29489_gb300", "_build", "c_abi_check")
    os.makedirs(d, exist_ok=True)
    src, exe = os.path.join(d, "abi_check.c"), os.path.join(d, "abi_check")
    with open(src, "w") as f:
        f.write(PROGRAM)
    libdir = os.path.dirname(lib)
    name = os.path.basename(lib)[3:-3]  # libmergepipe.so -> mergepipe
    subprocess.check_call(["gcc", "-std=c11", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"), src,
                           "-L", libdir, f"-l{name}", f"-Wl,-rpath,{libdir}", "-o", exe])
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "fails=0" in r.stdout
