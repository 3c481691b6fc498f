"""Mutation check of the oracle's pins.

Each case plants one plausible mistake in a copy of oracle.c — a dropped term, a wrong
sign, bound or index, a transposed operand, a missed special case — builds the copy and
runs the CPU pins (test_oracle_pins.py) against it in a child process: some pin must
fail.  An unmodified copy, built and run the same way, must pass every pin, so a broken
harness cannot pass for a caught mistake.  oracle.c itself is never changed; the copies
live in a temporary directory.

Left out on purpose: changes that swap one valid reading for another (the hash's key
rotation, the digest's byte layout, which Philox word feeds which element, rounding
p * 65536 down rather than up for the DARE threshold).  Those are
conventions the paper leaves open; the GPU parity tests hold both sides to the one the
implementation states.
"""
import concurrent.futures
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ORACLE_DIR = os.path.join(ROOT, "oracle")
sys.path.insert(0, ROOT)

from oracle import LIBRARY_UNDER_TEST_ENV  # noqa: E402
from oracle import build as oracle_build  # noqa: E402

# (name, text in oracle.c (must occur exactly once), replacement)
MUTANTS = [
    # element conversion
    ("bf16_rounds_half_down",
     "if (lower > 0x8000u || (lower == 0x8000u && (upper & 1u))) upper += 1u;",
     "if (lower > 0x8000u) upper += 1u;"),
    ("ties_key_truncates",
     "return (uint32_t)orc_f32_to_bf16(fabsf(delta)) & 0x7FFFu;",
     "return (f2u(fabsf(delta)) >> 16) & 0x7FFFu;"),
    ("bf16_nan_not_quieted", "return (uint16_t)((u >> 16) | 0x0040u);", "return (uint16_t)(u >> 16);"),
    # block statistics
    ("stats_accept_nonfinite", "    if (!is_finite_f(d)) return ORC_ENONFINITE;\n    float a = fabsf(d);",
     "    float a = fabsf(d);"),
    ("index_block_major", "uint64_t u = (uint64_t)i * f->n_blocks + b;", "uint64_t u = b * f->K + i;"),
    ("norm_without_sqrt", "if (norm) *norm = sqrtf(g[0]);", "if (norm) *norm = g[0];"),
    ("norm_drops_half_the_groups", "for (int s = 4; s >= 1; s >>= 1) {", "for (int s = 2; s >= 1; s >>= 1) {"),
    ("norm_drops_ragged_vector", "const uint64_t nvec = (n + V - 1) / V;", "const uint64_t nvec = n / V;"),
    ("norm_sums_deltas", "acc = fmaf(d, d, acc);", "acc = acc + d;"),
    ("nnz_counts_zeros", "if (d != 0.0f) ++cnt;", "++cnt;"),
    ("maxabs_signed", "float a = fabsf(d);", "float a = d;"),
    # TIES thresholds
    ("tau_off_by_one", "if (cum >= k) return (uint32_t)key;", "if (cum > k) return (uint32_t)key;"),
    ("tau_k_rounds_up", "uint64_t k = (uint64_t)floor((double)density * (double)numel);",
     "uint64_t k = (uint64_t)ceil((double)density * (double)numel);"),
    ("tau_zero_density_keeps_all", "if (k == 0) return ORC_TAU_NONE;", "if (k == 0) return 0;"),
    ("masked_tau_ignores_mask", "if ((mask[b] >> i) & 1u)\n", "if (1)\n"),
    ("masked_tau_omitted_as_largest", "h[0] += f->blk_len[b];", "h[0x7FFF] += f->blk_len[b];"),
    # hashes
    ("fnv1a_wrong_prime", "h *= 1099511628211ULL;", "h *= 1099511628213ULL;"),
    ("splitmix64_wrong_shift", "z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;", "z = (z ^ (z >> 31)) * 0xBF58476D1CE4E5B9ULL;"),
    ("hash_without_length", "return orc_splitmix64(orc_block_hash_sum(bytes, len) ^ len);",
     "return orc_splitmix64(orc_block_hash_sum(bytes, len));"),
    ("hash_even_key", "const uint64_t a = k | 1u,", "const uint64_t a = k,"),
    ("hash_key_not_per_vector", "const uint64_t k = orc_splitmix64(q);", "const uint64_t k = orc_splitmix64(0);"),
    ("index_hashes_block_major", "expert_hash[(uint64_t)i * f->n_blocks + b] = ", "expert_hash[b * f->K + i] = "),
    ("index_hashes_length_in_elements", "const uint64_t len = (uint64_t)f->blk_len[b] * es;",
     "const uint64_t len = (uint64_t)f->blk_len[b];"),
    ("key_hist_accepts_nonfinite", "    if (!is_finite_f(d)) return ORC_ENONFINITE;\n    hist[", "    hist["),
    # Alg. 1 plan
    ("plan_stops_at_first_overflow", "if (chat + q[r].cost <= budget) {",
     "if (chat + q[r].cost > budget) break;\n    {"),
    ("plan_strict_budget", "if (chat + q[r].cost <= budget) {", "if (chat + q[r].cost < budget) {"),
    ("plan_ascending_score", "if (x->score > y->score) return -1;\n  if (x->score < y->score) return 1;",
     "if (x->score < y->score) return -1;\n  if (x->score > y->score) return 1;"),
    ("plan_ties_broken_by_descending_unit", "return x->unit < y->unit ? -1 : (x->unit > y->unit ? 1 : 0);",
     "return x->unit > y->unit ? -1 : (x->unit < y->unit ? 1 : 0);"),
    ("plan_score_without_coefficient", "q[nq].score = fabsf(coef) * norm[s];", "q[nq].score = norm[s];"),
    ("plan_score_signed_coefficient", "q[nq].score = fabsf(coef) * norm[s];", "q[nq].score = coef * norm[s];"),
    ("plan_zero_blocks_are_candidates", "if (nnz[s] == 0) continue;", ""),
    ("plan_no_ties_pruning", "if (op->kind == ORC_TIES && orc_ties_key(maxabs[s])",
     "if (0 && orc_ties_key(maxabs[s])"),
    ("plan_ties_tau_of_first_group", "orc_ties_key(maxabs[s]) < tau[(size_t)i * n_groups + blk_group[b]]",
     "orc_ties_key(maxabs[s]) < tau[(size_t)i * n_groups]"),
    ("plan_ties_prunes_at_tau", "orc_ties_key(maxabs[s]) < tau[", "orc_ties_key(maxabs[s]) <= tau["),
    ("plan_unit_id_expert_major",
     "q[nq].unit = (uint32_t)(b * K + i);\n      q[nq].cost = (uint64_t)blk_len[b] * elem_size;",
     "q[nq].unit = (uint32_t)(i * n_blocks + b);\n      q[nq].cost = (uint64_t)blk_len[b] * elem_size;"),
    ("plan_score_per_byte_multiplies",
     "if (op->score_mode) q[nq].score = q[nq].score / (float)q[nq].cost;",
     "if (op->score_mode) q[nq].score = q[nq].score * (float)q[nq].cost;"),
    ("plan_cost_in_elements", "q[nq].cost = (uint64_t)blk_len[b] * elem_size;\n      if (op->score_mode)",
     "q[nq].cost = (uint64_t)blk_len[b];\n      if (op->score_mode)"),
    ("plan_set_hash_of_block", "set_hash += orc_splitmix64(q[r].unit);", "set_hash += orc_splitmix64(b);"),
    # tensor-level fallback
    ("fallback_sums_norms", "if (nnz[s2] != ORC_NNZ_MISSING) ss = fmaf(norm[s2], norm[s2], ss);",
     "if (nnz[s2] != ORC_NNZ_MISSING) ss = ss + norm[s2];"),
    ("fallback_masks_first_block_only",
     "for (uint64_t b2 = b; b2 < n_blocks && blk_tensor[b2] == blk_tensor[b]; ++b2) mask[b2] |= 1u << i;",
     "mask[b] |= 1u << i;"),
    ("fallback_cost_of_last_block", "cost += (uint64_t)blk_len[b2] * elem_size;",
     "cost = (uint64_t)blk_len[b2] * elem_size;"),
    ("fallback_one_unit_per_block", "if (b > 0 && blk_tensor[b - 1] == t) continue;", ""),
    ("fallback_unit_of_wrong_expert", "q[nq].unit = (uint32_t)(b * K + i);\n        q[nq].cost = cost;",
     "q[nq].unit = (uint32_t)(b * K + (K - 1 - i));\n        q[nq].cost = cost;"),
    ("fallback_per_byte_of_first_block", "if (op->score_mode) q[nq].score = q[nq].score / (float)cost;",
     "if (op->score_mode) q[nq].score = q[nq].score / (float)(blk_len[b] * elem_size);"),
    ("fallback_norm_includes_missing_entries", "if (nnz[s2] != ORC_NNZ_MISSING) ss = fmaf(norm[s2], norm[s2], ss);",
     "ss = fmaf(norm[s2], norm[s2], ss);"),
    ("fallback_without_coefficient", "q[nq].score = fabsf(coef) * sqrtf(ss);", "q[nq].score = sqrtf(ss);"),
    # Philox and DARE
    ("philox_multiplies_wrong_word", "uint64_t p0 = (uint64_t)0xD2511F53u * c0;",
     "uint64_t p0 = (uint64_t)0xD2511F53u * c1;"),
    ("philox_bumps_key_before_round_0", "if (r > 0) {\n      k0 += 0x9E3779B9u;", "{\n      k0 += 0x9E3779B9u;"),
    ("philox_output_words_swapped", "out[0] = c0;\n  out[1] = c1;", "out[0] = c1;\n  out[1] = c0;"),
    ("philox_nine_rounds", "for (int r = 0; r < 10; ++r) {", "for (int r = 0; r < 9; ++r) {"),
    ("dare_scales_by_keep_probability", "float sigma = op->drop_p < 1.0 ? (float)(1.0 / (1.0 - op->drop_p)) : 0.0f;",
     "float sigma = op->drop_p < 1.0 ? (float)(1.0 - op->drop_p) : 0.0f;"),
    ("dare_drops_at_threshold", "return r >= dare_threshold(p);", "return r > dare_threshold(p);"),
    ("dare_element_counter_restarts_per_block",
     "int rc = orc_merge_block(f->dtype, f->blk_len[b], off,", "int rc = orc_merge_block(f->dtype, f->blk_len[b], 0,"),
    ("dare_same_mask_for_every_expert", "uint32_t ctr[4] = {(uint32_t)g, (uint32_t)(g >> 32), expert, 0x44415245u};",
     "uint32_t ctr[4] = {(uint32_t)g, (uint32_t)(g >> 32), 0u, 0x44415245u};"),
    # operators (Eq. 4, App. A.1)
    ("avg_ignores_mask", "if (!((mask >> i) & 1u)) continue; /* omitted: zero entry, never read */",
     "if (!((mask >> i) & 1u) && !experts[i]) continue;"),
    ("avg_without_coefficient", "acc = fmaf(coef, d, acc);", "acc = acc + d;"),
    ("avg_delta_sign", "float d = load_elem(dtype, experts[i], k) - x0;\n        if (op->kind == ORC_DARE)",
     "float d = x0 - load_elem(dtype, experts[i], k);\n        if (op->kind == ORC_DARE)"),
    ("ties_elects_positive_on_balance", "if (P > -Nn) m = P / (float)cp;", "if (P >= -Nn) m = P / (float)cp;"),
    ("ties_mean_over_all_kept", "if (P > -Nn) m = P / (float)cp;", "if (P > -Nn) m = P / (float)(cp + cn);"),
    ("ties_sums_instead_of_mean", "if (P > -Nn) m = P / (float)cp;", "if (P > -Nn) m = P;"),
    ("ties_trims_at_tau", "if (orc_ties_key(d) >= tau_k[i]) dh = d;", "if (orc_ties_key(d) > tau_k[i]) dh = d;"),
    ("ties_ignores_mask", "if ((mask >> i) & 1u) {\n          float d", "if (((mask >> i) & 1u) || experts[i]) {\n          float d"),
    ("ties_without_lambda", "res = fmaf(op->lambda, m, x0);", "res = x0 + m;"),
    ("ties_elects_by_count", "if (P > -Nn) m = P / (float)cp;\n      else if (P < -Nn) m = Nn / (float)cn;",
     "if (cp > cn) m = P / (float)cp;\n      else if (cp < cn) m = Nn / (float)cn;"),
    ("dare_ties_trims", "} else if (orc_dare_keep(op->seed, i, j0 + k, op->drop_p)) {",
     "} else if (orc_ties_key(d) >= 0x3F80u) {"),
    ("renorm_ignores_known_zero", "if (((mask | known_zero) >> i) & 1u) {", "if ((mask >> i) & 1u) {"),
    ("renorm_accepts_nonpositive_alpha", "        if (!(op->alpha[i] > 0.0f)) return ORC_EINVAL;\n", ""),
    ("renorm_not_normalised", "op->kind == ORC_AVG_RENORM ? op->alpha[i] / s_sel : op->alpha[i];",
     "op->alpha[i];"),
    ("merge_tau_of_first_group", "tau_k[i] = tau[(size_t)i * f->n_groups + f->blk_group[b]];",
     "tau_k[i] = tau[(size_t)i * f->n_groups];"),
    ("merge_leaves_untouched_blocks_empty", "    int rc = orc_merge_block(f->dtype, f->blk_len[b], off,",
     "    if (mask && !mask[b]) continue;\n    int rc = orc_merge_block(f->dtype, f->blk_len[b], off,"),
    ("ties_negative_mean_over_positive_count", "else if (P < -Nn) m = Nn / (float)cn;",
     "else if (P < -Nn) m = Nn / (float)(cp > 0 ? cp : 1);"),
    ("renorm_sums_every_coefficient", "if (((mask | known_zero) >> i) & 1u) {", "if (1) {"),
    ("dare_ties_without_rescale", "            dh = d * sigma;\n", "            dh = d;\n"),
    ("full_read_mask_drops_last_expert", "((1u << f->K) - 1u);", "((1u << f->K) - 1u) >> 1;"),
    ("dare_counter_block_local_in_merge", "} else if (orc_dare_keep(op->seed, i, j0 + k, op->drop_p)) {",
     "} else if (orc_dare_keep(op->seed, i, k, op->drop_p)) {"),
    ("dare_adds_the_zero_of_a_dropped_entry",
     "if (!orc_dare_keep(op->seed, i, j0 + k, op->drop_p)) continue; /* dropped: omitted */\n          d = d * sigma;",
     "d = orc_dare_keep(op->seed, i, j0 + k, op->drop_p) ? d * sigma : 0.0f;"),
    ("merge_known_zero_from_nonzero", "if (nnz[(size_t)i * f->n_blocks + b] == 0) known_zero |= 1u << i;",
     "if (nnz[(size_t)i * f->n_blocks + b] != 0) known_zero |= 1u << i;"),
]

PIN_FILE = os.path.join(ROOT, "tests", "test_oracle_pins.py")


def _build_copy(d, name, old, new):
    with open(os.path.join(ORACLE_DIR, "oracle.c")) as f:
        src = f.read()
    if old is not None:
        assert src.count(old) == 1, f"{name}: the text to change occurs {src.count(old)} times in oracle.c"
        src = src.replace(old, new)
    os.makedirs(d, exist_ok=True)
    c = os.path.join(d, "oracle.c")
    with open(c, "w") as f:
        f.write(src)
    so = os.path.join(d, "liboracle.so")
    flags = [x for x in oracle_build.CFLAGS if x not in ("-Wall", "-Wextra")]
    subprocess.check_call(["gcc", *flags, "-I", ORACLE_DIR, c, "-o", so, "-lm"])
    return so


def _run_pins(so):
    env = dict(os.environ)
    env[LIBRARY_UNDER_TEST_ENV] = so
    r = subprocess.run([sys.executable, "-m", "pytest", PIN_FILE, "-x", "-q", "-p", "no:cacheprovider"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return r.returncode, (r.stdout + r.stderr)[-3000:]


@pytest.fixture(scope="module")
def outcomes(tmp_path_factory):
    root = tmp_path_factory.mktemp("oracle_mutants")
    cases = [("unmodified", None, None)] + MUTANTS
    libs = {name: _build_copy(str(root / name), name, old, new) for name, old, new in cases}
    workers = max(1, min(8, os.cpu_count() or 1))
    with concurrent.futures.ThreadPoolExecutor(workers) as ex:
        futs = {name: ex.submit(_run_pins, so) for name, so in libs.items()}
        return {name: f.result() for name, f in futs.items()}


def test_unmodified_copy_passes_every_pin(outcomes):
    rc, out = outcomes["unmodified"]
    assert rc == 0, out


@pytest.mark.parametrize("name", [m[0] for m in MUTANTS])
def test_a_pin_catches_the_planted_mistake(outcomes, name):
    assert outcomes["unmodified"][0] == 0, "the harness itself fails"
    rc, out = outcomes[name]
    assert rc != 0, f"every pin passes with the mistake '{name}' planted in the oracle"
    assert rc == 1, f"the pins did not run to a verdict with '{name}' planted (exit {rc}):\n{out}"
