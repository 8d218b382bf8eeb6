"""The pins must catch plausible mistakes in the oracle.

Each mutant below is a one-line textual change to a temporary copy of
oracle/bkv_oracle.c (a dropped term, a flipped sign, a wrong index or
aggregation, a transposed pairing).  The copy is compiled on the CPU and the
pin tests of tests/test_oracle_*.py are run against it: at least one must fail
for every mutant.  The committed oracle itself is never modified.
"""
import os
import shutil
import subprocess
import tempfile

import pytest

from oracle import oracle as O
from tests import test_oracle_beacons as TB
from tests import test_oracle_cfps as TC
from tests import test_oracle_numerics as TN
from tests import test_oracle_score_select as TS

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle", "bkv_oracle.c")

_SCORE = [(TS.test_score_matches_scipy_softmax_max, dict(M=3, L=50, d=8)),
          (TS.test_score_two_key_logistic_closed_form, {}), (TS.test_golden_worked_case, {}),
          (TS.test_score_single_query_sums_to_one_and_ranks_by_dot, {})]
_MEAN = [(TS.test_score_mean_matches_scipy_softmax_mean, dict(M=4, L=77, d=8)),
         (TS.test_score_mean_closed_forms_and_bounds, {}), (TS.test_score_mean_duplicated_query_weights, {})]
_CAUSAL = [(TS.test_score_causal_matches_scipy_softmax_over_visible_keys, dict(mean=False, M=6, L=40, d=8)),
           (TS.test_score_causal_closed_forms, {})]
_ROPE = [(TN.test_rope_is_complex_rotation_of_rotate_half_pairs, {}),
         (TN.test_rope_preserves_norm_and_relative_position, {})]
_FPS = [(TB.test_fps_matches_maxmin_brute_force, dict(seed=s)) for s in range(6)] + [
    (TB.test_fps_orthonormal_basis_ties_go_to_lowest_index, {}), (TB.test_fps_outlier_first, {})]
_CFPS = [(TC.test_fps_adopt_continues_from_a_dictated_pick, dict(seed=s)) for s in range(6)] + [
    (TC.test_fps_orthonormal_basis_takes_indices_in_order, {}), (TC.test_fps_zero_query_has_zero_similarity, {}),
    (TC.test_cfps_buffer_matches_fp64_brute_force_simulation, {}), (TC.test_cfps_closed_forms, {})]
_UPD = [(TB.test_update_planted_assignment_uses_cosine_not_dot, {}),
        (TB.test_update_single_beacon_is_global_mean, {}), (TB.test_update_centroid_is_mean_of_assigned, {})]
_SEL = [(TS.test_select_matches_lexsort_and_invariants, dict(L=130, budget=100, W=8, npre=3)),
        (TS.test_select_all_ties_take_lowest_indices, {})]

MUTANTS = [
    ("drop_inv_sqrt_d", "* inv_sqrt_d;", "* 1.0;", _SCORE),
    ("no_max_shift_in_lse", "double lse = m + log(s);", "double lse = log(s);", _SCORE),
    ("sum_instead_of_max", "else if (w > score[j])\n        score[j] = w;", "else\n        score[j] = score[j] + w;", _SCORE),
    ("mean_over_all_rows", "score[j] = score[j] / (double)n_valid;", "score[j] = score[j] / (double)M;", _MEAN),
    ("mean_takes_max", "      if (mean)\n        score[j] = score[j] + w;", "      if (mean && w > score[j])\n        score[j] = w;",
     _MEAN),
    ("causal_mask_inverted", "if (qpos && kpos[j] > qpos[q]) {", "if (qpos && kpos[j] < qpos[q]) {", _CAUSAL),
    ("causal_mask_hides_own_position", "if (qpos && kpos[j] > qpos[q]) {", "if (qpos && kpos[j] >= qpos[q]) {", _CAUSAL),
    ("causal_mask_ignored", "lg[j] = -INFINITY; /* masked: exp gives 0 below */\n        continue;",
     "lg[j] = -INFINITY; /* masked: exp gives 0 below */", _CAUSAL),
    ("rope_sign", "y[i] = x1 * cs - x2 * sn;", "y[i] = x1 * cs + x2 * sn;", _ROPE),
    ("rope_interleaved_pairs", "double x1 = x[i], x2 = x[i + h];", "double x1 = x[2 * i], x2 = x[2 * i + 1];",
     _ROPE),
    ("rope_frequency_exponent", "-(double)(2 * i) / (double)d", "-(double)(i) / (double)d", _ROPE),
    ("fps_min_update", "if (k == 0 || cj > val[j]) val[j] = cj;", "if (k == 0 || cj < val[j]) val[j] = cj;", _FPS),
    ("fps_first_pick_argmax", "val[i] = sum / (double)N;", "val[i] = -sum / (double)N;", _FPS),
    ("fps_forced_pick_ignored", "      c = forced[k];\n", "      c = r;\n", _CFPS),
    ("fps_first_similarity_not_reset", "if (k == 0 || cj > val[j]) val[j] = cj;", "if (cj > val[j]) val[j] = cj;",
     _FPS + _CFPS),
    ("cfps_compress_one_early", "    if (*size >= b_max) {", "    if (*size >= b_max - 1) {", _CFPS),
    ("cfps_keeps_arrival_order", "memcpy(tmp + (size_t)k * d, buf + (size_t)picks[k] * d,",
     "memcpy(tmp + (size_t)k * d, buf + (size_t)k * d,", _CFPS),
    ("assign_by_dot_product", "double cs = cosine(qn, c + (size_t)b * d, d, NULL);",
     "double cs = dot_seq(qn, c + (size_t)b * d, d);", _UPD),
    ("centroid_forgets_history", "sums[(size_t)b * d + i] = sums[(size_t)b * d + i] + x[(size_t)n * d + i];",
     "sums[(size_t)b * d + i] = x[(size_t)n * d + i];", _UPD),
    ("tie_break_high_index", "return (x->j < y->j) ? -1 : (x->j > y->j);",
     "return (x->j > y->j) ? -1 : (x->j < y->j);", _SEL),
    ("window_off_by_one", "for (int j = L - W; j < L; ++j) kept[n_keep++] = j;",
     "for (int j = L - W - 1; j < L - 1; ++j) kept[n_keep++] = j;", _SEL),
    ("bf16_round_half_up", "u += 0x7fffu + lsb;", "u += 0x8000u;",
     [(TN.test_bf16_known_patterns, {}), (TN.test_bf16_matches_torch_on_random_floats, {})]),
    ("gather_wrong_row", "memcpy(tk + (size_t)i * d, K + (size_t)kept[i] * d, row);",
     "memcpy(tk + (size_t)i * d, K + (size_t)i * d, row);", [(TS.test_gather_is_row_indexing, {})]),
]


@pytest.fixture(scope="module")
def workdir():
    d = tempfile.mkdtemp(prefix="bkv_mutants_")
    yield d
    shutil.rmtree(d, ignore_errors=True)


@pytest.mark.parametrize("name,old,new,checks", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_mutant(workdir, name, old, new, checks):
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation anchor for {name} not unique"
    path_c = os.path.join(workdir, f"{name}.c")
    path_so = os.path.join(workdir, f"lib{name}.so")
    with open(path_c, "w") as f:
        f.write(src.replace(old, new))
    subprocess.check_call(["gcc", *O.CFLAGS, "-o", path_so, path_c, "-lm"])
    lib = O.load(path_so)
    failed = []
    for fn, kw in checks:
        try:
            fn(lib, **kw)
        except Exception as exc:  # noqa: BLE001 - any failure counts as a catch
            failed.append((fn.__name__, type(exc).__name__))
    assert failed, f"no pin caught mutant {name}"
