"""Planted mistakes in the oracle must fail its pins.

Each case copies the oracle (the C source and its Python wrapper) to a
temporary directory with one plausible mistake planted -- a dropped weight, a
wrong sign, an inverted comparison, a wrong divisor or index -- builds that
copy, and runs the pins that should notice.  The mistake counts as caught when
at least one of them fails.  Nothing here touches a GPU.
"""
import importlib.util
import os
import shutil
import uuid

import pytest

import test_oracle_attend_fit as pins_af
import test_oracle_quant as pins_q

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ORACLE_DIR = os.path.join(ROOT, "oracle")

# (name, file, original text, planted text, pins to run: (function, kwargs))
MUTATIONS = [
    ("weight dropped from the Query-aware distance", "qwm_oracle.c",
     "acc = fmaf(wv[c], t2, acc); /* one fused multiply-add per term */",
     "acc = fmaf(1.0f, t2, acc);",
     [(pins_q.test_qsac_hand_cases, {}), (pins_q.test_topm_candidates_are_weighted_nearest, {})]),
    ("zero-point sign flipped", "qwm_oracle.c",
     "float zf = rint_even(-lo * inv);",
     "float zf = rint_even(lo * inv);",
     [(pins_q.test_int2_hand_example, {}), (pins_q.test_int2_round_trip_bound, {"G": 32})]),
    ("PSAC keep rule inverted", "qwm_oracle.c",
     "int keep = errq < err0;",
     "int keep = errq > err0;",
     [(pins_q.test_psac_keep_rule_and_projection, {}), (pins_q.test_psac_exact_when_error_in_span, {})]),
    ("secondary scale over 256 instead of 255", "qwm_oracle.c",
     "oracle_f32_to_f16_ru(mx / 255.0f)",
     "oracle_f32_to_f16_ru(mx / 256.0f)",
     [(pins_q.test_two_level_scales_hand_fixture, {}),
      (pins_q.test_two_level_scales_cover_minimal_and_round_trip, {})]),
    ("dequantisation sign flipped", "qwm_oracle.c",
     "double v = (double)oracle_bf16_to_f32(mu[c]) + s * (double)(q - z);",
     "double v = (double)oracle_bf16_to_f32(mu[c]) + s * (double)(z - q);",
     [(pins_q.test_two_level_scales_cover_minimal_and_round_trip, {}),
      (pins_q.test_psac_exact_when_error_in_span, {})]),
    ("k-means mean divides by count + 1", "qwm_oracle.c",
     "(float)(sum[(size_t)j * d + c] / (double)cnt[j])",
     "(float)(sum[(size_t)j * d + c] / (double)(cnt[j] + 1))",
     [(pins_af.test_fit_one_cluster_is_mean, {}), (pins_af.test_fit_objective_non_increasing_and_fixed_point, {})]),
    ("softmax scale left out of the logits", "qwm_oracle.c",
     "lg[j] = acc * scale;",
     "lg[j] = acc;",
     [(pins_af.test_attend_matches_torch_sdpa, {}), (pins_af.test_attend_single_key_returns_value, {})]),
    ("full-matrix distance uses the wrong channel", "qwm_oracle.c",
     "tc = fmaf(Mh[(size_t)c * d + c2], res[c2], tc);",
     "tc = fmaf(Mh[(size_t)c * d + c2], res[c], tc);",
     [(pins_q.test_full_matrix_distance_reduces_to_diagonal_and_matches_fp64, {})]),
    ("Query second moment over N - 1", "oracle.py",
     'M = np.einsum("nhc,nhe->hce", q, q) / N',
     'M = np.einsum("nhc,nhe->hce", q, q) / max(N - 1, 1)',
     [(pins_af.test_query_stats_hadamard_closed_form, {}), (pins_af.test_query_stats_diagonal_weights, {})]),
    ("PSAC INT8 codes truncated instead of rounded", "qwm_oracle.c",
     "float qq = rint_even(y);",
     "float qq = truncf(y);",
     [(pins_q.test_psac_int8_rounding_hand_fixture, {})]),
    ("k-means tie goes to the higher index", "qwm_oracle.c",
     "if (bj < 0 || acc < best) { best = acc; bj = j; }\n        }\n        lab[i] = bj;",
     "if (bj < 0 || acc <= best) { best = acc; bj = j; }\n        }\n        lab[i] = bj;",
     [(pins_af.test_fit_tie_goes_to_lower_index, {})]),
    ("k-means empty cluster reset to zero", "qwm_oracle.c",
     "if (cnt[j] == 0) continue;",
     "if (cnt[j] == 0) { for (int c = 0; c < d; ++c) mu[(size_t)j * d + c] = 0.0f; continue; }",
     [(pins_af.test_fit_empty_cluster_keeps_its_centroid, {})]),
    ("top-1 key by the smallest logit", "oracle.py",
     "idx[h] = np.argmax(L, axis=1)",
     "idx[h] = np.argmin(L, axis=1)",
     [(pins_af.test_top1_brute_force_and_ties, {}), (pins_af.test_top1_closed_form_and_shift_ratio, {})]),
]


def mutated_oracle(tmp_path, fname, old, new):
    d = tmp_path / ("oracle_" + uuid.uuid4().hex[:8])
    d.mkdir()
    for f in ("qwm_oracle.c", "oracle.py"):
        shutil.copy(os.path.join(ORACLE_DIR, f), d / f)
    path = d / fname
    src = path.read_text()
    assert src.count(old) == 1, f"the planted text's anchor is not unique in {fname}"
    path.write_text(src.replace(old, new))
    spec = importlib.util.spec_from_file_location("oracle_mutant_" + d.name, d / "oracle.py")
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    mod.build()
    return mod


@pytest.mark.parametrize("name,fname,old,new,pins", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_fails_a_pin(tmp_path, name, fname, old, new, pins):
    mod = mutated_oracle(tmp_path, fname, old, new)
    caught = []
    for fn, kw in pins:
        try:
            fn(mod, **kw)
        except Exception as e:  # a failed assertion, or an error the mistake provokes
            caught.append(f"{fn.__name__}: {type(e).__name__}")
    assert caught, f"no pin noticed: {name}"
