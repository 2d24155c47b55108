"""Pin strength: plant one plausible mistake at a time into a copy of the
oracle's C source, compile it on the CPU, and require that the pin suite
rejects every mutant. The real oracle is never modified."""
import os
import shutil

import pytest

import oracle
import oracle_pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "litevlm_oracle.c")

# (name, original text, planted text[, occurrence]). Without an occurrence the
# original text must appear exactly once; with one, the mistake is planted at
# that occurrence only (statements the visual-key and the full-key scores
# share are planted in each function separately).
MUTANTS = [
    ("gqa_head_map_modulo", "const int32_t g = h / group;", "const int32_t g = h % hkv;", 0),
    ("key_head_always_zero", "const int64_t krow = (j * hkv + g) * head_dim;",
     "const int64_t krow = (j * hkv + 0) * head_dim;", 0),
    ("key_rows_of_first_request", "kd[x] = litevlm_oracle_decode(dtype, k, n0 * hkv * head_dim + x);",
     "kd[x] = litevlm_oracle_decode(dtype, k, x);"),
    ("query_rows_of_first_request", "qd[x] = litevlm_oracle_decode(dtype, q, t0 * hq * head_dim + x);",
     "qd[x] = litevlm_oracle_decode(dtype, q, x);", 0),
    ("scale_1_over_d", "/ sqrt((double)head_dim)", "/ (double)head_dim", 0),
    ("logit_sign", "s[j] = dot * scale;", "s[j] = -dot * scale;", 0),
    ("no_mean_over_queries", "const double denom = (double)hq * (double)tb;", "const double denom = (double)hq;", 0),
    ("softmax_unnormalised", "const double p = exp(s[j] - m) / l;", "const double p = exp(s[j] - m);"),
    ("normaliser_without_max", "for (int64_t j = 0; j < nb; ++j) l += exp(s[j] - m);",
     "for (int64_t j = 0; j < nb; ++j) l += exp(s[j]);"),
    ("ascending_scores", "return a->key > b->key ? -1 : 1;", "return a->key > b->key ? 1 : -1;"),
    ("tie_to_higher_index",
     "return a->key > b->key ? -1 : 1;\n    return (a->idx > b->idx) - (a->idx < b->idx);",
     "return a->key > b->key ? -1 : 1;\n    return (a->idx < b->idx) - (a->idx > b->idx);"),
    ("nan_ranks_first", "if (an != bn) return an ? 1 : -1;", "if (an != bn) return an ? -1 : 1;"),
    ("ratio_rounds_to_nearest", "double kd = floor((double)keep_ratio * (double)n);",
     "double kd = floor((double)keep_ratio * (double)n + 0.5);"),
    ("kept_in_rank_order", "qsort(it, (size_t)kb, sizeof(oracle_item), oracle_index_cmp);", ""),
    ("e4m3_exponent_bias", "else v = ldexp((double)(8 + m), e - 10);", "else v = ldexp((double)(8 + m), e - 9);"),
    ("e4m3_subnormal_scale", "if (e == 0) v = ldexp((double)m, -9);", "if (e == 0) v = ldexp((double)m, -10);"),
    ("bf16_shift", "u = (uint32_t)h << 16;", "u = (uint32_t)h << 15;"),
    ("gather_wrong_row", "(const char*)src + (int64_t)kept_idx[r] * row_bytes",
     "(const char*)src + (int64_t)r * row_bytes"),
    ("full_keys_gqa_head_map_modulo", "const int32_t g = h / group;", "const int32_t g = h % hkv;", 1),
    ("full_keys_key_head_always_zero", "const int64_t krow = (j * hkv + g) * head_dim;",
     "const int64_t krow = (j * hkv + 0) * head_dim;", 1),
    ("full_keys_query_rows_of_first_request",
     "qd[x] = litevlm_oracle_decode(dtype, q, t0 * hq * head_dim + x);",
     "qd[x] = litevlm_oracle_decode(dtype, q, x);", 1),
    ("full_keys_scale_1_over_d", "/ sqrt((double)head_dim)", "/ (double)head_dim", 1),
    ("full_keys_logit_sign", "s[j] = dot * scale;", "s[j] = -dot * scale;", 1),
    ("full_keys_no_mean_over_queries", "const double denom = (double)hq * (double)tb;",
     "const double denom = (double)hq;", 1),
    ("full_keys_system_rows_of_first_request",
     "kd[x] = litevlm_oracle_decode(dtype, k_sys, s0 * row + x);", "kd[x] = litevlm_oracle_decode(dtype, k_sys, x);"),
    ("full_keys_text_rows_of_first_request",
     "kd[(sb + nb) * row + x] = litevlm_oracle_decode(dtype, k_txt, t0 * row + x);",
     "kd[(sb + nb) * row + x] = litevlm_oracle_decode(dtype, k_txt, x);"),
    ("full_keys_visual_column_offset", "const double p = exp(s[sb + j] - m) / z;",
     "const double p = exp(s[j] - m) / z;"),
    ("full_keys_not_causal", "const int64_t nk = sb + nb + i + 1;", "const int64_t nk = sb + nb + tb;"),
    ("full_keys_visual_normaliser", "for (int64_t j = 0; j < nk; ++j) z += exp(s[j] - m);",
     "for (int64_t j = sb; j < sb + nb; ++j) z += exp(s[j] - m);"),
    ("full_keys_no_system", "const int64_t nk = sb + nb + i + 1;", "const int64_t nk = nb + i + 1;"),
    ("views_threshold_not_strict", "const int sel = s[v] > threshold;", "const int sel = s[v] >= threshold;"),
    ("views_weights_swapped", "const float a = w_lex * lexical[(int64_t)b * num_views + v];",
     "const float a = w_logit * lexical[(int64_t)b * num_views + v];"),
    ("views_tie_to_higher_index", "    return ia < ib;\n", "    return ia > ib;\n"),
    ("views_nan_ranks_first", "    if (an != bn) return bn;\n", "    if (an != bn) return an;\n"),
    ("views_tokens_of_first_view", "ntok += tokens_per_view[v];", "ntok += tokens_per_view[0];"),
    ("views_no_fallback", "if (pass < min_views) {", "if (pass < 0) {"),
    ("project_rms_sum", "const double s = 1.0 / sqrt(ss / (double)hidden + eps);",
     "const double s = 1.0 / sqrt(ss + eps);"),
    ("project_eps_outside", "const double s = 1.0 / sqrt(ss / (double)hidden + eps);",
     "const double s = 1.0 / (sqrt(ss / (double)hidden) + eps);"),
    ("project_no_gamma", "xn[h] = xn[h] * s * (double)gamma[h];", "xn[h] = xn[h] * s;"),
    ("project_weight_transposed", "acc += xn[h] * litevlm_oracle_decode(OR_BF16, w, (int64_t)o * hidden + h);",
     "acc += xn[h] * litevlm_oracle_decode(OR_BF16, w, (int64_t)h * out_features + o);"),
    ("project_no_bias", "yr[o] = acc + (bias ? (double)bias[o] : 0.0);", "yr[o] = acc;"),
    ("project_rope_sign", "yr[h0 + j] = y1 * cos(a) - y2 * sin(a);", "yr[h0 + j] = y1 * cos(a) + y2 * sin(a);"),
    ("project_rope_frequency", "pow(rope_base, -2.0 * (double)j / (double)head_dim)",
     "pow(rope_base, -1.0 * (double)j / (double)head_dim)"),
    ("project_rope_adjacent_pairs", "const int32_t half = head_dim / 2;", "const int32_t half = 1;"),
    ("splice_visual_global_position", "position_ids[r] = S + (g - seq_offsets[b]);", "position_ids[r] = S + g;"),
    ("splice_text_renumbered", "position_ids[r] = S + N + t;", "position_ids[r] = S + k + t;"),
    ("splice_drops_visual", "for (int32_t i = 0; i < k; ++i, ++r) {", "for (int32_t i = 0; i < 0; ++i, ++r) {"),
]


def _plant(src, name, old, new, occurrence=None):
    if occurrence is None:
        assert src.count(old) == 1, f"mutation site for {name} not found exactly once"
        return src.replace(old, new)
    at = -1
    for _ in range(occurrence + 1):
        at = src.find(old, at + 1)
        assert at >= 0, f"mutation site {occurrence} for {name} not found"
    return src[:at] + new + src[at + len(old):]


@pytest.mark.parametrize("mutant", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_reject_mutant(tmp_path, mutant):
    name = mutant[0]
    src = open(SRC).read()
    mut = tmp_path / "mutant.c"
    mut.write_text(_plant(src, *mutant))
    so = oracle.build(str(mut), str(tmp_path / "libmutant.so"))
    lib = oracle.load(so)
    caught = []
    for pin in oracle_pins.ALL_PINS:
        try:
            pin(lib)
        except (AssertionError, oracle.OracleError) as e:
            caught.append(pin.__name__)
            break
    assert caught, f"no pin rejects the planted mistake {name}"
