"""Plant plausible mistakes in a copy of the oracle (on the CPU) and check that
the pins in test_oracle_pins.py fail for each one: a pin that no mistake can
trip pins nothing."""
import os

import numpy as np
import subprocess

import pytest

from oracle import focus_oracle as fo
import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(fo.__file__), "focus_oracle.c")

# (name, exact text in focus_oracle.c, replacement, pin functions that must fail)
MUTANTS = [
    ("ring_dropped", "int visible = (win[j] == win[i]) || (keep[j] == 1);",
     "int visible = (win[j] == win[i]);",
     [lambda: pins.test_lse_of_zero_scores_counts_visible_keys(),
      lambda: pins.test_attn_matches_streaming_simulation(40, 7, [2], 2, 16, 0)]),
    ("all_past_visible", "int visible = (win[j] == win[i]) || (keep[j] == 1);",
     "int visible = 1;",
     [lambda: pins.test_lse_of_zero_scores_counts_visible_keys()]),
    ("strict_causal", "for (int64_t j = 0; j <= i; ++j) {\n            int visible",
     "for (int64_t j = 0; j < i; ++j) {\n            int visible",
     [lambda: pins.test_no_compression_is_plain_causal()]),
    ("exp_sign", "double p = exp(s[j] - m);", "double p = exp(m - s[j]);",
     [lambda: pins.test_no_compression_is_plain_causal()]),
    ("k_for_v", "dot += qd[c] * bf16_to_f64(krows[j][c]);", "dot += qd[c] * bf16_to_f64(vrows[j][c]);",
     [lambda: pins.test_no_compression_is_plain_causal()]),
    ("scale_dropped", "s[j] = scale * s[j];", "s[j] = s[j];",
     [lambda: pins.test_no_compression_is_plain_causal()]),
    ("lse_no_max", "*lse = m + log(l);", "*lse = log(l);",
     [lambda: pins.test_first_row_sees_only_itself()]),
    ("summary_before_boundary", "if ((o + 1) % k == 0) return 1;", "if (o % k == 0) return 1;",
     [lambda: pins.test_layout_positions_closed_form(10), lambda: pins.test_layout_fig1_golden()]),
    ("partial_kmer_open", "return (o == n - 1) && close_partial;", "return 0;",
     [lambda: pins.test_layout_fig1_golden(),
      lambda: pins.test_layout_sizes_closed_form(5_000, 1_024, [100])]),
    ("retain_ordinary", "if (keep[j] != 1) continue;\n            if (R >= ring_cap)",
     "if (keep[j] != 0) continue;\n            if (R >= ring_cap)",
     [lambda: pins.test_sequential_equals_masked_parallel(700, 100, [10], 0)]),
    ("tail_off_by_one", "return tail > 0 && o >= n - tail;", "return tail > 0 && o > n - tail;",
     [lambda: pins.test_layout_tail_counts_closed_form(4_000, 1_000, [100], 3)]),
    ("tail_not_kept", "keep[t] = (uint8_t)in_tail(o, n, tail);", "keep[t] = 0;",
     [lambda: pins.test_attn_matches_streaming_simulation(40, 7, [2], 2, 16, 2),
      lambda: pins.test_tail_covering_every_base_is_causal_over_augmented()]),
    ("kmer_focus_in_next_kmer", "kmer[t++] = c;\n                c += 1;", "c += 1;\n                kmer[t++] = c;",
     [lambda: pins.test_kmer_ids_closed_form(4_000, 1_000, [100]),
      lambda: pins.test_kmer_local_lse_of_zero_scores_counts_visible_keys()]),
    ("local_no_boundary", "|| (same_window && kind[j] == 1) || j == boundary;", "|| (same_window && kind[j] == 1);",
     [lambda: pins.test_kmer_local_lse_of_zero_scores_counts_visible_keys(),
      lambda: pins.test_kmer_local_equals_appendix_mask_for_two_single_kmer_windows()]),
    ("local_all_focus_rows", "|| (same_window && kind[j] == 1) || j == boundary;", "|| kind[j] == 1;",
     [lambda: pins.test_kmer_local_lse_of_zero_scores_counts_visible_keys(),
      lambda: pins.test_kmer_local_invisible_rows_do_not_matter_and_visible_ones_do()]),
    ("local_no_in_window_focus", "|| (same_window && kind[j] == 1) || j == boundary;", "|| j == boundary;",
     [lambda: pins.test_kmer_local_lse_of_zero_scores_counts_visible_keys(),
      lambda: pins.test_kmer_local_invisible_rows_do_not_matter_and_visible_ones_do()]),
    ("local_whole_window", "int visible = (same_window && kmer[j] == kmer[i])", "int visible = (same_window)",
     [lambda: pins.test_kmer_local_lse_of_zero_scores_counts_visible_keys(),
      lambda: pins.test_kmer_local_invisible_rows_do_not_matter_and_visible_ones_do()]),
    ("boundary_is_first_focus", "if (kind[j] == 1) last_focus[win[j]] = j;",
     "if (kind[j] == 1 && last_focus[win[j]] < 0) last_focus[win[j]] = j;",
     [lambda: pins.test_kmer_local_invisible_rows_do_not_matter_and_visible_ones_do()]),
    ("rope_sin_sign", "yr[i + h] = hi * c + lo * s;", "yr[i + h] = hi * c - lo * s;",
     [lambda: pins.test_rope_one_hot_closed_form(64),
      lambda: pins.test_rope_position_zero_is_identity_and_pairs_keep_their_norm()]),
    ("rope_interleaved_pairs", "double lo = bf16_to_f64(xr[i]), hi = bf16_to_f64(xr[i + h]);",
     "double lo = bf16_to_f64(xr[(2 * i) % d]), hi = bf16_to_f64(xr[(2 * i + 1) % d]);",
     [lambda: pins.test_rope_one_hot_closed_form(64)]),
    ("rope_frequency", "double theta = pow(base, -2.0 * (double)i / (double)d);",
     "double theta = pow(base, -1.0 * (double)i / (double)d);",
     [lambda: pins.test_rope_one_hot_closed_form(128)]),
    ("rope_position_off_by_one", "double a = (double)pos[r] * theta;", "double a = (double)(pos[r] + 1) * theta;",
     [lambda: pins.test_rope_position_zero_is_identity_and_pairs_keep_their_norm()]),
    ("f64_attention_drops_ring", "if (!((win[j] == win[i]) || (keep[j] == 1))) continue;",
     "if (!(win[j] == win[i])) continue;",
     [lambda: pins.test_fp64_attention_variants_equal_the_pinned_bf16_ones()]),
    ("round_bf16_ties_away", "double r = nearbyint(ldexp(m, 8));", "double r = round(ldexp(m, 8));",
     [lambda: pins.test_round_bf16_is_nearest_even_and_matches_torch()]),
    ("last_window_full", "static int64_t window_bases(int64_t N, int64_t start, int32_t W) { return (N - start < W) ? (N - start) : W; }",
     "static int64_t window_bases(int64_t N, int64_t start, int32_t W) { (void)N; (void)start; return W; }",
     [lambda: pins.test_layout_sizes_closed_form(5_000, 1_024, [100]),
      lambda: pins.test_adaptive_windows_sizes_and_offsets_closed_form(1_037, [64, 1_000, 1_000], [8, 100, 3])]),
    ("summary_src_next_base", "kind[t] = 1; src[t] = (int32_t)base; pos[t] = (int32_t)t; win[t] = w;",
     "kind[t] = 1; src[t] = (int32_t)(base + 1); pos[t] = (int32_t)t; win[t] = w;",
     [lambda: pins.test_layout_fig1_golden()]),
    ("summary_token_id", "tok[(int64_t)b * T_total + t] = FO_SUMMARY_TOKEN;", "tok[(int64_t)b * T_total + t] = 0;",
     [lambda: pins.test_layout_matches_string_construction(*pins.LAYOUT_CASES[0], True)]),
    ("ring_offsets_one_ahead", "        ring_off[w] = (int32_t)r;", "        ring_off[w] = (int32_t)(r + 1);",
     [lambda: pins.test_layout_positions_closed_form(10), lambda: pins.test_layout_fig1_golden()]),
    ("decode_skips_self", "        kr[c] = k_new + (size_t)s * d;\n        vr[c] = v_new + (size_t)s * d;\n        c += 1;\n"
     "        softmax_row(d,", "        softmax_row(d,", [lambda: pins.test_decode_equals_prefill_row()]),
]


@pytest.mark.parametrize("name,old,new,checks", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_planted_mistake(tmp_path, name, old, new, checks):
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site for {name} not unique/found"
    mut = tmp_path / f"mut_{name}.c"
    mut.write_text(src.replace(old, new))
    so = tmp_path / f"libmut_{name}.so"
    subprocess.run(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", str(mut), "-o", str(so), "-lm"],
                   check=True)
    with fo.use_library(str(so)):
        for check in checks:
            with pytest.raises((AssertionError, ValueError, IndexError)):
                check()


# The token-embedding lookup is Python in the oracle: plant its mistakes by
# replacing the function for the duration of the pins.
_embed = fo.embed_tokens
EMBED_MUTANTS = [
    ("embed_token_off_by_one", lambda tok, table: _embed((np.asarray(tok).astype(np.int64) + 1) % 5, table)),
    ("embed_summary_as_base", lambda tok, table: _embed(np.where(np.asarray(tok) == fo.SUMMARY_TOKEN, 0, tok),
                                                         table)),
    ("embed_transposed_table", lambda tok, table: _embed(tok, np.ascontiguousarray(
        np.asarray(table)[:, ::-1]))),
]


@pytest.mark.parametrize("name,mutant", EMBED_MUTANTS, ids=[m[0] for m in EMBED_MUTANTS])
def test_embed_mutant_trips_a_pin(name, mutant, monkeypatch):
    monkeypatch.setattr(fo, "embed_tokens", mutant)
    tripped = False
    for pin in (pins.test_embed_tokens_one_hot_table_spells_the_string_layout,
                pins.test_embed_tokens_summary_rows_sit_at_summary_positions):
        try:
            pin()
        except (AssertionError, IndexError):      # a wrong row can name a token that does not exist
            tripped = True
    assert tripped, f"no embedding pin caught the mutant {name}"
