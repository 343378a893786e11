"""Planted mistakes in a copy of the oracle must each break at least one pin.

Each mutant edits one plausible step of rrq_oracle.c (a rounding rule, a
dropped term, a wrong sign, a transposed operand, a wrong index), compiles the
copy on the CPU and runs the pins of tests/_pins.py against it.  This shows
that the pins, not the oracle agreeing with itself, are what fix its
arithmetic."""
import os

import pytest

import oracle
import _pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "rrq_oracle.c")

MUTANTS = {
    "ties_round_up": ("return (fmodf(f, 2.0f) == 0.0f) ? f : f + 1.0f;", "return f + 1.0f;"),
    "ties_round_down": ("return (fmodf(f, 2.0f) == 0.0f) ? f : f + 1.0f;", "return f;"),
    "four_steps_not_three": ("float s = range / 3.0f;", "float s = range / 4.0f;"),
    "level_drops_offset": ("level[q] = lo + qs;", "level[q] = qs;"),
    "residual_sign": ("v[j] = v[j] - level[code];", "v[j] = v[j] + level[code];"),
    "transposed_difference": ("float d = v[j] - lo;", "float d = lo - v[j];"),
    "zero_sign_order_ignored": ("if (a == b && signbit(a) && !signbit(b)) return 1;", ""),
    "no_clamp": ("if (code > 3) code = 3;", "if (code > 4) code = 4;"),
    "packing_bit_order": ("codes[c / 4] |= (uint8_t)(q << (2 * (c % 4)));",
                          "codes[c / 4] |= (uint8_t)(q << (2 * (3 - c % 4)));"),
    "recon_drops_base": ("acc = (i == 0) ? value : acc + value;", "acc = (i == 0) ? 0.0f : acc + value;"),
    "recon_bf16_truncates": ("u += 0x7fffu + ((u >> 16) & 1u);", ""),
    "max_is_min": ("if (before(hi, v[j])) hi = v[j];", "if (before(v[j], hi)) hi = v[j];"),
    "range_of_input_not_residual": ("if (before(v[j], lo)) lo = v[j];\n      if (before(hi, v[j])) hi = v[j];",
                                    "if (before(x[j], lo)) lo = x[j];\n      if (before(hi, x[j])) hi = x[j];"),
    "scale_rounds_range_twice": ("float range = hi - lo;", "float range = (float)(double)(hi - lo) * 1.0000001f;"),
    "level_from_code_minus_one": ("float qs = (float)q * s;\n      level[q]", "float qs = (float)(q > 0 ? q - 1 : 0) * s;\n      level[q]"),
    # symmetric grid and binary16 scales
    "sym_zero_point_one": ("code = (int)round_half_even_signed(u) + 2;", "code = (int)round_half_even_signed(u) + 1;"),
    "sym_no_top_clamp": ("code = code > 3 ? 3 : code;", "code = code & 3;"),
    "sym_scale_not_rounded_to_f16": ("if (scale_f16) s = rrq_oracle_f16_to_f32(rrq_oracle_f32_to_f16(s));", ""),
    "sym_span_not_doubled": ("float span = 2.0f * amax;", "float span = amax;"),
    "sym_round_half_up": ("return u < 0.0f ? -round_half_even(-u) : round_half_even(u);", "return floorf(u + 0.5f);"),
    "sym_amax_signed": ("if (fabsf(v[j]) > amax) amax = fabsf(v[j]);", "if (v[j] > amax) amax = v[j];"),
    "sym_level_without_zero_point": ("float level = (float)(code - 2) * s;", "float level = (float)code * s;"),
    "sym_recon_zero_point_one": ("float level = (float)(q - 2) * s;", "float level = (float)(q - 1) * s;"),
    "sym_recon_drops_base": ("acc = (i == 0) ? level : acc + level;", "acc = (i == 0) ? 0.0f : acc + level;"),
    "f16_truncates": ("double frac = rhe_double((2.0 * m - 1.0) * 1024.0);", "double frac = floor((2.0 * m - 1.0) * 1024.0);"),
    "f16_bias_14": ("(uint16_t)((exp + 15) << 10)", "(uint16_t)((exp + 14) << 10)"),
    "f16_flushes_subnormals": ("const double n = rhe_double(a * ldexp(1.0, 24));", "const double n = 0.0;"),
    "f16_decode_exponent": ("else v = ldexp((double)(1024 + frac), e - 25);", "else v = ldexp((double)(1024 + frac), e - 24);"),
    "f16_ties_away": ("return (fmod(f, 2.0) == 0.0) ? f : f + 1.0;", "return f + 1.0;"),
    # Algorithm 1 with a base checkpoint
    "base_drops_zero": ("  return z + qs;", "  return qs;"),
    "base_sym_zero_point_one": ("if (grid_sym) return (float)(q - 2) * s;", "if (grid_sym) return (float)(q - 1) * s;"),
    "base_residual_sign": ("r[j] = x - base_level(grid_sym, q0, s0, z0);", "r[j] = x + base_level(grid_sym, q0, s0, z0);"),
    "base_ignored": ("r[j] = x - base_level(grid_sym, q0, s0, z0);", "r[j] = x - 0.0f * base_level(grid_sym, q0, s0, z0);"),
    "base_code_bit_order": ("const int q0 = (codes[0][c / 4] >> (2 * (c % 4))) & 3;",
                            "const int q0 = (codes[0][c / 4] >> (2 * (3 - c % 4))) & 3;"),
    # stage-wise product
    "gemv_drops_base": ("w = (i == 0) ? lv : w + lv;", "w = (i == 0) ? 0.0f : w + lv;"),
    "gemv_reversed_activation": ("(double)rrq_oracle_bf16_to_f32(A[(size_t)b * cols + j]);",
                                 "(double)rrq_oracle_bf16_to_f32(A[(size_t)b * cols + (cols - 1 - j)]);"),
    "gemv_wrong_output_row": ("Y[(size_t)b * rows + r] += (double)w", "Y[(size_t)b * rows + (rows - 1 - r)] += (double)w"),
    "gemv_bf16_weight": ("Y[(size_t)b * rows + r] += (double)w *",
                         "Y[(size_t)b * rows + r] += (double)rrq_oracle_bf16_to_f32(rrq_oracle_f32_to_bf16(w)) *"),
    # heterogeneous widths and the peak-to-mean ratio
    "bits_steps_pow2": ("const int m = (1 << bits[k]) - 1; /* steps of a b-bit grid */",
                        "const int m = (1 << bits[k]); /* steps of a b-bit grid */"),
    "bits_pack_msb_first": ("if ((q >> t) & 1) codes[bit / 8] |= (uint8_t)(1u << (bit % 8));",
                            "if ((q >> t) & 1) codes[bit / 8] |= (uint8_t)(1u << (7 - bit % 8));"),
    "bits_clamp_one_low": ("code = code < 0 ? 0 : (code > m ? m : code);", "code = code < 0 ? 0 : (code > m - 1 ? m - 1 : code);"),
    "bits_read_reversed": ("q |= ((codes[bit / 8] >> (bit % 8)) & 1) << t;", "q |= ((codes[bit / 8] >> (bit % 8)) & 1) << (b - 1 - t);"),
    "bits_level_drops_zero": ("      float lv = lo + qs;\n      v[j] = v[j] - lv;", "      float lv = qs;\n      v[j] = v[j] - lv;"),
    "pmr_sum_not_mean": ("pmr[gi] = sum > 0.0 ? peak / (sum / (double)group) : 0.0;", "pmr[gi] = sum > 0.0 ? peak / sum : 0.0;"),
    "pmr_signed_values": ("const double a = fabs((double)rrq_oracle_bf16_to_f32(W[gi * group + j]));",
                          "const double a = (double)rrq_oracle_bf16_to_f32(W[gi * group + j]);"),
    "gemv_one_stage_short": ("      for (int i = 0; i < k; ++i) {\n        const int q = (codes[i][c / 4] >> (2 * (c % 4))) & 3;\n        const float s = scale_f16 ? rrq_oracle_f16_to_f32(((const uint16_t*)scales[i])[gi])\n                                  : ((const float*)scales[i])[gi];\n        const float lv",
                             "      for (int i = 0; i < k - (k > 1); ++i) {\n        const int q = (codes[i][c / 4] >> (2 * (c % 4))) & 3;\n        const float s = scale_f16 ? rrq_oracle_f16_to_f32(((const uint16_t*)scales[i])[gi])\n                                  : ((const float*)scales[i])[gi];\n        const float lv"),
    # prefill product (bf16 weights)
    "prefill_drops_base": ("sum = st == 0 ? level : sum + level;", "sum = st == 0 ? 0.0f : sum + level;"),
    "prefill_weight_truncated": ("  return rrq_oracle_f32_to_bf16(sum);",
                                 "  uint32_t u; memcpy(&u, &sum, 4); return (uint16_t)(u >> 16);"),
    "prefill_reversed_activation": ("dot += wrow[j] * (double)rrq_oracle_bf16_to_f32(A[(size_t)t * cols + j]);",
                                    "dot += wrow[j] * (double)rrq_oracle_bf16_to_f32(A[(size_t)t * cols + (cols - 1 - j)]);"),
    "prefill_wrong_output_row": ("Y[(size_t)t * rows + r] = dot;", "Y[(size_t)t * rows + (rows - 1 - r)] = dot;"),
    "prefill_one_stage_short": ("for (int st = 0; st < k; ++st) {", "for (int st = 0; st < k - (k > 1); ++st) {"),
    "prefill_code_bit_order": ("const int code = (codes[st][c / 4] >> (2 * (c % 4))) & 3;",
                               "const int code = (codes[st][c / 4] >> (2 * (3 - c % 4))) & 3;"),
    "prefill_first_group_only": ("  const int64_t g = c / group;\n  float sum", "  const int64_t g = 0;\n  float sum"),
    # products with per-stage widths
    "pbits_drops_base": ("running = st == 0 ? lvl : running + lvl;", "running = st == 0 ? 0.0f : running + lvl;"),
    "pbits_ignores_widths": ("const int code = get_bits(codes[st], c, bits[st]);", "const int code = get_bits(codes[st], c, 2);"),
    "pbits_never_rounds": ("wts[j] = bf16_weights ? (double)rrq_oracle_bf16_to_f32(rrq_oracle_f32_to_bf16(running)) : (double)running;",
                           "wts[j] = (double)running;"),
    "pbits_wrong_output_row": ("Y[(size_t)t * rows + r] = sum;", "Y[(size_t)t * rows + (rows - 1 - r)] = sum;"),
    "pbits_first_stage_zero": ("const float lvl = zeros[st][g] + scaled;", "const float lvl = zeros[0][g] + scaled;"),
    # Algorithm 1 with a base checkpoint and per-stage widths
    "fbb_residual_sign": ("r0[j] = rrq_oracle_bf16_to_f32(W[first + j]) - base_level_w;",
                          "r0[j] = rrq_oracle_bf16_to_f32(W[first + j]) + base_level_w;"),
    "fbb_base_drops_zero": ("const float base_level_w = zeros[0][gi] + based;", "const float base_level_w = based;"),
    "fbb_base_read_at_width_two": ("const int q0 = get_bits(codes[0], first + j, bits[0]);",
                                   "const int q0 = get_bits(codes[0], first + j, 2);"),
    "fbb_widths_not_shifted": ("rrq_oracle_quantize_group_bits(r0, group, rest, bits + 1, Qr, sr, zr, NULL)",
                               "rrq_oracle_quantize_group_bits(r0, group, rest, bits, Qr, sr, zr, NULL)"),
    "fbb_first_scale_everywhere": ("scales[k][gi] = sr[k - 1];", "scales[k][gi] = sr[0];"),
}


@pytest.fixture(scope="module")
def source():
    with open(SRC) as f:
        return f.read()


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, source, tmp_path):
    old, new = MUTANTS[name]
    assert source.count(old) == 1, f"mutation site for {name} not found exactly once"
    src = tmp_path / "rrq_oracle.c"
    src.write_text(source.replace(old, new))
    lib = oracle.compile_oracle(str(src), str(tmp_path / "libmutant.so"))
    fails = _pins.all_failures(oracle.Oracle(lib))
    assert fails, f"mutant {name} passed every pin"
