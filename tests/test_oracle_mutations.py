"""Planted mistakes in the oracle must be caught by its pins.

Each case copies oracle/pic_oracle.c to a temporary directory, replaces one
expression with a plausible wrong one (a dropped term, a wrong sign or index,
a transposed operand, a swapped weight), compiles the copy and runs every pin
of tests/oracle_pins.py against it.  The case passes when at least one pin
fails, i.e. the pins would have exposed that mistake.  Every mutation keeps
all memory accesses in bounds.
"""
import os
import tempfile

import pytest

import oracle
import oracle_pins

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle",
                   "pic_oracle.c")

MUTATIONS = {
    "no_half_pixel_offset": (
        "double sx = ((double)x + 0.5) * ((double)Wl / (double)W) - 0.5;",
        "double sx = ((double)x) * ((double)Wl / (double)W);"),
    "x_uses_row_scale": (
        "double sx = ((double)x + 0.5) * ((double)Wl / (double)W) - 0.5;",
        "double sx = ((double)x + 0.5) * ((double)Hl / (double)H) - 0.5;"),
    "y_uses_x_coordinate": (
        "double sy = ((double)y + 0.5)",
        "double sy = ((double)x + 0.5)"),
    "align_corners_scale": (
        "double sx = ((double)x + 0.5) * ((double)Wl / (double)W) - 0.5;",
        "double sx = (W > 1) ? (double)x * ((double)(Wl - 1) / (double)(W - 1)) : 0.0;"),
    "no_lower_clamp": (
        "if (sx < 0.0) sx = 0.0;",
        "if (sx < -1.0) sx = 0.0;"),
    "swapped_column_weights": (
        "double top = (1.0 - a) * g[(int64_t)v0 * Wl + u0] + a * g[(int64_t)v0 * Wl + u1];",
        "double top = a * g[(int64_t)v0 * Wl + u0] + (1.0 - a) * g[(int64_t)v0 * Wl + u1];"),
    "swapped_row_weights": (
        "return (1.0 - b) * top + b * bot;",
        "return b * top + (1.0 - b) * bot;"),
    "wrapping_right_neighbour": (
        "int u1 = (u0 + 1 < Wl) ? u0 + 1 : Wl - 1;",
        "int u1 = (u0 + 1 < Wl) ? u0 + 1 : 0;"),
    "bottom_row_uses_top_row": (
        "double bot = (1.0 - a) * g[(int64_t)v1 * Wl + u0] + a * g[(int64_t)v1 * Wl + u1];",
        "double bot = (1.0 - a) * g[(int64_t)v0 * Wl + u0] + a * g[(int64_t)v0 * Wl + u1];"),
    "floor_level_size": (
        "return (int)(((int64_t)n + p - 1) / p);",
        "return (int)((int64_t)n / p > 0 ? (int64_t)n / p : 1);"),
    "step_ignored": (
        "y[i] = (double)q[i] * step;",
        "y[i] = (double)q[i];"),
    "transposed_weights": (
        "s += Wk[(int64_t)i * din + j] * h[j];",
        "s += Wk[(int64_t)(j % dout) * din + (i % din)] * h[j];"),
    "dropped_bias": (
        "z[i] = s + bk[i];",
        "z[i] = s;"),
    "activation_on_output_layer": (
        "h[i] = last ? z[i] : pic_oracle_act(z[i], act);",
        "h[i] = pic_oracle_act(z[i], act);"),
    "no_hidden_activation": (
        "h[i] = last ? z[i] : pic_oracle_act(z[i], act);",
        "h[i] = z[i];"),
    "gelu_wrong_scale": (
        "return 0.5 * z * (1.0 + erf(z / sqrt(2.0)));",
        "return 0.5 * z * (1.0 + erf(z / 2.0));"),
    "gelu_tanh_form": (
        "return 0.5 * z * (1.0 + erf(z / sqrt(2.0)));",
        "return 0.5 * z * (1.0 + tanh(0.7978845608028654 * (z + 0.044715 * z * z * z)));"),
    "leaky_relu": (
        "return z > 0.0 ? z : 0.0;",
        "return z > 0.0 ? z : 0.01 * z;"),
    "no_upper_clamp": (
        "if (v > 1.0) return 1.0;",
        "if (v > 1.0) return v;"),
    "levels_coarsest_first": (
        "f[d++] = pic_oracle_bilinear_at(y[l] + (int64_t)c * Hl * Wl, Hl, Wl, H, W, x, yy);",
        "f[(L - 1 - l) * C + c] = pic_oracle_bilinear_at(y[l] + (int64_t)c * Hl * Wl, Hl, Wl, H, W, x, yy); d++;"),
    "channel_major_features": (
        "f[d++] = pic_oracle_bilinear_at(y[l] + (int64_t)c * Hl * Wl, Hl, Wl, H, W, x, yy);",
        "f[c * L + l] = pic_oracle_bilinear_at(y[l] + (int64_t)c * Hl * Wl, Hl, Wl, H, W, x, yy); d++;"),
    "channel_offset_dropped": (
        "f[d++] = pic_oracle_bilinear_at(y[l] + (int64_t)c * Hl * Wl, Hl, Wl, H, W, x, yy);",
        "f[d++] = pic_oracle_bilinear_at(y[l], Hl, Wl, H, W, x, yy);"),
    "zigzag_direction_flipped": (
        "if (d % 2 == 0)\n            for (int row = hi; row >= lo; --row)",
        "if (d % 2 == 1)\n            for (int row = hi; row >= lo; --row)"),
    "run_code_off_by_one": (
        "symbols[n++] = eob - 17 + run;",
        "symbols[n++] = eob - 16 + run - (run == 16);"),
    "izpr_run_length_off_by_one": (
        "int run = s + 17 - eob;",
        "int run = s + 16 - eob;"),
    "no_trailing_trim": (
        "if (zz[k] != 0) last = k;",
        "last = 63;"),
    "idct_transposed_coefficients": (
        "s += dct_alpha(u) * dct_alpha(v) * S[u * 8 + v] *",
        "s += dct_alpha(u) * dct_alpha(v) * S[v * 8 + u] *"),
    "dct_dc_weight_unnormalised": (
        "return k == 0 ? sqrt(1.0 / 8.0) : sqrt(2.0 / 8.0);",
        "return k == 0 ? 0.5 : sqrt(2.0 / 8.0);"),
    "idct_no_half_sample": (
        "S[u * 8 + v] *\n                         cos((2 * m + 1) * u * PIC_ORACLE_PI / 16.0)",
        "S[u * 8 + v] *\n                         cos((2 * m) * u * PIC_ORACLE_PI / 16.0)"),
    "patches_column_major": (
        "for (int by = 0; by < (Hl + 7) / 8; ++by)\n                for (int bx = 0; bx < (Wl + 7) / 8; ++bx, ++b) {\n                    double S[64], x[64];",
        "for (int bx = 0; bx < (Wl + 7) / 8; ++bx)\n                for (int by = 0; by < (Hl + 7) / 8; ++by, ++b) {\n                    double S[64], x[64];"),
    "patch_step_ignored": (
        "S[k] = (double)symbols[64 * b + k] * steps[l];",
        "S[k] = (double)symbols[64 * b + k];"),
    "patch_written_transposed": (
        "if (r < Hl && q < Wl) g[(int64_t)r * Wl + q] = x[m * 8 + n];",
        "if (r < Hl && q < Wl) g[(int64_t)r * Wl + q] = x[n * 8 + m];"),
    "block_count_floor": (
        "n += (int64_t)C * ((level_size(H, l) + 7) / 8) * ((level_size(W, l) + 7) / 8);",
        "n += (int64_t)C * (level_size(H, l) / 8 + 1) * (level_size(W, l) / 8 + 1);"),
    "value_levels_ignore_channels": (
        "off += (int64_t)C * level_size(H, l) * level_size(W, l);\n    }\n}\n\n/* Steps 2-5",
        "off += (int64_t)level_size(H, l) * level_size(W, l);\n    }\n}\n\n/* Steps 2-5"),
    "sample_std_not_population": (
        "sigma[c] = sqrt(v / (double)N);\n    }\n}",
        "sigma[c] = sqrt(v / (double)(N - 1));\n    }\n}"),
    "fused_bias_sign": (
        "s += w[(int64_t)i * C + c] * (beta[c] - gamma[c] * mu[c] / sigma[c]);",
        "s += w[(int64_t)i * C + c] * (beta[c] + gamma[c] * mu[c] / sigma[c]);"),
    "fused_weight_times_sigma": (
        "w_out[(int64_t)i * C + c] = w[(int64_t)i * C + c] * gamma[c] / sigma[c];",
        "w_out[(int64_t)i * C + c] = w[(int64_t)i * C + c] * gamma[c] * sigma[c];"),
    "fused_bias_drops_beta": (
        "s += w[(int64_t)i * C + c] * (beta[c] - gamma[c] * mu[c] / sigma[c]);",
        "s += w[(int64_t)i * C + c] * (0.0 - gamma[c] * mu[c] / sigma[c]);"),
    "mlps_without_last_activation": (
        "z[i] = pic_oracle_act(acc + bk[i], act);",
        "z[i] = (k == n_layers - 2) ? acc + bk[i] : pic_oracle_act(acc + bk[i], act);"),
    "modulate_before_normalise": (
        "for (int c = 0; c < Cf; ++c) f[c] = gamma[c] * ((f[c] - mu[c]) / sigma[c]) + beta[c];",
        "for (int c = 0; c < Cf; ++c) f[c] = (gamma[c] * f[c] + beta[c] - mu[c]) / sigma[c];"),
    "stats_second_pass_unshifted": (
        "for (int c = 0; c < Cf; ++c) v[c] += (f[c] - mu[c]) * (f[c] - mu[c]);",
        "for (int c = 0; c < Cf; ++c) v[c] += f[c] * f[c];"),
    "u8_truncates": (
        "return (int)nearbyint(255.0 * pic_oracle_clamp01(v));",
        "return (int)floor(255.0 * pic_oracle_clamp01(v));"),
    "u8_scale_256": (
        "return (int)nearbyint(255.0 * pic_oracle_clamp01(v));",
        "return (int)nearbyint(256.0 * pic_oracle_clamp01(v)) > 255 ? 255 : (int)nearbyint(256.0 * pic_oracle_clamp01(v));"),
    "canonical_code_shift_order": (
        "if (k > 0) c = (c + 1) << (tab_len[k] - tab_len[k - 1]);",
        "if (k > 0) c = (c << (tab_len[k] - tab_len[k - 1])) + 1;"),
    "huffman_lsb_first": (
        "if ((code[k] >> b) & 1u) words[bit >> 5] |= 0x80000000u >> (bit & 31);",
        "if ((code[k] >> b) & 1u) words[bit >> 5] |= 1u << (bit & 31);"),
    "package_merge_takes_one_more": (
        "take[max_len] = 2 * m - 2;",
        "take[max_len] = 2 * m - 1;"),
    "canonical_ties_descending": (
        "(len[order[b]] == len[v] && value[order[b]] > value[v]))) {",
        "(len[order[b]] == len[v] && value[order[b]] < value[v]))) {"),
    "package_merge_no_packages": (
        "if (lv > 1) take[lv - 1] = 2 * packs;",
        "if (lv > 1) take[lv - 1] = packs;"),
    "izpr_raster_not_zigzag": (
        "blk[order[pos++]] = s;",
        "blk[pos++] = s;"),
}


def _compile_mutant(name: str, tmp: str) -> str:
    with open(SRC) as f:
        src = f.read()
    old, new = MUTATIONS[name]
    assert src.count(old) == 1, f"mutation anchor for {name!r} not found exactly once"
    path = os.path.join(tmp, f"{name}.c")
    with open(path, "w") as f:
        f.write(src.replace(old, new))
    return oracle.compile_oracle(src=path, out=os.path.join(tmp, f"lib{name}.so"))


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(name):
    with tempfile.TemporaryDirectory() as tmp:
        mutant = oracle.load(_compile_mutant(name, tmp))
        failed = []
        for pin in oracle_pins.PINS:
            try:
                pin(mutant)
            except (AssertionError, ValueError):
                failed.append(pin.__name__)
        assert failed, f"no pin exposes the planted mistake {name!r}"
