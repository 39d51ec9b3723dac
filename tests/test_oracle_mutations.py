"""Planted mistakes: each case below copies bisco_oracle.c with one
plausible slip (a dropped term, a wrong sign, index or bit order, a rounding
mode), builds the copy, and runs the pin suite against it.  The pins must
fail for every one of them -- otherwise they would not pin the oracle.  All
of it runs on the CPU; nothing here touches the CUDA library."""
import os
import subprocess
import sys

import pytest

import oracle

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)

# name -> (text in bisco_oracle.c, replacement)
MUTATIONS = {
    "residual_sign": ("v[k] = v[k] - rhat;", "v[k] = v[k] + rhat;"),
    "mask_dropped_after_stage_1": ("if (prot[8 * c + k]) v[k] = 0.0;", ";"),
    "bit_order_reversed": ("bits |= (uint8_t)(1u << k);", "bits |= (uint8_t)(1u << (7 - k));"),
    "zero_encoded_negative": ("if (v[k] < 0.0) bits", "if (v[k] <= 0.0) bits"),
    "decode_without_inv_sqrt8": ("double t = or_fp16_to_double(norms[e]) * inv_sqrt8;",
                                 "double t = or_fp16_to_double(norms[e]);"),
    "decode_drops_last_stage": (
        "for (int32_t s = 0; s < S; ++s) {\n                int64_t e = ((int64_t)s * N + i) * C + c;\n"
        "                double t = or_fp16_to_double(norms[e]) * inv_sqrt8;",
        "for (int32_t s = 0; s < S - 1; ++s) {\n                int64_t e = ((int64_t)s * N + i) * C + c;\n"
        "                double t = or_fp16_to_double(norms[e]) * inv_sqrt8;"),
    "protected_scatter_missing": (
        "acc = acc + (((codes[e] >> k) & 1) ? -t : t);\n            }\n            o[j] = acc;\n        }\n"
        "        for (int32_t t = 0; t < p; ++t)\n"
        "            o[idx[t]] = or_fp16_to_double(scale[t]) * (double)q8[(int64_t)i * pp + t];",
        "acc = acc + (((codes[e] >> k) & 1) ? -t : t);\n            }\n            o[j] = acc;\n        }\n"),
    "table_decode_protected_scatter_missing": (
        "acc = acc + or_fp16_to_double(norms[e]) * t;\n            }\n            o[j] = acc;\n        }\n"
        "        for (int32_t t = 0; t < p; ++t)\n"
        "            o[idx[t]] = or_fp16_to_double(scale[t]) * (double)q8[(int64_t)i * pp + t];",
        "acc = acc + or_fp16_to_double(norms[e]) * t;\n            }\n            o[j] = acc;\n        }\n"),
    "q8_truncates": ("q = nearbyint(or_bf16_to_double(W[(int64_t)i * K + j]) / s);",
                     "q = trunc(or_bf16_to_double(W[(int64_t)i * K + j]) / s);"),
    "q8_divides_by_unrounded_scale": (
        "double s = or_fp16_to_double(s16);\n        for (int32_t i = 0; i < N; ++i) {",
        "double s = m / 127.0;\n        for (int32_t i = 0; i < N; ++i) {"),
    "row_q8_divides_by_unrounded_scale": (
        "double s = or_fp16_to_double(s16);\n        for (int32_t k = 0; k < K; ++k) {",
        "double s = m / 127.0;\n        for (int32_t k = 0; k < K; ++k) {"),
    "selection_ties_to_higher_index": ("return (x->j < y->j) ? -1 : (x->j > y->j);",
                                       "return (x->j > y->j) ? -1 : (x->j < y->j);"),
    "fp16_rounds_toward_zero": ("double m = nearbyint(ldexp(a, 10 - E));",
                                "double m = floor(ldexp(a, 10 - E));"),
    "matmul_reversed_activation": ("or_bf16_to_double(X[(int64_t)b * K + j]);",
                                   "or_bf16_to_double(X[(int64_t)b * K + (K - 1 - j)]);"),
    "coupled_drops_down_term": ("double s = (tg + tu) + td;", "double s = tg + tu;"),
    "rows_not_masked": ("memset(Wm + (int64_t)idx[t] * K, 0, sizeof(uint16_t) * (size_t)K);", ";"),
    "row_scale_from_half_row": (
        "for (int32_t k = 0; k < K; ++k) {\n            double a = fabs(or_bf16_to_double(W[(int64_t)i * K + k]));",
        "for (int32_t k = 0; k < K / 2; ++k) {\n            double a = fabs(or_bf16_to_double(W[(int64_t)i * K + k]));"),
    "row_decode_keeps_bsq": ("out[(int64_t)(i - row0) * K + k] = s * (double)q8[(int64_t)t * kp + k];", ";"),
    "lora_bm_transposed": ("or_bf16_to_double(Bm[(int64_t)n * rank + r]) * t[r];",
                           "or_bf16_to_double(Bm[(int64_t)r * N + n]) * t[r];"),
    "lora_scale_dropped": ("Y0[(int64_t)b * N + n] + scale * acc;", "Y0[(int64_t)b * N + n] + acc;"),
    "fp8_rounds_toward_zero": ("double m = nearbyint(ldexp(a, mb - E));",
                               "double m = floor(ldexp(a, mb - E));"),
    "fp8_e4m3_bias_off_by_one": ("*mbits = 3; *bias = 7;", "*mbits = 3; *bias = 8;"),
    "fp8_scale_over_127": ("uint16_t s16 = or_double_to_fp16(m / maxf);",
                           "uint16_t s16 = or_double_to_fp16(m / 127.0);"),
    "fp8_subnormal_step_wrong": ("double m = nearbyint(ldexp(a, bias - 1 + mb));",
                                 "double m = nearbyint(ldexp(a, bias + mb));"),
    "decoder_table_ignores_stage": ("tables[((int64_t)s * 256 + codes[e]) * 8 + k]",
                                    "tables[((int64_t)0 * 256 + codes[e]) * 8 + k]"),
    "decoder_table_transposed": ("tables[((int64_t)s * 256 + codes[e]) * 8 + k]",
                                 "tables[(int64_t)s * 2048 + (int64_t)k * 256 + codes[e]]"),
    "linear_decoder_transposed": ("acc = acc + A[k * 8 + j] * or_code_elem(v, j);",
                                  "acc = acc + A[j * 8 + k] * or_code_elem(v, j);"),
    "code_element_sign_flipped": ("return ((v >> k) & 1) ? -t : t;", "return ((v >> k) & 1) ? t : -t;"),
    "mlp_residual_replaces_hidden": ("for (int32_t a = 0; a < hdim; ++a) h[a] = h[a] + g[a];",
                                     "for (int32_t a = 0; a < hdim; ++a) h[a] = g[a];"),
    "mlp_output_weights_transposed": ("acc = acc + W2[(int64_t)k * hdim + a] * h[a];",
                                      "acc = acc + W2[(int64_t)a * 8 + k] * h[a];"),
}


@pytest.fixture(scope="module")
def source():
    with open(os.path.join(ROOT, "oracle", "bisco_oracle.c")) as f:
        return f.read()


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, source, tmp_path):
    old, new = MUTATIONS[name]
    assert source.count(old) == 1, "mutation anchor not found once: " + name
    src = tmp_path / "bisco_oracle_mutant.c"
    src.write_text(source.replace(old, new))
    lib = tmp_path / "libbisco_oracle_mutant.so"
    subprocess.check_call(["gcc", *oracle.CFLAGS, "-o", str(lib), str(src), "-lm"])
    env = dict(os.environ, BISCO_ORACLE_LIB=str(lib))
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(HERE, "test_oracle_pins.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 1, "pins passed with the planted mistake %r:\n%s" % (
        name, r.stdout[-2000:])
