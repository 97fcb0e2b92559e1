"""The oracle's pins catch plausible mistakes.

Each case plants one mistake in a copy of ``oracle/oracle.c`` (on the CPU), builds it, and
runs the pin suite against that build in a child process; the suite must fail. A case whose
mistake the pins no longer detect fails here.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "oracle.c")

MUTANTS = {
    "silu_is_sigmoid": ("return u / (1.0 + exp(-u));", "return 1.0 / (1.0 + exp(-u));"),
    "silu_wrong_sign": ("return u / (1.0 + exp(-u));", "return u / (1.0 + exp(u));"),
    "down_transposed": ("Dl[(int64_t)k * d + j]", "Dl[(int64_t)j * r + k]"),
    "up_transposed": ("Ul[(int64_t)j * r + k]", "Ul[(int64_t)k * d + j]"),
    "residual_dropped": ("m[j] = x[j] + s;", "m[j] = s;"),
    "norm_sum_not_mean": ("sqrt(ss / (double)d + eps)", "sqrt(ss + eps)"),
    "eps_outside_sqrt": ("sqrt(ss / (double)d + eps)", "(sqrt(ss / (double)d) + eps)"),
    "gain_dropped": ("n[j] = gamma[j] * m[j] * inv;", "n[j] = m[j] * inv;"),
    "projection_transposed": ("bf16_to_f64(W[(int64_t)c * d + j])", "bf16_to_f64(W[(int64_t)j * kv + c])"),
    "bias_dropped": ("out[c] = s + (b ? bf16_to_f64(b[c]) : 0.0);", "out[c] = s;"),
    "rope_wrong_direction": ("x[j] = x1 * c - x2 * s;", "x[j] = x1 * c + x2 * s;"),
    "rope_interleaved_pairs": ("double x1 = x[j], x2 = x[j + half];", "double x1 = x[2 * j], x2 = x[2 * j + 1];"),
    "rope_frequency_exponent": ("pow(theta, -2.0 * (double)j / (double)head_dim)", "pow(theta, -(double)j / (double)head_dim)"),
    "mrope_axes_swapped": ("if (j >= section[0] + section[1]) return 2;", "if (j >= section[0] + section[1]) return 1;"),
    "mrope_interleave_offset": ("if (j % 3 == 1 && j < 3 * section[1]) return 1;",
                                "if (j % 3 == 0 && j < 3 * section[1]) return 1;"),
    "k_norm_over_whole_vector": ("oracle_head_rmsnorm(Dh, kgamma + (int64_t)l * Dh, c->k_norm_eps, kk + hh * Dh);",
                                 "{ if (hh == 0) { double ss = 0.0; for (int j = 0; j < kv; ++j) ss += kk[j] * kk[j]; "
                                 "const double inv = 1.0 / sqrt(ss / kv + c->k_norm_eps); for (int j = 0; j < kv; ++j) "
                                 "kk[j] *= bf16_to_f64(kgamma[(int64_t)l * Dh + j % Dh]) * inv; } }"),
    "k_norm_after_rope": ("  if (c->k_norm)\n    for (int hh = 0; hh < c->n_kv_heads; ++hh)\n"
                          "      oracle_head_rmsnorm(Dh, kgamma + (int64_t)l * Dh, c->k_norm_eps, kk + hh * Dh);\n"
                          "  for (int hh = 0; hh < c->n_kv_heads; ++hh)\n"
                          "    oracle_rope_head(Dh, c->rope_theta, c->rope, c->mrope_section, p3, kk + hh * Dh);",
                          "  for (int hh = 0; hh < c->n_kv_heads; ++hh)\n"
                          "    oracle_rope_head(Dh, c->rope_theta, c->rope, c->mrope_section, p3, kk + hh * Dh);\n"
                          "  if (c->k_norm)\n    for (int hh = 0; hh < c->n_kv_heads; ++hh)\n"
                          "      oracle_head_rmsnorm(Dh, kgamma + (int64_t)l * Dh, c->k_norm_eps, kk + hh * Dh);"),
    "k_norm_without_gain": ("x[j] = bf16_to_f64(g[j]) * x[j] * inv;", "x[j] = x[j] * inv;"),
    "attention_scale_dropped": ("const double w = exp(scale * dot - mx);", "const double w = exp(dot - mx);"),
    "attention_causal_off_by_one": ("for (int s = 0; s <= last; ++s) {\n          const double* kr = k + (((int64_t)b * S + s) * Hkv + h) * D;\n          const double* vr",
                                    "for (int s = 0; s < last; ++s) {\n          const double* kr = k + (((int64_t)b * S + s) * Hkv + h) * D;\n          const double* vr"),
    "attention_group_mapping": ("const int h = hq / G;", "const int h = hq % Hkv;"),
    "attention_not_normalised": ("for (int j = 0; j < D; ++j) o[j] /= den;", "(void)den;"),
    "k_norm_mean_as_sum": ("const double inv = 1.0 / sqrt(ss / (double)head_dim + eps);",
                           "const double inv = 1.0 / sqrt(ss + eps);"),
    "value_rotated": ("oracle_rope_head(Dh, c->rope_theta, c->rope, c->mrope_section, p3, kk + hh * Dh);",
                      "{ oracle_rope_head(Dh, c->rope_theta, c->rope, c->mrope_section, p3, kk + hh * Dh); "
                      "oracle_rope_head(Dh, c->rope_theta, c->rope, c->mrope_section, p3, vv + hh * Dh); }"),
    "position_of_wrong_batch": ("pos[(b * P + a) * n_vis + i]", "pos[a * n_vis + i]"),
    "recurrent_chain_not_carried": ("memcpy(prev, m, sizeof(double) * d);", ";"),
    "recurrent_starts_from_zero": ("prev[j] = bf16_to_f64(x0[t * d + j]);  /* M_0 = E */",
                                   "prev[j] = 0.0;"),
    "recurrent_down_of_next_layer": ("oracle_adapter_row(d, r, prev, D + (int64_t)l * r * d,",
                                     "oracle_adapter_row(d, r, prev, D + (int64_t)((l + 1) % L) * r * d,"),
    "recurrent_outputs_previous_state": ("memory_outputs(c, l, m, h, gamma, Wk, Wv, bk, bv, kgamma, p3, q * Ls + s,",
                                         "memory_outputs(c, l, prev, h, gamma, Wk, Wv, bk, bv, kgamma, p3, q * Ls + s,"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_reject_mutant(name, tmp_path):
    old, new = MUTANTS[name]
    src = open(SRC).read()
    assert src.count(old) >= 1, f"mutation site for {name} no longer in oracle.c"
    mutated = tmp_path / "oracle_mut.c"
    mutated.write_text(src.replace(old, new))
    lib = tmp_path / "liboracle_mut.so"
    subprocess.check_call(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-fopenmp", str(mutated),
                           "-o", str(lib), "-lm"])
    env = dict(os.environ, DV_ORACLE_LIB=str(lib), OMP_NUM_THREADS="2")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode != 0, f"pins did not catch mutant {name}:\n{r.stdout[-2000:]}"
