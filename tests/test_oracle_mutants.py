"""The oracle's pins catch plausible mistakes (CPU only).

Each case plants one mistake in a copy of the C oracle -- a flipped RoPE
sign, the router input stacked in the wrong order, a dropped gain, bias or
norm, a transposed projection, the wrong kv head for a grouped query, a
missing 1/sqrt(d), a prefill query reading its own slot, ... -- compiles the
copy, and runs the pin suite
(tests/test_oracle_pins.py) against it in a child process.  A mutant that
passes every pin would mean a wrong oracle could go unnoticed, so each one
must make at least one pin fail.  The unmodified copy, built the same way,
must pass them all.
"""
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "wm_oracle.c")

# (name, text in wm_oracle.c, its planted replacement); each text occurs once
MUTANTS = [
    ("rope_sign", "y[i] = x0 * c - x1 * s;", "y[i] = x0 * c + x1 * s;"),
    ("rope_frequency", "double a = pos * pow(theta, -2.0 * i / d);",
     "double a = pos * pow(theta, -1.0 * i / d);"),
    ("rmsnorm_eps_placement", "double r = 1.0 / sqrt(ss / n + eps);",
     "double r = 1.0 / (sqrt(ss / n) + eps);"),
    ("router_input_order", "int l = L - 1 - m * p;", "int l = m * p;"),
    ("router_reshape_order", "int j = o / L, l = o % L;", "int j = o % k, l = o / k;"),
    ("premix_gain_dropped", "orc_rmsnorm(x, D, eps, g, hhat + ((int64_t)X * L + l) * D);",
     "orc_rmsnorm(x, D, eps, NULL, hhat + ((int64_t)X * L + l) * D);"),
    ("mix_weight_index", "ht[e] += alpha_Xj[l] * hhat_X[(int64_t)l * D + e];",
     "ht[e] += alpha_Xj[L - 1 - l] * hhat_X[(int64_t)l * D + e];"),
    ("channel_norm_skipped", "orc_rmsnorm(ht, D, eps, g, xn);",
     "memcpy(xn, ht, sizeof(double) * D);"),
    ("qk_norm_skipped", "orc_rmsnorm(out + (int64_t)hh * d, d, eps_qk, gq, y);",
     "memcpy(y, out + (int64_t)hh * d, sizeof(double) * d);"),
    ("values_rotated_too", "if (is_key) {", "if (1) {"),
    ("decode_scale_missing", "s[t] = acc * inv_sqrt_d;", "s[t] = acc;"),
    ("decode_gqa_map", "int hkv = hq / group;\n    int S = seq_lens[b];",
     "int hkv = hq % Hkv;\n    int S = seq_lens[b];"),
    ("decode_reads_keys_as_values",
     "o[e] += wt * rd(v_pool, base[t] + e, dt);\n    }\n    for (int e = 0; e < d; ++e) o[e] /= wsum;\n    m_attn += 2 * (int64_t)S * d;",
     "o[e] += wt * rd(k_pool, base[t] + e, dt);\n    }\n    for (int e = 0; e < d; ++e) o[e] /= wsum;\n    m_attn += 2 * (int64_t)S * d;"),
    ("prefill_reads_own_slot", "int nslots = i + 1; /* slots 0 .. i */",
     "int nslots = i + 2; /* slots 0 .. i */"),
    ("prefill_scale_missing", "s[t] = acc * scale;", "s[t] = acc;"),
    ("router_bias_dropped", "double z = rd(br, (int64_t)X * k * L + o, dt);", "double z = 0.0;"),
    ("router_shared_by_branches", "const void* W = adv(Wr, (int64_t)X * k * L * in_dim, dt);",
     "const void* W = Wr;"),
    ("projection_transposed", "acc += rd(W_Xj, n * D + e, dt) * xn[e];",
     "acc += rd(W_Xj, (int64_t)e * n_out + n, dt) * xn[e];"),
]


def _build(tmp_path, name, text):
    src = tmp_path / f"{name}.c"
    src.write_text(text)
    lib = tmp_path / f"lib{name}.so"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-shared", "-fPIC", "-o",
                           str(lib), str(src), "-lm"])
    return str(lib)


def _pins_pass(lib) -> bool:
    env = dict(os.environ, WM_ORACLE_LIB=lib, OMP_NUM_THREADS="2")
    r = subprocess.run([sys.executable, "-m", "pytest", os.path.join(ROOT, "tests",
                        "test_oracle_pins.py"), "-x", "-q", "-p", "no:cacheprovider"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return r.returncode == 0


def test_unmodified_copy_passes_the_pins(tmp_path):
    with open(SRC) as f:
        text = f.read()
    assert _pins_pass(_build(tmp_path, "unmodified", text))


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(tmp_path, name, old, new):
    with open(SRC) as f:
        text = f.read()
    assert text.count(old) == 1, f"mutation site of {name} not unique"
    assert not _pins_pass(_build(tmp_path, name, text.replace(old, new)))
