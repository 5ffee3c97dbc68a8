"""The oracle pins catch planted mistakes.

Each case copies the oracle's C source, plants one plausible mistake (a
dropped term, a wrong sign, a wrong index, a transposed operand, ...),
compiles the copy and runs the pin suite against it in a subprocess.  The
pins must fail for every mutant; the unmodified source must pass.
"""
import os
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "dopr_oracle.c")
PINS = os.path.join(ROOT, "tests", "test_oracle_pins.py")

# (name, original text, planted text)
MUTANTS = [
    ("rmsnorm_no_eps", "sqrt(ss / (double)n + eps)", "sqrt(ss / (double)n)"),
    ("rmsnorm_sum_not_mean", "sqrt(ss / (double)n + eps)", "sqrt(ss + eps)"),
    ("rope_sign", "x[i] = x1 * c - x2 * s;", "x[i] = x1 * c + x2 * s;"),
    ("rope_freq", "pow(theta, -2.0 * (double)i / (double)D)", "pow(theta, -1.0 * (double)i / (double)D)"),
    ("positions_not_offset", "oracle_rope(qh, D, (double)(pos0 + t), M->rope_theta);",
     "oracle_rope(qh, D, (double)t, M->rope_theta);"),
    ("gqa_interleaved", "int g = h / G;", "int g = h % Hkv;"),
    ("not_causal", "Vall + (size_t)g * S * D, m + t + 1,", "Vall + (size_t)g * S * D, m + T,"),
    ("softmax_scale", "const double scale = 1.0 / sqrt((double)D);", "const double scale = 1.0 / (double)D;"),
    ("score_sign", "return yes - no;", "return no - yes;"),
    ("silu_sign", "return x / (1.0 + exp(-x));", "return x / (1.0 + exp(x));"),
    ("attn_residual_dropped", "for (size_t i = 0; i < (size_t)T * H; ++i) r[i] += dlt[i];\n        /* post",
     "for (size_t i = 0; i < (size_t)T * H; ++i) r[i] = dlt[i];\n        /* post"),
    ("linear_transposed", "const uint16_t *w = W + (size_t)o * in;\n            for (int i = 0; i < in; ++i) wrow[i] = oracle_bf16_to_f64(w[i]);",
     "const uint16_t *w = W + (size_t)o;\n            for (int i = 0; i < in; ++i) wrow[i] = oracle_bf16_to_f64(w[(size_t)i * out]);"),
    ("qnorm_uses_knorm_gain", "widen(M->q_norm[l], D, gw);", "widen(M->k_norm[l], D, gw);"),
    ("no_final_norm", "oracle_rmsnorm(h, g, H, M->rms_eps, hn);", "memcpy(hn, h, sizeof(double) * (size_t)H);"),
    ("score_token_dropped", "ids[L] = M->score_token_id;", "ids[L] = 0;"),
    ("stored_v_from_k", "const double *sv = pv + (((size_t)l * m + i) * Hkv + g) * D;",
     "const double *sv = pk + (((size_t)l * m + i) * Hkv + g) * D;"),
    ("pack_positions_unshifted", "tok_pos[off + j] = pair_m[p] + j;", "tok_pos[off + j] = j;"),
    ("salience_mean_over_all", "u[i] = acc / (double)k;", "u[i] = acc / (double)cnt;"),
    ("topk_ties_to_higher", "return (x->idx > y->idx) - (x->idx < y->idx);", "return (x->idx < y->idx) - (x->idx > y->idx);"),
    ("probs_average_over_kv_heads", "row[i] += pw[i] / (double)Hq;", "row[i] += pw[i] / (double)Hkv;"),
    ("probs_key_count", "Kall + (size_t)kvh * S * D, m + t + 1, D,", "Kall + (size_t)kvh * S * D, m + t, D,"),
    ("mlp_bias_dropped", "double z = oracle_bf16_to_f64(b1[j]);", "double z = 0.0;"),
    ("mlp_gelu_tanh_form", "a = 0.5 * z * (1.0 + erf(z / sqrt(2.0)));", "a = 0.5 * z * (1.0 + tanh(z / sqrt(2.0)));"),
]


def _run_pins(lib_path: str) -> int:
    env = dict(os.environ, DOPR_ORACLE_LIB=lib_path, OMP_NUM_THREADS="1")
    r = subprocess.run([sys.executable, "-m", "pytest", PINS, "-x", "-q", "-p", "no:cacheprovider"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return r.returncode


def _build_mutant(tmp, name, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, f"{name}: pattern must occur exactly once"
    path = os.path.join(tmp, f"{name}.c")
    with open(path, "w") as f:
        f.write(src.replace(old, new))
    return oracle.build(force=True, src=path, out=os.path.join(tmp, f"lib_{name}.so"))


def test_unmodified_oracle_passes_pins(tmp_path):
    lib = oracle.build(force=True, src=SRC, out=str(tmp_path / "lib_clean.so"))
    assert _run_pins(lib) == 0


def test_every_planted_mistake_is_caught(tmp_path):
    libs = {name: _build_mutant(str(tmp_path), name, old, new) for name, old, new in MUTANTS}
    with ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 2)) as ex:
        rcs = dict(zip(libs, ex.map(_run_pins, libs.values())))
    survived = [n for n, rc in rcs.items() if rc == 0]
    assert not survived, f"mutants not caught by the pins: {survived}"
