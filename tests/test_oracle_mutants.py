"""The pins in test_oracle_pins.py must catch plausible mistakes in the oracle.

Each case plants one mistake in a private copy of oracle/lla_oracle.c (compiled on the CPU
into a temporary directory), runs the pin tests against that copy, and expects them to fail.
The committed oracle is never modified.
"""
import os
import subprocess
import sys
import tempfile
from concurrent.futures import ThreadPoolExecutor

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "lla_oracle.c")

# (name, exact text in the oracle, planted replacement)
MUTANTS = [
    ("ratio_drops_factor_2", "return 2.0 * (double)T * (double)d_head",
     "return (double)T * (double)d_head"),
    ("encode_wrong_stacking", "xs[t * d + e] = x[((int64_t)t * N + n) * d + e];",
     "xs[e * T + t] = x[((int64_t)t * N + n) * d + e];"),
    ("encode_mu_sign", "xs[k] = xs[k] - mu[k];", "xs[k] = xs[k] + mu[k];"),
    ("decode_transposed_w_up", "acc += c[n * r + j] * w_up_t[(int64_t)e * r + j];",
     "acc += c[n * r + j] * w_up_t[(int64_t)j * d + e];"),
    ("decode_drops_mu_t", "xhat[n * d + e] = acc + (mu_t ? mu_t[e] : 0.0);",
     "xhat[n * d + e] = acc;"),
    ("decode_wrong_loop_slice",
     "lla_oracle_reconstruct(d, r_k, L, c_k, w_up_k + (int64_t)t * d * r_k,",
     "lla_oracle_reconstruct(d, r_k, L, c_k, w_up_k,"),
    ("attention_drops_scale", "s[i] = scale * dot;", "s[i] = dot;"),
    ("attention_no_max_subtraction", "s[i] = exp(s[i] - m);", "s[i] = exp(s[i]);"),
    ("pass1_value_is_key", "memcpy(V + L * d, cur_v,", "memcpy(V + L * d, cur_k,"),
    ("prefill_not_causal", "rc = lla_oracle_attention(d, i + 1, q + i * d, K, V, scale, out + i * d);",
     "rc = lla_oracle_attention(d, N, q + i * d, K, V, scale, out + i * d);"),
    ("rope_sin_sign", "y[a] = x[a] * c - x[b] * s;", "y[a] = x[a] * c + x[b] * s;"),
    ("rope_theta_exponent", "const double theta = pow(base, -2.0 * j / d);",
     "const double theta = pow(base, -1.0 * j / d);"),
    ("rope_pairing_mixed", "const int b = pairing ? 2 * j + 1 : j + h;",
     "const int b = pairing ? j + h : 2 * j + 1;"),
    ("rope_query_position", "lla_oracle_rope(d, pairing, base, pos0 + n - 1, q, qr);",
     "lla_oracle_rope(d, pairing, base, pos0 + L, q, qr);"),
    ("rope_keys_not_rotated",
     "for (int64_t i = 0; i < n; ++i)\n        lla_oracle_rope(d, pairing, base, pos0 + i, K + i * d, Kr + i * d);",
     "for (int64_t i = 0; i < n; ++i)\n        memcpy(Kr + i * d, K + i * d, sizeof(double) * (size_t)d);"),
    ("prefill_rope_query_position", "lla_oracle_rope(d, pairing, base, pos0 + i, q + i * d, qr);",
     "lla_oracle_rope(d, pairing, base, pos0, q + i * d, qr);"),
    ("decoupled_query_position",
     "lla_oracle_rope(d_rope, pairing, base, pos0 + n - 1, q_rope, qj + d);",
     "lla_oracle_rope(d_rope, pairing, base, pos0 + L, q_rope, qj + d);"),
    ("decoupled_key_position",
     "lla_oracle_rope(d_rope, pairing, base, pos0 + i, kr, J + i * w + d);",
     "lla_oracle_rope(d_rope, pairing, base, pos0, kr, J + i * w + d);"),
    ("decoupled_rotary_dropped", "for (int e = 0; e < w; ++e)\n            dot += qj[e] * J[i * w + e];",
     "for (int e = 0; e < d; ++e)\n            dot += qj[e] * J[i * w + e];"),
    ("decoupled_current_rotary_key", "const double *kr = i < L ? k_rope + i * d_rope : cur_k_rope;",
     "const double *kr = i < L ? k_rope + i * d_rope : k_rope;"),
    ("decoupled_drops_scale", "sj[i] = dot * scale;", "sj[i] = dot;"),
    ("ratio_2d_drops_heads",
     "return 2.0 * (double)T * (double)H * (double)d_head / (double)(r_k + r_v);",
     "return 2.0 * (double)T * (double)d_head / (double)(r_k + r_v);"),
    ("encode_2d_head_major_stack",
     "xs[((int64_t)t * H + h) * d + e] = x[(((int64_t)t * N + n) * H + h) * d + e];",
     "xs[((int64_t)h * T + t) * d + e] = x[(((int64_t)t * N + n) * H + h) * d + e];"),
    ("encode_2d_mu_sign", "xs[k] -= mu[k];", "xs[k] += mu[k];"),
    ("decode_2d_pass1_value_is_key", "V[L * d + e] = cur_v[e];", "V[L * d + e] = cur_k[e];"),
    ("decode_2d_head_major_slice", "const int64_t th = (int64_t)t * H + h;",
     "const int64_t th = (int64_t)h * T + t;"),
    ("decode_2d_mu_loop_slice", "mu_k ? mu_k + th * d : NULL, K);",
     "mu_k ? mu_k + (int64_t)t * d : NULL, K);"),
    ("decode_2d_value_loop_only", "lla_oracle_reconstruct(d, r_v, L, c_v, w_up_v + th * d * r_v,",
     "lla_oracle_reconstruct(d, r_v, L, c_v, w_up_v + (int64_t)t * d * r_v,"),
]


def _run_mutant(name, old, new, tmp):
    src = open(SRC).read()
    assert src.count(old) == 1, f"{name}: anchor text not found exactly once"
    path_c = os.path.join(tmp, f"{name}.c")
    path_so = os.path.join(tmp, f"lib{name}.so")
    with open(path_c, "w") as f:
        f.write(src.replace(old, new))
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-fopenmp", path_c, "-o",
                    path_so, "-lm"], check=True)
    # one OpenMP thread per mutant: the mutants already run side by side
    env = dict(os.environ, LLA_ORACLE_LIB=path_so, OMP_NUM_THREADS="1")
    res = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                          os.path.join(ROOT, "tests", "test_oracle_pins.py")],
                         cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return name, res.returncode


def test_pins_catch_every_planted_mistake():
    with tempfile.TemporaryDirectory() as tmp:
        with ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 2)) as ex:
            results = list(ex.map(lambda m: _run_mutant(*m, tmp), MUTANTS))
    survivors = [name for name, rc in results if rc == 0]
    assert not survivors, f"pins did not catch: {survivors}"
