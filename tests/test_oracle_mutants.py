"""Planted mistakes: each pin of the oracle must be able to fail.

Every case below copies the oracle's C source, plants one plausible mistake
in it (a dropped term, a flipped sign, a wrong index, a transposed operand,
an off-by-one in a window or a mask), builds the copy with the same compiler
flags, and runs the pin suite (``tests/test_oracle_pins.py``) against it in a
child process.  The case passes only when some pin fails on the copy: a
mistake that every pin lets through would mark a gap in the pins.

The passages each mistake breaks (Sec. III-B "SpeechKV"): Eq. (pool) -- a
softmax over the gate logits u . k_j of a window, the value pooled with the
key's weights, the last window holding the frames present, text rows kept,
pooling from layer l0 on --; Eq. (attn) -- softmax(q K^T / sqrt(d_h)) V per
query head over its KV head, at prefill over the compressed rows up to the
query's own position; Sec. III-C -- one appended row per decoded token.

CPU only: the planted mistakes live in copies of the oracle, never in the
CUDA path, and nothing here touches a GPU.
"""
import concurrent.futures
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "speechkv_oracle.c")
PINS = os.path.join(ROOT, "tests", "test_oracle_pins.py")

# (name, text in the oracle, replacement, which occurrence (0-based))
MUTANTS = [
    # Eq. (pool)
    ("pool_value_plain_mean",
     "vs += z[j - j0] * V[j * row + (int64_t)h * d + c];",
     "vs += V[j * row + (int64_t)h * d + c] / (double)(j1 - j0);", 0),
    ("pool_gate_sign", "z[j - j0] = s;", "z[j - j0] = -s;", 0),
    ("pool_gate_on_values",
     "s += gate[(int64_t)h * d + c] * K[j * row + (int64_t)h * d + c];",
     "s += gate[(int64_t)h * d + c] * V[j * row + (int64_t)h * d + c];", 0),
    ("pool_weights_unnormalised", "z[j - j0] /= sum;", "z[j - j0] /= 1.0;", 0),
    ("pool_last_partial_window_dropped", "while (n * we < (int64_t)T)",
     "while ((n + 1) * we <= (int64_t)T)", 0),
    ("pool_from_layer_after_l0", "return layer >= l0 ? w : 1;",
     "return layer > l0 ? w : 1;", 0),
    ("pool_suffix_read_at_compressed_offset",
     "const int64_t src = ((int64_t)P + T + t) * row;",
     "const int64_t src = ((int64_t)P + n + t) * row;", 0),
    ("pool_suffix_values_from_keys",
     "V_out[dst + e] = store(V[src + e], storage);",
     "V_out[dst + e] = store(K[src + e], storage);", 0),
    ("pool_prefix_not_rounded",
     "K_out[t * row + e] = store(K[t * row + e], storage);",
     "K_out[t * row + e] = K[t * row + e];", 0),
    ("pool_window_one_frame_short", "j1 = (int64_t)P + (i + 1) * we;",
     "j1 = (int64_t)P + (i + 1) * we - 1;", 0),
    ("pool_last_window_runs_into_text", "if (j1 > (int64_t)P + T)",
     "if (j1 > (int64_t)P + T + N)", 0),
    ("pool_gate_of_head_zero", "s += gate[(int64_t)h * d + c] * K[",
     "s += gate[c] * K[", 0),
    ("pool_alpha_indexed_by_window",
     "alpha[(j - P) * H_kv + h] = z[j - j0];",
     "alpha[(j - j0) * H_kv + h] = z[j - j0];", 0),
    # length bookkeeping
    ("len_ignores_generated", "return (int64_t)P + n + (int64_t)N + (int64_t)G;",
     "return (int64_t)P + n + (int64_t)N;", 0),
    # storage rounding
    ("bf16_truncates", "double r = ldexp(nearbyint(ldexp(x, -q)), q);",
     "double r = ldexp(trunc(ldexp(x, -q)), q);", 0),
    ("bf16_seven_bits", "return round_sig_bits(x, 8,",
     "return round_sig_bits(x, 7,", 0),
    ("f32_rounds_as_bf16", "return (double)(float)x;",
     "return oracle_round_bf16(x);", 0),
    # Sec. III-C append
    ("append_length_not_advanced", "return n + 1;", "return n;", 0),
    ("append_value_row_gets_key", "memcpy(V_cache + n * row, v_new,",
     "memcpy(V_cache + n * row, k_new,", 0),
    # Eq. (attn) at decode
    ("decode_scale_one_over_d", "scale = 1.0 / sqrt((double)d);",
     "scale = 1.0 / (double)d;", 0),
    ("decode_heads_interleaved", "const int32_t h = hq / group;",
     "const int32_t h = hq % H_kv;", 0),
    ("decode_query_of_kv_head", "s += q[(int64_t)hq * d + c] * K[j * row",
     "s += q[(int64_t)h * d + c] * K[j * row", 0),
    ("decode_weights_unnormalised", "p[j] /= sum;", "p[j] /= 1.0;", 0),
    ("decode_no_max_shift", "p[j] = exp(p[j] - m);", "p[j] = exp(p[j]);", 0),
    ("decode_values_from_keys",
     "acc += p[j] * V[j * row + (int64_t)h * d + c];",
     "acc += p[j] * K[j * row + (int64_t)h * d + c];", 0),
    ("decode_drops_newest_row",
     "const int32_t group = H_q / H_kv;\n    const int64_t row",
     "const int32_t group = H_q / H_kv;\n    if (n > 1)\n        n -= 1;\n"
     "    const int64_t row", 0),
    ("decode_output_not_rounded",
     "out[(int64_t)hq * d + c] = store(acc, storage);",
     "out[(int64_t)hq * d + c] = acc;", 0),
    # Eq. (attn) at prefill, adjusted causal mask
    ("prefill_scale_one_over_d", "scale = 1.0 / sqrt((double)d);",
     "scale = 1.0 / (double)d;", 1),
    ("prefill_heads_interleaved", "const int32_t h = hq / group;",
     "const int32_t h = hq % H_kv;", 1),
    ("prefill_suffix_position_off_by_one", "return t - T + n;",
     "return t - T + n - 1;", 0),
    ("prefill_window_visible_only_when_complete",
     "return P + (t - P) / w_eff;", "return P + (t - P + 1) / w_eff - 1;", 0),
    ("prefill_suffix_boundary_in_speech", "if (t < (int64_t)P + T)\n",
     "if (t <= (int64_t)P + T)\n", 0),
    ("prefill_query_of_kv_head", "const double *q = Q + t * qrow + (int64_t)hq * d;",
     "const double *q = Q + t * qrow + (int64_t)h * d;", 0),
    ("prefill_weights_unnormalised", "store(acc / sum, storage)", "store(acc, storage)", 0),
    ("prefill_values_from_keys",
     "acc += p[e] * V[e * krow + (int64_t)h * d + k];",
     "acc += p[e] * K[e * krow + (int64_t)h * d + k];", 0),
    ("prefill_output_not_rounded",
     "out[t * qrow + (int64_t)hq * d + k] = store(acc / sum, storage);",
     "out[t * qrow + (int64_t)hq * d + k] = acc / sum;", 0),
]


def _plant(src: str, old: str, new: str, nth: int) -> str:
    at = -1
    for _ in range(nth + 1):
        at = src.find(old, at + 1)
        assert at >= 0, f"mutation target not found: {old!r} (occurrence {nth})"
    return src[:at] + new + src[at + len(old):]


def _run_pins(lib: str) -> subprocess.CompletedProcess:
    env = dict(os.environ, SPEECHKV_ORACLE_LIB=lib)
    return subprocess.run(
        [sys.executable, "-m", "pytest", PINS, "-x", "-q", "-p", "no:cacheprovider",
         "-W", "ignore::RuntimeWarning"],
        cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)


@pytest.fixture(scope="module")
def mutant_runs(tmp_path_factory):
    src = open(SRC).read()
    tmp = tmp_path_factory.mktemp("oracle_mutants")
    libs = {}
    for name, old, new, nth in MUTANTS:
        c = tmp / f"{name}.c"
        c.write_text(_plant(src, old, new, nth))
        so = tmp / f"{name}.so"
        subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
                        "-o", str(so), str(c), "-lm"], check=True)
        libs[name] = str(so)
    # the unmodified source, built the same way, must pass every pin
    c = tmp / "unmodified.c"
    c.write_text(src)
    so = tmp / "unmodified.so"
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
                    "-o", str(so), str(c), "-lm"], check=True)
    libs["unmodified"] = str(so)
    workers = max(1, min(8, os.cpu_count() or 1))
    with concurrent.futures.ThreadPoolExecutor(workers) as ex:
        futs = {name: ex.submit(_run_pins, lib) for name, lib in libs.items()}
        return {name: f.result() for name, f in futs.items()}


def test_unmodified_copy_passes_the_pins(mutant_runs):
    r = mutant_runs["unmodified"]
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]


@pytest.mark.parametrize("name", [m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(mutant_runs, name):
    r = mutant_runs[name]
    # exit code 1: the suite ran and at least one pin failed (not a crash,
    # not a collection error)
    assert r.returncode == 1, (
        f"{name}: pins exit {r.returncode}\n" + r.stdout[-2000:] + r.stderr[-2000:])
    assert " failed" in r.stdout
