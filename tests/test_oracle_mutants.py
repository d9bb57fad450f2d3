"""Planted mistakes in the oracle are caught by its pins (CPU).

Each case copies oracle/reco_oracle.c, plants one plausible mistake (a flipped sign, a
dropped term, an off-by-one index, a swapped operand, a boundary moved), compiles the
mutant, and in a separate process swaps it in for the oracle library and runs the pins
meant to catch it: at least one must fail (a mutant that crashes counts as caught)."""
import ctypes
import multiprocessing as mp
import os
import subprocess
import sys

import pytest

import oracle
import test_oracle_pins as P

SRC = os.path.join(os.path.dirname(oracle.__file__), "reco_oracle.c")

MUTANTS = {
    "eq1 sign of the adjustment": (
        "return base - delta * ((vi - mean) / range);", "return base + delta * ((vi - mean) / range);",
        [P.test_eq1_golden_cases]),
    "eq1 statistics without v_i": (
        "for (int s = 0; s < n; ++s) {", "for (int s = 0; s < n - 1; ++s) {",
        [P.test_eq1_golden_cases]),
    "eq2 causal mask dropped": (
        "int visible = L - w + t + 1;", "int visible = L;",
        [P.test_eq2_zero_query_closed_form]),
    "eq2 window position off by one": (
        "int visible = L - w + t + 1;", "int visible = L - w + t;",
        [P.test_eq2_zero_query_closed_form]),
    "eq2 sum over heads instead of mean": (
        "raw[j] = acc[j] / (double)G;", "raw[j] = acc[j];",
        [P.test_eq2_mass_is_window_size]),
    "eq2 scale dropped": (
        "dot += (double)qr[c] * (double)k[(size_t)j * d + c];\n                logit[j] = scale * dot;",
        "dot += (double)qr[c] * (double)k[(size_t)j * d + c];\n                logit[j] = dot;",
        [P.test_eq2_single_query_is_a_softmax_row, P.test_eq2_scale_enters_the_logits]),
    "decode scale dropped": (
        "dot += (double)q[c] * (double)k[(size_t)j * d + c];\n        logit[j] = scale * dot;",
        "dot += (double)q[c] * (double)k[(size_t)j * d + c];\n        logit[j] = dot;",
        [P.test_decode_matches_torch_sdpa]),
    "eq2 transposed query/key index": (
        "dot += (double)qr[c] * (double)k[(size_t)j * d + c];", "dot += (double)qr[c] * (double)k[(size_t)c * d + j];",
        [P.test_eq2_single_query_is_a_softmax_row]),
    "top-m ties to the higher index": (
        "return (i < j) ? -1 : (i > j);", "return (i > j) ? -1 : (i < j);",
        [P.test_eq2_hand_example_and_selection]),
    "top-m window not counted in m": (
        "int nc = L - w, kc = m - w;", "int nc = L - w, kc = m;",
        [P.test_select_invariants_and_identity]),
    "max-pool window one too wide": (
        "int half = pool / 2;", "int half = pool / 2 + 1;",
        [P.test_maxpool_matches_scipy]),
    "decode lse without its max": (
        "if (lse) *lse = mx + log(Z);", "if (lse) *lse = log(Z);",
        [P.test_decode_lse_is_the_eq2_row_normaliser]),
    "decode normaliser misses the last key": (
        "for (int j = 0; j < len; ++j) Z += exp(logit[j] - mx);",
        "for (int j = 0; j < len - 1; ++j) Z += exp(logit[j] - mx);",
        [P.test_decode_lse_is_the_eq2_row_normaliser]),
    "decode multiplies by K instead of V": (
        "out[c] += p * (double)v[(size_t)j * d + c];", "out[c] += p * (double)k[(size_t)j * d + c];",
        [P.test_decode_matches_torch_sdpa]),
    "eq3 lower band edge exclusive": (
        "if (v <= tau_l) return 0;", "if (v < tau_l) return 0;",
        [P.test_eq3_bands_golden]),
    "eq3 full penalty in the middle band": (
        "band == 1 ? (double)beta / 2.0 : (double)beta", "band == 1 ? (double)beta : (double)beta",
        [P.test_eq3_bands_golden]),
    "eq5 sign of the mean log-probability": (
        "ppl[b] = exp(-sum_lp / (double)nv);", "ppl[b] = exp(sum_lp / (double)nv);",
        [P.test_eq5_golden]),
    "sampling boundary taken inclusive": (
        "if (c > u && p > 0.0) {", "if (c >= u && p > 0.0) {",
        [P.test_sample_golden_cdf_boundaries]),
    "sampling before the penalty": (
        "int bad = oracle_reflect_penalty(logits, B, V, ids, n_ids, rewards, tau_l, tau_h, beta, NULL);",
        "int bad = 0;",
        [P.test_sample_draws_after_the_penalty]),
    "sampling normaliser without the max shift": (
        "for (int j = 0; j < V; ++j) Z += exp((double)z[j] - M);", "for (int j = 0; j < V; ++j) Z += exp((double)z[j]);",
        [P.test_sample_golden_cdf_boundaries]),
    "eq5 log-sum-exp without the max": (
        "sum_lp += (double)z[x] - (M + log(Z));", "sum_lp += (double)z[x] - log(Z);",
        [P.test_eq5_matches_torch_cross_entropy_and_ragged_lengths]),
}


def _build_mutant(tmp_path, old, new):
    text = open(SRC).read()
    assert text.count(old) == 1, f"mutation site not unique: {old!r}"
    src = tmp_path / "mutant.c"
    src.write_text(text.replace(old, new))
    so = tmp_path / "libmutant.so"
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math", "-ffp-contract=off",
                    str(src), "-o", str(so), "-lm"], check=True)
    return so


def _child(name, so, q):
    sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))
    import oracle as O
    import test_oracle_pins as PP
    O._lib = O._bind(ctypes.CDLL(so))
    failures = 0
    for pin_name in [p.__name__ for p in MUTANTS[name][2]]:
        pin = getattr(PP, pin_name)
        args = {}
        if pin_name == "test_eq2_zero_query_closed_form":
            args = dict(G=3, w=5, L=20)
        if pin_name == "test_maxpool_matches_scipy":
            args = dict(pool=7)
        try:
            pin(**args)
        except AssertionError:
            failures += 1
    q.put(failures)


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name, tmp_path):
    old, new, pins = MUTANTS[name]
    so = _build_mutant(tmp_path, old, new)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    p = ctx.Process(target=_child, args=(name, str(so), q))
    p.start()
    p.join(300)
    assert p.exitcode is not None, "mutant check hung"
    if p.exitcode < 0:  # killed by a signal: the planted mistake crashed the pins' run
        return
    assert p.exitcode == 0
    failures = q.get(timeout=10)
    assert failures >= 1, f"planted mistake '{name}' passed every pin"
