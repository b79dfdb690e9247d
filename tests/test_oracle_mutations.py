"""The oracle's pins have teeth: plant a plausible mistake in a copy of the C oracle,
compile it on the CPU, and check that at least one pin test fails against it."""
import ctypes
import os
import subprocess

import pytest

import oracle
from tests import test_oracle_pins as pins

SRC = os.path.join(os.path.dirname(oracle.__file__), "precog_oracle.c")

MUTATIONS = {
    "dropped_beta": ("h[n] = h[n] * alpha + beta;", "h[n] = h[n] * alpha;"),
    "exponent_sign": ("exp(dt_td * A[d * N + n])", "exp(-dt_td * A[d * N + n])"),
    "transposed_A": ("exp(dt_td * A[d * N + n])", "exp(dt_td * A[n * D + d])"),
    "B_by_channel": ("B[t * N + n] * x_td", "B[t * N + (d % N)] * x_td"),
    "beta_without_dt": ("B[t * N + n] * x_td * dt_td", "B[t * N + n] * x_td"),
    "readout_wrong_state": ("C[t * N + n] * h[n]", "C[t * N + n] * h[(n + 1) % N]"),
    "chunk_end_off_by_one": ("t < offsets[c + 1]; ++t", "t + 1 < offsets[c + 1]; ++t"),
    "ties_go_high": ("if (s > best)", "if (s >= best)"),
    "initial_state_ignored": ("h[n] = (h0 != NULL) ? h0[(c * D + d) * N + n] : 0.0;", "h[n] = 0.0;"),
    "first_key_skipped": ("for (int64_t i = 0; i < M; ++i) {", "for (int64_t i = 1; i < M; ++i) {"),
    "dot_drops_last_dim": ("for (int64_t k = 0; k < dim; ++k)", "for (int64_t k = 0; k + 1 < dim; ++k)"),
    "empty_index_scores_minus_inf": ("best_score[q] = (arg < 0) ? NAN : best;", "best_score[q] = best;"),
    # the K-dial trajectory: the final state of a chunk whose length is not a multiple of
    # the stride is not kept (fewer writes, never more)
    "trajectory_final_state_dropped": ("if (step % stride == 0 || t + 1 == offsets[c + 1])",
                                       "if (step % stride == 0)"),
    # the complex-A scan (Eq. 1's complex diagonal)
    "complex_conjugate_rotation": ("A_re[d * N + n] + I * A_im[d * N + n]",
                                   "A_re[d * N + n] - I * A_im[d * N + n]"),
    "complex_parts_swapped": ("A_re[d * N + n] + I * A_im[d * N + n]",
                              "A_im[d * N + n] + I * A_re[d * N + n]"),
    "complex_rotation_dropped": ("cexp(dt_td * a)", "exp(dt_td * creal(a))"),
    "complex_beta_imaginary": ("const double complex alpha = cexp(dt_td * a);\n"
                               "                    const double beta = B[t * N + n] * x_td * dt_td;",
                               "const double complex alpha = cexp(dt_td * a);\n"
                               "                    const double complex beta = I * B[t * N + n] * x_td * dt_td;"),
    "complex_readout_imaginary": ("C[t * N + n] * creal(h[n])", "C[t * N + n] * cimag(h[n])"),
}

PIN_TESTS = [
    lambda: pins.test_theorem1_precog_equals_in_context(37, 11),
    pins.test_proposition_outputs_depend_on_context_only_through_state,
    pins.test_constant_gates_geometric_series,
    pins.test_A_zero_is_cumulative_sum_exact,
    pins.test_dyadic_gates_hand_expanded,
    pins.test_readout_uses_updated_state,
    lambda: pins.test_unroll_closed_form_and_linearity(5),
    pins.test_channel_isolation_and_state_index,
    pins.test_chunk_boundaries_and_empty_chunks,
    pins.test_stability_bound,
    pins.test_retrieve_matches_numpy_argmax_first_occurrence,
    pins.test_retrieve_ties_nan_and_empty,
    pins.test_retrieve_planted_tiny_workload,
    lambda: pins.test_trajectory_is_prefix_rollouts(7),
    pins.test_complex_scan_real_special_case,
    pins.test_complex_scan_theorem1_and_geometric_series,
]


def _compile(src_text, out_dir, name):
    c_path = os.path.join(out_dir, f"{name}.c")
    so_path = os.path.join(out_dir, f"{name}.so")
    with open(c_path, "w") as f:
        f.write(src_text)
    subprocess.run(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-shared", "-fPIC",
                    c_path, "-o", so_path, "-lm"], check=True)
    return so_path


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(name, tmp_path, monkeypatch):
    src = open(SRC).read()
    old, new = MUTATIONS[name]
    assert old in src, f"mutation anchor for {name} not found in the oracle source"
    so_path = _compile(src.replace(old, new), str(tmp_path), name)
    real = oracle._load()
    mutant = ctypes.CDLL(so_path)
    for fn in ("oracle_scan", "oracle_retrieve", "oracle_scan_complex", "oracle_trajectory"):
        getattr(mutant, fn).restype = getattr(real, fn).restype
        getattr(mutant, fn).argtypes = getattr(real, fn).argtypes
    monkeypatch.setattr(oracle, "_lib", mutant)
    failures = 0
    for pin in PIN_TESTS:
        try:
            pin()
        except AssertionError:
            failures += 1
    assert failures > 0, f"no pin caught the planted mistake '{name}'"


# Mistakes planted in the numpy routines of the oracle (top-k, composition, SMC).
PY_SRC = os.path.join(os.path.dirname(oracle.__file__), "__init__.py")

PY_MUTATIONS = {
    "topk_ties_go_high": ("retrieve_topk", "        cand.sort()\n",
                          "        cand.sort(key=lambda c: (c[0], -c[1]))\n"),
    "topk_keeps_nan": ("retrieve_topk", "for i in range(M) if not np.isnan(S[q, i])]",
                       "for i in range(M)]"),
    "compose_temperature_inverted": ("compose", "z = s[valid] / temperature", "z = s[valid] * temperature"),
    "compose_unnormalised": ("compose", "w = e / e.sum()", "w = e"),
    "smc_route_ignores_J": ("smc_route", "retrieve(sub[m, : int(J[m])], emb[c:c + 1])",
                            "retrieve(sub[m], emb[c:c + 1])"),
    "smc_forgetting_slot_deposits": ("smc_consolidate", "        if slot < 0:\n            continue\n", ""),
    "compose_missing_entries_weighted": ("compose", "valid = ~np.isnan(s)", "valid = np.ones(s.shape, dtype=bool)"),
    "smc_ema_weights_swapped": ("smc_consolidate", "out[slot] = (1.0 - alpha) * out[slot] + alpha * h[c]",
                                "out[slot] = alpha * out[slot] + (1.0 - alpha) * h[c]"),
}

PY_PIN_TESTS = [
    pins.test_topk_matches_numpy_stable_argsort,
    pins.test_topk_nan_and_short_index,
    pins.test_compose_softmax_weights,
    pins.test_composition_commutes_with_the_scan,
    pins.test_smc_route_two_levels,
    pins.test_smc_consolidate_closed_form,
]


@pytest.mark.parametrize("name", sorted(PY_MUTATIONS))
def test_planted_python_mistake_is_caught(name, monkeypatch):
    import types
    func, old, new = PY_MUTATIONS[name]
    src = open(PY_SRC).read()
    assert old in src, f"mutation anchor for {name} not found in the oracle source"
    mutant = types.ModuleType("oracle_mutant")
    mutant.__file__ = PY_SRC
    exec(compile(src.replace(old, new), PY_SRC, "exec"), mutant.__dict__)
    mutant._lib = oracle._load()                     # the unmutated C library
    monkeypatch.setattr(oracle, func, getattr(mutant, func))
    failures = 0
    for pin in PY_PIN_TESTS:
        try:
            pin()
        except AssertionError:
            failures += 1
    assert failures > 0, f"no pin caught the planted mistake '{name}'"
