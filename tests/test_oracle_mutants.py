"""Sensitivity of the oracle's pins. Each case plants one plausible mistake in
a copy of the C oracle (a wrong sign, a dropped term, a wrong index or
denominator, a transposed operand, a broken tie rule, a lost stability, an
off-by-one in the selection), builds it with the oracle's own flags, and runs
the pins of test_oracle.py against it (all but the 11-second exhaustive sweep
of the exponential): at least one pin must fail. A control build of the
unmodified source must pass them, so that a failure is the planted mistake's
and not the harness's. The mistakes are planted on the CPU only."""
import os
import subprocess
import sys

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
SRC = os.path.join(ROOT, "oracle", "elbow_oracle.c")

# (name, the oracle's line, the planted mistake)
MUTANTS = [
    ("deviation_sign_as_printed",  # Alg. 1 as printed: D = p' - x' (always k = 1)
     "float D = (1.0f - pn) - xn;", "float D = pn - xn;"),
    ("normalisation_drops_p_min",
     "float pn = (p[idx[i]] - p_min) / den;", "float pn = p[idx[i]] / den;"),
    ("normalisation_reciprocal_multiply",  # two roundings instead of Alg. 1's one quotient
     "float pn = (p[idx[i]] - p_min) / den;", "float pn = (p[idx[i]] - p_min) * (1.0f / den);"),
    ("softmax_reciprocal_multiply",
     "for (int j = 0; j < N; ++j) p[j] = e[j] / s;",
     "for (int j = 0; j < N; ++j) p[j] = e[j] * (1.0f / s);"),
    ("x_over_n_not_n_minus_1",
     "float xn = (float)i / (float)(N - 1);", "float xn = (float)i / (float)N;"),
    ("argmax_takes_last_tie",
     "if (i == 0 || D > d_best) {", "if (i == 0 || D >= d_best) {"),
    ("k_is_e_not_e_plus_1",
     "int k = (mode == 1) ? K : (e_arg + 1 < K ? e_arg + 1 : K);",
     "int k = (mode == 1) ? K : (e_arg < K ? e_arg : K);"),
    ("sort_ties_higher_id_first",
     "while (j >= 0 && p[idx[j]] < p[key]) {", "while (j >= 0 && p[idx[j]] <= p[key]) {"),
    ("softmax_sum_drops_last_level",
     "for (int h = N / 2; h >= 1; h /= 2)", "for (int h = N / 2; h >= 2; h /= 2)"),
    ("softmax_without_max_shift",
     "for (int j = 0; j < N; ++j) e[j] = oracle_exp(l[j] - m);",
     "for (int j = 0; j < N; ++j) e[j] = oracle_exp(l[j]);"),
    ("exp_wrong_second_coefficient",
     "(float)(1.0 / 1.0),   (float)(1.0 / 2.0),", "(float)(1.0 / 1.0),   (float)(1.0 / 3.0),"),
    ("gate_kept_at_slot_k",
     "gates[s] = (s < k) ? g : 0.0f;", "gates[s] = (s <= k) ? g : 0.0f;"),
    ("renorm_over_all_k_slots",
     "for (int s = 0; s < k; ++s) S = S + p[idx[s]];",
     "for (int s = 0; s < K; ++s) S = S + p[idx[s]];"),
    ("dispatch_not_stable",
     "  for (int64_t t = 0; t < T; ++t) {\n    for (int s = 0; s < K; ++s) {",
     "  for (int64_t t = T - 1; t >= 0; --t) {\n    for (int s = 0; s < K; ++s) {"),
    ("unselected_pair_pos_zero",
     "        pair_pos[t * K + s] = -1;", "        pair_pos[t * K + s] = 0;"),
    ("offsets_off_by_one",
     "for (int e = 0; e < N; ++e) offsets[e + 1] = offsets[e] + (int32_t)cnt[e];",
     "for (int e = 0; e < N; ++e) offsets[e + 1] = offsets[e] + (int32_t)cnt[e] + (e == 0);"),
    ("residual_dropped",
     "for (int c = 0; c < d; ++c) yr[c] += bf16_to_double(residual[t * d + c]);",
     "for (int c = 0; c < d; ++c) yr[c] += 0.0 * bf16_to_double(residual[t * d + c]);"),
    ("router_weight_transposed",
     "acc += bf16_to_double(xr[c]) * bf16_to_double(w_router[(int64_t)j * d + c]);",
     "acc += bf16_to_double(xr[c]) * bf16_to_double(w_router[(int64_t)c * N + j]);"),
    ("swiglu_gate_and_up_swapped",
     "double hv = g / (1.0 + exp(-g)) * u;", "double hv = u / (1.0 + exp(-u)) * g;"),
    ("down_weight_transposed",
     "o += bf16_to_double(wdn[(int64_t)c * I + i]) * h[i];",
     "o += bf16_to_double(wdn[(int64_t)i * d + c]) * h[i];"),
    ("combine_uses_first_gate",
     "yr[c] += (double)gates[s] * o;", "yr[c] += (double)gates[0] * o;"),
    ("elbow_angle_sign",
     "double ax = -x, ay = -y, bx = 1.0 - x, by = 1.0 - y;",
     "double ax = -x, ay = y, bx = 1.0 - x, by = 1.0 - y;"),
    ("randomised_tail_may_redraw_rank_k_minus_1",
     "int excl = (mode == 2) ? k : K;", "int excl = (mode == 2) ? (k > 1 ? k - 1 : k) : K;"),
]


def _build(tmp, name, old, new):
    with open(SRC) as f:
        src = f.read()
    if old is not None:
        assert src.count(old) == 1, f"{name}: the line to plant the mistake in is not unique"
        src = src.replace(old, new)
    path = os.path.join(tmp, name + ".c")
    with open(path, "w") as f:
        f.write(src)
    so = os.path.join(tmp, "lib" + name + ".so")
    subprocess.run(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
                    "-fPIC", "-shared", path, "-o", so, "-lm"], check=True)
    return so


def _run_pins(so):
    env = dict(os.environ, ORACLE_LIBRARY=so, OMP_NUM_THREADS="4")
    r = subprocess.run([sys.executable, "-m", "pytest", os.path.join(HERE, "test_oracle.py"), "-q",
                        "-x", "-p", "no:cacheprovider", "-k", "not exhaustive"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    return r.returncode, (r.stdout + r.stderr)[-3000:]


def test_control_build_passes_the_pins(tmp_path):
    rc, out = _run_pins(_build(str(tmp_path), "control", None, None))
    assert rc == 0, out


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_reject_planted_mistake(tmp_path, name, old, new):
    rc, out = _run_pins(_build(str(tmp_path), name, old, new))
    assert rc == 1, f"no pin failed on {name}:\n{out}"


# Mistakes planted in the oracle's Python part (the load metrics of App. A.3):
# the function is rebuilt from its source with one change and swapped in for
# the pins of test_oracle.py that exercise it.
LOAD_MUTANTS = [
    ("delta_sign", "delta = 1.0 - k_elb.mean() / K", "delta = k_elb.mean() / K"),
    ("elbow_load_counts_slot_k", "if s < k_elb[t]:", "if s <= k_elb[t]:"),
    ("l1_bound_missing_factor_2", "l1_bound=2 * delta / (1 - delta),",
     "l1_bound=delta / (1 - delta),"),
    ("cv2_bound_square_dropped", "cv2_bound=2 * N * delta / (1 - delta) ** 2,",
     "cv2_bound=2 * N * delta / (1 - delta),"),
    ("max_change_of_minima", "max_change=abs(q_elb.max() - q_top.max()),",
     "max_change=abs(q_elb.min() - q_top.min()),"),
    ("q_not_normalised", "q_elb = L_elb / L_elb.sum()", "q_elb = L_elb"),
]


@pytest.mark.parametrize("name,old,new", LOAD_MUTANTS, ids=[m[0] for m in LOAD_MUTANTS])
def test_load_pins_reject_planted_mistake(monkeypatch, name, old, new):
    import inspect

    import oracle
    import test_oracle as pins

    src = inspect.getsource(oracle.load_balance)
    assert src.count(old) == 1, f"{name}: the line to plant the mistake in is not unique"
    ns = dict(vars(oracle))
    exec(compile(src.replace(old, new), "<mutant>", "exec"), ns)
    monkeypatch.setattr(oracle, "load_balance", ns["load_balance"])
    failed = 0
    for pin in (pins.test_theorem1_and_corollaries, pins.test_load_balance_hand_example):
        try:
            pin()
        except AssertionError:
            failed += 1
    assert failed >= 1, f"no pin failed on {name}"
