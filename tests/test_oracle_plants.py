"""The oracle's pins catch plausible mistakes.

Each case copies oracle/pdb_oracle.c, plants one mistake in the copy (the
committed file is never touched), builds it here on the CPU, points the
oracle module at the planted build, and runs the pins that guard that
routine: at least one of them must fail.  The pins compare against
mathematics (fp64, exact sums, closed forms, brute force), so a mistake in
the oracle cannot hide behind a matching mistake in its check."""
import inspect
import subprocess
import textwrap
from collections import defaultdict

import pytest

import oracle
from oracle import history
from tests import test_history as th
from tests import test_oracle_numerics as num
from tests import test_oracle_schedule as sched
from tests import test_oracle_sgd as sgd

# name -> (text in pdb_oracle.c, planted text, pins that must catch it)
PLANTS = {
    "taylor-coefficient": (
        "p = fmaf(p, r, (float)(1.0 / 120.0));", "p = fmaf(p, r, (float)(1.0 / 121.0));",
        [num.test_expf_within_2ulp_dense_grid, num.test_expf_within_2ulp_random_and_small]),
    "cody-waite-tail-dropped": (
        "r = r - kf * ln2_lo;", "r = r;",
        [num.test_expf_within_2ulp_dense_grid, num.test_expf_within_2ulp_random_and_small]),
    "exp-argument-sign": (
        "return -y / (1.0f + orc_expf(y * m));", "return -y / (1.0f + orc_expf(-y * m));",
        [num.test_grad_logistic_closed_forms, num.test_grad_logistic_is_the_derivative_of_the_logistic_loss]),
    "logistic-numerator-sign": (
        "return -y / (1.0f + orc_expf(y * m));", "return y / (1.0f + orc_expf(y * m));",
        [num.test_grad_logistic_is_the_derivative_of_the_logistic_loss]),
    "butterfly-stage-missing": (
        "for (int off = 16; off >= 1; off >>= 1) {", "for (int off = 16; off >= 2; off >>= 1) {",
        [num.test_dot_exact_on_small_integers, num.test_dot_uses_32_partial_sums]),
    "sixteen-partial-sums": (
        "a[i % 32] = fmaf(w[col[i]], val ? val[i] : 1.0f, a[i % 32]);",
        "a[i % 16] = fmaf(w[col[i]], val ? val[i] : 1.0f, a[i % 16]);",
        [num.test_dot_uses_32_partial_sums, num.test_dot_error_bound_random]),
    "hinge-tie": (
        "return (y * m < 1.0f) ? -y : 0.0f;", "return (y * m <= 1.0f) ? -y : 0.0f;",
        [num.test_grad_squared_and_hinge]),
    "update-sign": (
        "w[col[b + i]] = w[col[b + i]] - c * x;", "w[col[b + i]] = w[col[b + i]] + c * x;",
        [sgd.test_one_logistic_step_from_zero, sgd.test_squared_loss_geometric_closed_form]),
    "chain-rank-off-by-one": (
        "rank[p] = (int32_t)cnt[j];", "rank[p] = (int32_t)cnt[j] + 1;",
        [lambda: sched.test_chains_brute_force(0), lambda: sched.test_chains_brute_force(1)]),
    "level-first-position-ignored": (
        "if (prev[p] >= 0 && level[row_of[prev[p]]] > lv)", "if (prev[p] > 0 && level[row_of[prev[p]]] > lv)",
        [sched.test_levels_single_predecessor_chain] +
        [lambda s=s: sched.test_levels_equal_brute_force(s) for s in range(16)]),
    "squared-loss-sign": (
        "if (loss == ORC_SQUARED) return m - y;", "if (loss == ORC_SQUARED) return y - m;",
        [num.test_grad_squared_and_hinge, sgd.test_squared_loss_geometric_closed_form]),
    "exp-scale-not-split": (
        "int h = k / 2;", "int h = k;",
        [num.test_expf_special_values, num.test_expf_subnormal_results_correctly_scaled,
         num.test_expf_within_2ulp_dense_grid]),
    "chain-next-not-linked": (
        "if (last[j] >= 0) next[last[j]] = (int32_t)p;", ";",
        [lambda: sched.test_chains_brute_force(0), lambda: sched.test_chains_brute_force(1)]),
    "level-order-reversed-in-level": (
        "for (int64_t t = 0; t < n_rows; ++t) order[fill[level[t]]++] = (int32_t)t;",
        "for (int64_t t = n_rows - 1; t >= 0; --t) order[fill[level[t]]++] = (int32_t)t;",
        [sched.test_level_order_is_stable_by_level_then_id]),
    "bsp-batch-not-snapshot": (
        "float m = orc_dot(w, col + b, val ? val + b : NULL, k);\n                c[t - b0] = eta * orc_grad(loss, m, y[t]);",
        "float m = orc_dot(w, col + b, val ? val + b : NULL, k);\n                c[t - b0] = eta * orc_grad(loss, m, y[t]);\n"
        "                for (int64_t p = b; p < b + k; ++p) w[col[p]] = w[col[p]] - c[t - b0] * (val ? val[p] : 1.0f);",
        [lambda: sgd.test_bsp_full_batch_is_gradient_descent(oracle.LOGISTIC),
         lambda: sgd.test_bsp_full_batch_is_gradient_descent(oracle.SQUARED)]),
    "bsp-sum-not-reset": (
        "delta[col[p]] = 0.0f;", ";",
        [lambda: sgd.test_bsp_batch_one_is_sequential(oracle.LOGISTIC), sgd.test_bsp_short_last_batch]),
}


@pytest.mark.parametrize("name", list(PLANTS))
def test_planted_mistake_fails_a_pin(name, tmp_path, monkeypatch):
    old, new, pins = PLANTS[name]
    src = open(oracle._SRC).read()
    assert src.count(old) == 1, "the planted text must name one place"
    planted = tmp_path / "pdb_oracle.c"
    planted.write_text(src.replace(old, new))
    lib = tmp_path / "liboracle.so"
    subprocess.run(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-ffp-contract=off", "-fno-fast-math",
                    "-o", str(lib), str(planted), "-lm"], check=True)
    monkeypatch.setattr(oracle, "build", lambda: str(lib))
    monkeypatch.setattr(oracle, "_lib", None)
    caught = 0
    for pin in pins:
        try:
            pin()
        except AssertionError:
            caught += 1
    assert caught > 0, f"no pin caught the planted mistake {name!r}"


# ------------------------------------------------------------------ history
# The checker of execution histories and traces (oracle/history.py) is
# pinned the same way: a copy of one predicate with a mistake replaces it.


def _rc_only(ops):
    """The Read Constraint alone (a checker that forgot the Write Constraint)."""
    pos_w = {}
    for q, (kind, _, chunk, it) in enumerate(ops):
        if kind == "w":
            pos_w[(chunk, it)] = q
    for q, (kind, _, chunk, it) in enumerate(ops):
        if kind == "r" and it > 1:
            wq = pos_w.get((chunk, it - 1))
            if wq is None or wq > q:
                return False
    return True


def _wc_only(ops):
    """The Write Constraint alone (a checker that forgot the Read Constraint)."""
    reads = defaultdict(list)
    for q, (kind, _, chunk, it) in enumerate(ops):
        if kind == "r":
            reads[(chunk, it)].append(q)
    for q, (kind, _, chunk, it) in enumerate(ops):
        if kind == "w" and any(rq > q for rq in reads[(chunk, it)]):
            return False
    return True


def _no_pair_breaks(row_ptr, col, n_epochs, trace):
    v = _order_violations(row_ptr, col, n_epochs, trace)
    v["rc"] = 0
    return v


_order_violations = history.trace_order_violations

PY_PLANTS = {
    "write-constraint-ignored": ("satisfies_rc_wc", _rc_only,
                                 [lambda r=r: th.test_paper_histories(*r) for r in th._golden()]),
    "read-constraint-ignored": ("satisfies_rc_wc", _wc_only,
                                [th.test_theorem2_random_executions, th.test_trace_batch_with_conflicts_is_rejected]),
    "trace-pairs-ignored": ("trace_order_violations", _no_pair_breaks,
                            [th.test_trace_batch_with_conflicts_is_rejected] +
                            [lambda s=s: th.test_trace_checkers_match_brute_force(s) for s in range(6)]),
}


@pytest.mark.parametrize("name", list(PY_PLANTS))
def test_planted_checker_mistake_fails_a_pin(name, monkeypatch):
    attr, fn, pins = PY_PLANTS[name]
    monkeypatch.setattr(history, attr, fn)
    caught = 0
    for pin in pins:
        try:
            pin()
        except AssertionError:
            caught += 1
    assert caught > 0, f"no pin caught the planted mistake {name!r}"


# Mistakes planted by editing one line of a copy of a checker's source.
PY_TEXT_PLANTS = {
    "delay-need-off-by-one": (
        "trace_delay_violations", "need = rank[(o[rd] - u.size)] - delay",
        "need = rank[(o[rd] - u.size)] - delay - 1"),
    "delay-group-first-write-dropped": (
        "trace_delay_violations", "done = cw - (cw[base] - is_w[base])", "done = cw - cw[base]"),
    "delay-ties-read-first": (
        "trace_delay_violations", "o = np.lexsort((kind, times, keys))", "o = np.lexsort((-kind, times, keys))"),
}
_DELAY_PINS = ([lambda s=s: th.test_trace_checkers_match_brute_force(s) for s in range(6)] +
               [th.test_trace_delay_fully_parallel_epoch, th.test_trace_sequential_and_level_traces_pass])


@pytest.mark.parametrize("name", list(PY_TEXT_PLANTS))
def test_planted_checker_line_fails_a_pin(name, monkeypatch):
    attr, old, new = PY_TEXT_PLANTS[name]
    src = textwrap.dedent(inspect.getsource(getattr(history, attr)))
    assert src.count(old) == 1, "the planted text must name one place"
    ns = dict(vars(history))
    exec(compile(src.replace(old, new), f"<planted {name}>", "exec"), ns)
    monkeypatch.setattr(history, attr, ns[attr])
    caught = 0
    for pin in _DELAY_PINS:
        try:
            pin()
        except AssertionError:
            caught += 1
    assert caught > 0, f"no pin caught the planted mistake {name!r}"
