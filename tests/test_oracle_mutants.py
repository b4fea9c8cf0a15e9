"""Plant plausible mistakes in copies of the oracle and check that the pins catch
every one of them.

Each mutant is the oracle's C source with one exact textual edit (a dropped
term, a flipped sign, a wrong operand, an off-by-one in the schedule), compiled
to a temporary library. The pins of tests/oracle_pins.py must reject each.
"""
import pytest

import oracle
from oracle_pins import failing_pins

MUTANTS = {
    "weight_decay_sign": ("double d = grad[j] + wd * theta[j];",
                          "double d = grad[j] - wd * theta[j];"),
    "momentum_operands_swapped": ("buf[j] = mu * buf[j] + d;",
                                  "buf[j] = mu * d + buf[j];"),
    "update_ignores_momentum": ("theta[j] = theta[j] - lr * buf[j];",
                                "theta[j] = theta[j] - lr * d;"),
    "grad_sum_not_mean": ("gbar[j] = s / (double)W;", "gbar[j] = s;", 1),
    "sync_step_uses_own_grad": ("sgd_momentum_update(N, lr, mu, wd, gbar,",
                                "sgd_momentum_update(N, lr, mu, wd, g + (int64_t)i * N,", 1),
    "param_mean_wrong_divisor": ("theta_avg[j] = s / (double)W;",
                                 "theta_avg[j] = s / (double)(W + 1);", 1),
    "localsgd_mean_wrong_divisor": ("theta_avg[j] = s / (double)W;",
                                    "theta_avg[j] = s / (double)(W + 1);", 2),
    "slowmo_drops_velocity": ("v[j] = beta * v[j] + delta;", "v[j] = delta;", 1),
    "slowmo_wrong_base": ("theta_new[j] = theta_ref[j] + alpha * v[j];",
                          "theta_new[j] = theta_avg[j] + alpha * v[j];", 1),
    "adamw_slowmo_wrong_base": ("theta_new[j] = theta_ref[j] + alpha * v[j];",
                                "theta_new[j] = theta_avg[j] + alpha * v[j];", 2),
    "delta_sign": ("double delta = theta_avg[j] - theta_ref[j];",
                   "double delta = theta_ref[j] - theta_avg[j];", 1),
    "adamw_delta_sign": ("double delta = theta_avg[j] - theta_ref[j];",
                         "double delta = theta_ref[j] - theta_avg[j];", 2),
    "no_epoch_end_sync": ("if (t == T) return 1;", "if (t == T) return 0;"),
    "schedule_off_by_one": ("if (t % K == 0) return 1;", "if (t % K == 1) return 1;"),
    "no_broadcast": ("for (int64_t j = 0; j < N; ++j) theta[(int64_t)i * N + j] = theta_new[j];",
                     "for (int64_t j = 0; j < 0; ++j) theta[(int64_t)i * N + j] = theta_new[j];", 1),
    "adamw_no_broadcast": ("for (int64_t j = 0; j < N; ++j) theta[(int64_t)i * N + j] = theta_new[j];",
                           "for (int64_t j = 0; j < 0; ++j) theta[(int64_t)i * N + j] = theta_new[j];", 2),
    "anchor_not_updated": ("for (int64_t j = 0; j < N; ++j) theta_ref[j] = theta_new[j];",
                           "for (int64_t j = 0; j < N; ++j) theta_ref[j] = theta_avg[j];", 1),
    "adamw_anchor_not_updated": ("for (int64_t j = 0; j < N; ++j) theta_ref[j] = theta_new[j];",
                                 "for (int64_t j = 0; j < N; ++j) theta_ref[j] = theta_avg[j];", 2),
    "momentum_init_nonzero": ("buf[(int64_t)i * N + j] = 0.0;",
                              "buf[(int64_t)i * N + j] = theta0[j];"),
    "velocity_init_nonzero": ("v[j] = 0.0;", "v[j] = theta0[j];"),
    "warmup_lr_off_by_one": ("return base_lr * (double)(s + 1) / (double)warmup_steps;",
                             "return base_lr * (double)(s) / (double)warmup_steps;"),
    "cosine_full_period": ("(1.0 + cos(3.14159265358979323846 * p))",
                           "(1.0 + cos(2.0 * 3.14159265358979323846 * p))"),
    "cosine_linear_instead": ("(1.0 + cos(3.14159265358979323846 * p))", "(2.0 - 2.0 * p)"),
    "warmup_epochs_ignored": ("if (epoch < warmup_epochs) return 1;", "if (epoch < 0) return 1;"),
    "localsgd_no_average": ("for (int64_t j = 0; j < N; ++j) theta[(int64_t)i * N + j] = theta_avg[j];",
                            "for (int64_t j = 0; j < 0; ++j) theta[(int64_t)i * N + j] = theta_avg[j];", 1),
    "localsgd_shared_gradient": ("/* each worker's local update with its own gradient */\n    for (int i = 0; i < W; ++i) {\n"
                                 "        sgd_momentum_update(N, lr, mu, wd, g + (int64_t)i * N,",
                                 "/* each worker's local update with its own gradient */\n    for (int i = 0; i < W; ++i) {\n"
                                 "        sgd_momentum_update(N, lr, mu, wd, g,"),
    "ddp_sum_not_mean": ("gbar[j] = s / (double)W;", "gbar[j] = s;", 2),
    "ddp_own_gradient": ("sgd_momentum_update(N, lr, mu, wd, gbar,",
                         "sgd_momentum_update(N, lr, mu, wd, g + (int64_t)i * N,", 2),
    "adamw_bias_correction_swapped": ("double bc2 = 1.0 - pow(beta2, (double)step);",
                                      "double bc2 = 1.0 - pow(beta1, (double)step);"),
    "adamw_no_sqrt": ("lr * m_hat / (sqrt(s_hat) + eps);", "lr * m_hat / (s_hat + eps);"),
    "adamw_first_moment_undamped": ("m[j] = beta1 * m[j] + (1.0 - beta1) * grad[j];",
                                    "m[j] = beta1 * m[j] + grad[j];"),
    "adamw_coupled_decay": ("theta[j] = theta[j] - lr * wd * theta[j];", "theta[j] = theta[j] - wd * theta[j];"),
    "adamw_sync_own_gradient": ("adamw_update(N, lr, beta1, beta2, eps, wd, step, gbar,",
                                "adamw_update(N, lr, beta1, beta2, eps, wd, step, g + (int64_t)i * N,", 1),
    "adamw_slowmo_drops_velocity": ("v[j] = beta * v[j] + delta;", "v[j] = delta;", 2),
    "adamw_ddp_own_gradient": ("adamw_update(N, lr, beta1, beta2, eps, wd, step, gbar,",
                               "adamw_update(N, lr, beta1, beta2, eps, wd, step, g + (int64_t)i * N,", 2),
    "state_average_sum_not_mean": ("mean[j] = acc / (double)W;", "mean[j] = acc;"),
    "state_average_row0_only": ("for (int64_t j = 0; j < N; ++j) state[(int64_t)i * N + j] = mean[j];",
                                "for (int64_t j = 0; j < N; ++j) state[j] = mean[j];"),
    "adamw_localsgd_no_average": ("for (int64_t j = 0; j < N; ++j) theta[(int64_t)i * N + j] = theta_avg[j];",
                                  "for (int64_t j = 0; j < 0; ++j) theta[(int64_t)i * N + j] = theta_avg[j];", 2),
}


def mutate(src: str, old: str, new: str, nth: int | None) -> str:
    """Replace the anchor `old` (which must occur exactly once, or, when `nth` is
    given, the nth of its occurrences in source order)."""
    if nth is None:
        assert src.count(old) == 1, "mutation anchor must occur exactly once"
        return src.replace(old, new)
    starts, pos = [], src.find(old)
    while pos >= 0:
        starts.append(pos)
        pos = src.find(old, pos + 1)
    assert len(starts) >= nth, "mutation anchor occurs fewer times than requested"
    at = starts[nth - 1]
    return src[:at] + new + src[at + len(old):]


@pytest.mark.parametrize("name", list(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    old, new, *nth = MUTANTS[name]
    src = oracle.SOURCE.read_text()
    mutant_src = tmp_path / "mutant.c"
    mutant_src.write_text(mutate(src, old, new, nth[0] if nth else None))
    lib_path = oracle.build_oracle(mutant_src, tmp_path / f"libmutant_{name}.so", force=True)
    failed = failing_pins(oracle.OracleLib(lib_path))
    assert failed, f"mutant {name} passed every pin"
