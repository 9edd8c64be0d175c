"""Planted mistakes in the oracle must fail at least one pin.

Each case copies the oracle's source, replaces one expression with a
plausible mistake (a dropped term, a swapped coefficient, a wrong sign or
index), loads the copy as a separate module and runs the named pins on it.
The mistake lives only in that in-memory copy, on the CPU.
"""
import importlib.util
import os
import sys

import pytest

import oracle_pins as P

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle", "dsm_oracle.py")

# (id, original text, planted mistake, pins expected to catch it)
MUTANTS = [
    ("global_beta_swapped", "u = T(f32(b1)) * m + c1 * delta\n    if sign_mode == 0:",
     "u = T(f32(b2)) * m + c1 * delta\n    if sign_mode == 0:",
     [P.pin_worked_example]),
    ("global_no_inv_gamma", "c1 = T((1.0 - f32(b1)) / f32(gamma))\n    c2 = T((1.0 - f32(b2)) / f32(gamma))\n    eg",
     "c1 = T((1.0 - f32(b1)))\n    c2 = T((1.0 - f32(b2)) / f32(gamma))\n    eg",
     [P.pin_worked_example]),
    ("global_mom_coeff", "    m_new = T(f32(b2)) * m + c2 * delta\n    return x_new, m_new, {\"delta\": delta, \"u\": u, \"sg\": sg,",
     "    m_new = T(f32(b2)) * m + c1 * delta\n    return x_new, m_new, {\"delta\": delta, \"u\": u, \"sg\": sg,",
     [P.pin_worked_example]),
    ("global_no_weight_decay", "x_new = x - eg * (sg + lam_e * x)", "x_new = x - eg * sg",
     [P.pin_worked_example]),
    ("global_diff_sign", "diffs = [x - X[i] for i in range(n)]", "diffs = [X[i] - x for i in range(n)]",
     [P.pin_worked_example]),
    ("global_mean_divisor", "return acc / dt.type(n), diffs", "return acc / dt.type(n + 1), diffs",
     [P.pin_worked_example]),
    ("global_eta_gamma", "eg = T(f32(eta) * f32(gamma))", "eg = T(f32(eta))",
     [P.pin_worked_example]),
    ("sign_at_zero", "return ((v > 0).astype(v.dtype) - (v < 0).astype(v.dtype))",
     "return ((v >= 0).astype(v.dtype) - (v < 0).astype(v.dtype))",
     [P.pin_worked_example]),
    ("adamw_bias_exponent", "bc1 = T(1.0 - beta_power(b1, j))", "bc1 = T(1.0 - beta_power(b1, j + 1))",
     [P.pin_adamw_constant_grad]),
    ("adamw_eps_inside_sqrt", "np.sqrt(vhat) + eps_", "np.sqrt(vhat + eps_)",
     [P.pin_adamw_vs_torch]),
    ("adamw_no_decay", "(mhat / (np.sqrt(vhat) + eps_) + wd_e * x)", "(mhat / (np.sqrt(vhat) + eps_))",
     [P.pin_adamw_vs_torch]),
    ("adamw_v_coeff", "v = b2_ * v + omb2 * (g * g)", "v = b2_ * v + omb1 * (g * g)",
     [P.pin_adamw_vs_torch]),
    ("adamw_v_bias", "vhat = v / bc2", "vhat = v / bc1",
     [P.pin_adamw_constant_grad]),
    ("sgdm_dampened", "buf = T(f32(mu)) * buf + g.astype(dt)",
     "buf = T(f32(mu)) * buf + T(1.0 - f32(mu)) * g.astype(dt)",
     [P.pin_sgdm_vs_torch]),
    ("rsign_pm_prob", "q = dt(0.5) + dt(0.5) * p", "q = p",
     [P.pin_lemma1]),
    ("rsign_zero_compare", "return np.where(r < p, s, dt(0.0)).astype(u.dtype)",
     "return np.where(r > p, s, dt(0.0)).astype(u.dtype)",
     [P.pin_lemma1]),
    ("philox_sbox", "c = [hi1 ^ c[1] ^ k0, lo1, hi0 ^ c[3] ^ k1, lo0]",
     "c = [hi0 ^ c[1] ^ k0, lo1, hi1 ^ c[3] ^ k1, lo0]",
     [P.pin_philox]),
    ("philox_word_index", "w = np.choose((e & U64(3)).astype(np.int64), words)",
     "w = np.choose(((e + U64(1)) & U64(3)).astype(np.int64), words)",
     [P.pin_philox_uniform_mapping]),
    ("splitmix_shift", "z = (z ^ (z >> U64(27))) * U64(_MIX_C2)", "z = (z ^ (z >> U64(28))) * U64(_MIX_C2)",
     [P.pin_splitmix64]),
    ("hash_fields_swapped", "shift = np.where((e & U64(1)) == 0, U64(40), U64(16))",
     "shift = np.where((e & U64(1)) == 0, U64(16), U64(40))",
     [P.pin_hash_fields]),
    ("bf16_round_half_up", "r = ((b + U64(0x7FFF) + kept_lsb) >> U64(16)) << U64(16)",
     "r = ((b + U64(0x8000)) >> U64(16)) << U64(16)",
     [P.pin_bf16]),
    ("grad_worker_scale", "s2 = (np.float32(0.1) * scale).astype(np.float32)",
     "s2 = (np.float32(0.3) * scale).astype(np.float32)",
     [P.pin_synthetic_grad]),
    ("stats_drift_uncentred", "drift_e += (dd - delta) ** 2", "drift_e += dd ** 2",
     [P.pin_stats]),
    ("stats_unanimous_any_worker",
     "    unanimous = np.ones(delta.shape, dtype=bool)\n    for dd_, dd in zip(inter[\"diffs\"], diffs):\n"
     "        unanimous &= sign(dd_) == sd",
     "    unanimous = np.zeros(delta.shape, dtype=bool)\n    for dd_, dd in zip(inter[\"diffs\"], diffs):\n"
     "        unanimous |= sign(dd_) == sd",
     [P.pin_stats_example]),
    ("stats_unanimous_skips_zero_differences", "        unanimous &= sign(dd_) == sd",
     "        unanimous &= (sign(dd_) == sd) | (dd_ == 0)",
     [P.pin_stats_example]),
    ("stats_flips_vs_applied_sign", "flip_e = sign(u) != sd", "flip_e = sg != sd",
     [P.pin_stats_example]),
    ("stats_flips_vs_worker_sign", "flip_e = sign(u) != sd", "flip_e = sign(u) != sign(inter[\"diffs\"][0])",
     [P.pin_worked_example, P.pin_stats_example]),
    ("stats_zero_of_unrandomized_sign", "zero_e = sg == 0", "zero_e = sign(u) == 0",
     [P.pin_stats_example]),
    ("stats_delta_sq_of_u", "sq = delta[sel] ** 2", "sq = u[sel].astype(np.float64) ** 2",
     [P.pin_worked_example]),
    ("stats_clamp_inclusive", "clamp_e = (np.abs(u) > np.asarray(f32(B), dtype=u.dtype))",
     "clamp_e = (np.abs(u) >= np.asarray(f32(B), dtype=u.dtype))",
     [P.pin_stats_example]),
    ("rsign_zero_inclusive", "return np.where(r < p, s, dt(0.0)).astype(u.dtype)",
     "return np.where(r <= p, s, dt(0.0)).astype(u.dtype)",
     [P.pin_stats_example]),
    ("stats_clamp_threshold", "clamp_e = (np.abs(u) > np.asarray(f32(B), dtype=u.dtype))",
     "clamp_e = (np.abs(u) > np.asarray(f32(B) / 2, dtype=u.dtype))",
     [P.pin_stats]),
    ("slowmo_no_inv_gamma", "u = T(f32(beta)) * m + inv_g * delta", "u = T(f32(beta)) * m + delta",
     [P.pin_slowmo_heavy_ball]),
    ("lookahead_signed", "    u = T(f32(b1)) * m + c1 * delta\n    x_new = x - T(f32(eta) * f32(gamma)) * u\n",
     "    u = T(f32(b1)) * m + c1 * delta\n    x_new = x - T(f32(eta) * f32(gamma)) * sign(u)\n",
     [P.pin_lookahead_slow_weights]),
    ("signed_slowmo_unsigned", "u = T(f32(b1)) * m + c1 * sd", "u = T(f32(b1)) * m + c1 * delta",
     [P.pin_signed_slowmo_signsgd]),
    ("global_adamw_bias", "mhat = m_new / T(1.0 - beta_power(b1, t + 1))", "mhat = m_new / T(1.0 - beta_power(b1, t + 2))",
     [P.pin_global_adamw_vs_torch]),
    ("global_adamw_no_inv_gamma", "g = T(1.0 / f32(gamma)) * delta", "g = delta",
     [P.pin_global_adamw_vs_torch]),
    ("reset_keeps_step_count", "j = self.k + 1 if self.reset_local else step + 1", "j = step + 1",
     [P.pin_local_state_across_rounds]),
    ("reset_keeps_moments", "            self.opt_m = [np.zeros_like(self.x) for _ in range(self.n)]\n",
     "            pass\n", [P.pin_local_state_across_rounds]),
    ("subset_tensor_lookup", "self.tensor_of = np.searchsorted(self.starts, self.elems, side=\"right\") - 1",
     "self.tensor_of = np.searchsorted(self.starts, self.elems, side=\"left\") - 1",
     [P.pin_subset_mode, P.pin_stats]),
]


def _mutant_module(name, old, new):
    with open(SRC) as f:
        src = f.read()
    assert src.count(old) == 1, f"mutation site not unique or missing: {old!r}"
    spec = importlib.util.spec_from_loader(f"_oracle_mutant_{name}", loader=None)
    mod = importlib.util.module_from_spec(spec)
    sys.modules[spec.name] = mod
    exec(compile(src.replace(old, new), f"<mutant {name}>", "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name,old,new,pins", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(name, old, new, pins):
    mod = _mutant_module(name, old, new)
    caught = []
    for pin in pins:
        try:
            with __import__("numpy").errstate(all="ignore"):
                pin(mod)
        except Exception as exc:  # AssertionError, or the mutant breaking outright
            caught.append((pin.__name__, type(exc).__name__))
    assert caught, f"mutant {name} passed every pin in {[p.__name__ for p in pins]}"
