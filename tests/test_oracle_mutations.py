"""Plant plausible mistakes in a temporary copy of the oracle and check that the pins fail.

Each mutation is applied to a copy of ``oracle/`` in a temporary directory;
the real oracle is never modified.  The pins in ``test_oracle_pins.py`` are
run against the mutated copy in a subprocess and must fail.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTATIONS = {
    "rope_sign": ("a * c - b * s, b * c + a * s", "a * c + b * s, b * c - a * s"),
    "rope_inverse_frequency": ("theta ** (-2.0 * i / head_dim)", "theta ** (-1.0 * i / head_dim)"),
    "dropped_attention_residual": ('x = x + o @ Lw["wo"].T', 'x = o @ Lw["wo"].T'),
    "transposed_wo": ('x = x + o @ Lw["wo"].T', 'x = x + o @ Lw["wo"]'),
    "gqa_head_index": ("g = h // group", "g = h % n_kv"),
    "eps_outside_sqrt": ("x / np.sqrt(ms + eps) * g", "x / (np.sqrt(ms) + eps) * g"),
    "dropped_q_norm": ('q = rms_norm(q, Lw["q_norm"], eps)', "q = q"),
    "attention_scale": ("/ np.sqrt(d)", "/ d"),
    "causal_mask_off_by_one": ("k_pos[None, :] <= q_pos[:, None]", "k_pos[None, :] < q_pos[:, None] + 2"),
    "gate_up_swapped": ('silu(u @ Lw["wg"].T) * (u @ Lw["wu"].T)', 'silu(u @ Lw["wu"].T) * (u @ Lw["wg"].T)'),
    "dropped_final_norm": ('return rms_norm(x, widen(W["final_norm"]), cfg.rms_eps)', "return x"),
    "log_softmax_sign": ("z - (m + np.log", "z + (m + np.log"),
    "layer_step_drops_new_key": ("V = np.concatenate([widen(v_cache[b, :, :p, :]).transpose(1, 0, 2), v[b:b + 1]])",
                                 "V = np.concatenate([widen(v_cache[b, :, :p, :]).transpose(1, 0, 2), v[b:b + 1] * 0])"),
}


# Mistakes in the GRPO token-loss oracle, caught by test_oracle_grpo.py.
GRPO_MUTATIONS = {
    "advantage_variance_normalised": ("return (g - g.mean(axis=1, keepdims=True)).reshape(-1)",
                                      "return ((g - g.mean(axis=1, keepdims=True)) / (g.std(axis=1, keepdims=True) + 1e-6)).reshape(-1)"),
    "clip_bounds_swapped": ("np.clip(rho, 1.0 - eps_low, 1.0 + eps_high)", "np.clip(rho, 1.0 - eps_high, 1.0 + eps_low)"),
    "max_instead_of_min": ("surrogate = np.minimum(", "surrogate = np.maximum("),
    "ratio_inverted": ("rho = np.exp(lp - np.asarray(lp_old, dtype=np.float64))",
                       "rho = np.exp(np.asarray(lp_old, dtype=np.float64) - lp)"),
    "kl_sign": ("loss = loss + beta * kl_k3(lp, lp_ref)", "loss = loss - beta * kl_k3(lp, lp_ref)"),
    "kl_k1_estimator": ("return np.exp(x) - x - 1.0", "return -x"),
}


# Mistakes in the sampling oracle, caught by test_oracle_sampling.py.
SAMPLING_MUTATIONS = {
    "gumbel_sign": ("return -np.log(-np.log(u))", "return np.log(-np.log(u))"),
    "temperature_multiplies": ("y = z / tau + gumbel(", "y = z * tau + gumbel("),
    "mix_constant": ("_M1 = np.uint64(0xBF58476D1CE4E5B9)", "_M1 = np.uint64(0xBF58476D1CE4E5B8)"),
    "counter_offset": ("(i + np.uint64(1)) * GAMMA", "i * GAMMA"),
    "uniform_grid": ("+ 0.5) * 2.0 ** -24", "+ 0.0) * 2.0 ** -24"),
}


# Mistakes in the backward oracle and the GRPO derivative, caught by test_oracle_backward.py.
BACKWARD_MUTATIONS = {
    "rms_dx_dropped_projection": ("dx = r * a - (r ** 3 / n) * x * np.sum(a * x, axis=-1, keepdims=True)",
                                  "dx = r * a"),
    "rms_gain_grad_unscaled": ("dg = np.sum((dy * x * r).reshape(-1, n), axis=0)",
                               "dg = np.sum((dy * x).reshape(-1, n), axis=0)"),
    "rope_backward_forward_rotation": ("d1 * c + d2 * s, -d1 * s + d2 * c", "d1 * c - d2 * s, d1 * s + d2 * c"),
    "softmax_backward_no_rowsum": ("dS = P * (dP - np.sum(dP * P, axis=-1, keepdims=True))", "dS = P * dP"),
    "gqa_dv_overwritten": ("dv[:, g] += P.T @ do[:, h]", "dv[:, g] = P.T @ do[:, h]"),
    "dk_missing_scale": ("dkr[:, g] += dS.T @ c[\"qr\"][:, h] / np.sqrt(d)", "dkr[:, g] += dS.T @ c[\"qr\"][:, h]"),
    "silu_derivative": ("sg * (1.0 + c[\"g\"] * (1.0 - sg))", "sg"),
    "mlp_residual_gradient_dropped": ("dx = dx + dxm", "dx = dxm"),
    "embedding_duplicates_lost": ("np.add.at(grads[\"embed\"], np.asarray(tok), dx)",
                                  "grads[\"embed\"][np.asarray(tok)] += dx"),
    "onehot_sign": ("dz[np.arange(T), tgt] -= 1.0", "dz[np.arange(T), tgt] += 1.0"),
    "target_not_shifted": ("tgt[:T - 1] = np.asarray(tok)[1:]", "tgt[:T - 1] = np.asarray(tok)[:-1]"),
    "du1_missing_value_path": ("du1 = dq @ Lw[\"wq\"] + dk @ Lw[\"wk\"] + dv @ Lw[\"wv\"]",
                               "du1 = dq @ Lw[\"wq\"] + dk @ Lw[\"wk\"]"),
}

GRPO_GRAD_MUTATIONS = {
    "clipped_branch_passes_gradient": ("g = -np.where(unclipped, rho * a, 0.0)", "g = -rho * a"),
    "kl_grad_sign": ("g = g + beta * (1.0 - np.exp(", "g = g - beta * (1.0 - np.exp("),
    "coef_not_normalised": ("return -m * g / n if n > 0 else np.zeros_like(g)", "return -m * g"),
}


def _run_mutated(tmp_path, module, before, after, name, pins):
    shutil.copytree(os.path.join(ROOT, "oracle"), tmp_path / "oracle",
                    ignore=shutil.ignore_patterns("__pycache__"))
    p = tmp_path / "oracle" / module
    src = p.read_text()
    assert src.count(before) >= 1, f"mutation anchor for {name} not found"
    p.write_text(src.replace(before, after))
    env = dict(os.environ, PYTHONPATH=os.pathsep.join([str(tmp_path), ROOT]))
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", pins)],
                       cwd=str(tmp_path), env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"pins did not catch {name}:\n{r.stdout[-2000:]}"


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_planted_mistake(name, tmp_path):
    before, after = MUTATIONS[name]
    _run_mutated(tmp_path, "qwen3.py", before, after, name, "test_oracle_pins.py")


@pytest.mark.parametrize("name", sorted(GRPO_MUTATIONS))
def test_grpo_pins_catch_planted_mistake(name, tmp_path):
    before, after = GRPO_MUTATIONS[name]
    _run_mutated(tmp_path, "grpo.py", before, after, name, "test_oracle_grpo.py")


@pytest.mark.parametrize("name", sorted(SAMPLING_MUTATIONS))
def test_sampling_pins_catch_planted_mistake(name, tmp_path):
    before, after = SAMPLING_MUTATIONS[name]
    _run_mutated(tmp_path, "sampling.py", before, after, name, "test_oracle_sampling.py")


@pytest.mark.parametrize("name", sorted(BACKWARD_MUTATIONS))
def test_backward_pins_catch_planted_mistake(name, tmp_path):
    before, after = BACKWARD_MUTATIONS[name]
    _run_mutated(tmp_path, "backward.py", before, after, name, "test_oracle_backward.py")


@pytest.mark.parametrize("name", sorted(GRPO_GRAD_MUTATIONS))
def test_grpo_grad_pins_catch_planted_mistake(name, tmp_path):
    before, after = GRPO_GRAD_MUTATIONS[name]
    _run_mutated(tmp_path, "grpo.py", before, after, name, "test_oracle_backward.py")
