"""The pins must catch plausible mistakes in the oracle.

Each case plants one mistake in a copy of the oracle (a flipped sign, a
dropped term, a transposed operand, an off-by-one rank, a missing factor)
and runs the pin suite against the copy: it must fail.  The copy lives in a
temporary directory; nothing here touches the CUDA path."""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTATIONS = {
    # OBS compensation of Eq. (gptq_update): its sign, its columns shifted by one
    "compensation_sign": ("native.outer_sub(W[rows, j + 1:], e[rows] / d, Hinv[j, j + 1:])",
                          "native.outer_sub(W[rows, j + 1:], -e[rows] / d, Hinv[j, j + 1:])"),
    "compensation_shift": ("native.outer_sub(W[rows, j + 1:], e[rows] / d, Hinv[j, j + 1:])",
                           "native.outer_sub(W[rows, j + 1:], e[rows] / d, np.roll(Hinv[j, j + 1:], 1))"),
    # the Schur-complement downdate dropped
    "no_downdate": ("native.outer_sub(Hinv[j + 1:, j + 1:], Hinv[j + 1:, j], Hinv[j, j + 1:], d)",
                    "native.outer_sub(Hinv[j + 1:, j + 1:], 0.0 * Hinv[j + 1:, j], Hinv[j, j + 1:], d)"),
    # the residual of the quantizer halved
    "residual": ("e = W[:, j] - dq ", "e = W[:, j] - 0.5 * dq "),
    # the cross-moment term transposed
    "dbar_transposed": ("P = P + W0 @ np.asarray(Dbar, dtype=np.float64)",
                        "P = P + W0 @ np.asarray(Dbar, dtype=np.float64).T"),
    # the 1/2 of the surrogate
    "surrogate_half": ("return 0.5 * acc / T", "return acc / T"),
    # Adam's second bias correction
    "adam_bias": ("vhat = v / (1.0 - self.beta2 ** self.t)", "vhat = v"),
    # the damping 1.5 times too large
    "damping_mean": ("lam = damp_frac * float(np.mean(np.diag(Hd)))",
                     "lam = damp_frac * float(np.mean(np.diag(Hd))) * 1.5"),
    # the sliding-window weight off by one block
    "alpha_index": ("return 1.0 - (b_global - 1) / (B_total - 1)", "return 1.0 - b_global / (B_total - 1)"),
    # the output clipping: rank off by one, the factor inverted, a missing
    # factor in the gradient
    "clip_factor": ("kappa[over] = (q[:, None] / np.where(over, a, 1.0))[over]",
                    "kappa[over] = (np.where(over, a, 1.0) / q[:, None])[over]"),
    "clip_gradient": ("return (kappa * Z).T @ Xh / float(Xh.shape[0])", "return Z.T @ Xh / float(Xh.shape[0])"),
    # the mini-batch moment not normalised by its own token count
    "minibatch_norm": ("Hstep = np.asarray(Hk, dtype=np.float64) / float(Tk)",
                       "Hstep = np.asarray(Hk, dtype=np.float64) / float(T)"),
    # the nearest-rank percentile of both clipping steps off by one, or
    # taken from the single-precision value of pct
    "percentile_rank": ("return min(max(r - 1, 0), count - 1)", "return min(max(r, 0), count - 1)"),
    "percentile_single": ("r = math.ceil(Fraction(repr(float(pct))) * count)",
                          "r = math.ceil(Fraction(float(np.float32(pct))) * count)"),
    # the tie following of another run's rounding: taken off the ties too
    "follow_off_ties": ("take = (margin < tau) & (other != mine)", "take = (other != mine)"),
    # the weighted Hessian without the weights
    "weighted_hessian": ("H[g] += (c * sc[:, g:g + 1]).T @ c", "H[g] += c.T @ c"),
    # the activation grid without its clipping ratio
    "act_clip": ("xmax = (np.float32(a_clip) * np.abs(x).max(axis=1)).astype(np.float32)",
                 "xmax = (np.abs(x).max(axis=1)).astype(np.float32)"),
}


# the decoder block of the exact sliding window (oracle/block.py)
BLOCK_MUTATIONS = {
    "silu_derivative": ("gzg = gm * zu * (sg * (1.0 + zg * (1.0 - sg)))", "gzg = gm * zu * sg"),
    "softmax_backward": ("gsc = p * (gp - np.sum(gp * p, axis=-1, keepdims=True)) / np.sqrt(dh)",
                         "gsc = p * gp / np.sqrt(dh)"),
    "rope_transpose": ("return np.concatenate([g1 * c + g2 * s, -g1 * s + g2 * c], axis=-1)",
                       "return np.concatenate([g1 * c - g2 * s, g1 * s + g2 * c], axis=-1)"),
    "rms_backward": ("return gxr * r - x * (r ** 3) * np.sum(gxr * x, axis=-1, keepdims=True) / d,",
                     "return gxr * r,"),
    "causal_mask": ("mask = np.triu(np.ones((L, L), dtype=bool), 1)", "mask = np.zeros((L, L), dtype=bool)"),
    "window_blend": ("g_h = alpha * (dh_ @ F_this) / T + (1.0 - alpha) * g_next\n    grad =",
                     "g_h = alpha * (dh_ @ F_this) / T + alpha * g_next\n    grad ="),
    # the module-level window with the current weights as its reference
    "module_reference": ("h_ref, _ = block_forward(x, P_this)\n    h, cache = block_forward(x if x_hat is None else "
                         "x_hat, P_cur)\n    dh_",
                         "h_ref, _ = block_forward(x, P_cur)\n    h, cache = block_forward(x if x_hat is None else "
                         "x_hat, P_cur)\n    dh_"),
    # the current pass run on the reference input instead of the perturbed one
    "current_input": ("h, cache = block_forward(x if x_hat is None else x_hat, P_cur)\n    dh_",
                      "h, cache = block_forward(x, P_cur)\n    dh_"),
    "kl_current_input": ("h, cache = block_forward(x if x_hat is None else x_hat, P_cur)\n    loss, g_h",
                         "h, cache = block_forward(x, P_cur)\n    loss, g_h"),
    # the KL head: the gradient's sign, the head's norm left out of the
    # backward, the Fisher's label weights dropped, the KL's direction swapped
    "kl_gradient_sign": ("gz = (np.exp(_log_softmax(z1)) - np.exp(_log_softmax(z0))) / T",
                         "gz = (np.exp(_log_softmax(z0)) - np.exp(_log_softmax(z1))) / T"),
    "head_norm_backward": ("gh, _ = _rms_vjp(h, head[\"gf\"], r, gz @ head[\"Wh\"])",
                           "gh = (gz @ head[\"Wh\"]) * head[\"gf\"] * r"),
    "fisher_weights": ("F += p[..., v, None, None] * g[..., :, None] * g[..., None, :]",
                       "F += g[..., :, None] * g[..., None, :] / p.shape[-1]"),
    "kl_direction": ("return np.sum(np.exp(lp) * (lp - lq), axis=-1)",
                     "return np.sum(np.exp(lq) * (lq - lp), axis=-1)"),
}


# the sweep's hook for the exact losses (oracle/realq.py), caught by the
# block pins: the gradient's columns shifted to the quantized side
SWEEP_HOOK_MUTATIONS = {
    "hook_columns": ("G = gfn(W, alpha, (b_global - 1) * steps + si)[1][:, be:]",
                     "G = gfn(W, alpha, (b_global - 1) * steps + si)[1][:, :n - be]"),
    "hook_blend": ("before = gfn(W, alpha, k0)[0] if record else None",
                   "before = gfn(W, 1.0, k0)[0] if record else None"),
    # the rotation over calibration mini-batches stuck at the first one
    "hook_rotation": ("G = gfn(W, alpha, (b_global - 1) * steps + si)[1][:, be:]",
                      "G = gfn(W, alpha, 0)[1][:, be:]"),
}


def _pins_on_copy(tmp_path, old=None, new=None, target="realq.py", pins="tests/test_oracle_pins.py"):
    for d in ("oracle", "synth", "tests"):
        shutil.copytree(os.path.join(ROOT, d), tmp_path / d, ignore=shutil.ignore_patterns("__pycache__"))
    if old is not None:
        src = (tmp_path / "oracle" / target).read_text()
        assert src.count(old) == 1, f"mutation anchor not found once: {old}"
        (tmp_path / "oracle" / target).write_text(src.replace(old, new))
    env = dict(os.environ, PYTHONPATH=str(tmp_path))
    return subprocess.run([sys.executable, "-m", "pytest", pins, "-x", "-q", "-p",
                           "no:cacheprovider", "-m", "not gpu"], cwd=tmp_path, env=env, capture_output=True,
                          text=True, timeout=600)


def test_unchanged_copy_passes(tmp_path):
    # the control: the copy itself passes, so a failure below is the mistake's
    r = _pins_on_copy(tmp_path)
    assert r.returncode == 0, r.stdout[-2000:]


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_the_mistake(name, tmp_path):
    r = _pins_on_copy(tmp_path, *MUTATIONS[name])
    assert r.returncode != 0, f"the pins did not catch '{name}':\n{r.stdout[-2000:]}"
    assert " failed" in r.stdout, r.stdout[-2000:]     # a failing pin, not a crash


def test_unchanged_block_copy_passes(tmp_path):
    r = _pins_on_copy(tmp_path, pins="tests/test_oracle_block_pins.py")
    assert r.returncode == 0, r.stdout[-2000:]


@pytest.mark.parametrize("name", sorted(BLOCK_MUTATIONS))
def test_block_pins_catch_the_mistake(name, tmp_path):
    old, new = BLOCK_MUTATIONS[name]
    r = _pins_on_copy(tmp_path, old, new, target="block.py", pins="tests/test_oracle_block_pins.py")
    assert r.returncode != 0, f"the pins did not catch '{name}':\n{r.stdout[-2000:]}"
    assert " failed" in r.stdout, r.stdout[-2000:]


@pytest.mark.parametrize("name", sorted(SWEEP_HOOK_MUTATIONS))
def test_block_pins_catch_the_sweep_hook_mistake(name, tmp_path):
    old, new = SWEEP_HOOK_MUTATIONS[name]
    r = _pins_on_copy(tmp_path, old, new, target="realq.py", pins="tests/test_oracle_block_pins.py")
    assert r.returncode != 0, f"the pins did not catch '{name}':\n{r.stdout[-2000:]}"
    assert " failed" in r.stdout, r.stdout[-2000:]
