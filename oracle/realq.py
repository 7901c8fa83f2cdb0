"""Plain fp64 statement of the REAL-Q per-layer sweep (test infrastructure only).

Notation follows the paper: W (m x n, out x in), calibration inputs x̂_t
(perturbed) and x_t (full precision), H the input second-moment matrix,
F the aggregated Fisher on the module-output space, B the column block size.

Sections cited:
  Sec. 3.2 "GPTQ Recap", Eq. (gptq_update) and the lazy batch update after it
  Sec. 4.2 "Objective", Eq. (fisher_full), Eq. (fisher_loss)
  Sec. 4.3 "Dynamic Block-wise Gradient Descent", Eq. (block_gd_update)
  Sec. 4.4 "Loss Sliding Window", Eq. (slide_window)
  Algorithm 1 "REAL-Q Quantization"
  App. "Reconstruction error of GPTQ" theorem and the Schur-complement proof
  App. "Full Setup": Adam hyper-parameters, Eq. (reverse_cosine)
  Sec. 3.3 Eq. (saliency_hessian) and App. "Hessian-side saliency clipping"
  Sec. 4.3 / Sec. 5.1 mini-batches and App. "Activation clipping
    (a_loss_clip) for small Qwen3 models"
  Sec. 5 "Weight-Activation Quantization" (per-token activation grid)

Everything is fp64 except the integer decisions of the quantizer (the code and
the zero point), which are taken in fp32 arithmetic: the paper does not fix the
precision of quant(.), and the CUDA path decides in fp32, so both sides decide
in fp32 on their own fp32-rounded operands.

Readings of points the paper leaves open are listed with each function.
The oracle performs the OBS compensation of every column immediately on all
remaining columns and downdates H^-1 explicitly (no lazy batching, no Cholesky
shortcut): the column sweep is the literal recursion of Eq. (gptq_update) with
the Schur-complement downdate named in the theorem's proof.
"""
from __future__ import annotations

import math
from fractions import Fraction
from typing import Iterable, Optional

import numpy as np

from . import native

__all__ = [
    "hessian_sum", "cross_moment_sum", "prepare", "inverse_upper_cholesky",
    "quant_params", "quantize", "rtn", "sliding_alpha", "reverse_cosine_lr", "Adam",
    "surrogate_tokens", "surrogate_moment", "gradient", "gradient_error_scale", "realq_sweep", "pack_codes",
    "round_bf16", "quantize_activations", "saliency_clip", "weighted_hessian_sum",
    "loss_clip_factors", "gradient_tokens", "surrogate_tokens_clipped", "nearest_rank",
]


# ---------------------------------------------------------------------------
# Step a2: Hessian accumulation.  Sec. 3.2 defines H from the calibration
# inputs; REAL-Q feeds the perturbed inputs x̂ (Sec. 1, Sec. 2 on GPTAQ).
# ---------------------------------------------------------------------------
def hessian_sum(xhat_chunks: Iterable[np.ndarray]):
    """H_sum = sum_t x̂_t x̂_t^T over all chunks, and the token count T."""
    H, T = None, 0
    for c in xhat_chunks:
        c = np.asarray(c, dtype=np.float64)
        if H is None:
            H = np.zeros((c.shape[1], c.shape[1]))
        H += c.T @ c
        T += c.shape[0]
    return H, T


def cross_moment_sum(xhat_chunks: Iterable[np.ndarray], x_chunks: Iterable[np.ndarray]):
    """D_sum[i, j] = sum_t (x̂_ti - x_ti) x̂_tj.

    With Δy_t = Ŵ x̂_t - W0 x_t, the surrogate gradient needs
    (1/T) sum_t Δy_t x̂_t^T = (Ŵ - W0) H̄ + W0 D̄ with D̄ = D_sum / T.
    """
    D = None
    for ch, cx in zip(xhat_chunks, x_chunks):
        ch = np.asarray(ch, dtype=np.float64)
        cx = np.asarray(cx, dtype=np.float64)
        if D is None:
            D = np.zeros((ch.shape[1], ch.shape[1]))
        D += (ch - cx).T @ ch
    return D


# ---------------------------------------------------------------------------
# Step a3: preparation of the OBS Hessian (Alg. 1, "Compute ... H_g and its
# inverse").  Readings: H̄ = H_sum / T (the factor 2/T of Sec. 3.2 cancels in
# every ratio the OBS step uses); channels that never fire (H_jj = 0) get
# H_jj = 1 and their weights are zeroed; damping lambda = damp * mean(diag H̄).
# ---------------------------------------------------------------------------
def prepare(H_sum: np.ndarray, T: int, damp_frac: float = 0.01):
    H_sum = np.asarray(H_sum, dtype=np.float64)
    n = H_sum.shape[0]
    Hbar = H_sum / float(T)
    dead = np.diag(H_sum) == 0.0
    Hd = Hbar.copy()
    idx = np.arange(n)
    Hd[idx[dead], idx[dead]] = 1.0
    lam = damp_frac * float(np.mean(np.diag(Hd)))
    Hd[idx, idx] += lam
    return {"Hbar": Hbar, "Hd": Hd, "dead": dead, "lam": lam}


def inverse_upper_cholesky(Hd: np.ndarray) -> np.ndarray:
    """U upper triangular with Hd^-1 = U^T U (the 'Cholesky-based inverse')."""
    Hinv = np.linalg.inv(Hd)
    L = np.linalg.cholesky(Hinv)       # Hinv = L L^T, L lower
    return L.T.copy()                  # U = L^T  =>  Hinv = U^T U


# ---------------------------------------------------------------------------
# quant(.) of Alg. 1: uniform b-bit grid.  Reading: asymmetric
# min/max grid that always contains 0 (xmin <= 0 <= xmax, degenerate rows get
# [-1, 1]), scale = (xmax - xmin) / (2^b - 1), integer zero point; symmetric
# variant: xmax = max(|xmin|, xmax), xmin = -xmax, zero = 2^(b-1).  Rounding is
# round-half-to-even.  Decisions in fp32 (module docstring).
# ---------------------------------------------------------------------------
def _grid(w_rows: np.ndarray, bits: int, symmetric: bool):
    """quant(.)'s per-row grid of a group: (scale fp32, zero int, zero margin, zero before rounding)."""
    w = np.asarray(w_rows, dtype=np.float64).astype(np.float32)
    maxq = np.float32(2 ** bits - 1)
    xmin = np.minimum(w.min(axis=1), np.float32(0.0))
    xmax = np.maximum(w.max(axis=1), np.float32(0.0))
    if symmetric:
        xmax = np.maximum(-xmin, xmax)
        xmin = -xmax
    both0 = (xmin == 0) & (xmax == 0)
    xmin = np.where(both0, np.float32(-1.0), xmin).astype(np.float32)
    xmax = np.where(both0, np.float32(1.0), xmax).astype(np.float32)
    scale = ((xmax - xmin) / maxq).astype(np.float32)
    if symmetric:
        zero = np.full(w.shape[0], 2 ** (bits - 1), dtype=np.int64)
        zmargin = np.full(w.shape[0], 0.5)
        zf = zero.astype(np.float64)
    else:
        zf = (-xmin / scale).astype(np.float32)
        zero = np.rint(zf).astype(np.int64)
        zf = zf.astype(np.float64)
        zmargin = np.abs(np.abs(zf - np.floor(zf)) - 0.5)
    return scale, zero, zmargin, zf


def quant_params(w_rows: np.ndarray, bits: int = 4, symmetric: bool = False):
    """Per-row (scale fp32, zero int) for a group of columns w_rows (m x g)."""
    scale, zero, zmargin, _ = _grid(w_rows, bits, symmetric)
    return scale, zero, zmargin


def _round(w: np.ndarray, scale: np.ndarray, zero: np.ndarray, bits: int):
    """(q, w/scale in fp32 as fp64, margin) of quant(.) on one column."""
    maxq = 2 ** bits - 1
    x = (np.asarray(w, dtype=np.float64).astype(np.float32) / scale.astype(np.float32)).astype(np.float32)
    r = np.rint(x)
    q = np.clip(r.astype(np.int64) + zero, 0, maxq)
    x64 = x.astype(np.float64)
    margin = np.abs(np.abs(x64 - np.floor(x64)) - 0.5)
    return q, x64, margin


def _round32(a: np.ndarray) -> None:
    """In place: every entry rounded to the nearest single-precision value."""
    a[...] = a.astype(np.float32)


def _dequant(q: np.ndarray, scale: np.ndarray, zero: np.ndarray) -> np.ndarray:
    return (scale.astype(np.float32) * (q.astype(np.float32) - zero.astype(np.float32))).astype(np.float32)


def quantize(w: np.ndarray, scale: np.ndarray, zero: np.ndarray, bits: int = 4):
    """q = clamp(rint(w / scale) + zero, 0, 2^b - 1); deq = scale * (q - zero).

    Returns (q int64, deq as fp64 of the fp32 value, margin) where margin is the
    distance of w/scale from the nearest rounding boundary, in grid steps.
    """
    q, _, margin = _round(w, scale, zero, bits)
    return q, _dequant(q, scale, zero).astype(np.float64), margin


def _follow_tie(mine: np.ndarray, value: np.ndarray, margin: np.ndarray, other: np.ndarray, tau,
                offset, lo: int, hi: int):
    """Where this run's rounding of `value` is a tie (margin < tau) and another
    run of the sweep took the other neighbour, take that one.  The two
    neighbours are clamp(floor(value) + offset) and clamp(ceil(value) +
    offset).  Returns (decisions, mask of those taken from `other`)."""
    other = np.asarray(other, dtype=np.int64)
    down = np.clip(np.floor(value).astype(np.int64) + offset, lo, hi)
    up = np.clip(np.ceil(value).astype(np.int64) + offset, lo, hi)
    take = (margin < tau) & (other != mine) & ((other == down) | (other == up))
    return np.where(take, other, mine), take


def rtn(W: np.ndarray, bits: int = 4, group_size: int = 128, symmetric: bool = False):
    """Round-to-nearest baseline: every group quantized from the original weights."""
    W = np.asarray(W, dtype=np.float64)
    m, n = W.shape
    g = group_size if group_size > 0 else n
    codes = np.zeros((m, n), dtype=np.int64)
    deq = np.zeros((m, n))
    scales, zeros = [], []
    for j0 in range(0, n, g):
        s, z, _ = quant_params(W[:, j0:j0 + g], bits, symmetric)
        for j in range(j0, min(j0 + g, n)):
            codes[:, j], deq[:, j], _ = quantize(W[:, j], s, z, bits)
        scales.append(s)
        zeros.append(z)
    return codes, deq, np.stack(scales, 1), np.stack(zeros, 1)


# ---------------------------------------------------------------------------
# Schedules.  Eq. (slide_window) and Eq. (reverse_cosine).
# ---------------------------------------------------------------------------
def sliding_alpha(b_global: int, B_total: int) -> float:
    """alpha = 1 - (b_global - 1) / (B_total - 1); 1 when there is one step only."""
    if B_total <= 1:
        return 1.0
    return 1.0 - (b_global - 1) / (B_total - 1)


def reverse_cosine_lr(i: int, L: int, eta_final: float, eta_base: Optional[float] = None) -> float:
    """Learning rate of transformer block i (1-based) of L; eta_base = 0.01 eta_final."""
    if eta_base is None:
        eta_base = 0.01 * eta_final
    if L <= 1:
        return eta_final
    return eta_base + (eta_final - eta_base) * math.sin(0.5 * math.pi * (i - 1) / (L - 1))


# ---------------------------------------------------------------------------
# Adam (App. "Full Setup": beta1 0.9, beta2 0.999, eps 1e-8, bias correction
# at every block step).  Reading: PyTorch placement of eps (outside the sqrt),
# no weight decay; one state per weight, reset per module.
# ---------------------------------------------------------------------------
class Adam:
    def __init__(self, shape, lr, beta1=0.9, beta2=0.999, eps=1e-8):
        self.m = np.zeros(shape)
        self.v = np.zeros(shape)
        self.t = 0
        self.lr, self.beta1, self.beta2, self.eps = lr, beta1, beta2, eps

    def direction(self, g: np.ndarray, cols: slice) -> np.ndarray:
        """Advance the moments of columns `cols` with gradient g; return the step.
        (Every entry is independent: large updates are shared among threads
        by rows, with the same operations on every entry.)"""
        self.t += 1
        step = np.empty_like(g)

        def rows(r0, r1):
            m = self.m[r0:r1, cols]
            v = self.v[r0:r1, cols]
            gr = g[r0:r1]
            m[...] = self.beta1 * m + (1.0 - self.beta1) * gr
            v[...] = self.beta2 * v + (1.0 - self.beta2) * gr * gr
            mhat = m / (1.0 - self.beta1 ** self.t)
            vhat = v / (1.0 - self.beta2 ** self.t)
            step[r0:r1] = self.lr * mhat / (np.sqrt(vhat) + self.eps)

        native.row_chunks(g.shape[0], g.size, rows)
        return step


# ---------------------------------------------------------------------------
# Surrogate, Eq. (fisher_loss), read at the layer level: Δy_t = Ŵ x̂_t - W0 x_t
# on the module-output space with an m x m Fisher F.
# ---------------------------------------------------------------------------
def surrogate_tokens(What, W0, Xhat, X, F) -> float:
    """(1/2)(1/T) sum_t Δy_t^T F Δy_t, evaluated token by token (matmul per chunk)."""
    What = np.asarray(What, dtype=np.float64)
    W0 = np.asarray(W0, dtype=np.float64)
    F = np.asarray(F, dtype=np.float64)
    Xhat = np.asarray(Xhat)
    X = Xhat if X is None else np.asarray(X)
    T = Xhat.shape[0]
    acc = 0.0
    for t0 in range(0, T, 4096):
        xh = Xhat[t0:t0 + 4096].astype(np.float64)
        xx = X[t0:t0 + 4096].astype(np.float64)
        dY = xh @ What.T - xx @ W0.T
        acc += float(np.sum((dY @ F) * dY))
    return 0.5 * acc / T


def surrogate_moment(What, W0, Hbar, F) -> float:
    """Same loss when X = X̂: (1/2) tr(F ΔW H̄ ΔW^T) with ΔW = Ŵ - W0."""
    dW = np.asarray(What, dtype=np.float64) - np.asarray(W0, dtype=np.float64)
    return 0.5 * float(np.sum((np.asarray(F, dtype=np.float64) @ dW) * (dW @ np.asarray(Hbar, dtype=np.float64))))


def _gradient_factor(What, W0, Hbar, Dbar, cols: slice) -> np.ndarray:
    """P = (1/T) sum_t Δy_t x̂_t^T = (Ŵ - W0) H̄ + W0 D̄, columns `cols`."""
    W0 = np.asarray(W0, dtype=np.float64)
    P = (np.asarray(What, dtype=np.float64) - W0) @ np.asarray(Hbar, dtype=np.float64)[:, cols]
    if Dbar is not None:
        P = P + W0 @ np.asarray(Dbar, dtype=np.float64)[:, cols]
    return P


def gradient(What, W0, Hbar, Dbar, F, cols: slice = slice(None)) -> np.ndarray:
    """dL/dŴ = F P for the columns `cols` of Ŵ (m x |cols|; every column of P
    is its own product)."""
    return np.asarray(F, dtype=np.float64) @ _gradient_factor(What, W0, Hbar, Dbar, cols)


def gradient_error_scale(What, W0, Hbar, Dbar, F, cols: slice = slice(None)) -> np.ndarray:
    """|F| |P| for the columns `cols`: the sum of the magnitudes of the terms
    of each gradient entry, the scale of its rounding error in any
    floating-point evaluation (a sensitivity probe; not part of the method)."""
    return np.abs(np.asarray(F, dtype=np.float64)) @ np.abs(_gradient_factor(What, W0, Hbar, Dbar, cols))


# ---------------------------------------------------------------------------
# Nearest-rank percentile, the rule of both clipping steps of the paper (App.
# "Hessian-side saliency clipping": the 99th percentile of the per-token
# saliency; App. "Activation clipping (a_loss_clip)": the 95th percentile of
# the output perturbation).  Reading: the pct-percentile of `count` values is
# the smallest of them with at least pct * count values at or below it, i.e.
# the ceil(pct * count)-th smallest.  pct is the number as written (0.99 is
# 99/100) and the product is exact, so 0.99 of 8000 values is the 7920th.
# ---------------------------------------------------------------------------
def nearest_rank(pct: float, count: int) -> int:
    """0-based position of the nearest-rank pct-percentile in `count` sorted values."""
    r = math.ceil(Fraction(repr(float(pct))) * count)
    return min(max(r - 1, 0), count - 1)


# ---------------------------------------------------------------------------
# Output-perturbation clipping of the Block-GD loss (App. "Activation
# clipping (a_loss_clip) for small Qwen3 models": a_loss_clip = 0.95 on
# Qwen3-0.6B, 1.7B and 4B).  Per token, the output channels whose |Δy| lies
# above the 95th percentile are scaled down by a detached factor, so that a
# few outlier channels cannot dominate the Fisher MSE while their gradient
# stays non-zero.
# Readings: the percentile is taken per token over its m output channels, as
# the nearest-rank one of the saliency clip (the ceil(pct m)-th smallest
# |Δy_t,i|, see nearest_rank); a channel above it is scaled by
# kappa = q_t / |Δy_t,i| (its scaled residual has magnitude q_t), every other
# channel by 1; kappa is a constant of the step (detached), so with
# L = (1/2T) sum_t (kappa_t ⊙ Δy_t)^T F (kappa_t ⊙ Δy_t)
# the gradient is dL/dŴ = (1/T) sum_t (kappa_t ⊙ F (kappa_t ⊙ Δy_t)) x̂_t^T.
# The factors depend on the tokens, so this gradient is taken in token form
# on the step's mini-batch.  kappa is continuous in Δy (it is 1 at the
# threshold), so rounding differences near the threshold move it by no more
# than they move Δy.
# ---------------------------------------------------------------------------
def loss_clip_factors(dY: np.ndarray, pct: float):
    """kappa (T x m) and the per-token thresholds q (T) for residuals dY (T x m)."""
    dY = np.asarray(dY, dtype=np.float64)
    m = dY.shape[1]
    k = nearest_rank(pct, m)
    a = np.abs(dY)
    q = np.sort(a, axis=1)[:, k]
    kappa = np.ones_like(a)
    over = a > q[:, None]
    kappa[over] = (q[:, None] / np.where(over, a, 1.0))[over]
    return kappa, q


def gradient_tokens(What, W0, Xhat, X, F, a_loss_clip: Optional[float] = None) -> np.ndarray:
    """dL/dŴ (m x n) on the tokens Xhat (T x n), in token form: Δy_t = Ŵ x̂_t - W0 x_t,
    (1/T) sum_t (kappa_t ⊙ F (kappa_t ⊙ Δy_t)) x̂_t^T with kappa = 1 without clipping."""
    What = np.asarray(What, dtype=np.float64)
    W0 = np.asarray(W0, dtype=np.float64)
    F = np.asarray(F, dtype=np.float64)
    Xh = np.asarray(Xhat, dtype=np.float64)
    Xf = Xh if X is None else np.asarray(X, dtype=np.float64)
    dY = Xh @ What.T - Xf @ W0.T
    kappa = np.ones_like(dY) if a_loss_clip is None else loss_clip_factors(dY, a_loss_clip)[0]
    Z = (kappa * dY) @ F
    return (kappa * Z).T @ Xh / float(Xh.shape[0])


def surrogate_tokens_clipped(What, W0, Xhat, F, kappa) -> float:
    """(1/2)(1/T) sum_t (kappa_t ⊙ Δy_t)^T F (kappa_t ⊙ Δy_t) with given factors."""
    Xh = np.asarray(Xhat, dtype=np.float64)
    dY = Xh @ (np.asarray(What, dtype=np.float64) - np.asarray(W0, dtype=np.float64)).T
    Y = np.asarray(kappa, dtype=np.float64) * dY
    return 0.5 * float(np.sum((Y @ np.asarray(F, dtype=np.float64)) * Y)) / Xh.shape[0]


def pack_codes(codes: np.ndarray) -> np.ndarray:
    """Two int4 codes per byte, even column in the low nibble (m x ceil(n/2) uint8)."""
    m, n = codes.shape
    c = np.zeros((m, n + (n & 1)), dtype=np.uint8)
    c[:, :n] = codes
    return (c[:, 0::2] | (c[:, 1::2] << 4)).astype(np.uint8)


# ---------------------------------------------------------------------------
# The sweep: Algorithm 1, inner loops for one linear module.
# ---------------------------------------------------------------------------
def realq_sweep(W0, H_sum, T, *, bits=4, group_size=128, block_size=128, symmetric=False,
                damp_frac=0.01, bgd=None, F=None, F_next=None, D_sum=None, record=True, obs_hessians=None,
                follow=None, columns=None, grad_noise=None, state32=False):
    """Quantize W0 column by column with OBS feedback and Block-GD after each block.

    bgd: None for the plain column sweep (GPTQ), else a dict with keys
      steps_per_block (1 in the paper), lr, beta1, beta2, eps,
      optimizer ("adam" | "sgd"), b_global_start (1-based cumulative block index
      of this module's first block), B_total (column-block steps in the
      transformer block; 1 disables the sliding window), and optionally
      minibatches: a list of K pairs (H_mb_sum, T_mb), the second moments of
      calibration mini-batches (Sec. 4.3: each Block-GD step evaluates the
      surrogate on a calibration mini-batch; Sec. 5.1: 32 sequences).  Step s
      (0-based) of the block with global index b_global uses mini-batch
      ((b_global - 1) * steps_per_block + s) mod K, so consecutive steps of a
      transformer block rotate through the calibration set; or
      minibatch_tokens: a list of K token blocks X̂_k (T_k x n) with the same
      rotation, whose gradient is taken in token form, and then optionally
      a_loss_clip: the per-token output clipping percentile (0.95 in the
      paper's small-model runs; see loss_clip_factors); or
      gradient_fn: a callable (W, alpha, k) -> (loss, G) that gives the
      surrogate and its gradient in W (m x n) at the current weights, in
      place of the layer-level surrogate: the exact two-block window of
      Sec. 4.4 and the final block's KL at the LM head (App. "Pre-computation
      of the aggregated Fisher and last-transformer-block handling"), both
      stated in oracle.block.  k = (b_global - 1) * steps_per_block + s is
      the step's place in the rotation over calibration mini-batches (Sec.
      4.3: each step's forward pass uses a calibration mini-batch), the same
      rotation as minibatches above.  The per-block values it records are its
      own loss before the block's steps (on the first step's mini-batch) and
      after them (on the last step's).

    Readings: group parameters are computed at the first column of each group
    from the current (compensated, Block-GD-updated) weights; group_size 0
    means one group per row; the gradient is the full-batch moment form of the
    layer-level surrogate; Block-GD updates all rows jointly on the columns
    after the block; the block after the last column is skipped (no columns
    remain).  Returns a dict of codes, scale, zero, deq (fp32 values as fp64),
    per-column residuals, tie margins and per-block surrogate values.

    obs_hessians: None (one Hessian for every row), or the row-grouped OBS of
    Alg. 1 ("for all row-groups g"): a list of N_g pairs (H_g_sum, norm_g).
    The rows are split into N_g contiguous groups of ceil(m / N_g) rows; group
    g's OBS step and lazy update use H̄_g = H_g_sum / norm_g (damped and with
    its own dead channels, as in prepare), while Block-GD keeps the
    surrogate's plain H̄ = H_sum / T.

    follow: None, or the rounding decisions of another run of the same sweep
    as a dict with "codes" (m x n ints), optionally "zero" (m x ngroups ints)
    and "tau" (grid steps, default 1e-3: a scalar, or an m x n array of
    per-decision tolerances with "tau_zero" an m x ngroups one for the zero
    points).  quant(.) rounds to the nearest
    grid point, and where w / scale (or -xmin / scale for the zero point)
    lies within tau of a rounding boundary both neighbours are the correctly
    rounded result up to the rounding of the operands (reading C3 of the
    rounding that Sec. 3.2's quant(.) leaves open).  At every such tie where
    the other run took the other neighbour, this run takes it too and
    carries it forward through the compensation and Block-GD; every other
    decision is this sweep's own.  n_followed counts the decisions taken.

    columns: None for the whole sweep, or stop after that many columns (a
    bounded sample of the work, for timing).

    grad_noise: None, or a sensitivity probe {"seed", "eta"}: every moment-form
    Block-GD gradient entry moves by eta times the magnitude of its terms
    (gradient_error_scale) times a seeded standard normal, the size of the
    rounding differences that any floating-point evaluation of the gradient
    may show.  Comparing a probed run with the plain one shows which
    decisions the sweep's arithmetic does not determine at that precision.
    The returned "x" holds every column's w / scale before rounding, "zf"
    every group's -xmin / scale.

    state32: a second sensitivity probe (not part of the method): the sweep's
    state (the Hessian, each downdated inverse, the weights after every
    compensation and every optimizer step, the gradient and Adam's moments)
    is rounded to single precision after every update, one realization of
    the rounding that an fp32 implementation carries along.
    """
    W0 = np.asarray(W0, dtype=np.float64)
    m, n = W0.shape
    B = block_size
    g = group_size if group_size > 0 else n
    if not (g % B == 0 or B % g == 0 or g == n):
        raise ValueError("group size must divide the block size or be a multiple of it")
    prep = prepare(H_sum, T, damp_frac)
    Hbar, Hd, dead = prep["Hbar"], prep["Hd"], prep["dead"]
    Dbar = None if D_sum is None else np.asarray(D_sum, dtype=np.float64) / float(T)

    W = W0.copy()
    if obs_hessians is None:
        groups = [(slice(0, m), Hd, dead)]
    else:
        mg = -(-m // len(obs_hessians))
        groups = []
        for k, (Hg, normg) in enumerate(obs_hessians):
            pg = prepare(Hg, normg, damp_frac)
            groups.append((slice(k * mg, min((k + 1) * mg, m)), pg["Hd"], pg["dead"]))
    for rows, _, dg in groups:
        W[rows, dg] = 0.0
    Hinvs = [np.linalg.inv(Hdg) for _, Hdg, _ in groups]
    r32 = _round32 if state32 else (lambda a: None)
    for Hinv in Hinvs:
        r32(Hinv)
    r32(W)
    ngroups = -(-n // g)
    codes = np.zeros((m, n), dtype=np.int64)
    scale = np.zeros((m, ngroups), dtype=np.float32)
    zero = np.zeros((m, ngroups), dtype=np.int64)
    margin = np.zeros((m, n))
    zmargin = np.zeros((m, ngroups))
    zfval = np.zeros((m, ngroups))
    eps_cols = np.zeros((m, n))
    xval = np.zeros((m, n))
    hinv_diag = np.zeros((len(groups), n))
    block_loss = []
    opt = None
    if bgd is not None:
        opt = Adam((m, n), bgd["lr"], bgd.get("beta1", 0.9), bgd.get("beta2", 0.999), bgd.get("eps", 1e-8))
    Fm = None if F is None else np.asarray(F, dtype=np.float64)
    Fn = None if F_next is None else np.asarray(F_next, dtype=np.float64)

    maxq = 2 ** bits - 1
    tau = 1e-3 if follow is None else follow.get("tau", 1e-3)
    tau_codes = np.broadcast_to(np.asarray(tau, dtype=np.float64), (m, n))
    tz = None if follow is None else follow.get("tau_zero")
    tau_zero = np.broadcast_to(np.asarray((tau if np.ndim(tau) == 0 else 1e-3) if tz is None else tz,
                                          dtype=np.float64), (m, ngroups))
    n_followed = n_followed_zero = 0
    for j in range(n if columns is None else min(int(columns), n)):
        if j % g == 0:
            gi = j // g
            scale[:, gi], zero[:, gi], zmargin[:, gi], zf = _grid(W[:, j:j + g], bits, symmetric)
            zfval[:, gi] = zf
            if follow is not None and follow.get("zero") is not None and not symmetric:
                zero[:, gi], took = _follow_tie(zero[:, gi], zf, zmargin[:, gi], follow["zero"][:, gi],
                                                tau_zero[:, gi], 0, 0, maxq)
                n_followed_zero += int(took.sum())
        gi = j // g
        q, x, mg = _round(W[:, j], scale[:, gi], zero[:, gi], bits)
        if follow is not None:
            q, took = _follow_tie(q, x, mg, follow["codes"][:, j], tau_codes[:, j], zero[:, gi], 0, maxq)
            n_followed += int(took.sum())
        dq = _dequant(q, scale[:, gi], zero[:, gi]).astype(np.float64)
        e = W[:, j] - dq                       # residual delta_j of Eq. (gptq_update)
        codes[:, j] = q
        margin[:, j] = mg
        xval[:, j] = x
        eps_cols[:, j] = e
        for k, ((rows, _, _), Hinv) in enumerate(zip(groups, Hinvs)):
            d = Hinv[j, j]
            hinv_diag[k, j] = d
            # Eq. (gptq_update): W[:, j+1:] -= delta_j H^-1[j, j+1:] / [H^-1]_jj
            native.outer_sub(W[rows, j + 1:], e[rows] / d, Hinv[j, j + 1:])
            r32(W[rows, j + 1:])
            # remove j from the free set: Schur-complement downdate of H^-1
            native.outer_sub(Hinv[j + 1:, j + 1:], Hinv[j + 1:, j], Hinv[j, j + 1:], d)
            r32(Hinv[j + 1:, j + 1:])
        W[:, j] = dq

        be = j + 1
        if opt is not None and (be % B == 0 or be == n) and be < n:
            b = j // B
            b_global = bgd.get("b_global_start", 1) + b
            alpha = sliding_alpha(b_global, bgd.get("B_total", 1))
            gfn = bgd.get("gradient_fn")
            if gfn is not None:
                Feff = None
                k0 = (b_global - 1) * bgd.get("steps_per_block", 1)
                before = gfn(W, alpha, k0)[0] if record else None
            else:
                Feff = Fm if Fn is None else alpha * Fm + (1.0 - alpha) * Fn
                before = surrogate_moment(W, W0, Hbar, Feff) if (record and Dbar is None) else None
            mbs = bgd.get("minibatches")
            mbt = bgd.get("minibatch_tokens")
            steps = bgd.get("steps_per_block", 1)
            for si in range(steps):
                Hstep = Hbar
                if gfn is not None:
                    G = gfn(W, alpha, (b_global - 1) * steps + si)[1][:, be:]
                elif mbt:
                    if Dbar is not None:
                        raise ValueError("mini-batch tokens with perturbed inputs are not supported")
                    Xk = mbt[((b_global - 1) * steps + si) % len(mbt)]
                    G = gradient_tokens(W, W0, Xk, None, Feff, bgd.get("a_loss_clip"))[:, be:]
                else:
                    if mbs:
                        if Dbar is not None:
                            raise ValueError("mini-batch moments with perturbed inputs are not supported")
                        Hk, Tk = mbs[((b_global - 1) * steps + si) % len(mbs)]
                        Hstep = np.asarray(Hk, dtype=np.float64) / float(Tk)
                    G = gradient(W, W0, Hstep, Dbar, Feff, slice(be, n))
                    if grad_noise is not None:
                        # sensitivity probe: each entry moved by a random
                        # multiple of its terms' magnitude (eta ~ the
                        # relative rounding of one floating-point product)
                        gen = np.random.default_rng([int(grad_noise["seed"]), int(opt.t)])
                        G = G + grad_noise["eta"] * gradient_error_scale(W, W0, Hstep, Dbar, Feff, slice(be, n)) \
                            * gen.standard_normal(G.shape)
                if bgd.get("optimizer", "adam") == "sgd":
                    opt.t += 1
                    W[:, be:] -= bgd["lr"] * G
                    r32(W[:, be:])
                else:
                    if state32:
                        G = G.astype(np.float32).astype(np.float64)
                    W[:, be:] -= opt.direction(G, slice(be, n))
                    r32(W[:, be:])
                    r32(opt.m[:, be:])
                    r32(opt.v[:, be:])
            if gfn is not None:
                after = gfn(W, alpha, (b_global - 1) * steps + steps - 1)[0] if record else None
            else:
                after = surrogate_moment(W, W0, Hbar, Feff) if (record and Dbar is None) else None
            block_loss.append((b, alpha, before, after))

    return {
        "codes": codes, "scale": scale, "zero": zero, "deq": W.copy(),
        "margin": margin, "zero_margin": zmargin, "eps": eps_cols,
        "hinv_diag": hinv_diag[0] if obs_hessians is None else hinv_diag,
        "block_loss": block_loss, "adam_t": 0 if opt is None else opt.t,
        "n_followed": n_followed, "n_followed_zero": n_followed_zero, "x": xval, "zf": zfval,
        "Hbar": Hbar, "Hd": Hd, "dead": dead, "lam": prep["lam"], "Dbar": Dbar,
    }


# ---------------------------------------------------------------------------
# Weight-activation setting (Sec. 5, "Weight-Activation Quantization"):
# activations are quantized per token with a clipping ratio (a_clip = 0.9 in
# the paper), and in the activation-aware variant the weights are quantized
# against the already-quantized activations (they are the x̂ of the Hessian,
# and the full-precision x stay the reference of the surrogate).
# Readings: the activation grid is the symmetric grid of quant(.) ("symmetric
# throughout", Sec. 5.1) on the clipped range [-a_clip max|x_t|, a_clip
# max|x_t|] of each token; values beyond it take the end levels; a token of
# all zeros gets the range [-1, 1]; the dequantized value is formed in fp32
# and stored in the input's format (bf16, round to nearest even).  As for the
# weights, the integer decisions are taken in fp32.
# ---------------------------------------------------------------------------
def round_bf16(a: np.ndarray) -> np.ndarray:
    """fp32 values rounded to the nearest bf16 (ties to even), as fp32."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) & np.uint64(0xFFFF0000)
    return u.astype(np.uint32).view(np.float32)


def quantize_activations(X: np.ndarray, bits: int = 4, a_clip: float = 0.9, out_bf16: bool = True):
    """Per-token symmetric b-bit quantization of X (T x n).

    Returns (codes int64 T x n, scale fp32 per token, dequantized X as fp64 of
    its stored value)."""
    x = np.asarray(X, dtype=np.float64).astype(np.float32)
    maxq = np.float32(2 ** bits - 1)
    zero = 2 ** (bits - 1)
    xmax = (np.float32(a_clip) * np.abs(x).max(axis=1)).astype(np.float32)
    xmax = np.where(xmax == 0, np.float32(1.0), xmax).astype(np.float32)
    scale = ((xmax - (-xmax)) / maxq).astype(np.float32)
    r = np.rint((x / scale[:, None]).astype(np.float32))
    q = np.clip(r.astype(np.int64) + zero, 0, 2 ** bits - 1)
    xq = (scale[:, None] * (q - zero).astype(np.float32)).astype(np.float32)
    if out_bf16:
        xq = round_bf16(xq)
    return q, scale, xq.astype(np.float64)


# ---------------------------------------------------------------------------
# Saliency-weighted grouped Hessian (Sec. 3.3 Eq. saliency_hessian, used by
# Alg. 1 "for all row-groups g" with N_g = 4; App. "Hessian-side saliency
# clipping": per-token saliency clipped to the 99th percentile first).
# Readings: the rows of W form N_g contiguous groups, s[t, g] >= 0 is token
# t's saliency for group g; the percentile is the nearest-rank one (the
# smallest saliency value with at least pct of the tokens at or below it, see
# nearest_rank), taken per group over the T tokens; H̄_g = H_g / sum_t s'[t, g] (the
# saliency-weighted mean of x x^T; the OBS step does not depend on the scale).
# ---------------------------------------------------------------------------
def saliency_clip(S: np.ndarray, pct: float = 0.99):
    """Returns (S clipped, per-group thresholds): the threshold of group g is
    the ceil(pct T)-th smallest saliency of its column (nearest_rank)."""
    S = np.asarray(S, dtype=np.float64)
    T = S.shape[0]
    k = nearest_rank(pct, T)
    c = np.sort(S, axis=0)[k]
    return np.minimum(S, c[None, :]), c


def weighted_hessian_sum(xhat_chunks: Iterable[np.ndarray], s_chunks: Iterable[np.ndarray]):
    """H_g = sum_t s[t, g] x̂_t x̂_t^T for every group g, and sum_t s[t, g]."""
    H, wsum = None, None
    for c, sc in zip(xhat_chunks, s_chunks):
        c = np.asarray(c, dtype=np.float64)
        sc = np.asarray(sc, dtype=np.float64)
        if H is None:
            H = np.zeros((sc.shape[1], c.shape[1], c.shape[1]))
            wsum = np.zeros(sc.shape[1])
        for g in range(sc.shape[1]):
            H[g] += (c * sc[:, g:g + 1]).T @ c
            wsum[g] += sc[:, g].sum()
    return H, wsum
