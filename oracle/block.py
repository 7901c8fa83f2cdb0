"""fp64 statement of one synthetic decoder block and of the exact two-block
sliding-window loss (test infrastructure only: the CUDA path never imports
it).

Sec. 4.4, Eq. (slide_window): while quantizing block l the surrogate blends
this block's Fisher loss with the next block's, L = alpha L(l) + (1 - alpha)
L(l+1), and the gradient of L(l+1) is taken by back-propagating from the
output of block l+1 into block l.  The layer-level sweep replaces L(l+1) by
a linearised pull-back F' of the next block's Fisher; this module states the
exact form: for any linear module of block l (sliding_window_module, through
block l's own backward), and the direct form for the module whose output is
block l's residual increment (sliding_window_down: h = r + W x, so
Δh_t = (Ŵ - W0) x_t exactly).

Readings (the paper names the modules q, k, v, o, gate, up, down and a SwiGLU
MLP, Sec. 3.1 and App. "cosine alignment"; the rest is the common structure
of the LLaMA-3.1 and Qwen3 blocks it evaluates):
  pre-norm block   a = RMSNorm(x; g1),  h = x + Attn(a),
                   b = RMSNorm(h; g2),  y = h + W_d (silu(W_g b) * (W_u b))
  RMSNorm          x / sqrt(mean(x^2) + eps) * g, eps = 1e-6
  attention        H query heads of width dh, H_kv key/value heads (query
                   head i reads key/value head i // (H / H_kv)), rotary
                   position embedding on q and k (pairs (j, j + dh/2), angle
                   pos * base^(-2j/dh), base 10000), causal softmax over each
                   sequence with scale 1/sqrt(dh), output projection W_o
  tokens           S sequences of L tokens, (S, L, d); the Fisher losses
                   average over the S L tokens.
The backward pass is written out by hand (no autograd) and pinned by central
finite differences.

The final block has no next block: it takes the true KL against the LM head
(Eq. kl_loss; App. "Pre-computation of the aggregated Fisher and
last-transformer-block handling").  Readings for that part:
  head             z = RMSNorm(h; g_f) W_h^T (a final norm, then the head,
                   as in the evaluated model families), V logits per token
  KL               (1/T) sum_t KL(p_t || q_t), p_t = softmax of the reference
                   logits, q_t = softmax of the perturbed ones (Eq. kl_loss's
                   direction: full precision first)
  Fisher           Eq. fisher_full with g_t the gradient of the NLL of a label
                   drawn from p_t (the draw is an input, fisher_sampled); its
                   exact expectation over the label is fisher_tokens, which is
                   the per-token Hessian H_t of Eq. taylor_expansion.
"""
from __future__ import annotations

from typing import Dict, Optional, Sequence, Tuple

import numpy as np

from . import realq as _sweep

__all__ = ["block_params", "block_forward", "block_vjp", "next_block_loss", "sliding_window_down",
           "sliding_window_module", "head_params", "head_logits", "kl_logits", "kl_head_loss", "nll_scores",
           "fisher_sampled", "fisher_tokens", "kl_final_module", "module_inputs", "window_gradient_fn",
           "kl_gradient_fn", "MODULES", "quantize_block", "quantize_model"]

EPS = 1e-6


def block_params(rng: np.random.Generator, d: int, n_heads: int, n_kv: int, dh: int, f: int,
                 scale: float = 0.2) -> Dict[str, np.ndarray]:
    """Random fp64 parameters of one block (weights ~ N(0, scale^2 / fan_in))."""
    def w(rows, cols):
        return rng.standard_normal((rows, cols)) * scale / np.sqrt(cols)
    return {"g1": 1.0 + 0.1 * rng.standard_normal(d), "Wq": w(n_heads * dh, d), "Wk": w(n_kv * dh, d),
            "Wv": w(n_kv * dh, d), "Wo": w(d, n_heads * dh), "g2": 1.0 + 0.1 * rng.standard_normal(d),
            "Wg": w(f, d), "Wu": w(f, d), "Wd": w(d, f), "n_heads": n_heads, "n_kv": n_kv, "dh": dh}


def _rms(x, g):
    r = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + EPS)
    return x * r * g, r


def _rms_vjp(x, g, r, gy):
    # y = x r g, r = (mean(x^2) + eps)^-1/2;  dr/dx = -r^3 x / d
    d = x.shape[-1]
    gxr = gy * g
    return gxr * r - x * (r ** 3) * np.sum(gxr * x, axis=-1, keepdims=True) / d, np.sum(gy * x * r, axis=(0, 1))


def _rope_tables(L, dh, base=10000.0):
    half = dh // 2
    inv = base ** (-np.arange(half) * 2.0 / dh)
    ang = np.arange(L)[:, None] * inv[None, :]
    return np.cos(ang), np.sin(ang)


def _rope(x, cos, sin):
    # x: (S, L, heads, dh); pairs (j, j + dh/2) rotated by the position's angle
    half = x.shape[-1] // 2
    x1, x2 = x[..., :half], x[..., half:]
    c, s = cos[None, :, None, :], sin[None, :, None, :]
    return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)


def _rope_t(gy, cos, sin):
    # the transpose (inverse) rotation
    half = gy.shape[-1] // 2
    g1, g2 = gy[..., :half], gy[..., half:]
    c, s = cos[None, :, None, :], sin[None, :, None, :]
    return np.concatenate([g1 * c + g2 * s, -g1 * s + g2 * c], axis=-1)


def _silu(z):
    return z / (1.0 + np.exp(-z))


def block_forward(x: np.ndarray, P: Dict) -> Tuple[np.ndarray, Dict]:
    """y = block(x) for x of shape (S, L, d); returns (y, cache for block_vjp)."""
    S, L, d = x.shape
    H, Hkv, dh = P["n_heads"], P["n_kv"], P["dh"]
    rep = H // Hkv
    a, r1 = _rms(x, P["g1"])
    q = (a @ P["Wq"].T).reshape(S, L, H, dh)
    k = (a @ P["Wk"].T).reshape(S, L, Hkv, dh)
    v = (a @ P["Wv"].T).reshape(S, L, Hkv, dh)
    cos, sin = _rope_tables(L, dh)
    qr, kr = _rope(q, cos, sin), _rope(k, cos, sin)
    kr_h = np.repeat(kr, rep, axis=2)                      # (S, L, H, dh)
    v_h = np.repeat(v, rep, axis=2)
    sc = np.einsum("sthe,suhe->shtu", qr, kr_h) / np.sqrt(dh)
    mask = np.triu(np.ones((L, L), dtype=bool), 1)
    sc = np.where(mask[None, None], -np.inf, sc)
    sc = sc - sc.max(axis=-1, keepdims=True)
    p = np.exp(sc)
    p = p / p.sum(axis=-1, keepdims=True)                  # (S, H, L, L)
    o = np.einsum("shtu,suhe->sthe", p, v_h).reshape(S, L, H * dh)
    h = x + o @ P["Wo"].T
    b, r2 = _rms(h, P["g2"])
    zg, zu = b @ P["Wg"].T, b @ P["Wu"].T
    m = _silu(zg) * zu
    y = h + m @ P["Wd"].T
    cache = dict(x=x, a=a, r1=r1, q=q, k=k, v=v, qr=qr, kr_h=kr_h, v_h=v_h, p=p, o=o, h=h, b=b, r2=r2, zg=zg,
                 zu=zu, m=m, cos=cos, sin=sin, P=P)
    return y, cache


def block_vjp(cache: Dict, gy: np.ndarray) -> Tuple[np.ndarray, Dict[str, np.ndarray]]:
    """(dL/dx, {dL/dparam}) for an upstream gradient gy = dL/dy."""
    P = cache["P"]
    S, L, d = cache["x"].shape
    H, Hkv, dh = P["n_heads"], P["n_kv"], P["dh"]
    rep = H // Hkv
    g = {}
    # MLP: y = h + m Wd^T, m = silu(zg) * zu
    g["Wd"] = np.einsum("sti,stj->ij", gy, cache["m"])
    gm = gy @ P["Wd"]
    zg, zu = cache["zg"], cache["zu"]
    sg = 1.0 / (1.0 + np.exp(-zg))
    gzu = gm * _silu(zg)
    gzg = gm * zu * (sg * (1.0 + zg * (1.0 - sg)))
    g["Wg"] = np.einsum("sti,stj->ij", gzg, cache["b"])
    g["Wu"] = np.einsum("sti,stj->ij", gzu, cache["b"])
    gb = gzg @ P["Wg"] + gzu @ P["Wu"]
    gh_n, g["g2"] = _rms_vjp(cache["h"], P["g2"], cache["r2"], gb)
    gh = gy + gh_n
    # attention: h = x + o Wo^T
    g["Wo"] = np.einsum("sti,stj->ij", gh, cache["o"])
    go = (gh @ P["Wo"]).reshape(S, L, H, dh)
    p, v_h = cache["p"], cache["v_h"]
    gp = np.einsum("sthe,suhe->shtu", go, v_h)
    gv_h = np.einsum("shtu,sthe->suhe", p, go)
    gsc = p * (gp - np.sum(gp * p, axis=-1, keepdims=True)) / np.sqrt(dh)
    gqr = np.einsum("shtu,suhe->sthe", gsc, cache["kr_h"])
    gkr_h = np.einsum("shtu,sthe->suhe", gsc, cache["qr"])
    gkr = gkr_h.reshape(S, L, Hkv, rep, dh).sum(axis=3)
    gv = gv_h.reshape(S, L, Hkv, rep, dh).sum(axis=3)
    gq = _rope_t(gqr, cache["cos"], cache["sin"]).reshape(S, L, H * dh)
    gk = _rope_t(gkr, cache["cos"], cache["sin"]).reshape(S, L, Hkv * dh)
    gv = gv.reshape(S, L, Hkv * dh)
    a = cache["a"]
    g["Wq"] = np.einsum("sti,stj->ij", gq, a)
    g["Wk"] = np.einsum("sti,stj->ij", gk, a)
    g["Wv"] = np.einsum("sti,stj->ij", gv, a)
    ga = gq @ P["Wq"] + gk @ P["Wk"] + gv @ P["Wv"]
    gx_n, g["g1"] = _rms_vjp(cache["x"], P["g1"], cache["r1"], ga)
    return gh + gx_n, g


def next_block_loss(h: np.ndarray, dh_: np.ndarray, P_next: Dict, F_next: np.ndarray):
    """L(l+1) = (1/2T) sum_t Δz_t^T F Δz_t with Δz = B(h + Δh) - B(h), and its
    gradient with respect to Δh (T = S L tokens)."""
    z0, _ = block_forward(h, P_next)
    z1, cache = block_forward(h + dh_, P_next)
    dz = z1 - z0
    T = h.shape[0] * h.shape[1]
    w = dz @ F_next
    loss = 0.5 * float(np.sum(w * dz)) / T
    g, _ = block_vjp(cache, w / T)
    return loss, g


def sliding_window_down(W: np.ndarray, W0: np.ndarray, X: np.ndarray, R: np.ndarray, alpha: float,
                        F_this: np.ndarray, F_next: np.ndarray, P_next: Dict, X_hat=None, R_hat=None):
    """The exact two-block sliding-window loss of a down_proj-type module and
    its gradient with respect to W (d x n).

    X: the module's inputs (S, L, n); R: block l's output without this
    module's contribution (S, L, d), so h = R + X W0^T is the reference output
    and R + X W^T the current one.  Block l's own Fisher loss is exact at the
    module level here: Δh_t = (W - W0) x_t.  With the current pass's X_hat
    and R_hat (the model quantized so far), the current output is
    R_hat + X_hat W^T and Δh its difference from the reference."""
    S, L, n = X.shape
    T = S * L
    W0 = np.asarray(W0, dtype=np.float64)
    h = R + X @ W0.T
    if X_hat is None and R_hat is None:
        dh_ = X @ (np.asarray(W, dtype=np.float64) - W0).T
        X_hat = X
    else:
        X_hat = X if X_hat is None else X_hat
        dh_ = (R if R_hat is None else R_hat) + X_hat @ np.asarray(W, dtype=np.float64).T - h
    l_this = 0.5 * float(np.sum((dh_ @ F_this) * dh_)) / T
    l_next, g_next = next_block_loss(h, dh_, P_next, F_next)
    g_h = alpha * (dh_ @ F_this) / T + (1.0 - alpha) * g_next
    grad = np.einsum("sti,stj->ij", g_h, X_hat)
    return alpha * l_this + (1.0 - alpha) * l_next, grad


_MODULE_WEIGHT = {"q_proj": "Wq", "k_proj": "Wk", "v_proj": "Wv", "o_proj": "Wo", "gate_proj": "Wg",
                  "up_proj": "Wu", "down_proj": "Wd"}


def _current(module: str, W: np.ndarray, P_this: Dict, P_hat) -> Tuple[str, Dict]:
    name = _MODULE_WEIGHT[module]
    P_cur = dict(P_this if P_hat is None else P_hat)
    P_cur[name] = np.asarray(W, dtype=np.float64)
    return name, P_cur


def sliding_window_module(module: str, W: np.ndarray, x: np.ndarray, P_this: Dict, P_next: Dict, alpha: float,
                          F_this: np.ndarray, F_next: np.ndarray, x_hat=None, P_hat=None):
    """The exact two-block sliding-window loss of any linear module of block l
    and its gradient with respect to that module's weight.

    x: block l's input (S, L, d); P_this: block l with its reference (full
    precision) weights; W replaces the module's weight.  Block l's output is
    h = B_l(x̂; Ŵ) and its reference h* = B_l(x; W0); the loss is
      alpha (1/2T) sum_t Δh_t^T F_this Δh_t
        + (1 - alpha) (1/2T) sum_t (B_{l+1}(h)_t - B_{l+1}(h*)_t)^T F_next (...),
    Δh = h - h*, both terms back-propagated through block l to W.

    The current pass (Sec. 4.3: the surrogate is evaluated by a forward pass
    through the current transformer block; Eq. fisher_loss: Δy_t = y_t - y*_t)
    takes x_hat, block l's input in the model quantized so far (the
    perturbed x̂ of Sec. 1), and P_hat, block l's weights with the modules
    quantized so far; both default to the reference (x, P_this).  W
    replaces the module's weight in P_hat."""
    name, P_cur = _current(module, W, P_this, P_hat)
    h_ref, _ = block_forward(x, P_this)
    h, cache = block_forward(x if x_hat is None else x_hat, P_cur)
    dh_ = h - h_ref
    T = x.shape[0] * x.shape[1]
    l_this = 0.5 * float(np.sum((dh_ @ F_this) * dh_)) / T
    l_next, g_next = next_block_loss(h_ref, dh_, P_next, F_next)
    g_h = alpha * (dh_ @ F_this) / T + (1.0 - alpha) * g_next
    _, grads = block_vjp(cache, g_h)
    return alpha * l_this + (1.0 - alpha) * l_next, grads[name]


# ---------------------------------------------------------------------------
# The final block: the true KL divergence against the LM head.


def head_params(rng: np.random.Generator, d: int, V: int, scale: float = 1.0) -> Dict[str, np.ndarray]:
    """Random fp64 final norm and LM head (W_h ~ N(0, scale^2 / d), V x d)."""
    return {"gf": 1.0 + 0.1 * rng.standard_normal(d), "Wh": rng.standard_normal((V, d)) * scale / np.sqrt(d)}


def head_logits(h: np.ndarray, head: Dict):
    """z = RMSNorm(h; g_f) W_h^T for h of shape (S, L, d); returns (z, cache)."""
    u, r = _rms(h, head["gf"])
    return u @ head["Wh"].T, (h, r)


def _head_vjp(hc, head, gz):
    h, r = hc
    gh, _ = _rms_vjp(h, head["gf"], r, gz @ head["Wh"])
    return gh


def _log_softmax(z):
    z = z - z.max(axis=-1, keepdims=True)
    return z - np.log(np.sum(np.exp(z), axis=-1, keepdims=True))


def kl_logits(z_ref: np.ndarray, z: np.ndarray) -> np.ndarray:
    """KL(softmax(z_ref) || softmax(z)) over the last axis, one value per token."""
    lp, lq = _log_softmax(z_ref), _log_softmax(z)
    return np.sum(np.exp(lp) * (lp - lq), axis=-1)


def kl_head_loss(h_ref: np.ndarray, dh_: np.ndarray, head: Dict):
    """L = (1/T) sum_t KL(p_t || q_t) with p from the reference block output
    h* and q from h* + Δh, and its gradient with respect to Δh.  The gradient
    of KL(p || softmax(z)) in z is softmax(z) - p."""
    z0, _ = head_logits(h_ref, head)
    z1, hc = head_logits(h_ref + dh_, head)
    T = h_ref.shape[0] * h_ref.shape[1]
    loss = float(np.sum(kl_logits(z0, z1))) / T
    gz = (np.exp(_log_softmax(z1)) - np.exp(_log_softmax(z0))) / T
    return loss, _head_vjp(hc, head, gz)


def nll_scores(h_ref: np.ndarray, head: Dict, labels: np.ndarray) -> np.ndarray:
    """g_t = the gradient in y_t of -log p(label_t | y_t) at the reference
    output (S, L, d); labels (S, L) are integers in [0, V)."""
    z, hc = head_logits(h_ref, head)
    p = np.exp(_log_softmax(z))
    onehot = np.zeros_like(p)
    np.put_along_axis(onehot, np.asarray(labels)[..., None], 1.0, axis=-1)
    return _head_vjp(hc, head, p - onehot)


def fisher_sampled(h_ref: np.ndarray, head: Dict, labels: np.ndarray) -> np.ndarray:
    """Eq. fisher_full: F = (1/T) sum_t g_t g_t^T with one label per token
    drawn from the reference distribution p_t (the draw is passed in)."""
    g = nll_scores(h_ref, head, labels)
    g = g.reshape(-1, g.shape[-1])
    return g.T @ g / g.shape[0]


def fisher_tokens(h_ref: np.ndarray, head: Dict) -> np.ndarray:
    """The per-token Fisher as the exact expectation over the label:
    F_t = sum_v p_t(v) g_t(v) g_t(v)^T, shape (S, L, d, d).  Its token mean is
    the expectation of fisher_sampled over the draw."""
    z, _ = head_logits(h_ref, head)
    p = np.exp(_log_softmax(z))
    S, L, d = h_ref.shape
    F = np.zeros((S, L, d, d))
    for v in range(p.shape[-1]):
        g = nll_scores(h_ref, head, np.full((S, L), v))
        F += p[..., v, None, None] * g[..., :, None] * g[..., None, :]
    return F


def kl_final_module(module: str, W: np.ndarray, x: np.ndarray, P_this: Dict, head: Dict, x_hat=None, P_hat=None):
    """The final block's loss for any linear module: the true KL at the LM
    head between the reference block output and the current one (input
    x_hat, weights P_hat with W in place of the module's weight; both default
    to the reference, as in sliding_window_module), and its gradient with
    respect to W."""
    name, P_cur = _current(module, W, P_this, P_hat)
    h_ref, _ = block_forward(x, P_this)
    h, cache = block_forward(x if x_hat is None else x_hat, P_cur)
    loss, g_h = kl_head_loss(h_ref, h - h_ref, head)
    _, grads = block_vjp(cache, g_h)
    return loss, grads[name]


# ---------------------------------------------------------------------------
# The sweep's Block-GD step on these losses (realq_sweep's gradient_fn).

_MODULE_INPUT = {"q_proj": "a", "k_proj": "a", "v_proj": "a", "o_proj": "o", "gate_proj": "b", "up_proj": "b",
                 "down_proj": "m"}


def module_inputs(module: str, x: np.ndarray, P: Dict) -> np.ndarray:
    """The inputs of a module of block l with input x and weights P, as the
    (S L) x n token matrix whose second moment is the module's OBS Hessian
    (in the sequential pipeline: the current pass's x̂ and weights)."""
    _, cache = block_forward(x, P)
    a = cache[_MODULE_INPUT[module]]
    return a.reshape(-1, a.shape[-1])


def _minibatch(x, k):
    """Mini-batch k of a rotation: x itself when it is one array, else
    x[k mod len(x)]."""
    if x is None or isinstance(x, np.ndarray):
        return x
    return x[k % len(x)]


def window_gradient_fn(module: str, x, P_this: Dict, P_next: Dict, F_this: np.ndarray, F_next: np.ndarray,
                       x_hat=None, P_hat=None):
    """(W, alpha, k) -> (loss, gradient) of the exact two-block window for
    the Block-GD step of the module's sweep (alpha is the step's blend
    weight).  x (and x_hat) are block l's inputs, or a list of calibration
    mini-batches of them, step k taking mini-batch k mod their number."""
    def fn(W, alpha, k=0):
        return sliding_window_module(module, W, _minibatch(x, k), P_this, P_next, alpha, F_this, F_next,
                                     _minibatch(x_hat, k), P_hat)
    return fn


def kl_gradient_fn(module: str, x, P_this: Dict, head: Dict, x_hat=None, P_hat=None):
    """(W, alpha, k) -> (loss, gradient) of the final block's KL at the LM
    head (no window: alpha is not used; x, x_hat and k as in
    window_gradient_fn)."""
    def fn(W, alpha, k=0):
        return kl_final_module(module, W, _minibatch(x, k), P_this, head, _minibatch(x_hat, k), P_hat)
    return fn


# ---------------------------------------------------------------------------
# Alg. 1's loop over the linear modules of one decoder block with the exact
# losses.

MODULES = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")


def quantize_block(x: np.ndarray, P_this: Dict, *, x_hat: Optional[np.ndarray] = None, P_next: Optional[Dict] = None,
                   F_this: Optional[np.ndarray] = None, F_next: Optional[np.ndarray] = None,
                   head: Optional[Dict] = None, lr: float, steps_per_block: int = 1, optimizer: str = "adam",
                   bits: int = 4, group_size: int = 128, block_size: int = 128, damp_frac: float = 0.01,
                   modules: Sequence[str] = MODULES, follow: Optional[Dict[str, Dict]] = None):
    """Quantize the linear modules of block l one after another (Alg. 1: for
    each linear module, the column sweep with a Block-GD step after every
    column block), each against the exact two-block window (P_next, F_this,
    F_next given) or, for the last block, the true KL at the LM head (head
    given).

    x: block l's full-precision input; x_hat: its input in the model
    quantized so far (default x).  The current weights start at P_this; as
    each module finishes, its dequantized weights replace it there, so the
    next module's current pass, OBS Hessian (the second moment of its inputs
    in that pass) and loss see every module quantized before it.  b_global
    runs over the column blocks of all the block's modules, B_total being
    their sum (Eq. slide_window; Alg. 1's note on b_global).  follow maps a
    module to the rounding decisions of another run that its sweep takes at
    rounding ties (realq_sweep's follow).  Returns the sweep result of every
    module and the final current weights."""
    x_hat = x if x_hat is None else x_hat
    P_hat = dict(P_this)
    nbs = {}
    for module in modules:
        n = P_this[_MODULE_WEIGHT[module]].shape[1]
        nbs[module] = -(-n // block_size)
    B_total = sum(nbs.values())
    b_start = 1
    out = {}
    for module in modules:
        name = _MODULE_WEIGHT[module]
        X = module_inputs(module, x_hat, P_hat)
        H_sum, T = _sweep.hessian_sum([X])
        cur = dict(P_hat)
        if head is not None:
            fn = kl_gradient_fn(module, x, P_this, head, x_hat, cur)
        else:
            fn = window_gradient_fn(module, x, P_this, P_next, F_this, F_next, x_hat, cur)
        bgd = {"lr": lr, "steps_per_block": steps_per_block, "optimizer": optimizer, "b_global_start": b_start,
               "B_total": B_total, "gradient_fn": fn}
        res = _sweep.realq_sweep(P_this[name], H_sum, T, bits=bits, group_size=group_size, block_size=block_size,
                                 damp_frac=damp_frac, bgd=bgd, follow=(follow or {}).get(module))
        P_hat[name] = res["deq"]
        out[module] = res
        b_start += nbs[module]
    return out, P_hat


def quantize_model(x: np.ndarray, blocks: Sequence[Dict], fishers: Sequence[np.ndarray], head: Dict, *,
                   lr_final: float, follow: Optional[Sequence[Dict[str, Dict]]] = None, **kw):
    """Alg. 1's outer loop (Stage 1) over a stack of L decoder blocks: block
    l is quantized with quantize_block against the exact two-block window
    with block l+1 (F^(l), F^(l+1) its aggregated Fishers) or, for the last
    block, the KL at the LM head, at the learning rate of the reverse-cosine
    schedule over blocks (eta_l from 0.01 eta_final up to eta_final).  The
    full-precision input of block l+1 is block l's full-precision output; its
    input in the model quantized so far is block l's output with its
    quantized weights on its own such input.  follow: per block, the
    quantize_block follow of that block.  kw go to quantize_block.  Returns
    each block's module results and its quantized weights."""
    L = len(blocks)
    x_ref, x_hat = x, x
    out = []
    for l, P in enumerate(blocks):
        last = l == L - 1
        lr = _sweep.reverse_cosine_lr(l + 1, L, lr_final)
        res, P_hat = quantize_block(x_ref, P, x_hat=x_hat, P_next=None if last else blocks[l + 1],
                                    F_this=fishers[l], F_next=None if last else fishers[l + 1],
                                    head=head if last else None, lr=lr,
                                    follow=None if follow is None else follow[l], **kw)
        out.append((res, P_hat))
        x_ref = block_forward(x_ref, P)[0]
        x_hat = block_forward(x_hat, P_hat)[0]
    return out
