"""Pins of the fp64 decoder block and of the exact two-block sliding window
(oracle/block.py): central finite differences of every hand-written
derivative, structural invariants of the attention, and the reduction of the
exact window to the layer-level one when the next block is the identity."""
import numpy as np
import pytest

import oracle
from oracle import block as ob


def _tiny(seed=0, d=16, H=4, Hkv=2, dh=4, f=24, S=2, L=5):
    r = np.random.default_rng(seed)
    P = ob.block_params(r, d, H, Hkv, dh, f, scale=0.8)
    x = r.standard_normal((S, L, d))
    return r, P, x


def test_block_vjp_matches_finite_differences():
    r, P, x = _tiny(1)
    y, cache = ob.block_forward(x, P)
    c = r.standard_normal(y.shape)
    gx, gp = ob.block_vjp(cache, c)

    def loss(xx, PP):
        return float(np.sum(ob.block_forward(xx, PP)[0] * c))

    h = 1e-6
    for idx in [(0, 0, 0), (1, 4, 7), (0, 2, 15), (1, 0, 3)]:
        e = np.zeros_like(x)
        e[idx] = h
        fd = (loss(x + e, P) - loss(x - e, P)) / (2 * h)
        assert abs(fd - gx[idx]) <= 1e-6 * max(1.0, abs(fd)), (idx, fd, gx[idx])
    for name in ("Wq", "Wk", "Wv", "Wo", "Wg", "Wu", "Wd", "g1", "g2"):
        for k in range(3):
            idx = tuple(int(r.integers(0, s)) for s in P[name].shape)
            Pp = dict(P)
            Pm = dict(P)
            Pp[name] = P[name].copy()
            Pm[name] = P[name].copy()
            Pp[name][idx] += h
            Pm[name][idx] -= h
            fd = (loss(x, Pp) - loss(x, Pm)) / (2 * h)
            assert abs(fd - gp[name][idx]) <= 1e-6 * max(1.0, abs(fd)), (name, idx, fd, gp[name][idx])


def test_attention_is_causal_within_each_sequence():
    r, P, x = _tiny(2)
    y0, _ = ob.block_forward(x, P)
    x1 = x.copy()
    x1[1, 2] += r.standard_normal(x.shape[2])
    y1, _ = ob.block_forward(x1, P)
    changed = np.abs(y1 - y0).max(axis=2) > 0
    assert not changed[0].any()                      # the other sequence
    assert not changed[1, :2].any()                  # earlier positions
    assert changed[1, 2:].all()                      # the token and every later one


def test_rotary_scores_depend_on_the_position_difference():
    r = np.random.default_rng(3)
    dh, L = 8, 12
    q = r.standard_normal((1, L, 1, dh))
    k = r.standard_normal((1, L, 1, dh))
    cos, sin = ob._rope_tables(L, dh)
    # the same two vectors placed at (i, j) and at (i + 4, j + 4)
    qs = np.repeat(q[:, :1], L, axis=1)
    ks = np.repeat(k[:, :1], L, axis=1)
    qr, kr = ob._rope(qs, cos, sin), ob._rope(ks, cos, sin)
    s1 = float(np.sum(qr[0, 5, 0] * kr[0, 2, 0]))
    s2 = float(np.sum(qr[0, 9, 0] * kr[0, 6, 0]))
    assert abs(s1 - s2) <= 1e-12 * max(1.0, abs(s1))
    # and the rotation is orthogonal (its transpose undoes it)
    assert np.allclose(ob._rope_t(ob._rope(q, cos, sin), cos, sin), q, atol=1e-14)


def _down_case(seed, zero_next):
    r = np.random.default_rng(seed)
    S, L, n, d = 2, 6, 12, 16
    P = ob.block_params(r, d, 4, 2, 4, 24, scale=0.8)
    if zero_next:
        P["Wo"] = np.zeros_like(P["Wo"])
        P["Wd"] = np.zeros_like(P["Wd"])
    X = r.standard_normal((S, L, n))
    R = r.standard_normal((S, L, d))
    W0 = r.standard_normal((d, n)) * 0.1
    W = W0 + r.standard_normal((d, n)) * 0.02
    Z = r.standard_normal((d, 3))
    F = 0.5 * np.eye(d) + Z @ Z.T / 6
    Z2 = r.standard_normal((d, 3))
    Fn = 0.5 * np.eye(d) + Z2 @ Z2.T / 6
    return X, R, W0, W, F, Fn, P


def test_identity_next_block_reduces_to_the_layer_level_window():
    # with its output projections zero the next block is the identity, so its
    # Fisher loss is the layer-level one with F' = F_next
    X, R, W0, W, F, Fn, P = _down_case(4, True)
    alpha = 0.3
    loss, grad = ob.sliding_window_down(W, W0, X, R, alpha, F, Fn, P)
    Xf = X.reshape(-1, X.shape[2])
    Hbar = Xf.T @ Xf / Xf.shape[0]
    Feff = alpha * F + (1 - alpha) * Fn
    np.testing.assert_allclose(grad, oracle.gradient(W, W0, Hbar, None, Feff), rtol=1e-11, atol=1e-14)
    assert abs(loss - oracle.surrogate_moment(W, W0, Hbar, Feff)) <= 1e-12 * abs(loss)


@pytest.mark.parametrize("alpha", [1.0, 0.4, 0.0])
def test_sliding_window_gradient_matches_finite_differences(alpha):
    X, R, W0, W, F, Fn, P = _down_case(5, False)
    _, grad = ob.sliding_window_down(W, W0, X, R, alpha, F, Fn, P)
    h = 1e-6
    r = np.random.default_rng(6)
    for _ in range(6):
        i, j = int(r.integers(0, W.shape[0])), int(r.integers(0, W.shape[1]))
        E = np.zeros_like(W)
        E[i, j] = h
        lp, _ = ob.sliding_window_down(W + E, W0, X, R, alpha, F, Fn, P)
        lm, _ = ob.sliding_window_down(W - E, W0, X, R, alpha, F, Fn, P)
        fd = (lp - lm) / (2 * h)
        assert abs(fd - grad[i, j]) <= 1e-6 * max(1e-3, abs(fd)), (i, j, fd, grad[i, j])


def test_next_block_loss_is_second_order_in_the_perturbation():
    # B(h + e u) - B(h) = e J u + O(e^2): the loss scales as e^2 for small e
    X, R, W0, W, F, Fn, P = _down_case(7, False)
    h = R + X @ W0.T
    u = np.random.default_rng(8).standard_normal(h.shape)
    l1, _ = ob.next_block_loss(h, 1e-3 * u, P, Fn)
    l2, _ = ob.next_block_loss(h, 2e-3 * u, P, Fn)
    assert abs(l2 / l1 - 4.0) < 1e-2


def _module_case(seed):
    r = np.random.default_rng(seed)
    d = 16
    P = ob.block_params(r, d, 4, 2, 4, 24, scale=0.8)
    Pn = ob.block_params(r, d, 4, 2, 4, 24, scale=0.8)
    x = r.standard_normal((2, 5, d))
    Z = r.standard_normal((d, 3))
    F = 0.5 * np.eye(d) + Z @ Z.T / 6
    Z2 = r.standard_normal((d, 3))
    Fn = 0.5 * np.eye(d) + Z2 @ Z2.T / 6
    return r, P, Pn, x, F, Fn


@pytest.mark.parametrize("module", ["q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj"])
def test_every_module_window_gradient_matches_finite_differences(module):
    r, P, Pn, x, F, Fn = _module_case(9)
    name = ob._MODULE_WEIGHT[module]
    W = P[name] + r.standard_normal(P[name].shape) * 0.05
    loss, grad = ob.sliding_window_module(module, W, x, P, Pn, 0.6, F, Fn)
    assert loss > 0
    h = 1e-6
    for _ in range(4):
        i, j = int(r.integers(0, W.shape[0])), int(r.integers(0, W.shape[1]))
        E = np.zeros_like(W)
        E[i, j] = h
        lp, _ = ob.sliding_window_module(module, W + E, x, P, Pn, 0.6, F, Fn)
        lm, _ = ob.sliding_window_module(module, W - E, x, P, Pn, 0.6, F, Fn)
        fd = (lp - lm) / (2 * h)
        assert abs(fd - grad[i, j]) <= 1e-6 * max(1e-3, abs(fd)), (module, i, j, fd, grad[i, j])


def test_module_window_agrees_with_the_down_proj_form():
    # for down_proj the block-level statement equals the module-level one
    # (h = r + W_d m, with m the SwiGLU product and r the rest of the block)
    r, P, Pn, x, F, Fn = _module_case(10)
    W = P["Wd"] + r.standard_normal(P["Wd"].shape) * 0.05
    loss, grad = ob.sliding_window_module("down_proj", W, x, P, Pn, 0.35, F, Fn)
    y, cache = ob.block_forward(x, P)
    m = cache["m"]
    R = y - m @ P["Wd"].T
    loss2, grad2 = ob.sliding_window_down(W, P["Wd"], m, R, 0.35, F, Fn, Pn)
    assert abs(loss - loss2) <= 1e-12 * abs(loss)
    np.testing.assert_allclose(grad, grad2, rtol=1e-10, atol=1e-15)


# --- the current pass: perturbed input, modules quantized so far -----------

def _current_pass(r, P, x, skip):
    # block l's input in the model quantized so far, and its weights with
    # every other module moved off the reference
    x_hat = x + 0.1 * r.standard_normal(x.shape)
    P_hat = dict(P)
    for k in ("Wq", "Wk", "Wv", "Wo", "Wg", "Wu", "Wd"):
        if k != skip:
            P_hat[k] = P[k] + 0.03 * r.standard_normal(P[k].shape)
    return x_hat, P_hat


@pytest.mark.parametrize("module", ["q_proj", "o_proj", "up_proj", "down_proj"])
def test_current_pass_window_gradient_matches_finite_differences(module):
    r, P, Pn, x, F, Fn = _module_case(21)
    name = ob._MODULE_WEIGHT[module]
    x_hat, P_hat = _current_pass(r, P, x, name)
    W = P[name] + r.standard_normal(P[name].shape) * 0.05
    args = (x, P, Pn, 0.6, F, Fn, x_hat, P_hat)
    loss, grad = ob.sliding_window_module(module, W, *args)
    # at the module's reference weight the loss is still positive: the input
    # and the other modules differ from the reference
    assert ob.sliding_window_module(module, P[name], *args)[0] > 0
    e = 1e-6
    for _ in range(4):
        i, j = int(r.integers(0, W.shape[0])), int(r.integers(0, W.shape[1]))
        E = np.zeros_like(W)
        E[i, j] = e
        fd = (ob.sliding_window_module(module, W + E, *args)[0] -
              ob.sliding_window_module(module, W - E, *args)[0]) / (2 * e)
        assert abs(fd - grad[i, j]) <= 1e-6 * max(1e-3, abs(fd)), (module, i, j, fd, grad[i, j])


def test_current_pass_agrees_with_the_down_proj_form():
    # Δh = (R̂ + X̂ Wᵀ) - (R + X W0ᵀ): the down_proj form from the two passes'
    # cached SwiGLU products and residuals against the block-level statement
    r, P, Pn, x, F, Fn = _module_case(22)
    x_hat, P_hat = _current_pass(r, P, x, "Wd")
    W = P["Wd"] + r.standard_normal(P["Wd"].shape) * 0.05
    loss, grad = ob.sliding_window_module("down_proj", W, x, P, Pn, 0.35, F, Fn, x_hat, P_hat)
    y, cache = ob.block_forward(x, P)
    y_hat, cache_hat = ob.block_forward(x_hat, P_hat)
    R = y - cache["m"] @ P["Wd"].T
    R_hat = y_hat - cache_hat["m"] @ P_hat["Wd"].T
    loss2, grad2 = ob.sliding_window_down(W, P["Wd"], cache["m"], R, 0.35, F, Fn, Pn, cache_hat["m"], R_hat)
    assert abs(loss - loss2) <= 1e-10 * abs(loss)
    np.testing.assert_allclose(grad, grad2, rtol=1e-8, atol=1e-12 * np.abs(grad).max())


@pytest.mark.parametrize("module", ["k_proj", "gate_proj"])
def test_current_pass_kl_gradient_matches_finite_differences(module):
    r, P, _, x, _, _ = _module_case(23)
    head = ob.head_params(r, x.shape[2], 11, scale=1.5)
    name = ob._MODULE_WEIGHT[module]
    x_hat, P_hat = _current_pass(r, P, x, name)
    W = P[name] + r.standard_normal(P[name].shape) * 0.05
    loss, grad = ob.kl_final_module(module, W, x, P, head, x_hat, P_hat)
    assert loss > 0
    e = 1e-6
    for _ in range(4):
        i, j = int(r.integers(0, W.shape[0])), int(r.integers(0, W.shape[1]))
        E = np.zeros_like(W)
        E[i, j] = e
        fd = (ob.kl_final_module(module, W + E, x, P, head, x_hat, P_hat)[0] -
              ob.kl_final_module(module, W - E, x, P, head, x_hat, P_hat)[0]) / (2 * e)
        assert abs(fd - grad[i, j]) <= 1e-6 * max(1e-4, abs(fd)), (module, i, j, fd, grad[i, j])


def test_current_pass_kl_agrees_with_the_down_proj_form():
    # down_proj's KL gradient is the head's gradient in Δh times the current
    # pass's SwiGLU product, Σ_t g_t m̂_tᵀ, with no backward through block l
    r, P, _, x, _, _ = _module_case(24)
    head = ob.head_params(r, x.shape[2], 11, scale=1.5)
    x_hat, P_hat = _current_pass(r, P, x, "Wd")
    W = P["Wd"] + r.standard_normal(P["Wd"].shape) * 0.05
    loss, grad = ob.kl_final_module("down_proj", W, x, P, head, x_hat, P_hat)
    y, _ = ob.block_forward(x, P)
    y_hat, cache_hat = ob.block_forward(x_hat, P_hat)
    m_hat = cache_hat["m"]
    h = y_hat + m_hat @ (W - P_hat["Wd"]).T
    loss2, g_h = ob.kl_head_loss(y, h - y, head)
    assert abs(loss - loss2) <= 1e-10 * abs(loss)
    np.testing.assert_allclose(grad, np.einsum("sti,stj->ij", g_h, m_hat), rtol=1e-8,
                               atol=1e-12 * np.abs(grad).max())


# --- the final block: the true KL at the LM head ---------------------------

def _head_case(seed, d=6, V=7, S=2, L=3):
    r = np.random.default_rng(seed)
    head = ob.head_params(r, d, V, scale=1.5)
    h = r.standard_normal((S, L, d))
    return r, head, h


def test_kl_of_two_hand_computed_distributions():
    # p = softmax(0, ln 3) = (1/4, 3/4), q = softmax(0, 0) = (1/2, 1/2)
    z_ref = np.array([[0.0, np.log(3.0)]])
    z = np.zeros((1, 2))
    want = 0.25 * np.log(0.5) + 0.75 * np.log(1.5)
    assert abs(ob.kl_logits(z_ref, z)[0] - want) <= 1e-15
    # a constant shift of either side's logits changes neither distribution
    assert abs(ob.kl_logits(z_ref + 7.0, z - 3.0)[0] - want) <= 1e-14
    assert ob.kl_logits(z_ref, z_ref)[0] == 0.0


def test_kl_head_loss_is_zero_with_a_zero_gradient_at_the_reference():
    r, head, h = _head_case(11)
    loss, g = ob.kl_head_loss(h, np.zeros_like(h), head)
    assert loss == 0.0 and np.abs(g).max() == 0.0
    loss, _ = ob.kl_head_loss(h, 0.3 * r.standard_normal(h.shape), head)
    assert loss > 0.0


def test_kl_head_gradient_matches_finite_differences():
    r, head, h = _head_case(12)
    dh0 = 0.4 * r.standard_normal(h.shape)
    _, g = ob.kl_head_loss(h, dh0, head)
    e = 1e-6
    for idx in [(0, 0, 0), (1, 2, 5), (0, 1, 3), (1, 0, 1)]:
        E = np.zeros_like(h)
        E[idx] = e
        fd = (ob.kl_head_loss(h, dh0 + E, head)[0] - ob.kl_head_loss(h, dh0 - E, head)[0]) / (2 * e)
        assert abs(fd - g[idx]) <= 1e-7 * max(1e-3, abs(fd)), (idx, fd, g[idx])


def test_fisher_is_the_kl_hessian_at_the_reference_output():
    # at h* the first-order term of KL vanishes and its Hessian in y_t is the
    # expected outer product of the NLL score (Eq. taylor_expansion and the
    # Fisher-Hessian identity); per token, (1/T) F_t u_t is the derivative of
    # the KL gradient along u
    r, head, h = _head_case(13)
    S, L, d = h.shape
    F = ob.fisher_tokens(h, head)
    u = r.standard_normal(h.shape)
    e = 1e-5
    gp = ob.kl_head_loss(h, e * u, head)[1]
    gm = ob.kl_head_loss(h, -e * u, head)[1]
    hv = (gp - gm) / (2 * e)
    want = np.einsum("stij,stj->sti", F, u) / (S * L)
    np.testing.assert_allclose(hv, want, rtol=1e-6, atol=1e-9 * np.abs(want).max())
    # and the loss itself: KL(h* + e u) / e^2 -> (1/2T) sum_t u_t^T F_t u_t
    quad = 0.5 * float(np.einsum("sti,stij,stj->", u, F, u)) / (S * L)
    r1 = ob.kl_head_loss(h, 2e-3 * u, head)[0] / 4e-6
    r2 = ob.kl_head_loss(h, 1e-3 * u, head)[0] / 1e-6
    assert abs((2 * r2 - r1) - quad) <= 1e-5 * quad        # Richardson: O(e^2) left
    # each F_t is symmetric positive semidefinite with the head's null
    # direction: the score is orthogonal to h_t (RMSNorm is scale-free up to eps)
    assert np.allclose(F, np.swapaxes(F, -1, -2), atol=1e-15)
    assert np.linalg.eigvalsh(F).min() > -1e-12
    assert np.abs(np.einsum("stij,stj->sti", F, h)).max() <= 1e-5 * np.abs(F).max() * np.abs(h).max()


def test_sampled_fisher_averages_to_the_exact_expectation():
    # Eq. fisher_full with labels drawn from p_t: its mean over many draws is
    # the token mean of the per-token expectation (fixed seed: deterministic)
    r, head, h = _head_case(14, d=4, V=5)
    z, _ = ob.head_logits(h, head)
    p = np.exp(z - z.max(axis=-1, keepdims=True))
    p /= p.sum(axis=-1, keepdims=True)
    want = ob.fisher_tokens(h, head).mean(axis=(0, 1))
    K = 4000
    cdf = np.cumsum(p, axis=-1)
    draws = []
    for _ in range(K):
        lab = (r.random(p.shape[:-1])[..., None] > cdf).sum(axis=-1)
        draws.append(ob.fisher_sampled(h, head, np.minimum(lab, p.shape[-1] - 1)))
    draws = np.array(draws)
    se = draws.std(axis=0) / np.sqrt(K)
    assert np.all(np.abs(draws.mean(axis=0) - want) <= 5 * se + 1e-12)
    # the test has the power to see a wrong expectation: labels drawn
    # uniformly instead of from p_t fall outside the bound
    V = p.shape[-1]
    gs = [ob.nll_scores(h, head, np.full(h.shape[:2], v)) for v in range(V)]
    uniform = sum(np.einsum("sti,stj->ij", g, g) for g in gs) / (V * h.shape[0] * h.shape[1])
    assert not np.all(np.abs(draws.mean(axis=0) - uniform) <= 5 * se + 1e-12)


@pytest.mark.parametrize("module", ["q_proj", "v_proj", "gate_proj", "down_proj"])
def test_final_block_kl_gradient_matches_finite_differences(module):
    r, P, _, x, _, _ = _module_case(15)
    head = ob.head_params(r, x.shape[2], 11, scale=1.5)
    name = ob._MODULE_WEIGHT[module]
    l0, g0 = ob.kl_final_module(module, P[name], x, P, head)
    assert l0 == 0.0 and np.abs(g0).max() == 0.0
    W = P[name] + r.standard_normal(P[name].shape) * 0.05
    loss, grad = ob.kl_final_module(module, W, x, P, head)
    assert loss > 0
    e = 1e-6
    for _ in range(4):
        i, j = int(r.integers(0, W.shape[0])), int(r.integers(0, W.shape[1]))
        E = np.zeros_like(W)
        E[i, j] = e
        fd = (ob.kl_final_module(module, W + E, x, P, head)[0] - ob.kl_final_module(module, W - E, x, P, head)[0]) / (2 * e)
        assert abs(fd - grad[i, j]) <= 1e-6 * max(1e-4, abs(fd)), (module, i, j, fd, grad[i, j])


# --- the sweep's Block-GD step on the exact losses ---------------------------

def _spd(r, d, k=3):
    Z = r.standard_normal((d, k))
    return 0.5 * np.eye(d) + Z @ Z.T / (2 * k)


def test_exact_window_sweep_reduces_to_the_layer_level_sweep():
    # down_proj with an identity next block: the exact window's gradient is
    # F_eff ΔW H̄ and its loss the layer-level surrogate, so the whole sweep
    # (codes, weights, per-block losses) is the layer-level one
    r = np.random.default_rng(20)
    d, f = 16, 64
    P = ob.block_params(r, d, 4, 2, 4, f, scale=0.8)
    Pn = ob.block_params(r, d, 4, 2, 4, f, scale=0.8)
    Pn["Wo"] = np.zeros_like(Pn["Wo"])
    Pn["Wd"] = np.zeros_like(Pn["Wd"])
    x = r.standard_normal((4, 8, d))
    F, Fn = _spd(r, d), _spd(r, d)
    Xm = ob.module_inputs("down_proj", x, P)
    H_sum, T = Xm.T @ Xm, Xm.shape[0]
    bgd = dict(lr=1e-3, steps_per_block=1, b_global_start=2, B_total=6)
    kw = dict(block_size=16, group_size=16)
    ref = oracle.realq_sweep(P["Wd"], H_sum, T, bgd=bgd, F=F, F_next=Fn, **kw)
    ex = oracle.realq_sweep(P["Wd"], H_sum, T, bgd=dict(bgd, gradient_fn=ob.window_gradient_fn("down_proj", x, P, Pn, F, Fn)),
                            **kw)
    assert np.array_equal(ref["codes"], ex["codes"])
    np.testing.assert_allclose(ex["deq"], ref["deq"], rtol=1e-9, atol=1e-12)
    assert len(ex["block_loss"]) == 3 and ex["adam_t"] == ref["adam_t"] == 3
    for (b1, a1, bf1, af1), (b2, a2, bf2, af2) in zip(ref["block_loss"], ex["block_loss"]):
        assert (b1, a1) == (b2, a2)
        assert abs(bf1 - bf2) <= 1e-10 * bf1 and abs(af1 - af2) <= 1e-10 * af1


@pytest.mark.parametrize("module", ["q_proj", "v_proj", "gate_proj"])
def test_exact_window_sweep_descends_with_small_sgd_steps(module):
    # a small enough gradient step lowers a smooth loss: every block's loss
    # after its Block-GD step is below the loss before it
    r = np.random.default_rng(21)
    d, f = 32, 48
    P = ob.block_params(r, d, 4, 2, 8, f, scale=0.8)
    Pn = ob.block_params(r, d, 4, 2, 8, f, scale=0.8)
    x = r.standard_normal((2, 8, d))
    F, Fn = _spd(r, d), _spd(r, d)
    name = ob._MODULE_WEIGHT[module]
    Xm = ob.module_inputs(module, x, P)
    bgd = dict(optimizer="sgd", lr=1e-2, steps_per_block=1, b_global_start=1, B_total=4,
               gradient_fn=ob.window_gradient_fn(module, x, P, Pn, F, Fn))
    out = oracle.realq_sweep(P[name], Xm.T @ Xm, Xm.shape[0], block_size=8, group_size=8, bgd=bgd)
    assert len(out["block_loss"]) == P[name].shape[1] // 8 - 1
    for b, alpha, before, after in out["block_loss"]:
        assert abs(alpha - (1.0 - b / 3.0)) <= 1e-15
        assert 0.0 < after < before, (module, b, before, after)


def test_final_block_kl_sweep_descends_with_small_sgd_steps():
    r = np.random.default_rng(22)
    d, f = 32, 48
    P = ob.block_params(r, d, 4, 2, 8, f, scale=0.8)
    head = ob.head_params(r, d, 40, scale=2.0)
    x = r.standard_normal((2, 8, d))
    Xm = ob.module_inputs("up_proj", x, P)
    bgd = dict(optimizer="sgd", lr=1e-1, steps_per_block=1, b_global_start=1, B_total=1,
               gradient_fn=ob.kl_gradient_fn("up_proj", x, P, head))
    out = oracle.realq_sweep(P["Wu"], Xm.T @ Xm, Xm.shape[0], block_size=8, group_size=8, bgd=bgd)
    assert len(out["block_loss"]) == 3
    for b, alpha, before, after in out["block_loss"]:
        assert 0.0 < after < before, (b, before, after)
    # the Block-GD steps moved the weights: the sweep differs from the plain
    # column sweep on the same Hessian
    plain = oracle.realq_sweep(P["Wu"], Xm.T @ Xm, Xm.shape[0], block_size=8, group_size=8)
    assert np.abs(out["deq"] - plain["deq"]).max() > 0.0


# --- Alg. 1's loop over the block's modules with the exact losses ------------

def _driver_case(seed=31):
    r = np.random.default_rng(seed)
    d, H, Hkv, dh, f, S, L = 32, 4, 2, 8, 48, 2, 24
    P = ob.block_params(r, d, H, Hkv, dh, f, scale=0.8)
    Pn = ob.block_params(r, d, H, Hkv, dh, f, scale=0.8)
    x = r.standard_normal((S, L, d))
    x_hat = x + 0.05 * r.standard_normal(x.shape)
    F, Fn = _spd(r, d), _spd(r, d)
    return r, P, Pn, x, x_hat, F, Fn


def test_block_driver_runs_the_global_block_index_over_all_modules():
    # Eq. slide_window: b_global counts the column blocks of every module of
    # the block in order, B_total is their sum; each recorded step's alpha is
    # 1 - (b_global - 1)/(B_total - 1) (a module's last block takes no step)
    r, P, Pn, x, x_hat, F, Fn = _driver_case()
    out, _ = ob.quantize_block(x, P, x_hat=x_hat, P_next=Pn, F_this=F, F_next=Fn, lr=1e-3, group_size=16,
                               block_size=16)
    widths = {"q_proj": 32, "k_proj": 32, "v_proj": 32, "o_proj": 32, "gate_proj": 32, "up_proj": 32,
              "down_proj": 48}
    B_total = sum(w // 16 for w in widths.values())
    assert B_total == 15
    b_global = 1
    for module in ob.MODULES:
        nb = widths[module] // 16
        got = [a for _, a, _, _ in out[module]["block_loss"]]
        assert got == pytest.approx([1.0 - (b_global + b - 1) / (B_total - 1) for b in range(nb - 1)], abs=1e-15)
        assert out[module]["adam_t"] == nb - 1
        b_global += nb
    assert out["q_proj"]["block_loss"][0][1] == 1.0


def test_block_driver_threads_the_modules_quantized_so_far():
    # o_proj's OBS Hessian and current pass see q, k, v quantized: the
    # driver's o_proj sweep equals one run from those weights by hand
    r, P, Pn, x, x_hat, F, Fn = _driver_case(32)
    kw = dict(lr=1e-3, group_size=16, block_size=16)
    out, P_hat = ob.quantize_block(x, P, x_hat=x_hat, P_next=Pn, F_this=F, F_next=Fn, **kw)
    cur = dict(P)
    for module in ("q_proj", "k_proj", "v_proj"):
        cur[ob._MODULE_WEIGHT[module]] = out[module]["deq"]
        assert not np.allclose(out[module]["deq"], P[ob._MODULE_WEIGHT[module]])
    X = ob.module_inputs("o_proj", x_hat, cur)
    H_sum, T = oracle.hessian_sum([X])
    fn = ob.window_gradient_fn("o_proj", x, P, Pn, F, Fn, x_hat, cur)
    bgd = {"lr": 1e-3, "b_global_start": 7, "B_total": 15, "gradient_fn": fn}
    want = oracle.realq_sweep(P["Wo"], H_sum, T, group_size=16, block_size=16, bgd=bgd)
    assert np.array_equal(out["o_proj"]["codes"], want["codes"])
    np.testing.assert_allclose(out["o_proj"]["deq"], want["deq"], rtol=0, atol=1e-15)
    # and the final current weights are every module's dequantized weights
    for module in ob.MODULES:
        assert P_hat[ob._MODULE_WEIGHT[module]] is out[module]["deq"]


def test_block_driver_with_small_sgd_steps_lowers_every_modules_loss():
    # with small plain gradient steps each block step lowers the exact
    # window's loss (the descent lemma of Sec. 4.3's analysis), module after
    # module through the whole block, and the final block's KL likewise
    r, P, Pn, x, x_hat, F, Fn = _driver_case(33)
    out, _ = ob.quantize_block(x, P, x_hat=x_hat, P_next=Pn, F_this=F, F_next=Fn, lr=0.5, optimizer="sgd",
                               group_size=16, block_size=16)
    head = ob.head_params(r, x.shape[2], 13, scale=1.5)
    out_kl, _ = ob.quantize_block(x, P, x_hat=x_hat, head=head, lr=2.0, optimizer="sgd", group_size=16,
                                  block_size=16)
    for res in list(out.values()) + list(out_kl.values()):
        for _, _, before, after in res["block_loss"]:
            assert after < before, (before, after)


# --- calibration mini-batches of the exact losses (Sec. 4.3) ---------------

def test_minibatch_losses_average_to_the_full_batch_loss():
    # the losses are means over tokens and attention stays within a
    # sequence, so over mini-batches of whole sequences of equal size the
    # mean of the mini-batch losses and gradients is the full batch's
    r, P, Pn, x, x_hat, F, Fn = _driver_case(34)
    x = np.concatenate([x, r.standard_normal(x.shape)], axis=0)            # 4 sequences
    x_hat = x + 0.05 * r.standard_normal(x.shape)
    head = ob.head_params(r, x.shape[2], 13, scale=1.5)
    W = P["Wg"] + 0.05 * r.standard_normal(P["Wg"].shape)
    mb = [x[i:i + 2] for i in (0, 2)]
    mbh = [x_hat[i:i + 2] for i in (0, 2)]
    for full, part in ((ob.window_gradient_fn("gate_proj", x, P, Pn, F, Fn, x_hat),
                        ob.window_gradient_fn("gate_proj", mb, P, Pn, F, Fn, mbh)),
                       (ob.kl_gradient_fn("gate_proj", x, P, head, x_hat),
                        ob.kl_gradient_fn("gate_proj", mb, P, head, mbh))):
        lf, gf = full(W, 0.4)
        parts = [part(W, 0.4, k) for k in range(2)]
        assert parts[0][0] != parts[1][0]
        assert abs(np.mean([p[0] for p in parts]) - lf) <= 1e-12 * abs(lf)
        np.testing.assert_allclose(np.mean([p[1] for p in parts], axis=0), gf, rtol=0,
                                   atol=1e-12 * np.abs(gf).max())


def test_sweep_rotation_over_minibatches_is_a_full_batch_step_to_first_order():
    # K plain gradient steps per block over K mini-batches (the rotation
    # starting at mini-batch 0 for every block when steps_per_block = K) sum
    # to K lr times the full-batch gradient up to O(lr^2): with a small lr the
    # sweep equals the full-batch one with a single step of K lr
    r, P, Pn, x, x_hat, F, Fn = _driver_case(35)
    x = np.concatenate([x, r.standard_normal(x.shape)], axis=0)
    x_hat = x + 0.05 * r.standard_normal(x.shape)
    mb, mbh = [x[i:i + 2] for i in (0, 2)], [x_hat[i:i + 2] for i in (0, 2)]
    X = ob.module_inputs("up_proj", x_hat, P)
    H_sum, T = oracle.hessian_sum([X])
    lr = 1e-3
    kw = dict(group_size=16, block_size=16)
    rot = oracle.realq_sweep(P["Wu"], H_sum, T, bgd={
        "lr": lr, "optimizer": "sgd", "steps_per_block": 2, "B_total": 1,
        "gradient_fn": ob.window_gradient_fn("up_proj", mb, P, Pn, F, Fn, mbh)}, **kw)
    full = oracle.realq_sweep(P["Wu"], H_sum, T, bgd={
        "lr": 2 * lr, "optimizer": "sgd", "steps_per_block": 1, "B_total": 1,
        "gradient_fn": ob.window_gradient_fn("up_proj", x, P, Pn, F, Fn, x_hat)}, **kw)
    first = oracle.realq_sweep(P["Wu"], H_sum, T, bgd={
        "lr": 2 * lr, "optimizer": "sgd", "steps_per_block": 1, "B_total": 1,
        "gradient_fn": ob.window_gradient_fn("up_proj", mb[:1], P, Pn, F, Fn, mbh[:1])}, **kw)
    assert np.array_equal(rot["codes"], full["codes"])
    d_rot = np.abs(rot["deq"] - full["deq"]).max()
    d_first = np.abs(first["deq"] - full["deq"]).max()
    # (the scales are fp32, so an O(lr^2) change of a group's extreme weight
    # can move its scale, and every weight of the group, by one fp32 step)
    assert d_rot <= 1e-6 and d_rot <= 1e-2 * d_first, (d_rot, d_first)


def test_model_loop_feeds_each_block_the_quantized_stack_and_its_schedule():
    # Alg. 1's outer loop: block l+1's perturbed input is the quantized
    # block l's output on its own perturbed input, its reference input the
    # full-precision output; the learning rate follows the reverse-cosine
    # schedule over blocks; the last block takes the KL at the LM head
    r = np.random.default_rng(36)
    d, H, Hkv, dh, f, S, L = 32, 4, 2, 8, 48, 2, 12
    blocks = [ob.block_params(r, d, H, Hkv, dh, f, scale=0.8) for _ in range(3)]
    fishers = [_spd(r, d) for _ in range(3)]
    head = ob.head_params(r, d, 13, scale=1.5)
    x = r.standard_normal((S, L, d))
    kw = dict(group_size=16, block_size=16, optimizer="sgd")
    out = ob.quantize_model(x, blocks, fishers, head, lr_final=0.3, **kw)
    assert len(out) == 3
    # block 2 by hand: its inputs from blocks 0 and 1 as the loop left them
    x1 = ob.block_forward(ob.block_forward(x, blocks[0])[0], blocks[1])[0]
    x1_hat = ob.block_forward(ob.block_forward(x, out[0][1])[0], out[1][1])[0]
    res, _ = ob.quantize_block(x1, blocks[2], x_hat=x1_hat, head=head, lr=0.3, **kw)
    for module in ob.MODULES:
        assert np.array_equal(res[module]["codes"], out[2][0][module]["codes"])
        np.testing.assert_allclose(res[module]["deq"], out[2][0][module]["deq"], rtol=0, atol=1e-15)
    # block 0 at the first rate of the schedule (0.01 lr_final), with the
    # window to block 1
    res0, _ = ob.quantize_block(x, blocks[0], P_next=blocks[1], F_this=fishers[0], F_next=fishers[1], lr=0.003,
                                **kw)
    for module in ob.MODULES:
        np.testing.assert_allclose(res0[module]["deq"], out[0][0][module]["deq"], rtol=0, atol=1e-15)
    # the quantized stack's output is off the reference, and block 1 saw it
    assert not np.allclose(x1, x1_hat)
