"""Parity of the decoder block of the exact two-block sliding window
(realq_block_forward, realq_block_window) with the fp64 oracle
(oracle/block.py: block_forward, next_block_loss), through the C ABI.

Tolerances (fp32 arithmetic, fp32 accumulation over at most max(d, f, L)
unit-scale terms): the forward within 1e-5 of the output's scale; the
window's Δz is the difference of two forward passes about |h|/|Δh| = 10
times larger than it, so the loss and the gradient within 1e-4 of their
scale.  Inputs and parameters are rounded to fp32 first, so that both sides
see the same block.  Collected after the other parity files and before the
no-allocation entry point's test, which runs last."""
import numpy as np
import pytest
import torch

from oracle import block as ob
import paper_2609_00049_gb300 as rq

pytestmark = pytest.mark.gpu

_KEYS = ("g1", "Wq", "Wk", "Wv", "Wo", "g2", "Wg", "Wu", "Wd")

CASES = [
    # (S, L, d, H, Hkv, dh, f): grouped queries over a ragged length; one
    # key/value head per query head; one token per sequence; wide heads; and
    # a case that spans several GEMM tiles and thread blocks in every launch
    (2, 7, 16, 4, 2, 4, 24),
    (3, 5, 24, 3, 3, 8, 40),
    (2, 1, 16, 4, 1, 4, 20),
    (1, 9, 32, 2, 1, 16, 48),
    (4, 96, 256, 8, 2, 32, 704),
]


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_00049_gb300 import build as b
    b.build()
    rq.lib()


def _f32(a):
    return np.asarray(a, dtype=np.float32).astype(np.float64)


def _case(seed, S, L, d, H, Hkv, dh, f):
    r = np.random.default_rng(seed)
    P = ob.block_params(r, d, H, Hkv, dh, f, scale=0.8)
    for k in _KEYS:
        P[k] = _f32(P[k])
    W = {k: torch.from_numpy(P[k].astype(np.float32)).cuda() for k in _KEYS}
    dims = rq.block_dims(d, H, Hkv, dh, f)
    ws = rq.workspace(rq.realq_block_workspace_size(dims, S, L))
    return r, P, W, dims, ws


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


@pytest.mark.parametrize("case", CASES)
def test_block_forward_matches_the_oracle(case):
    S, L, d, H, Hkv, dh, f = case
    r, P, W, dims, ws = _case(1, *case)
    x = _f32(r.standard_normal((S, L, d)))
    want, _ = ob.block_forward(x, P)
    y = torch.empty((S, L, d), dtype=torch.float32, device="cuda")
    rq.realq_block_forward(dims, W, _dev(x), y, ws)
    got = y.cpu().numpy()
    assert np.isfinite(got).all()
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-5 * np.abs(want).max())


@pytest.mark.parametrize("case", CASES)
def test_block_window_matches_the_oracle(case):
    S, L, d, H, Hkv, dh, f = case
    r, P, W, dims, ws = _case(2, *case)
    h = _f32(r.standard_normal((S, L, d)))
    dh_ = _f32(0.1 * r.standard_normal((S, L, d)))
    Z = r.standard_normal((d, 3))
    F = _f32(0.5 * np.eye(d) + Z @ Z.T / 6)
    want_loss, want_g = ob.next_block_loss(h, dh_, P, F)
    g = torch.empty((S, L, d), dtype=torch.float32, device="cuda")
    loss = torch.zeros(1, dtype=torch.float32, device="cuda")
    rq.realq_block_window(dims, W, _dev(h), _dev(dh_), _dev(F), g, ws, loss=loss)
    got_g, got_loss = g.cpu().numpy(), float(loss.item())
    assert abs(got_loss - want_loss) <= 1e-4 * abs(want_loss), (got_loss, want_loss)
    np.testing.assert_allclose(got_g, want_g, rtol=0, atol=1e-4 * np.abs(want_g).max())


def test_block_window_is_deterministic_and_zero_at_zero():
    S, L, d, H, Hkv, dh, f = CASES[4]
    r, P, W, dims, ws = _case(3, *CASES[4])
    h = _dev(r.standard_normal((S, L, d)))
    dh_ = _dev(0.1 * r.standard_normal((S, L, d)))
    F = _dev(np.eye(d))
    outs = []
    for _ in range(2):
        g = torch.empty((S, L, d), dtype=torch.float32, device="cuda")
        loss = torch.zeros(1, dtype=torch.float32, device="cuda")
        rq.realq_block_window(dims, W, h, dh_, F, g, ws, loss=loss)
        outs.append((g.clone(), loss.clone()))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])
    g = torch.empty((S, L, d), dtype=torch.float32, device="cuda")
    loss = torch.ones(1, dtype=torch.float32, device="cuda")
    rq.realq_block_window(dims, W, h, torch.zeros_like(h), F, g, ws, loss=loss)
    assert loss.item() == 0.0 and g.abs().max().item() == 0.0


MODULES = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")


def _spd(r, d):
    Z = r.standard_normal((d, 3))
    return _f32(0.5 * np.eye(d) + Z @ Z.T / 6)


def _weights(P):
    return {k: torch.from_numpy(P[k].astype(np.float32)).cuda() for k in _KEYS}


@pytest.mark.parametrize("case", [CASES[0], CASES[4]])
@pytest.mark.parametrize("module", MODULES)
def test_module_window_matches_the_oracle(case, module):
    # block l's own backward to the module's weight with the next block's
    # window (Eq. slide_window), against oracle.block.sliding_window_module
    S, L, d, H, Hkv, dh, f = case
    r, P, W, dims, _ = _case(4, *case)
    _, Pn, Wn, _, _ = _case(104, *case)
    name = ob._MODULE_WEIGHT[module]
    Wm = _f32(P[name] + 0.05 * r.standard_normal(P[name].shape))
    x = _f32(r.standard_normal((S, L, d)))
    F, Fn = _spd(r, d), _spd(r, d)
    want_loss, want_g = ob.sliding_window_module(module, Wm, x, P, Pn, 0.6, F, Fn)
    grad = torch.empty(Wm.shape, dtype=torch.float32, device="cuda")
    loss = torch.zeros(1, dtype=torch.float32, device="cuda")
    ws = rq.workspace(rq.realq_block_module_workspace_size(dims, S, L))
    rq.realq_block_module_window(dims, W, Wn, _dev(x), module, _dev(Wm), 0.6, _dev(F), _dev(Fn), grad, ws, loss=loss)
    got = grad.cpu().numpy()
    assert abs(loss.item() - want_loss) <= 1e-4 * abs(want_loss), (loss.item(), want_loss)
    np.testing.assert_allclose(got, want_g, rtol=0, atol=1e-4 * np.abs(want_g).max())


def test_head_kl_matches_the_oracle():
    r = np.random.default_rng(5)
    S, L, d, V = 4, 33, 64, 1000
    head = {k: _f32(v) for k, v in ob.head_params(r, d, V, scale=1.5).items()}
    h = _f32(r.standard_normal((S, L, d)))
    dh_ = _f32(0.1 * r.standard_normal((S, L, d)))
    want_loss, want_g = ob.kl_head_loss(h, dh_, head)
    g = torch.empty((S, L, d), dtype=torch.float32, device="cuda")
    loss = torch.zeros(1, dtype=torch.float32, device="cuda")
    ws = rq.workspace(rq.realq_block_head_workspace_size(d, S, L, V))
    rq.realq_block_head_kl(_dev(head["gf"]), _dev(head["Wh"]), _dev(h), _dev(dh_), g, ws, loss=loss)
    assert abs(loss.item() - want_loss) <= 1e-4 * abs(want_loss), (loss.item(), want_loss)
    np.testing.assert_allclose(g.cpu().numpy(), want_g, rtol=0, atol=1e-4 * np.abs(want_g).max())


@pytest.mark.parametrize("module", ("k_proj", "o_proj", "up_proj", "down_proj"))
def test_final_block_module_kl_matches_the_oracle(module):
    case = CASES[1]
    S, L, d, H, Hkv, dh, f = case
    r, P, W, dims, _ = _case(6, *case)
    name = ob._MODULE_WEIGHT[module]
    Wm = _f32(P[name] + 0.05 * r.standard_normal(P[name].shape))
    x = _f32(r.standard_normal((S, L, d)))
    V = 29
    head = {k: _f32(v) for k, v in ob.head_params(r, d, V, scale=1.5).items()}
    want_loss, want_g = ob.kl_final_module(module, Wm, x, P, head)
    grad = torch.empty(Wm.shape, dtype=torch.float32, device="cuda")
    loss = torch.zeros(1, dtype=torch.float32, device="cuda")
    ws = rq.workspace(rq.realq_block_module_workspace_size(dims, S, L, V))
    rq.realq_block_module_kl(dims, W, _dev(x), module, _dev(Wm), _dev(head["gf"]), _dev(head["Wh"]), grad, ws,
                             loss=loss)
    assert abs(loss.item() - want_loss) <= 1e-4 * abs(want_loss), (loss.item(), want_loss)
    np.testing.assert_allclose(grad.cpu().numpy(), want_g, rtol=0, atol=1e-4 * np.abs(want_g).max())
