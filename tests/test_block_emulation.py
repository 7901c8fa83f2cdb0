"""The decoder block's launch sequence (csrc/block_ops.cuh) run on the host
against the fp64 oracle (oracle/block.py).

The header's per-thread bodies and the order and arguments of its launches
and GEMMs are compiled with g++ into a test-only library whose executor calls
each body for every index of its launch and does each GEMM as a plain loop
(tests/emu/block_emu.cpp).  The fp32 results must match the oracle within a
tolerance derived below; this checks the index arithmetic and the argument
of every step before the CUDA build of the same header runs on a GPU.  Each
launch also runs with its indices reversed (the result must not change: the
GPU orders no index before another), and every GEMM is checked for an output
that overlaps its operands."""
import ctypes
import os
import shutil
import subprocess

import numpy as np
import pytest

from oracle import block as ob

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_00049_gb300", "csrc")
SRC = os.path.join(ROOT, "tests", "emu", "block_emu.cpp")


@pytest.fixture(scope="module")
def emu(tmp_path_factory):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no C++ compiler")
    out = str(tmp_path_factory.mktemp("emu") / "libblock_emu.so")
    subprocess.run([cxx, "-O2", "-std=c++17", "-shared", "-fPIC", "-Wall", "-Wextra", "-Werror", "-I", CSRC, SRC,
                    "-o", out], check=True, capture_output=True, text=True)
    lib = ctypes.CDLL(out)
    lib.emu_block_workspace.restype = ctypes.c_size_t
    lib.emu_block_workspace.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    lib.emu_block_forward.restype = ctypes.c_int
    lib.emu_block_window.restype = ctypes.c_int
    lib.emu_set_order.argtypes = [ctypes.c_int]
    lib.emu_set_order(0)
    return lib


_ORDER = ("g1", "Wq", "Wk", "Wv", "Wo", "g2", "Wg", "Wu", "Wd")


class _Block:
    def __init__(self, lib, P, S, L):
        self.lib = lib
        d = P["g1"].shape[0]
        self.iv = np.array([S, L, d, P["n_heads"], P["n_kv"], P["dh"], P["Wg"].shape[0]], dtype=np.int64)
        self.fv = np.array([1e-6, 10000.0], dtype=np.float32)
        self.w32 = [np.ascontiguousarray(P[k], dtype=np.float32) for k in _ORDER]
        self.wptr = (ctypes.c_void_p * 9)(*[a.ctypes.data for a in self.w32])
        n = lib.emu_block_workspace(self.iv.ctypes.data, self.fv.ctypes.data)
        self.ws = np.zeros(n // 4 + 64, dtype=np.float32)
        self.shape = (S, L, d)

    def forward(self, x, rcs=None):
        x32 = np.ascontiguousarray(x, dtype=np.float32)
        y = np.zeros(self.shape, dtype=np.float32)
        rc = self.lib.emu_block_forward(ctypes.c_void_p(self.iv.ctypes.data), ctypes.c_void_p(self.fv.ctypes.data),
                                        self.wptr, ctypes.c_void_p(x32.ctypes.data), ctypes.c_void_p(y.ctypes.data),
                                        ctypes.c_void_p(self.ws.ctypes.data))
        if rcs is None:
            assert rc == 0
        else:
            rcs.append(rc)
        return y

    def window(self, h, dh_, F, rcs=None):
        h32, d32 = (np.ascontiguousarray(a, dtype=np.float32) for a in (h, dh_))
        F32 = np.ascontiguousarray(F, dtype=np.float32)
        g = np.zeros(self.shape, dtype=np.float32)
        loss = np.zeros(1, dtype=np.float32)
        rc = self.lib.emu_block_window(ctypes.c_void_p(self.iv.ctypes.data), ctypes.c_void_p(self.fv.ctypes.data),
                                       self.wptr, *(ctypes.c_void_p(a.ctypes.data) for a in (h32, d32, F32, g, loss)),
                                       ctypes.c_void_p(self.ws.ctypes.data))
        if rcs is None:
            assert rc == 0
        else:
            rcs.append(rc)
        return float(loss[0]), g


CASES = [
    # (S, L, d, H, Hkv, dh, f): grouped queries over a ragged length; one
    # key/value head per query head; a single token per sequence; wide heads
    (2, 7, 16, 4, 2, 4, 24),
    (3, 5, 24, 3, 3, 8, 40),
    (2, 1, 16, 4, 1, 4, 20),
    (1, 9, 32, 2, 1, 16, 48),
    (4, 96, 256, 8, 2, 32, 704),
]


def _case(seed, S, L, d, H, Hkv, dh, f):
    r = np.random.default_rng(seed)
    P = ob.block_params(r, d, H, Hkv, dh, f, scale=0.8)
    # round the parameters to fp32 so that both sides see the same block
    for k in _ORDER:
        P[k] = P[k].astype(np.float32).astype(np.float64)
    return r, P


@pytest.mark.parametrize("case", CASES)
def test_forward_matches_the_oracle(emu, case):
    S, L, d, H, Hkv, dh, f = case
    r, P = _case(1, *case)
    x = r.standard_normal((S, L, d)).astype(np.float32).astype(np.float64)
    want, _ = ob.block_forward(x, P)
    got = _Block(emu, P, S, L).forward(x)
    # fp32 arithmetic with fp32 accumulation over at most max(d, f, L) terms
    # of unit size: a few 1e-7 relative per operation, well inside 1e-5 of
    # the output's scale
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-5 * np.abs(want).max())


@pytest.mark.parametrize("case", CASES)
def test_window_loss_and_gradient_match_the_oracle(emu, case):
    S, L, d, H, Hkv, dh, f = case
    r, P = _case(2, *case)
    h = r.standard_normal((S, L, d)).astype(np.float32).astype(np.float64)
    dh_ = (0.1 * r.standard_normal((S, L, d))).astype(np.float32).astype(np.float64)
    Z = r.standard_normal((d, 3))
    F = (0.5 * np.eye(d) + Z @ Z.T / 6).astype(np.float32).astype(np.float64)
    want_loss, want_g = ob.next_block_loss(h, dh_, P, F)
    loss, g = _Block(emu, P, S, L).window(h, dh_, F)
    # Δz is the difference of two fp32 forward passes whose outputs are about
    # |h| / |Δh| = 10 times larger than Δz, so its relative error is ~10x the
    # forward's (1e-5 of scale): 1e-4 of the gradient's and the loss's scale
    assert abs(loss - want_loss) <= 1e-4 * abs(want_loss), (loss, want_loss)
    np.testing.assert_allclose(g, want_g, rtol=0, atol=1e-4 * np.abs(want_g).max())


def test_window_of_a_zero_perturbation_is_zero(emu):
    S, L, d, H, Hkv, dh, f = CASES[0]
    r, P = _case(3, *CASES[0])
    h = r.standard_normal((S, L, d))
    F = np.eye(d)
    loss, g = _Block(emu, P, S, L).window(h, np.zeros_like(h), F)
    assert loss == 0.0 and np.abs(g).max() == 0.0


MODULES = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")


def _ptrs(P):
    arrs = [np.ascontiguousarray(P[k], dtype=np.float32) for k in _ORDER]
    return arrs, (ctypes.c_void_p * 9)(*[a.ctypes.data for a in arrs])


def _c(a):
    return ctypes.c_void_p(a.ctypes.data)


def _spd32(r, d):
    Z = r.standard_normal((d, 3))
    return (0.5 * np.eye(d) + Z @ Z.T / 6).astype(np.float32).astype(np.float64)


def _module_case(seed, case, module):
    S, L, d, H, Hkv, dh, f = case
    r, P = _case(seed, *case)
    _, Pn = _case(seed + 100, *case)
    name = ob._MODULE_WEIGHT[module]
    Wm = (P[name] + 0.05 * r.standard_normal(P[name].shape)).astype(np.float32).astype(np.float64)
    x = r.standard_normal((S, L, d)).astype(np.float32).astype(np.float64)
    return r, P, Pn, name, Wm, x


def _iv(P, S, L):
    d = P["g1"].shape[0]
    return (np.array([S, L, d, P["n_heads"], P["n_kv"], P["dh"], P["Wg"].shape[0]], dtype=np.int64),
            np.array([1e-6, 10000.0], dtype=np.float32))


def _ws(emu, iv, fv, V=0):
    emu.emu_module_workspace.restype = ctypes.c_size_t
    emu.emu_module_workspace.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64]
    return np.zeros(emu.emu_module_workspace(iv.ctypes.data, fv.ctypes.data, V) // 4 + 64, dtype=np.float32)


@pytest.mark.parametrize("module", MODULES)
def test_module_inputs_match_the_oracle(emu, module):
    # the module's calibration inputs from a forward pass (its OBS Hessian's
    # tokens): the attention norm's output, the attention output, the MLP
    # norm's output or the SwiGLU product
    case = CASES[0]
    S, L, d = case[0], case[1], case[2]
    r, P = _case(8, *case)
    x = r.standard_normal((S, L, d)).astype(np.float32).astype(np.float64)
    want = ob.module_inputs(module, x, P)
    iv, fv = _iv(P, S, L)
    al, pl = _ptrs(P)
    x32 = np.ascontiguousarray(x, dtype=np.float32)
    got = np.zeros(want.shape, dtype=np.float32)
    ws = np.zeros(emu.emu_block_workspace(iv.ctypes.data, fv.ctypes.data) // 4 + 64, dtype=np.float32)
    assert emu.emu_module_inputs(_c(iv), _c(fv), pl, _c(x32), ctypes.c_int(MODULES.index(module)), _c(got),
                                 _c(ws)) == 0
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-5 * np.abs(want).max())


def _current_pass32(r, P, x, name):
    # block l's input and weights in the model quantized so far (the other
    # modules moved off the reference), rounded to fp32
    x_hat = (x + 0.1 * r.standard_normal(x.shape)).astype(np.float32).astype(np.float64)
    P_hat = dict(P)
    for k in ("Wq", "Wk", "Wv", "Wo", "Wg", "Wu", "Wd"):
        if k != name:
            P_hat[k] = (P[k] + 0.03 * r.standard_normal(P[k].shape)).astype(np.float32).astype(np.float64)
    return x_hat, P_hat


@pytest.mark.parametrize("current", [False, True])
@pytest.mark.parametrize("module", MODULES)
def test_module_window_matches_the_oracle(emu, module, current):
    # block l's own backward to each module's weight, with the next block's
    # window (Eq. slide_window); the case with grouped queries and a ragged
    # length; with current, block l's current pass takes a perturbed input
    # and other weights than the reference
    case = CASES[0]
    S, L, d = case[0], case[1], case[2]
    r, P, Pn, name, Wm, x = _module_case(4, case, module)
    F, Fn = _spd32(r, d), _spd32(r, d)
    alpha = 0.6
    x_hat, P_hat = _current_pass32(r, P, x, name) if current else (None, None)
    want_loss, want_g = ob.sliding_window_module(module, Wm, x, P, Pn, alpha, F, Fn, x_hat, P_hat)
    iv, fv = _iv(P, S, L)
    al, pl = _ptrs(P)
    an, pn = _ptrs(Pn)
    ah, ph = _ptrs(P_hat) if current else (None, None)
    xh32 = np.ascontiguousarray(x_hat, dtype=np.float32) if current else None
    x32, W32, F32, Fn32 = (np.ascontiguousarray(a, dtype=np.float32) for a in (x, Wm, F, Fn))
    g = np.zeros(Wm.shape, dtype=np.float32)
    loss = np.zeros(1, dtype=np.float32)
    ws = _ws(emu, iv, fv)
    rc = emu.emu_module_window(_c(iv), _c(fv), pl, ph, pn, _c(x32), _c(xh32) if current else None,
                               ctypes.c_int(MODULES.index(module)), _c(W32), ctypes.c_float(alpha), _c(F32), _c(Fn32),
                               _c(g), _c(loss), _c(ws))
    assert rc == 0
    # Δh is a difference of two fp32 forward passes, as in the window
    assert abs(float(loss[0]) - want_loss) <= 1e-4 * abs(want_loss), (float(loss[0]), want_loss)
    np.testing.assert_allclose(g, want_g, rtol=0, atol=1e-4 * np.abs(want_g).max())


def test_kl_head_matches_the_oracle(emu):
    r = np.random.default_rng(5)
    S, L, d, V = 3, 5, 16, 37
    head = ob.head_params(r, d, V, scale=1.5)
    head = {k: v.astype(np.float32).astype(np.float64) for k, v in head.items()}
    h = r.standard_normal((S, L, d)).astype(np.float32).astype(np.float64)
    dh_ = (0.1 * r.standard_normal((S, L, d))).astype(np.float32).astype(np.float64)
    want_loss, want_g = ob.kl_head_loss(h, dh_, head)
    iv = np.array([S, L, d, 1, 1, 2, 1], dtype=np.int64)
    fv = np.array([1e-6, 10000.0], dtype=np.float32)
    gf, Wh, h32, d32 = (np.ascontiguousarray(a, dtype=np.float32) for a in (head["gf"], head["Wh"], h, dh_))
    g = np.zeros((S, L, d), dtype=np.float32)
    loss = np.zeros(1, dtype=np.float32)
    ws = _ws(emu, iv, fv, V)
    rc = emu.emu_head_kl(_c(iv), _c(fv), _c(gf), _c(Wh), ctypes.c_int64(V), _c(h32), _c(d32), _c(g), _c(loss),
                         _c(ws))
    assert rc == 0
    # the KL of distributions 1e-1 apart is second order: its fp32 value is
    # a sum of p (log p - log q) terms 10x larger than the result
    assert abs(float(loss[0]) - want_loss) <= 1e-4 * abs(want_loss), (float(loss[0]), want_loss)
    np.testing.assert_allclose(g, want_g, rtol=0, atol=1e-4 * np.abs(want_g).max())


@pytest.mark.parametrize("current", [False, True])
@pytest.mark.parametrize("module", ("k_proj", "o_proj", "up_proj", "down_proj"))
def test_final_block_module_kl_matches_the_oracle(emu, module, current):
    case = CASES[1]
    S, L, d = case[0], case[1], case[2]
    r, P, _, name, Wm, x = _module_case(6, case, module)
    V = 29
    head = {k: v.astype(np.float32).astype(np.float64) for k, v in ob.head_params(r, d, V, scale=1.5).items()}
    x_hat, P_hat = _current_pass32(r, P, x, name) if current else (None, None)
    want_loss, want_g = ob.kl_final_module(module, Wm, x, P, head, x_hat, P_hat)
    iv, fv = _iv(P, S, L)
    al, pl = _ptrs(P)
    ah, ph = _ptrs(P_hat) if current else (None, None)
    xh32 = np.ascontiguousarray(x_hat, dtype=np.float32) if current else None
    x32, W32, gf, Wh = (np.ascontiguousarray(a, dtype=np.float32) for a in (x, Wm, head["gf"], head["Wh"]))
    g = np.zeros(Wm.shape, dtype=np.float32)
    loss = np.zeros(1, dtype=np.float32)
    ws = _ws(emu, iv, fv, V)
    rc = emu.emu_module_kl(_c(iv), _c(fv), pl, ph, _c(x32), _c(xh32) if current else None,
                           ctypes.c_int(MODULES.index(module)), _c(W32), _c(gf), _c(Wh), ctypes.c_int64(V), _c(g),
                           _c(loss), _c(ws))
    assert rc == 0
    assert abs(float(loss[0]) - want_loss) <= 1e-4 * abs(want_loss), (float(loss[0]), want_loss)
    np.testing.assert_allclose(g, want_g, rtol=0, atol=1e-4 * np.abs(want_g).max())


# Plausible mistakes planted in a copy of the header must fail the check:
# the transpose rotation's sign, the softmax backward's row term, the
# RMSNorm backward's correction, the key/value head of a query head, the
# SiLU derivative, and a GEMM fed the untransposed weight.
PLANTED = {
    "rope_inverse": ("p[j] = x1 * c + x2 * s;", "p[j] = x1 * c - x2 * s;"),
    "softmax_row_term": ("const float ds = p * (dp - Dt);", "const float ds = p * dp;"),
    "rms_correction": ("const float v = gr[k] * g[k] * rr - xr[k] * c;", "const float v = gr[k] * g[k] * rr;"),
    "kv_head": ("const int64_t kvh = h / a.rep();\n        const int64_t off",
                "const int64_t kvh = h % a.Hkv;\n        const int64_t off"),
    "silu_derivative": ("zg[i] = c * u * (sg * (1.f + g * (1.f - sg)));", "zg[i] = c * u * sg;"),
    "untransposed_weight": ("gemm_rr(T, d, qw, B.o, B.WoT, B.h, B.x)", "gemm_rr(T, d, qw, B.o, W.Wo, B.h, B.x)"),
    # module-level: q_proj's gradient taken before the transpose rotation,
    # the blend of the two blocks' gradients, the KL gradient's sign
    "wgrad_before_rope": ("if (module == M_Q) return e | x.gemm(gemm_wgrad(T, qw, d, B.o, B.a, gW), \"blk_wgrad\");\n",
                          ""),
    "module_blend": ("Axpy{M.tmp, M.wthis, M.gh, alpha}", "Axpy{M.tmp, M.wthis, M.gh, 1.f - alpha}"),
    "kl_sign": ("b[v] = (q - p) * inv_T;", "b[v] = (p - q) * inv_T;"),
    # the current pass run on the reference input
    "current_input": ("e |= forward(x, dm, Wcur, Bl, xhat, M.dh);", "e |= forward(x, dm, Wcur, Bl, xin, M.dh);"),
}
# the check each planted mistake is run against
_PLANTED_CHECK = {"wgrad_before_rope": "module_q", "module_blend": "module_q", "kl_sign": "kl",
                  "current_input": "module_q_current"}


@pytest.mark.parametrize("name", sorted(PLANTED))
def test_the_check_catches_a_planted_mistake(name, tmp_path):
    old, new = PLANTED[name]
    src = open(os.path.join(CSRC, "block_ops.cuh")).read()
    assert src.count(old) == 1, f"anchor not found once: {old}"
    if name == "wgrad_before_rope":
        # move q_proj's weight gradient ahead of the transpose rotation
        new = old
        src = src.replace(old, "")
        anchor = '    e |= x.map(T * dm.H * (dm.dh / 2), Rope{B.o, qw'
        assert src.count(anchor) == 1
        src = src.replace(anchor, old + anchor)
        old = new
    (tmp_path / "block_ops.cuh").write_text(src.replace(old, new))
    out = str(tmp_path / "libmut.so")
    subprocess.run([shutil.which("g++") or "c++", "-O2", "-std=c++17", "-shared", "-fPIC", "-I", str(tmp_path), SRC,
                    "-o", out], check=True, capture_output=True, text=True)
    lib = ctypes.CDLL(out)
    lib.emu_block_workspace.restype = ctypes.c_size_t
    lib.emu_block_workspace.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    check = _PLANTED_CHECK.get(name, "window")
    if check != "window":
        assert _planted_module_or_kl_differs(lib, check), f"the planted mistake '{name}' went unnoticed"
        return
    S, L, d, H, Hkv, dh, f = CASES[0]
    r, P = _case(2, *CASES[0])
    h = r.standard_normal((S, L, d)).astype(np.float32).astype(np.float64)
    dh_ = (0.1 * r.standard_normal((S, L, d))).astype(np.float32).astype(np.float64)
    F = np.eye(d)
    want_loss, want_g = ob.next_block_loss(h, dh_, P, F)
    loss, g = _Block(lib, P, S, L).window(h, dh_, F)
    bad = abs(loss - want_loss) > 1e-4 * abs(want_loss) or np.abs(g - want_g).max() > 1e-4 * np.abs(want_g).max()
    assert bad, f"the planted mistake '{name}' went unnoticed"


def _planted_module_or_kl_differs(lib, check):
    case = CASES[0]
    S, L, d = case[0], case[1], case[2]
    if check == "kl":
        r = np.random.default_rng(5)
        V = 37
        head = {k: v.astype(np.float32).astype(np.float64) for k, v in ob.head_params(r, d, V, scale=1.5).items()}
        h = r.standard_normal((S, L, d)).astype(np.float32).astype(np.float64)
        dh_ = (0.1 * r.standard_normal((S, L, d))).astype(np.float32).astype(np.float64)
        want_loss, want_g = ob.kl_head_loss(h, dh_, head)
        iv = np.array([S, L, d, 1, 1, 2, 1], dtype=np.int64)
        fv = np.array([1e-6, 10000.0], dtype=np.float32)
        gf, Wh, h32, d32 = (np.ascontiguousarray(a, dtype=np.float32) for a in (head["gf"], head["Wh"], h, dh_))
        g = np.zeros((S, L, d), dtype=np.float32)
        loss = np.zeros(1, dtype=np.float32)
        ws = _ws(lib, iv, fv, V)
        assert lib.emu_head_kl(_c(iv), _c(fv), _c(gf), _c(Wh), ctypes.c_int64(V), _c(h32), _c(d32), _c(g), _c(loss),
                               _c(ws)) == 0
    else:
        r, P, Pn, name, Wm, x = _module_case(4, case, "q_proj")
        F, Fn = _spd32(r, d), _spd32(r, d)
        current = check == "module_q_current"
        x_hat, P_hat = _current_pass32(r, P, x, name) if current else (None, None)
        want_loss, want_g = ob.sliding_window_module("q_proj", Wm, x, P, Pn, 0.6, F, Fn, x_hat, P_hat)
        iv, fv = _iv(P, S, L)
        al, pl = _ptrs(P)
        an, pn = _ptrs(Pn)
        ah, ph = _ptrs(P_hat) if current else (None, None)
        xh32 = np.ascontiguousarray(x_hat, dtype=np.float32) if current else None
        x32, W32, F32, Fn32 = (np.ascontiguousarray(a, dtype=np.float32) for a in (x, Wm, F, Fn))
        g = np.zeros(Wm.shape, dtype=np.float32)
        loss = np.zeros(1, dtype=np.float32)
        ws = _ws(lib, iv, fv)
        assert lib.emu_module_window(_c(iv), _c(fv), pl, ph, pn, _c(x32), _c(xh32) if current else None,
                                     ctypes.c_int(0), _c(W32), ctypes.c_float(0.6), _c(F32), _c(Fn32), _c(g),
                                     _c(loss), _c(ws)) == 0
    return (abs(float(loss[0]) - want_loss) > 1e-4 * abs(want_loss)
            or np.abs(g - want_g).max() > 1e-4 * np.abs(want_g).max())


def _all_ops(lib, case, V=23):
    """Every op of the header on one case (forward, window, the module
    window and the final block's KL for all seven modules with a current
    pass off the reference, the KL head), as one flat fp32 vector, with the
    return codes."""
    S, L, d, H, Hkv, dh, f = case
    r, P = _case(7, *case)
    _, Pn = _case(107, *case)
    out, rcs = [], []
    blk = _Block(lib, P, S, L)
    x = r.standard_normal((S, L, d))
    dh_ = 0.1 * r.standard_normal((S, L, d))
    F, Fn = _spd32(r, d), _spd32(r, d)
    out.append(blk.forward(x, rcs).ravel())
    loss, g = blk.window(x, dh_, F, rcs)
    out += [g.ravel(), np.float32([loss])]
    iv, fv = _iv(P, S, L)
    al, pl = _ptrs(P)
    an, pn = _ptrs(Pn)
    head = {k: np.ascontiguousarray(v, dtype=np.float32) for k, v in ob.head_params(r, d, V, scale=1.5).items()}
    x32, d32, F32, Fn32 = (np.ascontiguousarray(a, dtype=np.float32) for a in (x, dh_, F, Fn))
    x_hat, P_hat = _current_pass32(r, P, x, None)
    xh32 = np.ascontiguousarray(x_hat, dtype=np.float32)
    ah, ph = _ptrs(P_hat)
    for i, module in enumerate(MODULES):
        W32 = np.ascontiguousarray(P[ob._MODULE_WEIGHT[module]] + 0.05 * r.standard_normal(
            P[ob._MODULE_WEIGHT[module]].shape), dtype=np.float32)
        for kind in ("window", "kl"):
            gW = np.zeros(W32.shape, dtype=np.float32)
            lo = np.zeros(1, dtype=np.float32)
            if kind == "window":
                ws = _ws(lib, iv, fv)
                rcs.append(lib.emu_module_window(_c(iv), _c(fv), pl, ph, pn, _c(x32), _c(xh32), ctypes.c_int(i),
                                                 _c(W32), ctypes.c_float(0.6), _c(F32), _c(Fn32), _c(gW), _c(lo),
                                                 _c(ws)))
            else:
                ws = _ws(lib, iv, fv, V)
                rcs.append(lib.emu_module_kl(_c(iv), _c(fv), pl, ph, _c(x32), _c(xh32), ctypes.c_int(i), _c(W32),
                                             _c(head["gf"]), _c(head["Wh"]), ctypes.c_int64(V), _c(gW), _c(lo),
                                             _c(ws)))
            out += [gW.ravel(), lo]
    g = np.zeros((S, L, d), dtype=np.float32)
    lo = np.zeros(1, dtype=np.float32)
    ws = _ws(lib, iv, fv, V)
    rcs.append(lib.emu_head_kl(_c(iv), _c(fv), _c(head["gf"]), _c(head["Wh"]), ctypes.c_int64(V), _c(x32), _c(d32),
                               _c(g), _c(lo), _c(ws)))
    out += [g.ravel(), lo]
    return np.concatenate(out), rcs


# grouped queries over a ragged length, one key/value head per query head,
# and more than one 1024-token chunk of the fixed-order loss sum
ORDER_CASES = [CASES[0], CASES[1], (1, 1100, 8, 2, 1, 4, 12)]


@pytest.mark.parametrize("case", ORDER_CASES)
def test_launches_do_not_depend_on_the_order_of_their_indices(emu, case):
    # The GPU runs the indices of one launch in no fixed order, so no index
    # may read what another index of the same launch writes: every op run
    # with each launch's indices reversed gives the same bits.  Every GEMM's
    # output also shares no memory with its A and B operands (the host
    # executor returns an error code if one does).
    try:
        emu.emu_set_order(0)
        a, rca = _all_ops(emu, case)
        emu.emu_set_order(1)
        b, rcb = _all_ops(emu, case)
    finally:
        emu.emu_set_order(0)
    assert rca == [0] * len(rca) and rcb == [0] * len(rcb)
    assert np.isfinite(a).all()
    assert a.tobytes() == b.tobytes()


# A launch whose indices depend on each other, and a GEMM that overwrites
# its own operand, planted in a copy of the header, must each be caught.
PLANTED_ORDER = {
    # the attention output written over the values that later queries read
    "attn_output_over_values": ("AttnFwd{B.q, B.k, B.v, B.o, B.lse, as}", "AttnFwd{B.q, B.k, B.v, B.v, B.lse, as}"),
    # the gate's input gradient written over the gate gradient it reads
    "gemm_over_its_operand": ("e |= x.gemm(gemm_rr(T, d, f, B.zg, W.Wg, B.b), \"blk_proj_bwd\");",
                              "e |= x.gemm(gemm_rr(T, d, f, B.zg, W.Wg, B.zg), \"blk_proj_bwd\");"),
}


@pytest.mark.parametrize("name", sorted(PLANTED_ORDER))
def test_the_order_check_catches_a_planted_dependence(name, tmp_path):
    old, new = PLANTED_ORDER[name]
    src = open(os.path.join(CSRC, "block_ops.cuh")).read()
    assert src.count(old) == 1, f"anchor not found once: {old}"
    (tmp_path / "block_ops.cuh").write_text(src.replace(old, new))
    out = str(tmp_path / "libmut.so")
    subprocess.run([shutil.which("g++") or "c++", "-O2", "-std=c++17", "-shared", "-fPIC", "-I", str(tmp_path), SRC,
                    "-o", out], check=True, capture_output=True, text=True)
    lib = ctypes.CDLL(out)
    lib.emu_block_workspace.restype = ctypes.c_size_t
    lib.emu_block_workspace.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    lib.emu_set_order.argtypes = [ctypes.c_int]
    case = CASES[1]     # H = H_kv, so that the attention output and the values have one width
    lib.emu_set_order(0)
    a, rca = _all_ops(lib, case)
    lib.emu_set_order(1)
    b, rcb = _all_ops(lib, case)
    caught = any(rca) or any(rcb) or a.tobytes() != b.tobytes()
    assert caught, f"the planted dependence '{name}' went unnoticed"
