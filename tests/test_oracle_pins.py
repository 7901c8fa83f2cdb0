"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a closed
form, a brute-force search, a special case that reduces to a textbook routine,
an independent route to the same quantity, or a library implementation.
"""
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth
from oracle import brute


def _correlated_case(seed, m, n, T, w_std=0.02):
    r = synth.rng(seed, "pin-corr", m, n, T)
    Z = r.standard_normal((T, n))
    M = np.eye(n) + 0.6 * r.standard_normal((n, n)) / math.sqrt(n)
    X = Z @ M
    W0 = r.standard_normal((m, n)) * w_std
    return W0.astype(np.float32).astype(np.float64), X


# ---------------------------------------------------------------------------
# quantizer: the grid point chosen is the nearest one among all 2^b codes
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("bits,sym", [(4, False), (4, True), (3, False), (2, True)])
def test_quantizer_is_nearest_grid_point(bits, sym):
    r = synth.rng(1, "quant", bits, int(sym))
    w = r.standard_normal((64, 128)) * 0.02
    w[:, 5] *= 4.0                      # values outside the grid range get clamped
    s, z, _ = oracle.quant_params(w[:, :100], bits, sym)
    levels = 2 ** bits
    grid = (s[:, None].astype(np.float32) * (np.arange(levels, dtype=np.float32)[None, :] - z[:, None].astype(np.float32)))
    for j in range(w.shape[1]):
        q, dq, _ = oracle.quantize(w[:, j], s, z, bits)
        dist = np.abs(grid.astype(np.float64) - w[:, j:j + 1].astype(np.float32).astype(np.float64))
        chosen = dist[np.arange(64), q]
        # the chosen code is a nearest grid point (up to fp32 rounding of w/scale)
        assert np.all(chosen <= dist.min(axis=1) + 1e-6 * s)
        assert np.array_equal(dq, grid[np.arange(64), q].astype(np.float64))
        unique = np.sort(dist, axis=1)[:, 1] - dist.min(axis=1) > 1e-6 * s
        assert np.array_equal(q[unique], np.argmin(dist, axis=1)[unique])
    # the grid holds 0 exactly and spans the group's range
    assert np.all(np.min(np.abs(grid), axis=1) == 0.0)
    lo = np.minimum(w[:, :100].min(1), 0)
    hi = np.maximum(w[:, :100].max(1), 0)
    assert np.all(grid.min(1) <= lo + s) and np.all(grid.max(1) >= hi - s)


def test_degenerate_group_gets_unit_range():
    s, z, _ = oracle.quant_params(np.zeros((3, 8)), 4, False)
    # -xmin/scale = 1/(2/15) evaluates to 7.4999997 in fp32, so the zero point is 7
    assert np.allclose(s, 2.0 / 15.0) and np.all(z == 7)


# ---------------------------------------------------------------------------
# RTN special case: no Block-GD and H = I leave no error feedback
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("group,sym,bits", [(128, False, 4), (0, True, 4), (32, False, 3)])
def test_identity_hessian_reduces_to_rtn(group, sym, bits):
    r = synth.rng(2, "rtn")
    W0 = r.standard_normal((48, 256)) * 0.02
    T = 1000
    res = oracle.realq_sweep(W0, T * np.eye(256), T, bits=bits, group_size=group, symmetric=sym, damp_frac=0.01)
    codes, deq, s, z = oracle.rtn(W0, bits, group, sym)
    assert np.array_equal(res["codes"], codes)
    assert np.array_equal(res["deq"], deq)
    assert np.array_equal(res["scale"], s) and np.array_equal(res["zero"], z)


# ---------------------------------------------------------------------------
# OBS step against the definition: at column j the compensation uses row j of
# the inverse of H restricted to the columns still free (Schur complement),
# and the same sweep through rows of the upper Cholesky factor of H^-1,
# immediate or lazily batched, gives the same result.
# ---------------------------------------------------------------------------
def _sweep_submatrix_inverse(W0, Hd, bits, g, sym):
    W = W0.copy()
    m, n = W.shape
    codes = np.zeros((m, n), dtype=np.int64)
    for j in range(n):
        if j % g == 0:
            s, z, _ = oracle.quant_params(W[:, j:j + g], bits, sym)
        q, dq, _ = oracle.quantize(W[:, j], s, z, bits)
        eps = W[:, j] - dq
        Hinv_free = np.linalg.inv(Hd[j:, j:])          # free set {j, ..., n-1}
        v = np.zeros(n)
        v[j] = -1.0
        v[j + 1:] = -Hinv_free[0, 1:] / Hinv_free[0, 0]  # the lemma's compensation vector
        W += np.outer(eps, v)                          # ΔW^(j) = eps_j v_j^T
        W[:, j] = dq
        codes[:, j] = q
    return codes, W


def _sweep_cholesky_lazy(W0, Hd, bits, g, sym, B):
    U = np.linalg.cholesky(np.linalg.inv(Hd)).T
    W = W0.copy()
    m, n = W.shape
    codes = np.zeros((m, n), dtype=np.int64)
    for b0 in range(0, n, B):
        b1 = min(b0 + B, n)
        E = np.zeros((m, b1 - b0))
        for j in range(b0, b1):
            if j % g == 0:
                s, z, _ = oracle.quant_params(W[:, j:j + g], bits, sym)
            q, dq, _ = oracle.quantize(W[:, j], s, z, bits)
            err = (W[:, j] - dq) / U[j, j]
            W[:, j + 1:b1] -= np.outer(err, U[j, j + 1:b1])
            W[:, j] = dq
            E[:, j - b0] = err
            codes[:, j] = q
        W[:, b1:] -= E @ U[b0:b1, b1:]
    return codes, W


@pytest.mark.parametrize("n,g,B", [(3, 3, 1), (8, 8, 2), (12, 4, 4), (16, 8, 4)])
def test_obs_recursion_matches_definitions(n, g, B):
    W0, X = _correlated_case(3, 4, n, 200)
    H = X.T @ X
    ref = oracle.realq_sweep(W0, H, 200, bits=4, group_size=g, block_size=B, damp_frac=0.01)
    Hd = ref["Hd"]
    c1, w1 = _sweep_submatrix_inverse(W0, Hd, 4, g, False)
    c2, w2 = _sweep_cholesky_lazy(W0, Hd, 4, g, False, B)
    assert np.array_equal(ref["codes"], c1) and np.array_equal(ref["codes"], c2)
    assert np.allclose(ref["deq"], w1, rtol=0, atol=1e-12)
    assert np.allclose(ref["deq"], w2, rtol=0, atol=1e-12)


# ---------------------------------------------------------------------------
# Theorem "Reconstruction error of GPTQ": sum_j ||eps_j||^2 / [H^-1]_jj equals
# tr(ΔW H ΔW^T) exactly under the fixed Hessian.
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("seed,m,n,g", [(4, 16, 64, 16), (5, 8, 96, 32), (6, 32, 40, 0)])
def test_gptq_error_theorem(seed, m, n, g):
    W0, X = _correlated_case(seed, m, n, 500)
    res = oracle.realq_sweep(W0, X.T @ X, 500, bits=3, group_size=g, block_size=8)
    lhs = np.sum(np.sum(res["eps"] ** 2, axis=0) / res["hinv_diag"])
    dW = res["deq"] - W0
    rhs = np.trace(dW @ res["Hd"] @ dW.T)
    assert abs(lhs - rhs) <= 1e-10 * abs(rhs)


# ---------------------------------------------------------------------------
# Closed-form inverse: the Kac-Murdock-Szego matrix A_ij = rho^|i-j| has a
# tridiagonal inverse, and every trailing principal block is again KMS.
# ---------------------------------------------------------------------------
def _kms_inverse(n, rho):
    Ainv = np.zeros((n, n))
    c = 1.0 / (1.0 - rho * rho)
    for i in range(n):
        Ainv[i, i] = c * (1.0 + rho * rho) if 0 < i < n - 1 else c
        if i + 1 < n:
            Ainv[i, i + 1] = Ainv[i + 1, i] = -rho * c
    if n == 1:
        Ainv[0, 0] = 1.0
    return Ainv


def test_kms_closed_form_inverse_and_downdate():
    n, rho, T = 24, 0.7, 10
    A = rho ** np.abs(np.subtract.outer(np.arange(n), np.arange(n)))
    U = oracle.inverse_upper_cholesky(A)
    assert np.allclose(U.T @ U, _kms_inverse(n, rho), atol=1e-12)
    assert np.allclose(np.tril(U, -1), 0.0)
    r = synth.rng(7, "kms")
    W0 = r.standard_normal((5, n)) * 0.02
    res = oracle.realq_sweep(W0, T * A, T, damp_frac=0.0, group_size=0)
    want = np.array([_kms_inverse(n - j, rho)[0, 0] for j in range(n)])
    assert np.allclose(res["hinv_diag"], want, rtol=1e-12)


# ---------------------------------------------------------------------------
# Hessian: integer inputs give an exact H; compare with exact integer sums.
# ---------------------------------------------------------------------------
def test_hessian_exact_on_integer_inputs():
    r = synth.rng(8, "hint")
    X = r.integers(-2, 3, size=(300, 7))
    H, T = oracle.hessian_sum([X[:128], X[128:]])
    assert T == 300
    for i in range(7):
        for j in range(7):
            assert H[i, j] == sum(int(X[t, i]) * int(X[t, j]) for t in range(300))
    Xfp = r.integers(-2, 3, size=(300, 7))
    D = oracle.cross_moment_sum([X], [Xfp])
    for i in range(7):
        for j in range(7):
            assert D[i, j] == sum((int(X[t, i]) - int(Xfp[t, i])) * int(X[t, j]) for t in range(300))


def test_dead_columns():
    case = synth.layer_case(9, 6, 20, 64, dead_cols=(3, 11))
    H, T = oracle.hessian_sum([case.Xhat])
    res = oracle.realq_sweep(case.W0, H, T, group_size=0)
    assert list(np.nonzero(res["dead"])[0]) == [3, 11]
    assert np.all(res["deq"][:, [3, 11]] == 0.0)
    assert np.all(res["codes"][:, [3, 11]] == res["zero"][:, [0]])
    Hd = res["Hd"]
    assert Hd[3, 3] == 1.0 + res["lam"] and np.all(Hd[3, :3] == 0.0)
    # reading: the damping mean is taken after the dead channels got H_jj = 1
    d = np.where(res["dead"], 1.0, np.diag(H) / T)
    assert res["lam"] == pytest.approx(0.01 * d.mean(), rel=1e-15)


# ---------------------------------------------------------------------------
# Surrogate and gradient: token form vs moment form; finite differences.
# ---------------------------------------------------------------------------
def test_surrogate_two_routes():
    case = synth.layer_case(10, 12, 20, 300)
    H, T = oracle.hessian_sum([case.Xhat])
    r = synth.rng(10, "what")
    What = case.W0 + 0.003 * r.standard_normal(case.W0.shape)
    a = oracle.surrogate_tokens(What, case.W0, case.Xhat, None, case.F)
    b = oracle.surrogate_moment(What, case.W0, H / T, case.F)
    assert abs(a - b) <= 1e-12 * abs(a)


def test_gradient_finite_differences_with_perturbed_inputs():
    case = synth.layer_case(11, 5, 7, 200, perturbed=True)
    H, T = oracle.hessian_sum([case.Xhat])
    D = oracle.cross_moment_sum([case.Xhat], [case.X])
    r = synth.rng(11, "what")
    What = case.W0 + 0.01 * r.standard_normal(case.W0.shape)
    G = oracle.gradient(What, case.W0, H / T, D / T, case.F)
    h = 1e-6
    for (i, j) in [(0, 0), (2, 3), (4, 6), (1, 5)]:
        Wp = What.copy(); Wp[i, j] += h
        Wm = What.copy(); Wm[i, j] -= h
        fd = (oracle.surrogate_tokens(Wp, case.W0, case.Xhat, case.X, case.F)
              - oracle.surrogate_tokens(Wm, case.W0, case.Xhat, case.X, case.F)) / (2 * h)
        assert abs(fd - G[i, j]) <= 1e-6 * max(1e-3, abs(G[i, j]))


# ---------------------------------------------------------------------------
# Descent lemma (Sec. 5, SGD form): the surrogate is quadratic in the free
# columns, so one SGD step changes it by exactly
#   -eta ||G||^2 + (eta^2/2) <G, F G H̄_rr>,
# negative whenever eta < 2 / (lambda_max(F) lambda_max(H̄_rr)).
# ---------------------------------------------------------------------------
def test_sgd_step_descent_lemma():
    case = synth.layer_case(12, 16, 48, 400, outliers=2)
    H, T = oracle.hessian_sum([case.Xhat])
    Hbar = H / T
    F = case.F.astype(np.float64)
    B = 16
    be = B
    lmax = np.linalg.eigvalsh(F)[-1] * np.linalg.eigvalsh(Hbar[be:, be:])[-1]
    eta = 1.0 / lmax
    res = oracle.realq_sweep(case.W0, H, T, block_size=B, group_size=16,
                             bgd={"lr": eta, "optimizer": "sgd"}, F=F)
    assert len(res["block_loss"]) == 2
    for (b, alpha, before, after) in res["block_loss"]:
        assert after < before
    # quadratic identity at a random point, loss evaluated token by token
    r = synth.rng(12, "quad")
    What = case.W0 + 0.004 * r.standard_normal(case.W0.shape)
    G = oracle.gradient(What, case.W0, Hbar, None, F)[:, be:]
    Wn = What.copy(); Wn[:, be:] -= eta * G
    d_loss = oracle.surrogate_tokens(Wn, case.W0, case.Xhat, None, F) - oracle.surrogate_tokens(What, case.W0, case.Xhat, None, F)
    pred = -eta * np.sum(G * G) + 0.5 * eta * eta * np.sum(G * (F @ G @ Hbar[be:, be:]))
    assert abs(d_loss - pred) <= 1e-9 * abs(pred)
    assert pred < 0


# ---------------------------------------------------------------------------
# Adam against torch.optim.Adam in fp64 (library implementation).
# ---------------------------------------------------------------------------
def test_adam_matches_torch():
    torch = pytest.importorskip("torch")
    r = synth.rng(13, "adam")
    p0 = r.standard_normal((6, 9))
    grads = [r.standard_normal((6, 9)) * 10 ** r.uniform(-3, 1) for _ in range(6)]
    opt = oracle.Adam(p0.shape, lr=3e-4)
    p = p0.copy()
    tp = torch.tensor(p0, dtype=torch.float64, requires_grad=True)
    topt = torch.optim.Adam([tp], lr=3e-4, betas=(0.9, 0.999), eps=1e-8)
    for g in grads:
        p -= opt.direction(g, slice(0, 9))
        tp.grad = torch.tensor(g, dtype=torch.float64)
        topt.step()
    assert np.allclose(p, tp.detach().numpy(), rtol=0, atol=1e-15)
    # first step is lr * g / (|g| + eps): a sign step
    o2 = oracle.Adam((1, 3), lr=0.5)
    d = o2.direction(np.array([[2.0, -1e-3, 0.0]]), slice(0, 3))
    assert np.allclose(d, [[0.5 * 2 / (2 + 1e-8), -0.5 * 1e-3 / (1e-3 + 1e-8), 0.0]], rtol=1e-14)


# ---------------------------------------------------------------------------
# Schedules: Eq. (slide_window) and Eq. (reverse_cosine).
# ---------------------------------------------------------------------------
def test_schedules():
    assert oracle.sliding_alpha(1, 304) == 1.0
    assert oracle.sliding_alpha(304, 304) == 0.0
    a = [oracle.sliding_alpha(b, 11) for b in range(1, 12)]
    assert np.allclose(np.diff(a), -0.1)
    assert oracle.sliding_alpha(1, 1) == 1.0
    assert math.isclose(oracle.reverse_cosine_lr(1, 32, 1e-5), 1e-7)
    assert math.isclose(oracle.reverse_cosine_lr(32, 32, 1e-5), 1e-5)
    mid = oracle.reverse_cosine_lr(17, 33, 1.0)
    assert math.isclose(mid, 0.01 + 0.99 * math.sin(math.pi / 4))


def test_sliding_window_blends_fishers():
    case = synth.layer_case(14, 8, 24, 100, with_next=True)
    H, T = oracle.hessian_sum([case.Xhat])
    bgd = {"lr": 1e-4, "b_global_start": 3, "B_total": 7}
    res = oracle.realq_sweep(case.W0, H, T, block_size=8, group_size=8, bgd=bgd, F=case.F, F_next=case.F_next)
    alphas = [x[1] for x in res["block_loss"]]
    assert np.allclose(alphas, [1 - 2 / 6, 1 - 3 / 6])
    assert res["adam_t"] == 2


# ---------------------------------------------------------------------------
# Output invariants of a full sweep.
# ---------------------------------------------------------------------------
def test_sweep_output_invariants():
    case = synth.layer_case(15, 20, 300, 400, outliers=3)
    H, T = oracle.hessian_sum([case.Xhat])
    res = oracle.realq_sweep(case.W0, H, T, block_size=128, group_size=128,
                             bgd={"lr": 1e-4}, F=case.F)
    codes, s, z = res["codes"], res["scale"], res["zero"]
    assert codes.min() >= 0 and codes.max() <= 15
    gi = np.arange(300) // 128
    deq = (s[:, gi] * (codes.astype(np.float32) - z[:, gi].astype(np.float32))).astype(np.float64)
    assert np.array_equal(deq, res["deq"])
    assert res["adam_t"] == 2
    packed = oracle.pack_codes(codes)
    assert packed.shape == (20, 150)
    assert np.array_equal(packed[:, 7] & 15, codes[:, 14]) and np.array_equal(packed[:, 7] >> 4, codes[:, 15])


# ---------------------------------------------------------------------------
# The rank-one updates in C are numpy's outer-product updates, bit for bit.
# ---------------------------------------------------------------------------
def test_native_rank_one_updates_are_numpys():
    from oracle import native
    r = np.random.default_rng(7)
    A = r.standard_normal((70, 90))
    for d in (None, 0.37):
        B, C = A.copy(), A.copy()
        u, v = B[5:, 3], B[2, 11:]            # a strided column and a row, outside the updated block
        native.outer_sub(B[5:, 11:], u, v, d)
        if d is None:
            C[5:, 11:] -= np.outer(C[5:, 3], C[2, 11:])
        else:
            C[5:, 11:] -= np.outer(C[5:, 3], C[2, 11:]) / d
        assert np.array_equal(B, C)
        assert not np.array_equal(B, A)


# ---------------------------------------------------------------------------
# Following another run's decisions at rounding ties (reading C3).  With
# H = I there is no compensation and the sweep is round-to-nearest (P1).  Row
# 0's group spans [-7, 8]: scale 1 and zero point 7 exactly, so w = 2.5 is an
# exact tie (rint gives 2, code 9; the other neighbour is code 10).  Row 1's
# spans [-7.5, 7.5]: scale 1 and -xmin/scale = 7.5, a zero-point tie (rint
# gives 8; the other neighbour is 7).
# ---------------------------------------------------------------------------
def _tie_case():
    r = np.random.default_rng(8)
    W0 = r.uniform(-3.0, 3.0, (4, 8))
    W0[0, :3] = (-7.0, 8.0, 2.5)
    W0[1, :2] = (-7.5, 7.5)
    T = 10
    return W0, T * np.eye(8), T


def test_following_own_decisions_changes_nothing():
    W0, H, T = _tie_case()
    a = oracle.realq_sweep(W0, H, T, group_size=8, block_size=8)
    assert a["codes"][0, 2] == 9 and a["zero"][0, 0] == 7 and a["zero"][1, 0] == 8
    assert a["margin"][0, 2] == 0.0 and a["zero_margin"][1, 0] == 0.0
    b = oracle.realq_sweep(W0, H, T, group_size=8, block_size=8, follow={"codes": a["codes"], "zero": a["zero"]})
    assert b["n_followed"] == 0 and b["n_followed_zero"] == 0
    for k in ("codes", "zero", "scale", "deq"):
        assert np.array_equal(a[k], b[k]), k


def test_following_takes_the_other_neighbour_only_at_ties():
    W0, H, T = _tie_case()
    a = oracle.realq_sweep(W0, H, T, group_size=8, block_size=8)
    # the other neighbour at the code tie and at the zero-point tie: taken
    other = a["codes"].copy()
    other[0, 2] = 10
    zo = a["zero"].copy()
    zo[1, 0] = 7
    b = oracle.realq_sweep(W0, H, T, group_size=8, block_size=8, follow={"codes": other, "zero": zo})
    assert b["n_followed"] == 1 and b["n_followed_zero"] == 1
    assert b["codes"][0, 2] == 10 and b["deq"][0, 2] == 3.0
    assert b["zero"][1, 0] == 7
    assert np.array_equal(b["deq"][1], b["scale"][1, 0] * (b["codes"][1] - 7.0))
    assert np.array_equal(b["codes"][2:], a["codes"][2:])
    # a code two levels away at the tie is not a rounding of w: ignored
    other[0, 2] = 11
    c = oracle.realq_sweep(W0, H, T, group_size=8, block_size=8, follow={"codes": other})
    assert c["n_followed"] == 0 and c["codes"][0, 2] == 9
    # every code moved up by one: only decisions at a tie follow
    up = np.minimum(a["codes"] + 1, 15)
    d = oracle.realq_sweep(W0, H, T, group_size=8, block_size=8, follow={"codes": up})
    changed = d["codes"] != a["codes"]
    assert changed[0, 2] and np.all(a["margin"][changed] < 1e-3)
    assert d["n_followed"] == int(changed.sum())


def test_following_a_decision_changes_only_its_row_from_there_on():
    # compensation on (a correlated H), no Block-GD: rows are independent, so
    # a decision taken from the other run (a wide tau makes every decision
    # eligible) leaves every other row and the row's earlier columns alone
    W0, X = _correlated_case(9, 6, 40, 200)
    H, T = oracle.hessian_sum([X])
    a = oracle.realq_sweep(W0, H, T, group_size=8, block_size=8)
    i0, j0 = 3, 17
    other = a["codes"].copy()                   # a code next to the oracle's at (i0, j0)
    other[i0, j0] = a["codes"][i0, j0] + (1 if a["codes"][i0, j0] < 15 else -1)
    b = oracle.realq_sweep(W0, H, T, group_size=8, block_size=8, follow={"codes": other, "tau": 0.5})
    # (later decisions of row i0, taken from the changed state, may follow
    # the other run back to its codes: those count too)
    assert b["codes"][i0, j0] == other[i0, j0] and b["n_followed"] >= 1
    keep = np.ones_like(a["codes"], dtype=bool)
    keep[i0, j0:] = False
    assert np.array_equal(a["codes"][keep], b["codes"][keep])
    assert not np.array_equal(a["deq"][i0, j0:], b["deq"][i0, j0:])


def test_per_decision_tolerances_follow_only_where_they_are_wide():
    # tau as an m x n array: the decision at (i0, j0) may follow (tau 0.5
    # there), none other may (tau 0), so a run whose codes all differ by one
    # level changes (i0, j0) and nothing before it in its row or in other rows
    W0, X = _correlated_case(9, 6, 40, 200)
    H, T = oracle.hessian_sum([X])
    a = oracle.realq_sweep(W0, H, T, group_size=8, block_size=8)
    i0, j0 = 2, 21
    other = np.where(a["codes"] < 15, a["codes"] + 1, a["codes"] - 1)
    tau = np.zeros(a["codes"].shape)
    tau[i0, j0] = 0.5
    b = oracle.realq_sweep(W0, H, T, group_size=8, block_size=8, follow={"codes": other, "tau": tau})
    assert b["n_followed"] == 1 and b["codes"][i0, j0] == other[i0, j0]
    keep = np.ones_like(a["codes"], dtype=bool)
    keep[i0, j0:] = False
    assert np.array_equal(a["codes"][keep], b["codes"][keep])
    # a zero tolerance everywhere follows nothing, whatever the other run says
    c = oracle.realq_sweep(W0, H, T, group_size=8, block_size=8,
                           follow={"codes": other, "zero": a["zero"] + 1, "tau": np.zeros_like(tau),
                                   "tau_zero": np.zeros(a["zero"].shape)})
    assert c["n_followed"] == 0 and c["n_followed_zero"] == 0 and np.array_equal(a["codes"], c["codes"])


# ---------------------------------------------------------------------------
# Brute force over all int4 codes of a 4 x 8 layer (diagonal Fisher: rows
# decouple).  The surrogate evaluator agrees with the independent C evaluator;
# no code vector beats the global minimum; the sweep does not lose to RTN; with
# one column the sweep is the exact minimiser.
# ---------------------------------------------------------------------------
@pytest.mark.slow
def test_brute_force_4x8():
    W0, X = _correlated_case(16, 4, 8, 64)
    T = X.shape[0]
    H = X.T @ X
    F = np.diag(synth.rng(16, "fd").uniform(0.5, 2.0, size=4))
    gptq = oracle.realq_sweep(W0, H, T, group_size=0, block_size=8)
    realq = oracle.realq_sweep(W0, H, T, group_size=0, block_size=2, bgd={"lr": 2e-4}, F=F)
    codes_rtn, _, s_rtn, z_rtn = oracle.rtn(W0, 4, 0)
    s, z = gptq["scale"][:, 0], gptq["zero"][:, 0]
    assert np.array_equal(s, s_rtn[:, 0]) and np.array_equal(z, z_rtn[:, 0])
    Hbar = H / T
    mins, argmins = brute.layer_min(W0, s, z, Hbar)
    f = np.diag(F)
    for name, res in (("gptq", gptq), ("realq", realq)):
        per_row = np.array([brute.row_eval(W0[i], s[i], z[i], Hbar, res["codes"][i]) for i in range(4)])
        L_or = oracle.surrogate_moment(res["deq"], W0, Hbar, F)
        assert abs(0.5 * np.sum(f * per_row) - L_or) <= 1e-12 * L_or, name
        assert np.all(mins <= per_row * (1 + 1e-12)), name
    # n = 8 is small enough that the greedy sweep may lose to RTN on a row; over
    # many rows of the same input it must win (a sign or index error would not)
    Wm, _ = _correlated_case(16, 256, 8, 64)
    gm = oracle.realq_sweep(Wm, H, T, group_size=0, block_size=8)
    cr, dr, _, _ = oracle.rtn(Wm, 4, 0)
    Fi = np.eye(256)
    assert oracle.surrogate_moment(gm["deq"], Wm, Hbar, Fi) < 0.9 * oracle.surrogate_moment(dr, Wm, Hbar, Fi)


def test_single_column_sweep_is_exact_minimiser():
    r = synth.rng(17, "n1")
    W0 = r.standard_normal((32, 1)) * 0.02
    H = np.array([[3.7]])
    res = oracle.realq_sweep(W0, H, 1, group_size=0)
    s, z = res["scale"][:, 0], res["zero"][:, 0]
    for i in range(32):
        best, arg = brute.row_min(W0[i], s[i], z[i], H / 1.0)
        val = brute.row_eval(W0[i], s[i], z[i], H / 1.0, res["codes"][i])
        assert val <= best * (1 + 1e-12) + 1e-300


# ------------------------------------------------ activation quantizer ---
def test_activation_quantizer_worked_example():
    # Sec. 5 weight-activation setting, per-token symmetric 4-bit, a_clip 0.9:
    # max|x| = 2 -> clipped range 1.8 -> step 3.6 / 15 = 0.24, zero point 8;
    # x / 0.24 = (2.08, -4.17, 1.04, 8.33) -> (2, -4, 1, 8), and 8 + 8 = 16 is
    # clamped to the last level 15; the dequantized values 0.48, -0.96, 0.24,
    # 1.68 stored in bf16 (steps 2^-9, 2^-8, 2^-10, 2^-7) are
    # 246 * 2^-9, -246 * 2^-8, 246 * 2^-10 and 215 * 2^-7.
    x = np.array([[0.5, -1.0, 0.25, 2.0]])
    q, scale, xq = oracle.quantize_activations(x, bits=4, a_clip=0.9)
    assert q.tolist() == [[10, 4, 9, 15]]
    assert abs(float(scale[0]) - 0.24) < 1e-7
    assert xq.tolist() == [[246 / 512, -246 / 256, 246 / 1024, 215 / 128]]


def test_activation_quantizer_nearest_level_and_clipping():
    r = np.random.default_rng(5)
    X = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(r.standard_normal((64, 200)) * np.exp(r.standard_normal((64, 1)))))
    X[3] = 0.0
    for bits, clip in ((4, 0.9), (4, 1.0), (3, 0.8), (8, 0.9)):
        q, scale, xq = oracle.quantize_activations(X, bits=bits, a_clip=clip, out_bf16=False)
        z = 2 ** (bits - 1)
        levels = np.arange(2 ** bits) - z
        x = X.astype(np.float64)
        # brute force over all 2^b levels of each token's grid
        cand = scale[:, None, None].astype(np.float64) * levels[None, None, :]
        dist = np.abs(x[:, :, None] - cand)
        best = dist.argmin(axis=2)
        srt = np.sort(dist, axis=2)
        # not a tie, beyond the fp32 rounding of x / scale (2^-24 relative)
        clear = (srt[:, :, 1] - srt[:, :, 0]) > 1e-6 * scale[:, None] + 2.0 ** -22 * np.abs(x)
        assert np.array_equal(q[clear], best[clear])
        # the clipped range: values beyond +-(levels) sit on the end levels
        amax = np.abs(x).max(axis=1)
        assert np.all(q[3] == z) and abs(float(scale[3]) - 2.0 / (2 ** bits - 1)) < 1e-7
        xmax = np.where(amax == 0, 1.0, clip * amax)
        np.testing.assert_allclose(scale, 2 * xmax / (2 ** bits - 1), rtol=1e-6)
        ref = scale[:, None].astype(np.float64) * (q - z)
        assert np.all(np.abs(xq - ref) <= 2.0 ** -24 * np.abs(ref))
        inside = np.abs(x) <= (z - 1) * scale[:, None]
        half = 0.5 * scale[:, None] * (1 + 1e-6) + 2.0 ** -22 * np.abs(x)
        assert np.all((np.abs(x - xq) <= half)[inside])


def test_bf16_rounding_matches_the_input_generator_cast():
    r = np.random.default_rng(6)
    a = (r.standard_normal(10000) * 10 ** r.uniform(-3, 3, 10000)).astype(np.float32)
    assert np.array_equal(oracle.round_bf16(a), synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(a)))


# ------------------------------------------ saliency-weighted grouped OBS ---
def _grouped_case(seed, m=32, n=48, T=400):
    r = np.random.default_rng(seed)
    X = r.standard_normal((T, n))
    X[:, 3] *= 6.0
    W0 = r.standard_normal((m, n)) * 0.02
    Z = r.standard_normal((m, 4))
    F = 0.5 * np.eye(m) + Z @ Z.T / 8
    return r, X, W0, F


def test_grouped_sweep_reduces_to_one_hessian_for_uniform_saliency():
    r, X, W0, F = _grouped_case(61)
    H, T = oracle.hessian_sum([X])
    S = np.full((X.shape[0], 4), 3.0)
    Hg, wsum = oracle.weighted_hessian_sum([X], [S])
    np.testing.assert_allclose(Hg, 3.0 * np.broadcast_to(H, Hg.shape), rtol=0, atol=1e-12 * np.abs(Hg).max())
    bgd = {"lr": 2e-4, "steps_per_block": 1, "b_global_start": 1, "B_total": 1}
    a = oracle.realq_sweep(W0, H, T, group_size=16, block_size=16, bgd=bgd, F=F)
    b = oracle.realq_sweep(W0, H, T, group_size=16, block_size=16, bgd=bgd, F=F,
                           obs_hessians=[(Hg[g], wsum[g]) for g in range(4)])
    assert np.array_equal(a["codes"], b["codes"])
    np.testing.assert_allclose(b["deq"], a["deq"], rtol=0, atol=1e-12)


def test_grouped_gptq_rows_are_independent_sweeps():
    # without Block-GD every row group is GPTQ on its own rows with its own H_g
    r, X, W0, F = _grouped_case(62, m=30)
    H, T = oracle.hessian_sum([X])
    S = np.exp(2.0 * r.standard_normal((X.shape[0], 3)))
    Hg, wsum = oracle.weighted_hessian_sum([X], [S])
    b = oracle.realq_sweep(W0, H, T, group_size=16, block_size=16, obs_hessians=[(Hg[g], wsum[g]) for g in range(3)])
    for g in range(3):
        rows = slice(10 * g, 10 * (g + 1))
        a = oracle.realq_sweep(W0[rows], Hg[g], wsum[g], group_size=16, block_size=16)
        assert np.array_equal(a["codes"], b["codes"][rows])
        assert np.array_equal(a["deq"], b["deq"][rows])
    # and the groups really differ from the unweighted sweep
    u = oracle.realq_sweep(W0, H, T, group_size=16, block_size=16)
    assert not np.array_equal(u["codes"], b["codes"])


def test_weighted_hessian_exact_on_integers():
    r = np.random.default_rng(63)
    X = r.integers(-3, 4, (50, 7)).astype(np.float64)
    S = r.integers(0, 5, (50, 2)).astype(np.float64)
    Hg, wsum = oracle.weighted_hessian_sum([X[:20], X[20:]], [S[:20], S[20:]])
    for g in range(2):
        ref = np.zeros((7, 7))
        for t in range(50):
            for i in range(7):
                for j in range(7):
                    ref[i, j] += S[t, g] * X[t, i] * X[t, j]
        assert np.array_equal(Hg[g], ref)
        assert wsum[g] == S[:, g].sum()


def test_saliency_clip_is_the_nearest_rank_percentile():
    r = np.random.default_rng(64)
    S = np.exp(3.0 * r.standard_normal((1000, 4)))
    S[r.integers(0, 1000, 50), 1] = 7.0                 # ties
    S[5, 2] = 1e15                                       # an extreme outlier
    for pct in (0.99, 0.5, 1.0, 1e-9, 0.973):
        Sc, c = oracle.saliency_clip(S, pct)
        frac = Fraction(repr(pct))
        for g in range(4):
            v = S[:, g]
            # brute-force counting with the exact product pct * T
            cand = [x for x in np.unique(v) if (v <= x).sum() >= frac * len(v)]
            assert c[g] == min(cand)
            assert np.array_equal(Sc[:, g], np.minimum(v, c[g]))
    Sc, c = oracle.saliency_clip(S, 0.99)
    assert c[2] < 1e15 and Sc[5, 2] == c[2]
    # the 99th percentile of 8000 values is the 7920th smallest (0.99 * 8000 is
    # exactly 7920, so its ceiling is 7920 and not 7921)
    assert oracle.saliency_clip(np.arange(8000.0)[:, None], 0.99)[1][0] == 7919.0
    assert oracle.saliency_clip(np.arange(8001.0)[:, None], 0.99)[1][0] == 7920.0   # 7920.99 -> 7921st


def test_saliency_clipping_prevents_rank_one_collapse():
    # App. "Hessian-side saliency clipping": one token with a saliency ~1e12 x
    # the median makes H_g nearly rank one; clipping at the 99th percentile
    # restores a well-spread spectrum
    r = np.random.default_rng(65)
    X = r.standard_normal((2000, 16))
    S = np.exp(r.standard_normal((2000, 1)))
    S[17, 0] = 1e12
    Hg, _ = oracle.weighted_hessian_sum([X], [S])
    ev = np.linalg.eigvalsh(Hg[0])
    assert ev[-1] / ev.sum() > 0.99
    Sc, _ = oracle.saliency_clip(S, 0.99)
    Hc, _ = oracle.weighted_hessian_sum([X], [Sc])
    ev = np.linalg.eigvalsh(Hc[0])
    assert ev[-1] / ev.sum() < 0.2


# ------------------------------------------------- mini-batch Block-GD ---
def test_minibatch_of_all_tokens_is_the_full_batch():
    r, X, W0, F = _grouped_case(66)
    H, T = oracle.hessian_sum([X])
    base = {"lr": 2e-4, "steps_per_block": 1, "b_global_start": 1, "B_total": 1}
    a = oracle.realq_sweep(W0, H, T, group_size=16, block_size=16, bgd=base, F=F)
    b = oracle.realq_sweep(W0, H, T, group_size=16, block_size=16, bgd={**base, "minibatches": [(H, T)]}, F=F)
    assert np.array_equal(a["codes"], b["codes"]) and np.array_equal(a["deq"], b["deq"])


def test_minibatch_rotation_rule():
    # two mini-batches, the second with no second moment: steps that draw it
    # see a zero gradient and Adam does not move (m = v = 0 there); the
    # rotation (b_global - 1) * steps + s mod 2 decides which blocks move
    r, X, W0, F = _grouped_case(67)
    H, T = oracle.hessian_sum([X])
    zero = np.zeros_like(H)
    for start in (1, 2):
        bgd = {"lr": 2e-4, "steps_per_block": 1, "b_global_start": start, "B_total": 1,
               "minibatches": [(H, T), (zero, T)]}
        res = oracle.realq_sweep(W0, H, T, group_size=16, block_size=16, bgd=bgd, F=F)
        gptq = oracle.realq_sweep(W0, H, T, group_size=16, block_size=16)
        # block 0's step is the first optimizer step: it moves only if it
        # draws mini-batch 0, i.e. when b_global_start is odd
        moved_first = start % 2 == 1
        assert (not np.array_equal(res["codes"][:, 16:32], gptq["codes"][:, 16:32])
                or not np.array_equal(res["deq"][:, 16:32], gptq["deq"][:, 16:32])) == moved_first
    # the mean of the mini-batch moments is the full-batch moment
    Hs = [oracle.hessian_sum([X[k * 100:(k + 1) * 100]])[0] for k in range(4)]
    np.testing.assert_allclose(sum(Hs) / T, H / T, rtol=1e-13, atol=1e-15)


# ---------------------------------------------------------------------------
# output-perturbation clipping of the Block-GD loss (a_loss_clip) and the
# token-form gradient it needs
# ---------------------------------------------------------------------------
def test_loss_clip_worked_example():
    # one token with residuals 1..20 (shuffled, signs alternating): the 95th
    # nearest-rank percentile of 20 channels is the 19th smallest |Δy| = 19
    # (0.95 * 20 = 19 exactly), so only the channel with |Δy| = 20 is
    # scaled, by 19/20
    perm = np.random.default_rng(5).permutation(20)
    dY = (np.arange(1, 21, dtype=np.float64) * np.where(np.arange(20) % 2, -1.0, 1.0))[perm][None, :]
    kappa, q = oracle.loss_clip_factors(dY, 0.95)
    assert q[0] == 19.0
    expect = np.ones(20)
    expect[np.abs(dY[0]) == 20.0] = 19.0 / 20.0
    assert np.array_equal(kappa[0], expect)
    # 0.99 of 100 channels: rank 99 exactly, so the threshold is 99 and the
    # largest channel is scaled by 99/100; 0.98 of 100: rank 98, threshold
    # 98, the two largest scaled; 0.995 of 100: 99.5 -> rank 100, nothing
    dY = np.arange(1, 101, dtype=np.float64)[None, :]
    kappa, q = oracle.loss_clip_factors(dY, 0.99)
    assert q[0] == 99.0 and np.all(kappa[0, :99] == 1.0) and kappa[0, 99] == 99.0 / 100.0
    kappa, q = oracle.loss_clip_factors(dY, 0.98)
    assert q[0] == 98.0 and np.all(kappa[0, :98] == 1.0)
    assert kappa[0, 98] == 98.0 / 99.0 and kappa[0, 99] == 98.0 / 100.0
    kappa, q = oracle.loss_clip_factors(dY, 0.995)
    assert q[0] == 100.0 and np.all(kappa == 1.0)


def test_loss_clip_invariants():
    # per token: the scaled residuals never exceed the threshold, those above
    # it land exactly on it, and m - rank channels are scaled (distinct values)
    r = np.random.default_rng(6)
    dY = r.standard_t(3, size=(50, 64)) * np.exp(r.standard_normal((50, 1)))
    kappa, q = oracle.loss_clip_factors(dY, 0.95)
    k = math.ceil(Fraction(95, 100) * 64)
    Y = np.abs(kappa * dY)
    assert np.all(Y <= q[:, None] * (1 + 1e-15))
    np.testing.assert_allclose(Y.max(axis=1), q, rtol=1e-15)
    assert np.all((kappa < 1.0).sum(axis=1) == 64 - k)
    assert np.all((kappa > 0) & (kappa <= 1.0))


def test_token_gradient_without_clipping_is_the_moment_gradient():
    # kappa = 1: the token form equals F (Ŵ - W0) H̄ on the same tokens
    r, X, W0, F = _grouped_case(68)
    What = W0 + r.standard_normal(W0.shape) * 0.003
    H, T = oracle.hessian_sum([X])
    Gm = oracle.gradient(What, W0, H / T, None, F)
    Gt = oracle.gradient_tokens(What, W0, X, None, F)
    np.testing.assert_allclose(Gt, Gm, rtol=1e-11, atol=1e-15)
    # a percentile at the maximum scales nothing
    Gc = oracle.gradient_tokens(What, W0, X, None, F, a_loss_clip=1.0)
    np.testing.assert_allclose(Gc, Gm, rtol=1e-11, atol=1e-15)


def test_clipped_gradient_is_the_gradient_of_the_detached_loss():
    # central differences of L_kappa (kappa frozen at Ŵ) on sampled entries:
    # the loss is quadratic in Ŵ for fixed kappa, so they are exact up to
    # rounding
    r, X, W0, F = _grouped_case(69, m=12, n=10, T=60)
    X[:, 2] *= 40.0                                  # a few large residual channels
    What = W0 + r.standard_normal(W0.shape) * 0.01
    dY = X @ (What - W0).T
    kappa, _ = oracle.loss_clip_factors(dY, 0.9)
    assert (kappa < 1).any()
    G = oracle.gradient_tokens(What, W0, X, None, F, a_loss_clip=0.9)
    h = 1e-4
    for i, j in [(0, 0), (3, 2), (11, 9), (5, 7)]:
        E = np.zeros_like(What)
        E[i, j] = h
        fd = (oracle.surrogate_tokens_clipped(What + E, W0, X, F, kappa)
              - oracle.surrogate_tokens_clipped(What - E, W0, X, F, kappa)) / (2 * h)
        assert abs(fd - G[i, j]) <= 1e-8 * max(1.0, abs(G[i, j])), (i, j, fd, G[i, j])


def test_token_minibatch_sweep_reduces_to_the_moment_minibatch_sweep():
    # without clipping the token-form mini-batch sweep is the moment-form one
    r, X, W0, F = _grouped_case(70)
    H, T = oracle.hessian_sum([X])
    parts = [X[k * 100:(k + 1) * 100] for k in range(4)]
    base = {"lr": 2e-4, "steps_per_block": 1, "b_global_start": 2, "B_total": 1}
    a = oracle.realq_sweep(W0, H, T, group_size=16, block_size=16, F=F,
                           bgd={**base, "minibatches": [oracle.hessian_sum([p]) for p in parts]})
    b = oracle.realq_sweep(W0, H, T, group_size=16, block_size=16, F=F, bgd={**base, "minibatch_tokens": parts})
    assert np.array_equal(a["codes"], b["codes"])
    np.testing.assert_allclose(b["deq"], a["deq"], rtol=0, atol=1e-12)
    # with clipping the sweep differs, and only after the first block
    c = oracle.realq_sweep(W0, H, T, group_size=16, block_size=16, F=F,
                           bgd={**base, "minibatch_tokens": parts, "a_loss_clip": 0.95})
    assert np.array_equal(c["codes"][:, :16], a["codes"][:, :16])
    assert not np.allclose(c["deq"][:, 16:], a["deq"][:, 16:], rtol=0, atol=1e-9)


# ---------------------------------------------------------------------------
# The gradient of a column range is those columns of the full gradient; its
# error scale |F| |P| bounds it (triangle inequality) and equals it when no
# term cancels; the sensitivity probe with eta = 0 is the plain sweep, and
# the sweep's pre-rounding values give its codes and zero points.
# ---------------------------------------------------------------------------
def test_gradient_columns_error_scale_and_probe():
    case = synth.layer_case(16, 24, 96, 500, outliers=2, perturbed=True)
    H, T = oracle.hessian_sum([case.Xhat])
    D = oracle.cross_moment_sum([case.Xhat], [case.X])
    r = np.random.default_rng(17)
    What = case.W0 + r.standard_normal(case.W0.shape) * 0.003
    full = oracle.gradient(What, case.W0, H / T, D / T, case.F)
    part = oracle.gradient(What, case.W0, H / T, D / T, case.F, slice(40, 96))
    np.testing.assert_allclose(part, full[:, 40:], rtol=1e-12, atol=1e-15 * np.abs(full).max())
    scale = oracle.gradient_error_scale(What, case.W0, H / T, D / T, case.F, slice(40, 96))
    assert np.all(np.abs(part) <= scale * (1 + 1e-12))
    pos = oracle.gradient_error_scale(np.abs(What) + 1.0, np.zeros_like(What), np.abs(H) / T, None,
                                      np.abs(case.F))
    np.testing.assert_allclose(pos, oracle.gradient(np.abs(What) + 1.0, np.zeros_like(What), np.abs(H) / T, None,
                                                    np.abs(case.F)), rtol=1e-12)
    c2 = synth.layer_case(18, 20, 256, 600, outliers=2)
    H2, T2 = oracle.hessian_sum([c2.Xhat])
    kw = dict(group_size=64, block_size=64, bgd={"lr": 1e-4}, F=c2.F)
    a = oracle.realq_sweep(c2.W0, H2, T2, **kw)
    b = oracle.realq_sweep(c2.W0, H2, T2, grad_noise={"seed": 3, "eta": 0.0}, **kw)
    for k in ("codes", "scale", "zero", "deq", "x"):
        assert np.array_equal(a[k], b[k]), k
    p = oracle.realq_sweep(c2.W0, H2, T2, grad_noise={"seed": 3, "eta": 1e-6}, **kw)
    assert not np.array_equal(a["x"][:, 64:], p["x"][:, 64:])     # the probe moves the later blocks
    assert np.array_equal(a["x"][:, :64], p["x"][:, :64])         # and nothing before the first step
    g = np.arange(256) // 64
    assert np.array_equal(a["codes"], np.clip(np.rint(a["x"]).astype(np.int64) + a["zero"][:, g], 0, 15))
    assert np.array_equal(a["zero"], np.rint(a["zf"]).astype(np.int64))
