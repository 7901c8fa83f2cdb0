"""CUDA path vs the fp64 oracle on the same seeded inputs, through the C ABI.

Tolerances (derived in the design notes from the arithmetic):
  Hessian   bit-exact on integer inputs; otherwise |ΔH| <= 1e-5 * rms-scaled
            bound of fp32 accumulation over the token count.
  U         max |ΔU| <= 2e-4 * max |U| (fp32 blocked factorisation, damped H).
  codes     >= 99.9 % identical, every mismatch a rounding tie or downstream
            of one (tests/parity.py).
  scale     relative error <= 1e-5 on >= 99.9 % of groups.
  surrogate relative error <= 1e-3 (the path's own loss vs the oracle's).
"""
import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2609_00049_gb300 as rq
from paper_2609_00049_gb300 import layer
from parity import OracleSweep, check_codes_and_scales, follow_ties, unpack

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_00049_gb300 import build as b
    b.build()
    rq.lib()


def dev(a, dtype=torch.float32):
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda", dtype)


def bf16_dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to("cuda").view(torch.bfloat16)


def gpu_loss(Wq, W0, Hbar, F):
    m, n = Wq.shape
    out = torch.zeros(1, dtype=torch.float32, device="cuda")
    ws = rq.workspace(rq.realq_surrogate_workspace_size(m, n))
    rq.realq_surrogate_loss(Wq, W0, Hbar, F, out, ws)
    return float(out.item())


# --------------------------------------------------------------- Hessian ---
def test_hessian_exact_on_integer_inputs():
    case = synth.layer_case(20, 4, 200, 3000, integer_x=True)
    H = torch.zeros(200, 200, device="cuda")
    X = dev(case.Xhat)
    rq.realq_hessian_accumulate(X[:1700], H)
    rq.realq_hessian_accumulate(X[1700:], H)
    Href, _ = oracle.hessian_sum([case.Xhat])
    assert np.array_equal(H.cpu().numpy().astype(np.float64), Href)


def test_hessian_tensor_core_exact_on_integer_inputs():
    # integer activations are exact in bf16 and every partial sum is exact in fp32
    for n, T in ((256, 4160), (384, 20000), (136, 777), (1024, 65536)):
        case = synth.layer_case(33, 4, n, T, integer_x=True)
        X = dev(case.Xhat, torch.bfloat16)
        H, _, _ = layer.accumulate([X], n)
        Href, _ = oracle.hessian_sum([case.Xhat])
        assert np.array_equal(H.cpu().numpy().astype(np.float64), Href), (n, T)


@pytest.mark.parametrize("n,T", [(300, 5000), (128, 65536), (97, 4099), (512, 70000)])
def test_hessian_bf16_and_cross_moment(n, T):
    case = synth.layer_case(21, 4, n, T, perturbed=True, bf16=True, outliers=2)
    Xh = dev(case.Xhat, torch.bfloat16)
    Xf = dev(case.X, torch.bfloat16)
    H, D, T_ = layer.accumulate([Xh], n, [Xf])
    Href, _ = oracle.hessian_sum([case.Xhat])
    Dref = oracle.cross_moment_sum([case.Xhat], [case.X])
    scale = np.sqrt(np.outer(np.diag(Href), np.diag(Href)))
    err = np.abs(H.cpu().numpy() - Href) / scale
    assert err.max() < 2e-6 * np.sqrt(T)
    dscale = np.sqrt(np.outer(np.diag(Dref @ Dref.T / T) + 1e-30, np.diag(Href)))
    derr = np.abs(D.cpu().numpy() - Dref) / (np.abs(Dref).max())
    assert derr.max() < 1e-4, dscale.shape
    # bitwise repeatable (fixed-order split reduction)
    H2, _, _ = layer.accumulate([Xh], n)
    assert torch.equal(H, H2)


# --------------------------------------------------------------- prepare ---
# n = 1500 and 2052 take the tensor-core rank-64 updates and the tensor-core
# triangular-inverse product (n > 512, n % 4 == 0), 2052 with a ragged first
# 4-column panel; 1498 (n % 4 != 0) keeps the fp32 tiles
@pytest.mark.parametrize("n,dead", [(256, ()), (300, (5, 77, 299)), (64, ()), (1500, (3, 700)), (2052, ()),
                                    (1498, ())])
def test_prepare_matches_oracle(n, dead):
    case = synth.layer_case(22, 4, n, 4 * n, outliers=3, dead_cols=dead)
    Href, T = oracle.hessian_sum([case.Xhat])
    prep = layer.prepare(dev(Href), T, 0.01)
    ref = oracle.prepare(Href, T, 0.01)
    Uref = oracle.inverse_upper_cholesky(ref["Hd"])
    U = prep.U.cpu().numpy().astype(np.float64)
    assert np.abs(U - Uref).max() <= 2e-4 * np.abs(Uref).max()
    assert np.all(np.tril(U, -1) == 0)
    assert np.array_equal(prep.dead.cpu().numpy().astype(bool), ref["dead"])
    assert np.allclose(prep.Hbar.cpu().numpy(), ref["Hbar"], rtol=1e-6, atol=0)


def test_prepare_reports_not_spd():
    n = 96
    H = -torch.eye(n, device="cuda") * 10.0
    with pytest.raises(rq.RealqError) as ei:
        layer.prepare(H, 10, 0.01)
    assert ei.value.status == rq.REALQ_ERR_NOT_SPD
    assert ei.value.fail_col == n - 1


# ------------------------------------------------------------ the sweep ---
def _oracle_and_gpu(case, qkw, bgd=None, steps=1, with_next=False, b_global_start=1, B_total=1, use_dbar=False,
                    w_bf16=False):
    Hs, T = oracle.hessian_sum([case.Xhat])
    Ds = oracle.cross_moment_sum([case.Xhat], [case.X]) if use_dbar else None
    obgd = None if bgd is None else {"lr": bgd, "steps_per_block": steps, "b_global_start": b_global_start,
                                     "B_total": B_total}
    orc = OracleSweep(lambda follow, grad_noise=None: oracle.realq_sweep(
        case.W0, Hs, T, bits=qkw.get("bits", 4), group_size=qkw.get("group_size", 128),
        block_size=qkw.get("block_size", 128), symmetric=bool(qkw.get("symmetric", 0)), bgd=obgd, F=case.F,
        F_next=case.F_next if with_next else None, D_sum=Ds, follow=follow, grad_noise=grad_noise))
    Xh = dev(case.Xhat)
    Xf = dev(case.X) if use_dbar else None
    H, D, T_ = layer.accumulate([Xh], case.Xhat.shape[1], [Xf] if use_dbar else None)
    prep = layer.prepare(H, T_, qkw.get("damp_frac", 0.01), D_sum=D)
    q = rq.quant_cfg(**qkw)
    b = None if bgd is None else rq.bgd_cfg(bgd, steps_per_block=steps, b_global_start=b_global_start,
                                            B_total=B_total)
    W0 = dev(case.W0, torch.bfloat16) if w_bf16 else dev(case.W0)
    F = dev(case.F) if bgd is not None else None
    Fn = dev(case.F_next) if (with_next and bgd is not None) else None
    out = layer.quantize(W0, prep, q, b, F=F, F_next=Fn, use_dbar=use_dbar)
    torch.cuda.synchronize()
    return orc, out, prep, W0


def _check(orc, out, case, qkw, bgd, loss_tol=1e-3, prep=None, W0=None, lr=0.0, steps=1):
    n = case.W0.shape[1]
    codes = unpack(out.codes.cpu().numpy(), n)
    _, fol, rep = check_codes_and_scales(orc, codes, out.zero.cpu().numpy(), out.scale.cpu().numpy(), n, qkw, bgd,
                                         lr, steps)
    # dequantized values are the grid points of the returned codes
    g = qkw.get("group_size", 128) or n
    s = out.scale.cpu().numpy()[:, np.arange(n) // g]
    z = out.zero.cpu().numpy()[:, np.arange(n) // g].astype(np.float32)
    deq = (s * (codes.astype(np.float32) - z)).astype(np.float32)
    assert np.array_equal(deq, out.W.cpu().numpy())
    # (the oracle's result on the CUDA path's branch at rounding ties)
    L_or = oracle.surrogate_tokens(fol["deq"], case.W0, case.Xhat, case.X, case.F)
    if prep is not None and case.X is None:
        L_gpu = gpu_loss(out.W, W0, prep.Hbar, dev(case.F))
        assert abs(L_gpu - L_or) <= loss_tol * L_or, (L_gpu, L_or)
    return rep


def test_identity_hessian_gives_rtn_codes():
    r = synth.rng(23, "rtn-gpu")
    m, n, T = 64, 384, 1000
    W0 = (r.standard_normal((m, n)) * 0.02).astype(np.float32)
    prep = layer.prepare(torch.eye(n, device="cuda") * T, T, 0.01)
    for qkw in (dict(group_size=128), dict(group_size=0, symmetric=1), dict(group_size=32, bits=3),
                dict(group_size=256, block_size=64)):
        out = layer.quantize(dev(W0), prep, rq.quant_cfg(**qkw))
        codes, deq, s, z = oracle.rtn(W0, qkw.get("bits", 4), qkw.get("group_size", 128), bool(qkw.get("symmetric", 0)))
        assert np.array_equal(unpack(out.codes.cpu().numpy(), n), codes), qkw
        assert np.array_equal(out.scale.cpu().numpy(), s)
        assert np.array_equal(out.W.cpu().numpy().astype(np.float64), deq)


def _fc_case():
    wl = synth.workloads()["fc256x512"]
    mod = wl.modules[0]
    W0 = synth.weights(wl, mod)
    X = synth.xhat_full(wl, "x")
    return wl, synth.LayerCase(W0=W0, Xhat=X, X=None, F=synth.fisher(wl, mod))


def test_fc256x512_gptq_mode():
    wl, case = _fc_case()
    qkw = dict(group_size=128, block_size=128)
    orc, out, prep, W0 = _oracle_and_gpu(case, qkw)
    _check(orc, out, case, qkw, False, prep=prep, W0=W0)


@pytest.mark.parametrize("steps", [1, 4])
def test_fc256x512_realq(steps):
    wl, case = _fc_case()
    qkw = dict(group_size=128, block_size=128)
    orc, out, prep, W0 = _oracle_and_gpu(case, qkw, bgd=wl.lr, steps=steps)
    assert out.adam_t == orc["adam_t"] == 3 * steps
    _check(orc, out, case, qkw, True, prep=prep, W0=W0, lr=wl.lr, steps=steps)


@pytest.mark.parametrize("qkw", [dict(group_size=64, block_size=64), dict(group_size=0, symmetric=1),
                                 dict(group_size=32, block_size=128, bits=3), dict(group_size=256, block_size=128)])
def test_ragged_shapes_and_quantizer_modes(qkw):
    case = synth.layer_case(24, 200, 300, 1500, outliers=2, dead_cols=(7,))
    orc, out, prep, W0 = _oracle_and_gpu(case, qkw, bgd=2e-4)
    _check(orc, out, case, qkw, True, prep=prep, W0=W0, lr=2e-4)


def test_simt_fallback_shape():
    # n not a multiple of 4: the Block-GD GEMMs take the fp32 CUDA-core path
    case = synth.layer_case(34, 60, 197, 900, outliers=2)
    qkw = dict(group_size=64, block_size=64)
    orc, out, prep, W0 = _oracle_and_gpu(case, qkw, bgd=2e-4)
    _check(orc, out, case, qkw, True, prep=prep, W0=W0, lr=2e-4)


def test_block_narrower_than_layer_and_single_block():
    case = synth.layer_case(25, 40, 100, 800)
    qkw = dict(group_size=0, block_size=128)
    orc, out, prep, W0 = _oracle_and_gpu(case, qkw, bgd=1e-4)
    assert out.adam_t == 0
    _check(orc, out, case, qkw, True, prep=prep, W0=W0, lr=1e-4)


def test_sliding_window():
    case = synth.layer_case(26, 96, 320, 1200, with_next=True)
    qkw = dict(group_size=64, block_size=64)
    orc, out, prep, W0 = _oracle_and_gpu(case, qkw, bgd=2e-4, with_next=True, b_global_start=3, B_total=9)
    assert [round(x[1], 6) for x in orc["block_loss"]] == [round(1 - k / 8, 6) for k in range(2, 6)]
    _check(orc, out, case, qkw, True, prep=prep, W0=W0, lr=2e-4)


def test_perturbed_inputs_cross_moment():
    case = synth.layer_case(27, 64, 192, 900, perturbed=True)
    qkw = dict(group_size=64, block_size=64)
    orc, out, prep, W0 = _oracle_and_gpu(case, qkw, bgd=2e-4, use_dbar=True)
    _check(orc, out, case, qkw, True, lr=2e-4)


def test_bf16_weights():
    case = synth.layer_case(28, 128, 256, 1024, bf16=True)
    qkw = dict(group_size=128, block_size=128)
    orc, out, prep, W0 = _oracle_and_gpu(case, qkw, bgd=3e-4, w_bf16=True)
    _check(orc, out, case, qkw, True, prep=prep, W0=W0, lr=3e-4)


def test_resume_matches_single_call():
    case = synth.layer_case(29, 64, 384, 1000)
    Xh = dev(case.Xhat)
    H, _, T = layer.accumulate([Xh], 384)
    prep = layer.prepare(H, T)
    q = rq.quant_cfg(group_size=128, block_size=128)
    b = rq.bgd_cfg(1e-4)
    F = dev(case.F)
    W0 = dev(case.W0)
    full = layer.quantize(W0, prep, q, b, F=F)
    m, n = 64, 384
    W = torch.empty(m, n, device="cuda")
    codes = torch.empty(m, n // 2, dtype=torch.uint8, device="cuda")
    scale = torch.empty(m, 3, device="cuda")
    zero = torch.empty(m, 3, dtype=torch.uint8, device="cuda")
    am, av = torch.empty(m, n, device="cuda"), torch.empty(m, n, device="cuda")
    disp = torch.empty(m, n, device="cuda")
    ws = rq.workspace(rq.realq_quantize_workspace_size(m, n, q, b))
    t = 0
    for (b0, b1) in ((0, 1), (1, 3)):
        t = rq.realq_quantize_layer(W0, prep.U, prep.Hbar, q, W, codes, scale, zero, dead=prep.dead, bcfg=b, F=F,
                                    adam_m=am, adam_v=av, bgd_disp=disp, adam_t=t, block_begin=b0, block_end=b1,
                                    ws=ws)
    assert t == full.adam_t == 2
    assert torch.equal(codes, full.codes) and torch.equal(W, full.W)


def test_nonfinite_weight_is_reported():
    case = synth.layer_case(30, 32, 128, 400)
    W0 = case.W0.copy()
    W0[3, 5] = np.nan
    H, _, T = layer.accumulate([dev(case.Xhat)], 128)
    prep = layer.prepare(H, T)
    q = rq.quant_cfg()
    ws = rq.workspace(rq.realq_quantize_workspace_size(32, 128, q))
    layer.quantize(dev(W0), prep, q, ws=ws)
    with pytest.raises(rq.RealqError) as ei:
        rq.realq_workspace_status(ws)
    assert ei.value.status == rq.REALQ_ERR_NONFINITE


def test_bgd_refine_single_adam_step():
    case = synth.layer_case(31, 96, 256, 900)
    Hs, T = oracle.hessian_sum([case.Xhat])
    r = synth.rng(31, "what")
    What = (case.W0 + 0.004 * r.standard_normal(case.W0.shape)).astype(np.float32)
    c0 = 100
    Hbar = Hs / T
    G = oracle.gradient(What.astype(np.float64), case.W0, Hbar, None, case.F)[:, c0:]
    opt = oracle.Adam(What.shape, lr=1e-3)
    ref = What.astype(np.float64).copy()
    ref[:, c0:] -= opt.direction(G, slice(c0, 256))
    W = dev(What)
    am, av = torch.zeros_like(W), torch.zeros_like(W)
    b = rq.bgd_cfg(1e-3)
    ws = rq.workspace(rq.realq_bgd_workspace_size(96, 256))
    t = rq.realq_bgd_refine(W, dev(case.W0), c0, dev(Hbar), dev(case.F), b, adam_m=am, adam_v=av, ws=ws)
    assert t == 1
    got = W.cpu().numpy().astype(np.float64)
    assert np.array_equal(got[:, :c0], What[:, :c0].astype(np.float64))
    # the first Adam step is lr * sign(g) unless |g| is near the fp32 rounding level of the gradient
    sure = np.abs(G) > 1e-5 * np.abs(G).max()
    d = np.abs(got[:, c0:] - ref[:, c0:])
    assert d[sure].max() <= 1e-3 * 1e-3 + 2e-7 * np.abs(What).max()
    assert d[~sure].max(initial=0.0) <= 2.0 * 1e-3 + 1e-6


def test_surrogate_loss_matches_oracle():
    case = synth.layer_case(32, 80, 160, 700)
    Hs, T = oracle.hessian_sum([case.Xhat])
    r = synth.rng(32, "what")
    What = (case.W0 + 0.003 * r.standard_normal(case.W0.shape)).astype(np.float32)
    L_or = oracle.surrogate_tokens(What, case.W0, case.Xhat, None, case.F)
    L_gpu = gpu_loss(dev(What), dev(case.W0), dev(Hs / T), dev(case.F))
    assert abs(L_gpu - L_or) <= 1e-4 * L_or


# ------------------------------------------------ activation quantizer ---
@pytest.mark.parametrize("T,n,bits,clip", [(1000, 1024, 4, 0.9), (333, 197, 4, 0.9), (64, 4096, 3, 0.8),
                                           (50, 96, 8, 1.0), (1, 31, 4, 0.9)])
def test_activation_quantizer_bit_exact(T, n, bits, clip):
    r = synth.rng(41, "act-quant", T, n)
    x = r.standard_normal((T, n)) * np.exp(r.standard_normal((T, 1)))
    x[:, r.integers(0, n, 3)] *= 30.0                      # outlier channels
    x[T // 2] = 0.0                                        # a token of zeros
    bits16 = synth.f32_to_bf16_bits(x)
    xb = synth.bf16_bits_to_f32(bits16)
    q_or, s_or, xq_or = oracle.quantize_activations(xb, bits=bits, a_clip=clip)
    X = bf16_dev(bits16)
    ncb = (n + 1) // 2 if bits <= 4 else n
    codes = torch.empty(T, ncb, dtype=torch.uint8, device="cuda")
    scale = torch.empty(T, dtype=torch.float32, device="cuda")
    Xq = rq.realq_quantize_activations(X, bits, clip, codes=codes, scale=scale)
    assert np.array_equal(scale.cpu().numpy(), s_or)
    assert np.array_equal(Xq.float().cpu().numpy().astype(np.float64), xq_or)
    c = codes.cpu().numpy()
    q = unpack(c, n) if bits <= 4 else c.astype(np.int64)
    assert np.array_equal(q, q_or)
    # fp32 activations: the same codes, the dequantized values kept in fp32
    Xf = dev(xb)
    Xqf = rq.realq_quantize_activations(Xf, bits, clip)
    _, _, xq32 = oracle.quantize_activations(xb, bits=bits, a_clip=clip, out_bf16=False)
    assert np.array_equal(Xqf.cpu().numpy().astype(np.float64), xq32)
    # in place
    rq.realq_quantize_activations(X, bits, clip, X_q=X)
    assert torch.equal(X, Xq)


def test_activation_aware_sweep():
    # W4A4 activation-aware: the weights see the quantized activations (x̂), the
    # surrogate keeps the full-precision ones (x) through the cross moment
    case = synth.layer_case(42, 96, 256, 1500, bf16=True, outliers=3)
    x_bits = synth.f32_to_bf16_bits(case.Xhat)
    _, _, xhat = oracle.quantize_activations(case.Xhat, bits=4, a_clip=0.9)
    X = bf16_dev(x_bits)
    Xq = rq.realq_quantize_activations(X, 4, 0.9)
    assert np.array_equal(Xq.float().cpu().numpy().astype(np.float64), xhat)
    qkw = dict(group_size=128, block_size=128)
    Hs, T = oracle.hessian_sum([xhat])
    Ds = oracle.cross_moment_sum([xhat], [case.Xhat])
    orc = OracleSweep(lambda follow, grad_noise=None: oracle.realq_sweep(
        case.W0, Hs, T, group_size=128, block_size=128,
        bgd={"lr": 2e-4, "steps_per_block": 1, "b_global_start": 1, "B_total": 1}, F=case.F, D_sum=Ds,
        follow=follow, grad_noise=grad_noise))
    H, D, T_ = layer.accumulate([Xq], 256, [X])
    prep = layer.prepare(H, T_, 0.01, D_sum=D)
    out = layer.quantize(dev(case.W0), prep, rq.quant_cfg(**qkw), rq.bgd_cfg(2e-4), F=dev(case.F), use_dbar=True)
    torch.cuda.synchronize()
    n = 256
    codes = unpack(out.codes.cpu().numpy(), n)
    check_codes_and_scales(orc, codes, out.zero.cpu().numpy(), out.scale.cpu().numpy(), n, qkw, True, 2e-4, 1,
                           "activation-aware ")


def test_block_scheduler_activation_aware():
    # the block scheduler's W4A4 variant on a small two-input block: every
    # module matches the oracle sweep on the oracle's quantized activations
    from paper_2609_00049_gb300.block import BlockInput, BlockModule, BlockQuantizer
    r = synth.rng(43, "block-w4a4")
    T = 3000
    ins = {"a": 128, "b": 256}
    mods = [("m1", 64, "a"), ("m2", 96, "a"), ("m3", 64, "b")]
    x_bits = {k: synth.f32_to_bf16_bits(r.standard_normal((T, n)) * (1 + 9 * (r.random(n) < 0.02)))
              for k, n in ins.items()}
    Wf = {nm: synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(r.standard_normal((m, ins[i])) * 0.02))
          for nm, m, i in mods}
    Ff = {}
    for nm, m, _ in mods:
        z = r.standard_normal((m, 4))
        Ff[nm] = (np.eye(m) * 0.5 + z @ z.T / 8).astype(np.float32)
    qcfg = rq.quant_cfg(4, 64, 64, 0, 0.01)
    bq = BlockQuantizer([BlockInput(k, n, T) for k, n in ins.items()], [BlockModule(nm, m, ins[i], i) for nm, m, i in mods],
                        qcfg, 2e-4, 1, act_quant=(4, 0.9))
    bq.run({k: bf16_dev(v) for k, v in x_bits.items()}, {nm: dev(w) for nm, w in Wf.items()},
           {nm: dev(f) for nm, f in Ff.items()})
    torch.cuda.synchronize()
    bq.check_status()
    bstart = 1
    for nm, m, i in mods:
        x = synth.bf16_bits_to_f32(x_bits[i]).astype(np.float64)
        _, _, xhat = oracle.quantize_activations(x, 4, 0.9)
        Hs, _ = oracle.hessian_sum([xhat])
        Ds = oracle.cross_moment_sum([xhat], [x])
        orc = OracleSweep(lambda follow, grad_noise=None, W=Wf[nm], F=Ff[nm], Hs=Hs, Ds=Ds, b0=bstart: oracle.realq_sweep(
            W.astype(np.float64), Hs, T, group_size=64, block_size=64,
            bgd={"lr": 2e-4, "steps_per_block": 1, "b_global_start": b0, "B_total": 1}, F=F, D_sum=Ds,
            follow=follow, grad_noise=grad_noise))
        bstart += ins[i] // 64
        o = bq.out[nm]
        codes = unpack(o["codes"].cpu().numpy(), ins[i])
        qkw = dict(group_size=64, block_size=64)
        check_codes_and_scales(orc, codes, o["zero"].cpu().numpy(), o["scale"].cpu().numpy(), ins[i], qkw, True,
                               2e-4, 1, f"block W4A4 {nm} ")


# ------------------------------------------ saliency-weighted Hessians ---
@pytest.mark.parametrize("T,pct", [(4096, 0.99), (999, 0.99), (1000, 0.5), (77, 1.0), (1, 0.99), (8000, 0.99)])
def test_saliency_clip_bit_exact(T, pct):
    r = synth.rng(51, "saliency-clip", T)
    S = np.exp(3.0 * r.standard_normal((T, 4))).astype(np.float32)
    S[r.integers(0, T, max(1, T // 20)), 1] = 7.0
    S[0, 2] = 1e30
    S[T // 2, 3] = 0.0
    Sc_or, c_or = oracle.saliency_clip(S.astype(np.float64), pct)
    Sd = dev(S)
    Sc, c = rq.realq_saliency_clip(Sd, pct)
    assert np.array_equal(c.cpu().numpy().astype(np.float64), c_or)
    assert np.array_equal(Sc.cpu().numpy().astype(np.float64), Sc_or)
    rq.realq_saliency_clip(Sd, pct, S_out=Sd)          # in place
    assert torch.equal(Sd, Sc)


def _weighted_gpu(Xb, S, n, ng, chunks=(0,)):
    Hg = torch.zeros(ng, n, n, device="cuda")
    wsum = torch.zeros(ng, dtype=torch.float64, device="cuda")
    T = Xb.shape[0]
    bounds = list(chunks) + [T]
    ws = rq.workspace(rq.realq_hessian_weighted_workspace_size(n, max(b - a for a, b in zip(bounds[:-1], bounds[1:]))))
    for a, b in zip(bounds[:-1], bounds[1:]):
        rq.realq_hessian_accumulate_weighted(Xb[a:b], S[a:b], Hg, wsum, ws)
    rq.realq_workspace_status(ws)
    return Hg, wsum


def test_weighted_hessian_exact_on_perfect_squares():
    # s x is an integer that bf16 holds exactly (the low part is zero), every
    # product and partial sum is an integer below 2^24: the result is exact
    r = synth.rng(52, "weighted-exact")
    for n, T in ((128, 3000), (256, 5000), (96, 777)):
        X = r.integers(-7, 8, (T, n)).astype(np.float64)
        S = r.choice([0.0, 1.0, 4.0, 9.0, 16.0], size=(T, 4))
        Hg, wsum = _weighted_gpu(bf16_dev(synth.f32_to_bf16_bits(X)), dev(S), n, 4, chunks=(0, T // 3))
        Href, wref = oracle.weighted_hessian_sum([X], [S])
        assert np.array_equal(Hg.cpu().numpy().astype(np.float64), Href), (n, T)
        assert np.array_equal(wsum.cpu().numpy(), wref)


def test_weighted_hessian_within_the_split_rounding():
    r = synth.rng(53, "weighted-real")
    n, T = 256, 20000
    x = r.standard_normal((T, n))
    x[:, 7] *= 15.0
    X = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(x)).astype(np.float64)
    S, _ = oracle.saliency_clip(np.exp(1.0 * r.standard_normal((T, 4))), 0.99)
    S = S.astype(np.float32).astype(np.float64)
    Hg, wsum = _weighted_gpu(bf16_dev(synth.f32_to_bf16_bits(X)), dev(S), n, 4)
    Href, wref = oracle.weighted_hessian_sum([X], [S])
    A = np.abs(X)
    for g in range(4):
        absum = (A * S[:, g:g + 1]).T @ A                  # sum_t s |x_i x_j|
        d = np.sqrt(np.diag(Href[g]))
        # split of s x into two bf16 parts (2^-17) plus the tensor core's fp32
        # accumulation within a 1024-token chunk (64 MMAs, each adding its 16
        # products through a few truncating adds: ~64 x 5 x 2^-23 < 2^-14.5),
        # relative to the absolute sum; then the fp32 bound of the small cases
        bound = 2.0 ** -14 * absum + 2e-6 * np.sqrt(T) * np.outer(d, d)
        err = np.abs(Hg[g].cpu().numpy() - Href[g])
        assert np.all(err <= bound), (g, (err / bound).max())
        print(f"\ngroup {g}: max error / bound = {(err / bound).max():.3e}")
    np.testing.assert_allclose(wsum.cpu().numpy(), wref, rtol=1e-12)


def test_prepare_scaled_matches_oracle():
    # integer activations and perfect-square weights: the weighted Hessians are
    # exact on both sides, so this compares the scaled preparation alone
    r = synth.rng(54, "prepare-scaled")
    n, T = 192, 6000
    X = r.integers(-7, 8, (T, n)).astype(np.float64)
    X[:, 5] *= 3.0
    S = r.choice([1.0, 4.0, 9.0, 16.0], size=(T, 2), p=[0.7, 0.2, 0.07, 0.03])
    Hg, wsum = _weighted_gpu(bf16_dev(synth.f32_to_bf16_bits(X)), dev(S), n, 2)
    Href, wref = oracle.weighted_hessian_sum([X], [S])
    ws = rq.workspace(rq.realq_prepare_workspace_size(n))
    for g in range(2):
        U = torch.empty(n, n, device="cuda")
        Hb = torch.empty(n, n, device="cuda")
        dead = torch.empty(n, dtype=torch.uint8, device="cuda")
        rq.realq_hessian_prepare_scaled(Hg[g], float(wsum[g].item()), 0.01, U, Hb, dead, ws)
        ref = oracle.prepare(Href[g], wref[g], 0.01)
        Uref = oracle.inverse_upper_cholesky(ref["Hd"])
        assert np.abs(U.cpu().numpy() - Uref).max() <= 2e-4 * np.abs(Uref).max()
        np.testing.assert_allclose(Hb.cpu().numpy(), ref["Hbar"], rtol=1e-5, atol=1e-6 * np.abs(ref["Hbar"]).max())


# ------------------------------------------------ row-grouped OBS sweep ---
def _grouped_run(seed, m, n, T, ng, qkw, lr=None, correlated=False):
    # log-normal saliency (sigma 0.7) with three extreme tokens that the clipping
    # removes: after clipping, each H_g is as well conditioned as H (a
    # near rank-deficient H_g would make U_g depend on the last bits of H_g,
    # which no fp32 path reproduces against an fp64 oracle)
    case = synth.layer_case(seed, m, n, T, bf16=True, outliers=3)
    r = synth.rng(seed, "saliency")
    S = np.exp(0.7 * r.standard_normal((T, ng)))
    if correlated:
        # saliency that follows the outlier channels changes the shape of H_g
        oc = int(np.argmax(case.Xhat.var(axis=0)))
        S *= 1.0 + 5.0 * np.abs(case.Xhat[:, oc:oc + 1])
    S[r.integers(0, T, 3)] *= 1e8                           # gradient outliers (clipped)
    S = S.astype(np.float32).astype(np.float64)
    # oracle, from its own clipped saliency and Hessians
    Sc_or, _ = oracle.saliency_clip(S, 0.99)
    Hg_or, w_or = oracle.weighted_hessian_sum([case.Xhat], [Sc_or])
    H_or, T_ = oracle.hessian_sum([case.Xhat])
    bgd = None if lr is None else {"lr": lr, "steps_per_block": 1, "b_global_start": 1, "B_total": 1}
    kappa = max(np.linalg.cond(oracle.prepare(Hg_or[g], w_or[g])["Hd"]) for g in range(ng))
    orc = OracleSweep(lambda follow, grad_noise=None: oracle.realq_sweep(
        case.W0, H_or, T_, bits=qkw.get("bits", 4), group_size=qkw.get("group_size", 128),
        block_size=qkw.get("block_size", 128), bgd=bgd, F=case.F,
        obs_hessians=[(Hg_or[g], w_or[g]) for g in range(ng)], follow=follow, grad_noise=grad_noise))
    # GPU path
    X = bf16_dev(synth.f32_to_bf16_bits(case.Xhat))
    Sc, _ = rq.realq_saliency_clip(dev(S), 0.99)
    Hg, wsum = _weighted_gpu(X, Sc, n, ng)
    H, _, T_ = layer.accumulate([X], n)
    prep = layer.prepare(H, T_)
    ws = rq.workspace(rq.realq_prepare_workspace_size(n))
    Ug = torch.empty(ng, n, n, device="cuda")
    Hbg = torch.empty(ng, n, n, device="cuda")
    dg = torch.empty(ng, n, dtype=torch.uint8, device="cuda")
    for g in range(ng):
        rq.realq_hessian_prepare_scaled(Hg[g], float(wsum[g].item()), 0.01, Ug[g], Hbg[g], dg[g], ws)
    q = rq.quant_cfg(**qkw)
    b = None if lr is None else rq.bgd_cfg(lr)
    ngrp = -(-n // (qkw.get("group_size", 128) or n))
    W = torch.empty(m, n, device="cuda")
    codes = torch.empty(m, (n + 1) // 2, dtype=torch.uint8, device="cuda")
    scale = torch.empty(m, ngrp, device="cuda")
    zero = torch.empty(m, ngrp, dtype=torch.uint8, device="cuda")
    st = {}
    if lr is not None:
        st = {k: torch.empty(m, n, device="cuda") for k in ("adam_m", "adam_v", "bgd_disp")}
    wsq = rq.workspace(rq.realq_quantize_grouped_workspace_size(m, n, ng, q, b))
    t = rq.realq_quantize_layer_grouped(dev(case.W0), Ug, Hbg, dg, prep.Hbar, q, W, codes, scale, zero, bcfg=b,
                                        F=dev(case.F) if lr is not None else None, ws=wsq, **st)
    rq.realq_workspace_status(wsq)
    codes_np = unpack(codes.cpu().numpy(), n)
    _, _, rep = check_codes_and_scales(orc, codes_np, zero.cpu().numpy(), scale.cpu().numpy(), n, qkw,
                                       lr is not None, lr or 0.0, 1,
                                       f"grouped ng={ng} max cond(H_g,d)={kappa:.1f} ")
    if lr is not None:
        assert t == orc["adam_t"]
    g_ = qkw.get("group_size", 128) or n
    s_ = scale.cpu().numpy()[:, np.arange(n) // g_]
    z_ = zero.cpu().numpy()[:, np.arange(n) // g_].astype(np.float32)
    assert np.array_equal((s_ * (codes_np.astype(np.float32) - z_)).astype(np.float32), W.cpu().numpy())
    return rep


def test_grouped_sweep_gptq_mode():
    _grouped_run(55, 128, 256, 8000, 4, dict(group_size=64, block_size=64))


def test_grouped_sweep_with_block_gd():
    _grouped_run(56, 128, 384, 12000, 4, dict(group_size=128, block_size=128), lr=2e-4, correlated=True)


def test_grouped_sweep_ragged_rows_and_one_group():
    _grouped_run(57, 100, 192, 8000, 4, dict(group_size=64, block_size=64), lr=2e-4)
    _grouped_run(58, 96, 256, 8000, 1, dict(group_size=128, block_size=128), lr=2e-4, correlated=True)



def test_grouped_sweep_exact_hessians():
    # integer activations and integer saliencies: every weighted Hessian is
    # exact on both sides, so this checks the grouped sweep's logic alone
    r = synth.rng(59, "grouped-exact")
    m, n, T, ng = 128, 192, 3000, 4
    X = r.integers(-7, 8, (T, n)).astype(np.float64)
    X[:, 11] *= 4.0
    S = r.choice([1.0, 2.0, 4.0, 8.0], size=(T, ng), p=[0.6, 0.25, 0.1, 0.05])
    W0 = (r.standard_normal((m, n)) * 0.02).astype(np.float32).astype(np.float64)
    Z = r.standard_normal((m, 8))
    F = (0.5 * np.eye(m) + Z @ Z.T / 16).astype(np.float32).astype(np.float64)
    Hg_or, w_or = oracle.weighted_hessian_sum([X], [S])
    H_or, _ = oracle.hessian_sum([X])
    Xd = bf16_dev(synth.f32_to_bf16_bits(X))
    Hg, wsum = _weighted_gpu(Xd, dev(S), n, ng)
    assert np.array_equal(Hg.cpu().numpy().astype(np.float64), Hg_or)
    H, _, _ = layer.accumulate([Xd], n)
    prep = layer.prepare(H, T)
    ws = rq.workspace(rq.realq_prepare_workspace_size(n))
    Ug = torch.empty(ng, n, n, device="cuda")
    Hbg = torch.empty(ng, n, n, device="cuda")
    dg = torch.empty(ng, n, dtype=torch.uint8, device="cuda")
    for g in range(ng):
        rq.realq_hessian_prepare_scaled(Hg[g], float(wsum[g].item()), 0.01, Ug[g], Hbg[g], dg[g], ws)
    for lr in (None, 2e-4):
        qkw = dict(group_size=64, block_size=64)
        bgd = None if lr is None else {"lr": lr, "steps_per_block": 1, "b_global_start": 1, "B_total": 1}
        orc = OracleSweep(lambda follow, grad_noise=None, bgd=bgd: oracle.realq_sweep(
            W0, H_or, T, group_size=64, block_size=64, bgd=bgd, F=F,
            obs_hessians=[(Hg_or[g], w_or[g]) for g in range(ng)], follow=follow, grad_noise=grad_noise))
        q = rq.quant_cfg(**qkw)
        b = None if lr is None else rq.bgd_cfg(lr)
        W = torch.empty(m, n, device="cuda")
        codes = torch.empty(m, n // 2, dtype=torch.uint8, device="cuda")
        scale = torch.empty(m, 3, device="cuda")
        zero = torch.empty(m, 3, dtype=torch.uint8, device="cuda")
        st = {} if lr is None else {k: torch.empty(m, n, device="cuda") for k in ("adam_m", "adam_v", "bgd_disp")}
        wsq = rq.workspace(rq.realq_quantize_grouped_workspace_size(m, n, ng, q, b))
        rq.realq_quantize_layer_grouped(dev(W0), Ug, Hbg, dg, prep.Hbar, q, W, codes, scale, zero, bcfg=b,
                                        F=dev(F) if lr else None, ws=wsq, **st)
        codes_np = unpack(codes.cpu().numpy(), n)
        check_codes_and_scales(orc, codes_np, zero.cpu().numpy(), scale.cpu().numpy(), n, qkw, lr is not None,
                               lr or 0.0, 1, "grouped exact-H ")


def test_block_scheduler_saliency_groups():
    # the scheduler's grouped variant on a small two-input block: every module
    # matches the oracle's row-grouped sweep from its own clipped saliency
    from paper_2609_00049_gb300.block import BlockInput, BlockModule, BlockQuantizer
    r = synth.rng(60, "block-grouped")
    T, ng = 6000, 4
    ins = {"a": 128, "b": 256}
    mods = [("m1", 64, "a"), ("m2", 128, "a"), ("m3", 96, "b")]
    x_bits = {k: synth.f32_to_bf16_bits(r.standard_normal((T, n)) * (1 + 9 * (r.random(n) < 0.02)))
              for k, n in ins.items()}
    Wf = {nm: synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(r.standard_normal((m, ins[i])) * 0.02))
          for nm, m, i in mods}
    Ff, Sal = {}, {}
    for nm, m, _ in mods:
        z = r.standard_normal((m, 4))
        Ff[nm] = (np.eye(m) * 0.5 + z @ z.T / 8).astype(np.float32)
        s = np.exp(0.7 * r.standard_normal((T, ng)))
        s[r.integers(0, T, 4)] *= 1e7
        Sal[nm] = s.astype(np.float32)
    qcfg = rq.quant_cfg(4, 64, 64, 0, 0.01)
    bq = BlockQuantizer([BlockInput(k, n, T) for k, n in ins.items()],
                        [BlockModule(nm, m, ins[i], i) for nm, m, i in mods], qcfg, 2e-4, 1, saliency_groups=ng)
    bq.run({k: bf16_dev(v) for k, v in x_bits.items()}, {nm: dev(w) for nm, w in Wf.items()},
           {nm: dev(f) for nm, f in Ff.items()}, saliency={nm: dev(v) for nm, v in Sal.items()})
    torch.cuda.synchronize()
    bq.check_status()
    bstart = 1
    for nm, m, i in mods:
        x = synth.bf16_bits_to_f32(x_bits[i]).astype(np.float64)
        Sc, _ = oracle.saliency_clip(Sal[nm].astype(np.float64), 0.99)
        Hg, w = oracle.weighted_hessian_sum([x], [Sc])
        Hs, _ = oracle.hessian_sum([x])
        orc = OracleSweep(lambda follow, grad_noise=None, W=Wf[nm], F=Ff[nm], Hs=Hs, Hg=Hg, w=w, b0=bstart: oracle.realq_sweep(
            W.astype(np.float64), Hs, T, group_size=64, block_size=64,
            bgd={"lr": 2e-4, "steps_per_block": 1, "b_global_start": b0, "B_total": 1}, F=F,
            obs_hessians=[(Hg[g], w[g]) for g in range(ng)], follow=follow, grad_noise=grad_noise))
        bstart += ins[i] // 64
        o = bq.out[nm]
        codes = unpack(o["codes"].cpu().numpy(), ins[i])
        qkw = dict(group_size=64, block_size=64)
        check_codes_and_scales(orc, codes, o["zero"].cpu().numpy(), o["scale"].cpu().numpy(), ins[i], qkw, True,
                               2e-4, 1, f"block grouped {nm} ")


# ------------------------------------------------- mini-batch Block-GD ---
@pytest.mark.parametrize("start,steps", [(1, 1), (3, 1), (2, 2)])
def test_minibatch_block_gd(start, steps):
    case = synth.layer_case(61, 128, 384, 8000, bf16=True, outliers=3)
    K, Tm = 4, 2000
    qkw = dict(group_size=128, block_size=128)
    mbs = [oracle.hessian_sum([case.Xhat[k * Tm:(k + 1) * Tm]]) for k in range(K)]
    Hs, T = oracle.hessian_sum([case.Xhat])
    bgd = {"lr": 2e-4, "steps_per_block": steps, "b_global_start": start, "B_total": 1, "minibatches": mbs}
    orc = OracleSweep(lambda follow, grad_noise=None: oracle.realq_sweep(case.W0, Hs, T, group_size=128, block_size=128, bgd=bgd,
                                                        F=case.F, follow=follow, grad_noise=grad_noise))
    X = bf16_dev(synth.f32_to_bf16_bits(case.Xhat))
    H, _, _ = layer.accumulate([X], 384)
    prep = layer.prepare(H, T)
    Hmb = torch.empty(K, 384, 384, device="cuda")
    for k in range(K):
        Hk, _, _ = layer.accumulate([X[k * Tm:(k + 1) * Tm]], 384)
        rq.realq_scale_moment(Hk, Tm, Hmb[k])
    q = rq.quant_cfg(**qkw)
    b = rq.bgd_cfg(2e-4, steps_per_block=steps, b_global_start=start)
    m, n = 128, 384
    W = torch.empty(m, n, device="cuda")
    codes = torch.empty(m, n // 2, dtype=torch.uint8, device="cuda")
    scale = torch.empty(m, 3, device="cuda")
    zero = torch.empty(m, 3, dtype=torch.uint8, device="cuda")
    st = {k: torch.empty(m, n, device="cuda") for k in ("adam_m", "adam_v", "bgd_disp")}
    ws = rq.workspace(rq.realq_quantize_minibatch_workspace_size(m, n, K, q, b))
    t = rq.realq_quantize_layer_minibatch(dev(case.W0), prep.U, prep.Hbar, Hmb, q, W, codes, scale, zero,
                                          dead=prep.dead, bcfg=b, F=dev(case.F), ws=ws, **st)
    rq.realq_workspace_status(ws)
    assert t == orc["adam_t"] == 2 * steps
    c = unpack(codes.cpu().numpy(), n)
    check_codes_and_scales(orc, c, zero.cpu().numpy(), scale.cpu().numpy(), n, qkw, True, 2e-4, steps,
                           f"mini-batch start={start} steps={steps} ")


def test_prepare_deferred_status():
    # the capturable prepare leaves the failing column in its workspace
    n = 96
    H = -torch.eye(n, device="cuda") * 10.0
    U, Hbar = torch.empty(n, n, device="cuda"), torch.empty(n, n, device="cuda")
    dead = torch.empty(n, dtype=torch.uint8, device="cuda")
    ws = rq.workspace(rq.realq_prepare_workspace_size(n))
    rq.realq_hessian_prepare_deferred(H, 10, 0.01, U, Hbar, dead, ws)
    with pytest.raises(rq.RealqError) as ei:
        rq.realq_prepare_status(ws)
    assert ei.value.status == rq.REALQ_ERR_NOT_SPD and ei.value.fail_col == n - 1
    case = synth.layer_case(23, 4, n, 4 * n, outliers=2)
    Href, T = oracle.hessian_sum([case.Xhat])
    rq.realq_hessian_prepare_deferred(dev(Href), T, 0.01, U, Hbar, dead, ws)
    assert rq.realq_prepare_status(ws) == -1
    ref = oracle.prepare(Href, T, 0.01)
    Uref = oracle.inverse_upper_cholesky(ref["Hd"])
    assert np.abs(U.cpu().numpy() - Uref).max() <= 2e-4 * np.abs(Uref).max()


@pytest.mark.parametrize("variant", ["plain", "minibatch", "w4a4", "host"])
def test_block_graph_replay_matches_eager(variant):
    # capture() / capture_host() and replay() give the eager step's outputs
    # bit for bit, and a replay recomputes them (outputs are cleared first)
    from paper_2609_00049_gb300.block import BlockInput, BlockModule, BlockQuantizer
    r = synth.rng(44, "block-graph-" + variant)
    T = 4096 + 320
    ins = {"a": 128, "b": 192}
    mods = [("m1", 64, "a"), ("m2", 200, "a"), ("m3", 96, "b")]
    x_bits = {k: synth.f32_to_bf16_bits(r.standard_normal((T, n)) * (1 + 9 * (r.random(n) < 0.02)))
              for k, n in ins.items()}
    Wf = {nm: synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(r.standard_normal((m, ins[i])) * 0.02))
          for nm, m, i in mods}
    Ff = {}
    for nm, m, _ in mods:
        z = r.standard_normal((m, 4))
        Ff[nm] = (np.eye(m) * 0.5 + z @ z.T / 8).astype(np.float32)
    qcfg = rq.quant_cfg(4, 64, 64, 0, 0.01)
    kw = dict(minibatch_tokens=1024) if variant == "minibatch" else {}
    if variant == "w4a4":
        kw = dict(act_quant=(4, 0.9))
    if variant == "host":
        kw = dict(host_chunk_tokens=1024)   # five chunks, the last one ragged
    bq = BlockQuantizer([BlockInput(k, n, T) for k, n in ins.items()],
                        [BlockModule(nm, m, ins[i], i) for nm, m, i in mods], qcfg, 2e-4, 1, **kw)
    X = {k: bf16_dev(v) for k, v in x_bits.items()}
    W0 = {nm: dev(w) for nm, w in Wf.items()}
    F = {nm: dev(f) for nm, f in Ff.items()}
    keys = ("codes", "scale", "zero", "W")
    if variant == "host":
        # chunked accumulation sums in another order than the one-shot
        # Hessian: the eager reference is run_host itself
        X_h = {k: v.cpu().pin_memory() for k, v in X.items()}
        W_h = {k: v.cpu().pin_memory() for k, v in W0.items()}
        F_h = {k: v.cpu().pin_memory() for k, v in F.items()}
        out_h = {nm: {k: torch.empty_like(bq.out[nm][k], device="cpu").pin_memory() for k in keys[:3]}
                 for nm, _, _ in mods}
        bq.run_host(X_h, W_h, F_h, out_h)
    else:
        bq.run(X, W0, F)
    torch.cuda.synchronize()
    bq.check_status()
    eager = {nm: {k: bq.out[nm][k].clone() for k in keys} for nm, _, _ in mods}
    if variant == "host":
        h2d, d2h = bq.capture_host(X_h, W_h, F_h, out_h)
        assert h2d == sum(v.numel() * v.element_size() for d in (X_h, W_h, F_h) for v in d.values())
        assert d2h == sum(v.numel() * v.element_size() for d in out_h.values() for v in d.values())
    else:
        bq.capture(X, W0, F)
    for _ in range(2):
        for nm, _, _ in mods:
            for k in keys:
                bq.out[nm][k].fill_(0 if bq.out[nm][k].dtype == torch.uint8 else float("nan"))
            if variant == "host":
                for k in keys[:3]:
                    out_h[nm][k].fill_(0 if out_h[nm][k].dtype == torch.uint8 else float("nan"))
        bq.replay()
        torch.cuda.synchronize()
        bq.check_status()
        for nm, _, _ in mods:
            for k in keys:
                assert torch.equal(bq.out[nm][k], eager[nm][k]), (variant, nm, k)
            if variant == "host":
                for k in keys[:3]:
                    assert torch.equal(out_h[nm][k], eager[nm][k].cpu()), (variant, nm, k)


@pytest.mark.parametrize("clip,start,steps", [(0.95, 1, 1), (0.95, 2, 2), (0.9, 3, 1), (1.0, 1, 1)])
def test_token_block_gd_with_output_clipping(clip, start, steps):
    # token-form mini-batch Block-GD with per-token output clipping against
    # the oracle's token-form sweep; 8000 tokens in mini-batches of 2048 (the
    # last one 1856 tokens); clip = 1 scales nothing (the moment form)
    case = synth.layer_case(62, 128, 384, 8000, bf16=True, outliers=3)
    Tm = 2048
    parts = [case.Xhat[k * Tm:(k + 1) * Tm] for k in range(-(-8000 // Tm))]
    Hs, T = oracle.hessian_sum([case.Xhat])
    bgd = {"lr": 2e-4, "steps_per_block": steps, "b_global_start": start, "B_total": 1,
           "minibatch_tokens": parts, "a_loss_clip": clip}
    orc = OracleSweep(lambda follow, grad_noise=None: oracle.realq_sweep(case.W0, Hs, T, group_size=128, block_size=128, bgd=bgd,
                                                        F=case.F, follow=follow, grad_noise=grad_noise))
    qkw = dict(group_size=128, block_size=128)
    X = bf16_dev(synth.f32_to_bf16_bits(case.Xhat))
    H, _, _ = layer.accumulate([X], 384)
    prep = layer.prepare(H, T)
    q = rq.quant_cfg(**qkw)
    b = rq.bgd_cfg(2e-4, steps_per_block=steps, b_global_start=start)
    m, n = 128, 384
    W = torch.empty(m, n, device="cuda")
    codes = torch.empty(m, n // 2, dtype=torch.uint8, device="cuda")
    scale = torch.empty(m, 3, device="cuda")
    zero = torch.empty(m, 3, dtype=torch.uint8, device="cuda")
    st = {k: torch.empty(m, n, device="cuda") for k in ("adam_m", "adam_v", "bgd_disp")}
    ws = rq.workspace(rq.realq_quantize_tokens_workspace_size(m, n, Tm, q, b))
    t = rq.realq_quantize_layer_tokens(dev(case.W0), prep.U, prep.Hbar, X, Tm, clip, q, W, codes, scale, zero,
                                       dead=prep.dead, bcfg=b, F=dev(case.F), ws=ws, **st)
    rq.realq_workspace_status(ws)
    assert t == orc["adam_t"] == 2 * steps
    c = unpack(codes.cpu().numpy(), n)
    _, fol, _ = check_codes_and_scales(orc, c, zero.cpu().numpy(), scale.cpu().numpy(), n, qkw, True, 2e-4, steps,
                                       f"token form clip={clip} start={start} steps={steps} ")
    print(f"max|deq - oracle|={np.abs(W.cpu().numpy() - fol['deq']).max():.2e}")



@pytest.mark.parametrize("with_next", [False, True])
def test_traced_block_losses(with_next):
    # the surrogate before and after every block's Block-GD step against the
    # oracle's record of the same values (1e-3 relative, the loss tolerance);
    # with the sliding window the trace uses each block's blended F_eff
    case = synth.layer_case(28, 96, 320, 1200, with_next=True)
    qkw = dict(group_size=64, block_size=64)
    kw = dict(b_global_start=3, B_total=9) if with_next else {}
    Hs, T = oracle.hessian_sum([case.Xhat])
    orc = OracleSweep(lambda follow, grad_noise=None: oracle.realq_sweep(
        case.W0, Hs, T, group_size=64, block_size=64,
        bgd={"lr": 2e-4, "steps_per_block": 1, "b_global_start": kw.get("b_global_start", 1),
             "B_total": kw.get("B_total", 1)},
        F=case.F, F_next=case.F_next if with_next else None, follow=follow, grad_noise=grad_noise))
    H, _, T_ = layer.accumulate([dev(case.Xhat)], 320)
    prep = layer.prepare(H, T_)
    q = rq.quant_cfg(**qkw)
    b = rq.bgd_cfg(2e-4, **kw)
    m, n = 96, 320
    nb = n // 64
    W = torch.empty(m, n, device="cuda")
    codes = torch.empty(m, n // 2, dtype=torch.uint8, device="cuda")
    scale = torch.empty(m, n // 64, device="cuda")
    zero = torch.empty(m, n // 64, dtype=torch.uint8, device="cuda")
    st = {k: torch.empty(m, n, device="cuda") for k in ("adam_m", "adam_v", "bgd_disp")}
    ws = rq.workspace(rq.realq_quantize_workspace_size(m, n, q, b, with_next))
    bl = torch.full((nb, 2), float("nan"), device="cuda")
    tws = rq.workspace(rq.realq_quantize_trace_workspace_size(m, n))
    rq.realq_quantize_layer(dev(case.W0), prep.U, prep.Hbar, q, W, codes, scale, zero, dead=prep.dead, bcfg=b,
                            F=dev(case.F), F_next=dev(case.F_next) if with_next else None, ws=ws,
                            block_loss=bl, trace_ws=tws, **st)
    rq.realq_workspace_status(ws)
    got = bl.cpu().numpy()
    assert np.isnan(got[nb - 1]).all()          # the last block takes no step
    # on the CUDA path's branch at rounding ties (tests/parity.py)
    _, fol, _ = check_codes_and_scales(orc, unpack(codes.cpu().numpy(), n), zero.cpu().numpy(),
                                       scale.cpu().numpy(), n, qkw, True, 2e-4, 1, "traced ")
    for blk, alpha, before, after in fol["block_loss"]:
        print(f"\nblock {blk} alpha {alpha:.3f}: before {got[blk, 0]:.6e} / {before:.6e}, "
              f"after {got[blk, 1]:.6e} / {after:.6e}")
        assert abs(got[blk, 0] - before) <= 1e-3 * abs(before)
        assert abs(got[blk, 1] - after) <= 1e-3 * abs(after)


# ----------------------------------------------- Block-GD product precision ---
@pytest.mark.parametrize("products,tile", [(0, 0), (1, 1), (1, 2)])
def test_bgd_products_match_the_oracle(products, tile):
    # the plain Block-GD products as tf32x3 (0) and as f16x3 (1, the default
    # where m, n and the block are multiples of 8: fp16 planes with
    # power-of-two row scales) on either output tile: shapes no multiple of a
    # tile, a dead channel, the sliding window with perturbed inputs, bf16
    # weights, and a sweep resumed mid-way (M rebuilt from the displacement)
    rq.realq_set_bgd_products(products)
    rq.realq_set_tensor_tile(tile)
    try:
        case = synth.layer_case(27, 200, 328, 1500, outliers=2, dead_cols=(7,))
        for qkw in (dict(group_size=64, block_size=64), dict(group_size=128, block_size=128)):
            orc, out, prep, W0 = _oracle_and_gpu(case, qkw, bgd=2e-4)
            _check(orc, out, case, qkw, True, prep=prep, W0=W0, lr=2e-4)
        case = synth.layer_case(26, 96, 320, 1200, with_next=True, perturbed=True)
        qkw = dict(group_size=64, block_size=64)
        orc, out, prep, W0 = _oracle_and_gpu(case, qkw, bgd=2e-4, with_next=True, b_global_start=3, B_total=9,
                                             use_dbar=True)
        _check(orc, out, case, qkw, True, lr=2e-4)
        test_bf16_weights()
        test_resume_matches_single_call()
    finally:
        rq.realq_set_bgd_products(1)
        rq.realq_set_tensor_tile(0)


@pytest.mark.parametrize("qkw,m,n,bf16", [(dict(group_size=128, block_size=128), 200, 328, False),
                                          (dict(group_size=64, block_size=64), 1024, 1536, True),
                                          (dict(group_size=128, block_size=128), 512, 2048, False)])
def test_persistent_products_are_bit_identical(qkw, m, n, bf16):
    # the wide-tile f16x3 products as persistent kernels (the epilogue of one
    # tile overlapping the next tile's MMAs, two TMEM accumulators) and as one
    # tile per CTA: the same MMAs per tile and the same epilogue arithmetic,
    # so the whole sweep with Block-GD (ragged tiles, several tiles per CTA,
    # the K-split store of the next block's columns) gives the same bits
    case = synth.layer_case(79, m, n, 2 * n, outliers=2, bf16=bf16)
    H, _, T = layer.accumulate([dev(case.Xhat)], n)
    prep = layer.prepare(H, T)
    W0 = dev(case.W0, torch.bfloat16) if bf16 else dev(case.W0)
    outs = []
    rq.realq_set_tensor_tile(2)
    try:
        for mode in (0, 2, 1):   # (1 last: the default stays set)
            rq.realq_set_tensor_overlap(mode)
            outs.append(layer.quantize(W0, prep, rq.quant_cfg(**qkw), rq.bgd_cfg(2e-4, steps_per_block=2),
                                       F=dev(case.F)))
            torch.cuda.synchronize()
    finally:
        rq.realq_set_tensor_overlap(1)
        rq.realq_set_tensor_tile(0)
    for o in outs[1:]:
        for k in ("codes", "scale", "zero", "W"):
            assert torch.equal(getattr(outs[0], k), getattr(o, k)), k


# ------------------------------------------------- tensor-core tile shapes ---
@pytest.mark.parametrize("tile", [1, 2])
def test_tensor_tiles_match_the_oracle(tile):
    # every tf32x3 product forced onto one output tile (1: 128 x 128 with
    # 32-wide K slices, 2: 128 x 256 with 16-wide slices): the plain sweep with
    # Block-GD on ragged shapes (M and N no multiple of either tile), the
    # sliding window with perturbed inputs, the row-grouped sweep (the
    # corrected gradient factor), mini-batch moments and the token form (the
    # store epilogue and the K split)
    rq.realq_set_tensor_tile(tile)
    try:
        case = synth.layer_case(24, 200, 300, 1500, outliers=2, dead_cols=(7,))
        for qkw in (dict(group_size=64, block_size=64), dict(group_size=128, block_size=128)):
            orc, out, prep, W0 = _oracle_and_gpu(case, qkw, bgd=2e-4)
            _check(orc, out, case, qkw, True, prep=prep, W0=W0, lr=2e-4)
        case = synth.layer_case(26, 96, 320, 1200, with_next=True, perturbed=True)
        qkw = dict(group_size=64, block_size=64)
        orc, out, prep, W0 = _oracle_and_gpu(case, qkw, bgd=2e-4, with_next=True, b_global_start=3, B_total=9,
                                             use_dbar=True)
        _check(orc, out, case, qkw, True, lr=2e-4)
        _grouped_run(56, 128, 384, 12000, 4, dict(group_size=128, block_size=128), lr=2e-4, correlated=True)
        test_minibatch_block_gd(2, 2)
        test_token_block_gd_with_output_clipping(0.95, 2, 2)
    finally:
        rq.realq_set_tensor_tile(0)


# --------------------------------------------------- the quantizer kernels ---
@pytest.mark.parametrize("qkw,m,n", [(dict(group_size=128, block_size=128), 200, 384),
                                     (dict(group_size=0, block_size=64, symmetric=1), 96, 200),
                                     (dict(group_size=32, block_size=32), 64, 96),
                                     (dict(group_size=128, block_size=128), 1024, 520)])
def test_quantizer_kernels_agree_bit_for_bit(qkw, m, n):
    # the pipelined column-serial kernel and the barrier-phased one perform
    # the same operations in the same order: the whole sweep (with Block-GD,
    # ragged last blocks, per-row groups, 1024 rows = 32 CTAs) is the same
    # bits with either
    case = synth.layer_case(77, m, n, 3 * n, outliers=2)
    H, _, T = layer.accumulate([dev(case.Xhat)], n)
    prep = layer.prepare(H, T)
    outs = []
    for mode in (0, 1):
        rq.realq_set_quant_kernel(mode)
        try:
            outs.append(layer.quantize(dev(case.W0), prep, rq.quant_cfg(**qkw), rq.bgd_cfg(2e-4), F=dev(case.F)))
            torch.cuda.synchronize()
        finally:
            rq.realq_set_quant_kernel(0)
    for k in ("codes", "scale", "zero", "W"):
        assert torch.equal(getattr(outs[0], k), getattr(outs[1], k)), k
