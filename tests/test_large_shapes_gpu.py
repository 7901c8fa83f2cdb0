"""Full-size parity of the three larger decoder-block shapes with the fp64
oracle, run as the benchmark runs them (the block scheduler's step captured
into a CUDA graph and replayed, Block-GD at each shape's learning rate):

  llama3.1-8b   hidden 4096, Student-t(4) activations, the two-block sliding
                window (B_total = 304): q, k, v and o_proj (n = 4096) on the
                attention input and the attention output
  qwen3-32b     hidden 5120, 0.5 % outlier channels x50: k and v_proj
                (n = 5120) on the attention input
  llama3.1-70b  hidden 8192, 524,288 tokens of Student-t(3): k and v_proj
                (n = 8192) on the attention input; and down_proj on the MLP
                hidden state, n = 28672, whose H, U and H̄ (3.3 GB each) the
                one GPU holds

Each subset runs with the column-block indices (b_global, B_total) it has in
the whole block.  For every input the oracle can factor, it computes its own
fp64 Hessian over all T tokens and the literal sweep (every compensation and
Schur downdate applied at once, Block-GD with Adam), and the CUDA path must
match it:
  Hessian    every entry within 2e-6 sqrt(T) sqrt(H_ii H_jj) (fp32
             accumulation over T tokens)
  U          max |ΔU| <= 2e-4 max |U|
  codes      >= 99.9 % identical, none unexplained on the CUDA path's branch
             at rounding ties (tests/parity.py); scales within 1e-5 apart
             from the counted Adam-sign groups of reading R18
  surrogate  the CUDA path's loss of its output within 1e-3 relative of the
             oracle's loss of the oracle's output (moment form with the
             oracle's fp64 H̄, equal to the token form for these unperturbed
             inputs)
For down_in (n = 28672), whose literal downdating sweep would move 8 10^12
words on the host, the checks are sampled: the oracle's X̂_Sᵀ X̂_S on 48
columns and its whole diagonal, U H_d Uᵀ v = v on probes (relative residual
below 1e-4 = 10 sqrt(n) u), and the grid properties of down_proj's output.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2609_00049_gb300 as rq
from paper_2609_00049_gb300.block import BlockInput, BlockModule, BlockQuantizer
from parity import OracleSweep, check_codes_and_scales, unpack

pytestmark = pytest.mark.gpu

# (inputs, modules) run on the GPU; the oracle sweeps every module whose input is in ORACLE_INPUTS
RUN = {
    "llama3.1-8b": (("attn_in", "o_in"), ("q_proj", "k_proj", "v_proj", "o_proj")),
    "qwen3-32b": (("attn_in",), ("k_proj", "v_proj")),
    "llama3.1-70b": (("attn_in", "down_in"), ("k_proj", "v_proj", "down_proj")),
}
ORACLE_INPUTS = ("attn_in", "o_in")


def _global_blocks(wl):
    start, b = {}, 1
    for md in wl.modules:
        start[md.name] = b
        b += -(-md.n // wl.block_size)
    return start, b - 1


def _x64(bits):
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


@pytest.fixture(scope="module", params=list(RUN))
def shape_run(request):
    from paper_2609_00049_gb300 import build as b
    b.build()
    rq.lib()
    wl = synth.workloads()[request.param]
    ins, mods = RUN[wl.name]
    dev = torch.device("cuda", 0)
    x_bits, X = {}, {}
    for nm in ins:
        x_bits[nm] = synth.xhat_full(wl, nm, as_bits=True, threads=16)
        X[nm] = torch.from_numpy(x_bits[nm].view(np.int16)).to(dev).view(torch.bfloat16)
    modules = [md for md in wl.modules if md.name in mods]
    w_bits = {md.name: synth.weights(wl, md) for md in modules}
    W0 = {k: torch.from_numpy(v.view(np.int16)).to(dev).view(torch.bfloat16) for k, v in w_bits.items()}
    F_np = {md.name: synth.fisher(wl, md) for md in modules}
    F = {k: torch.from_numpy(v).to(dev) for k, v in F_np.items()}
    Fn_np, F_next = None, None
    if wl.sliding_window:
        Fn_np = {md.name: synth.fisher(wl, md, "F_next") for md in modules}
        F_next = {k: torch.from_numpy(v).to(dev) for k, v in Fn_np.items()}
    start, B_total = _global_blocks(wl)
    qcfg = rq.quant_cfg(wl.bits, wl.group_size, wl.block_size, wl.symmetric, wl.damp_frac)
    bq = BlockQuantizer([BlockInput(nm, wl.inputs[nm].n, wl.inputs[nm].T) for nm in ins],
                        [BlockModule(md.name, md.m, md.n, md.input) for md in modules], qcfg, wl.lr,
                        wl.steps_per_block, sliding_window=wl.sliding_window, device=dev,
                        b_global_start=start, B_total=B_total)
    bq.capture(X, W0, F, F_next)
    for o in bq.out.values():
        for k in ("codes", "scale", "zero", "W"):
            o[k].fill_(0 if o[k].dtype == torch.uint8 else float("nan"))
    bq.replay()
    torch.cuda.synchronize()
    bq.check_status()
    del X
    yield dict(wl=wl, bq=bq, x_bits=x_bits, w_bits=w_bits, modules=modules, F=F_np, F_next=Fn_np,
               start=start, B_total=B_total)
    del bq
    torch.cuda.empty_cache()


@pytest.fixture(scope="module")
def oracle_H(shape_run):
    """The oracle's own Hessian of every input it can factor, over all T tokens."""
    wl, out = shape_run["wl"], {}
    for nm, bits in shape_run["x_bits"].items():
        if nm not in ORACLE_INPUTS:
            continue
        spec = wl.inputs[nm]
        H, T = oracle.hessian_sum(_x64(bits[c:c + 8192]) for c in range(0, spec.T, 8192))
        assert T == spec.T
        out[nm] = H
    return out


def test_hessians_against_the_oracle(shape_run, oracle_H):
    wl, bq = shape_run["wl"], shape_run["bq"]
    for nm, Href in oracle_H.items():
        spec = wl.inputs[nm]
        H = bq.state[nm]["H"].cpu().numpy().astype(np.float64)
        scale = np.sqrt(np.outer(np.diag(Href), np.diag(Href)))
        err = np.abs(H - Href) / scale
        print(f"\n{wl.name} {nm}: n={spec.n} T={spec.T} max scaled error {err.max():.2e} "
              f"(bound {2e-6 * np.sqrt(spec.T):.2e})")
        assert err.max() < 2e-6 * np.sqrt(spec.T)
        ref = oracle.prepare(Href, spec.T, wl.damp_frac)
        Uref = oracle.inverse_upper_cholesky(ref["Hd"])
        U = bq.state[nm]["U"].cpu().numpy().astype(np.float64)
        rel = np.abs(U - Uref).max() / np.abs(Uref).max()
        print(f"{wl.name} {nm}: max|dU|/max|U| = {rel:.2e}")
        assert rel <= 2e-4
        assert np.all(np.tril(U, -1) == 0)
        assert np.array_equal(bq.state[nm]["dead"].cpu().numpy().astype(bool), ref["dead"])


def test_sweeps_against_the_oracle(shape_run, oracle_H):
    wl, bq = shape_run["wl"], shape_run["bq"]
    qkw = dict(bits=wl.bits, group_size=wl.group_size, block_size=wl.block_size)
    for md in shape_run["modules"]:
        if md.input not in oracle_H:
            continue
        spec = wl.inputs[md.input]
        W0 = synth.bf16_bits_to_f32(shape_run["w_bits"][md.name]).astype(np.float64)
        bgd = dict(lr=wl.lr, steps_per_block=wl.steps_per_block, b_global_start=shape_run["start"][md.name],
                   B_total=shape_run["B_total"] if wl.sliding_window else 1)
        Fn = shape_run["F_next"][md.name] if wl.sliding_window else None
        orc = OracleSweep(lambda follow, grad_noise=None: oracle.realq_sweep(
            W0, oracle_H[md.input], spec.T, bits=wl.bits, group_size=wl.group_size, block_size=wl.block_size,
            symmetric=bool(wl.symmetric), damp_frac=wl.damp_frac, bgd=bgd, F=shape_run["F"][md.name],
            F_next=Fn, record=False, follow=follow, grad_noise=grad_noise), eager=False)
        o = bq.out[md.name]
        nb = -(-md.n // wl.block_size)
        codes = unpack(o["codes"].cpu().numpy(), md.n)
        # (one oracle run, on the CUDA path's branch at rounding ties)
        _, fol, rep = check_codes_and_scales(orc, codes, o["zero"].cpu().numpy(), o["scale"].cpu().numpy(),
                                             md.n, qkw, True, wl.lr, wl.steps_per_block,
                                             f"{wl.name} {md.name} {md.m}x{md.n} ", plain_first=False,
                                             probe_scales=False)
        assert o["adam_t"] == fol["adam_t"] == (nb - 1) * wl.steps_per_block
        # the surrogate (Eq. fisher_loss at the layer level, the last block's
        # F_eff): the CUDA path's own value of its output against the
        # oracle's token form of the oracle's output
        alpha = oracle.sliding_alpha(bgd["b_global_start"] + nb - 1, bgd["B_total"])
        Feff = shape_run["F"][md.name].astype(np.float64)
        if Fn is not None:
            Feff = alpha * Feff + (1.0 - alpha) * Fn.astype(np.float64)
        # (the moment form with the oracle's own fp64 H̄: the token form's
        # value for unperturbed inputs, pinned to 1e-12 in the oracle's pins;
        # over all 262,144-524,288 tokens the token form costs minutes here)
        L_or = oracle.surrogate_moment(fol["deq"], W0, oracle_H[md.input] / spec.T, Feff)
        s_in = bq.state[md.input]
        ws = rq.workspace(rq.realq_surrogate_workspace_size(md.m, md.n))
        loss = torch.zeros(1, device="cuda")
        W0d = torch.from_numpy(W0.astype(np.float32)).cuda()
        rq.realq_surrogate_loss(o["W"], W0d, s_in["Hbar"], torch.from_numpy(Feff.astype(np.float32)).cuda(), loss,
                                ws)
        L_gpu = float(loss.item())
        print(f"{wl.name} {md.name}: surrogate gpu {L_gpu:.6e} oracle {L_or:.6e} "
              f"(rel {abs(L_gpu - L_or) / L_or:.2e})")
        assert abs(L_gpu - L_or) <= 1e-3 * L_or
        del W0d, ws


def test_wide_input_sampled_hessian_and_factor(shape_run):
    wl, bq = shape_run["wl"], shape_run["bq"]
    r = synth.rng(81, "large-hessian", wl.name)
    for nm, bits in shape_run["x_bits"].items():
        if nm in ORACLE_INPUTS:
            continue
        spec = wl.inputs[nm]
        out = synth.outlier_channels(wl, spec)
        S = np.sort(np.unique(np.concatenate([out[:16], r.choice(spec.n, 48, replace=False)]))[:48])
        Hs, T = oracle.hessian_sum(_x64(bits[c:c + 8192][:, S]) for c in range(0, spec.T, 8192))
        assert T == spec.T
        Sd = torch.from_numpy(S).cuda()
        Hg = bq.state[nm]["H"][Sd][:, Sd].double().cpu().numpy()
        err = np.abs(Hg - Hs) / np.sqrt(np.outer(np.diag(Hs), np.diag(Hs)))
        # the whole diagonal, H_jj = sum_t x_tj^2 (a bf16 square is exact in
        # fp32; the sum is taken in fp64)
        diag = np.zeros(spec.n)
        for c in range(0, spec.T, 4096):
            x = synth.bf16_bits_to_f32(bits[c:c + 4096])
            diag += np.sum(x * x, axis=0, dtype=np.float64)
        dg = torch.diagonal(bq.state[nm]["H"]).double().cpu().numpy()
        derr = np.abs(dg - diag) / diag
        print(f"\n{wl.name} {nm}: n={spec.n} T={spec.T} sampled max scaled error {err.max():.2e}, "
              f"diagonal max rel error {derr.max():.2e} (bound {2e-6 * np.sqrt(spec.T):.2e})")
        assert err.max() < 2e-6 * np.sqrt(spec.T)
        assert derr.max() < 2e-6 * np.sqrt(spec.T)
        assert np.array_equal(bq.state[nm]["dead"].cpu().numpy().astype(bool), diag == 0)
        # U H_d Uᵀ = I on fp64 probes (H_d the damped H̄ the kernels factor)
        s = bq.state[nm]
        U = s["U"]
        assert torch.count_nonzero(torch.tril(U, -1)).item() == 0
        Hd = s["Hbar"].double()
        d = torch.diagonal(Hd)
        d[s["dead"].bool()] = 1.0
        d += wl.damp_frac * d.mean()
        g = torch.Generator(device="cuda").manual_seed(82)
        v = torch.randn(spec.n, 8, device="cuda", dtype=torch.float64, generator=g)
        Ud = U.double()
        rel = ((Ud @ (Hd @ (Ud.T @ v)) - v).norm(dim=0) / v.norm(dim=0)).max().item()
        print(f"{wl.name} {nm}: max |U H_d Uᵀ v - v| / |v| = {rel:.2e}")
        assert rel < 1e-4
        del Hd, Ud


def test_sweep_outputs(shape_run):
    wl, bq = shape_run["wl"], shape_run["bq"]
    g, bits = wl.group_size, wl.bits
    for md in shape_run["modules"]:
        o = bq.out[md.name]
        n = md.n
        codes = unpack(o["codes"].cpu().numpy(), n)
        scale = o["scale"].cpu().numpy()
        zero = o["zero"].cpu().numpy().astype(np.float32)
        assert codes.min() >= 0 and codes.max() <= 2 ** bits - 1
        assert np.all(np.isfinite(scale)) and np.all(scale > 0)
        assert zero.max() <= 2 ** bits - 1
        deq = (scale[:, np.arange(n) // g] * (codes.astype(np.float32) - zero[:, np.arange(n) // g])).astype(np.float32)
        assert np.array_equal(deq, o["W"].cpu().numpy()), md.name
        assert o["adam_t"] == (-(-n // wl.block_size) - 1) * wl.steps_per_block
