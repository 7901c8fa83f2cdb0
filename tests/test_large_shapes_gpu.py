"""Full-size checks of the three larger decoder-block shapes, run as the
benchmark runs them (the block scheduler's step captured into a CUDA graph
and replayed, with Block-GD at each shape's learning rate):

  llama3.1-8b   hidden 4096, MLP 14336, Student-t(4) activations, the
                two-block sliding window (B_total = 304)
  qwen3-32b     hidden 5120, q 8192, MLP 25600, 0.5 % outlier channels x50
  llama3.1-70b  hidden 8192, MLP 28672, 524,288 tokens of Student-t(3): H, U
                and H̄ of n = 28672 (3.3 GB each) held on one GPU.  To keep
                the run short this shape runs the inputs and modules that
                set it apart: down_in with down_proj (n = 28672) and attn_in
                with k_proj and v_proj.

At these sizes the fp64 oracle cannot form whole Hessians or factors on the
host (2 T n^2 flops), so the checks are the oracle on sampled outputs and
properties that hold at any size:
  Hessian  the oracle's X̂_Sᵀ X̂_S for 48 sampled columns S of every input
           (outlier channels first): every entry within the fp32
           accumulation bound of the small cases, 2e-6 sqrt(T) sqrt(H_ii H_jj);
           the oracle's diagonal over all n columns, and with it the dead
           flags, bit for bit.
  U        upper triangular with exact zeros below; U H_d Uᵀ = I on random
           probe vectors in fp64 (H_d the damped H̄ the kernels factor, with
           λ = damp · mean diag), relative residual below 1e-4 = 10 sqrt(n) u
           at the largest n = 28672 (u = 2^-24, fp32 sums of length up to n,
           condition numbers of a few units for these damped moments); a
           dropped update or a wrong sign leaves a residual of order one.
  sweep    every module: codes in [0, 15], the dequantized weights equal
           scale · (q - zero) bit for bit, scales finite and positive, zero
           points in range, one Adam step per column block but the last;
           the surrogate against RTN is printed.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2609_00049_gb300 as rq
from paper_2609_00049_gb300.block import BlockInput, BlockModule, BlockQuantizer
from parity import unpack

pytestmark = pytest.mark.gpu

SUBSET = {"llama3.1-70b": (("attn_in", "down_in"), ("k_proj", "v_proj", "down_proj"))}


@pytest.fixture(scope="module", params=["llama3.1-8b", "qwen3-32b", "llama3.1-70b"])
def shape_run(request):
    from paper_2609_00049_gb300 import build as b
    b.build()
    rq.lib()
    wl = synth.workloads()[request.param]
    ins, mods = SUBSET.get(wl.name, (tuple(wl.inputs), tuple(md.name for md in wl.modules)))
    dev = torch.device("cuda", 0)
    x_bits, X = {}, {}
    for nm in ins:
        x_bits[nm] = synth.xhat_full(wl, nm, as_bits=True, threads=16)
        X[nm] = torch.from_numpy(x_bits[nm].view(np.int16)).to(dev).view(torch.bfloat16)
    modules = [md for md in wl.modules if md.name in mods]
    w_bits = {md.name: synth.weights(wl, md) for md in modules}
    W0 = {k: torch.from_numpy(v.view(np.int16)).to(dev).view(torch.bfloat16) for k, v in w_bits.items()}
    F = {md.name: torch.from_numpy(synth.fisher(wl, md)).to(dev) for md in modules}
    F_next = None
    if wl.sliding_window:
        F_next = {md.name: torch.from_numpy(synth.fisher(wl, md, "F_next")).to(dev) for md in modules}
    qcfg = rq.quant_cfg(wl.bits, wl.group_size, wl.block_size, wl.symmetric, wl.damp_frac)
    bq = BlockQuantizer([BlockInput(nm, wl.inputs[nm].n, wl.inputs[nm].T) for nm in ins],
                        [BlockModule(md.name, md.m, md.n, md.input) for md in modules], qcfg, wl.lr,
                        wl.steps_per_block, sliding_window=wl.sliding_window, device=dev)
    bq.capture(X, W0, F, F_next)
    for o in bq.out.values():
        for k in ("codes", "scale", "zero", "W"):
            o[k].fill_(0 if o[k].dtype == torch.uint8 else float("nan"))
    bq.replay()
    torch.cuda.synchronize()
    bq.check_status()
    del X
    yield wl, bq, x_bits, w_bits, modules
    del bq
    torch.cuda.empty_cache()


def test_hessian_sampled_entries(shape_run):
    wl, bq, x_bits, _, _ = shape_run
    r = synth.rng(81, "large-hessian", wl.name)
    for nm, bits in x_bits.items():
        spec = wl.inputs[nm]
        out = synth.outlier_channels(wl, spec)
        S = np.unique(np.concatenate([out[:16], r.choice(spec.n, 48, replace=False)]))[:48]
        S = np.sort(S)
        xs = lambda c: synth.bf16_bits_to_f32(bits[c:c + 8192][:, S]).astype(np.float64)
        Hs, T = oracle.hessian_sum(xs(c) for c in range(0, spec.T, 8192))
        assert T == spec.T
        Hg = bq.state[nm]["H"][torch.from_numpy(S).cuda()][:, torch.from_numpy(S).cuda()].double().cpu().numpy()
        scale = np.sqrt(np.outer(np.diag(Hs), np.diag(Hs)))
        err = np.abs(Hg - Hs) / scale
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


def test_factor_identity(shape_run):
    wl, bq, x_bits, _, _ = shape_run
    for nm in x_bits:
        s = bq.state[nm]
        n = wl.inputs[nm].n
        U = s["U"]
        assert torch.count_nonzero(torch.tril(U, -1)).item() == 0
        Hd = s["Hbar"].double()
        dead = s["dead"].bool()
        d = torch.diagonal(Hd)
        d[dead] = 1.0
        lam = wl.damp_frac * d.mean()
        d += lam
        g = torch.Generator(device="cuda").manual_seed(82)
        v = torch.randn(n, 8, device="cuda", dtype=torch.float64, generator=g)
        Ud = U.double()
        res = Ud @ (Hd @ (Ud.T @ v)) - v
        rel = (res.norm(dim=0) / v.norm(dim=0)).max().item()
        print(f"\n{wl.name} {nm}: n={n} max |U H_d Uᵀ v - v| / |v| = {rel:.2e}")
        assert rel < 1e-4
        del Hd, Ud


def test_sweep_outputs(shape_run):
    wl, bq, _, w_bits, modules = shape_run
    g, bits = wl.group_size, wl.bits
    for md in modules:
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
        assert o["adam_t"] == -(-n // wl.block_size) - 1
        s_in = bq.state[md.input]
        W0 = torch.from_numpy(synth.bf16_bits_to_f32(w_bits[md.name])).cuda()
        Fd = torch.from_numpy(synth.fisher(wl, md)).cuda()
        ws = rq.workspace(rq.realq_surrogate_workspace_size(md.m, n))
        loss = torch.zeros(1, device="cuda")
        rtn = oracle.rtn(synth.bf16_bits_to_f32(w_bits[md.name]).astype(np.float64), bits=bits, group_size=g)
        rq.realq_surrogate_loss(o["W"], W0, s_in["Hbar"], Fd, loss, ws)
        L_q = float(loss.item())
        rq.realq_surrogate_loss(torch.from_numpy(np.asarray(rtn[1], np.float32)).cuda(), W0, s_in["Hbar"], Fd, loss, ws)
        L_rtn = float(loss.item())
        print(f"\n{wl.name} {md.name} {md.m}x{n}: surrogate REAL-Q {L_q:.4e} vs RTN {L_rtn:.4e} "
              f"(ratio {L_q / L_rtn:.3f})")
        del W0, Fd, ws
