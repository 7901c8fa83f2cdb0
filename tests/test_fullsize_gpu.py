"""Parity at the full size of the Qwen3-0.6B-shaped decoder block (4 inputs of
262,144 tokens, 7 modules, asymmetric g128 W4, Block-GD with Adam at lr 3e-4),
run exactly as the benchmark times it: the library's concurrent block
scheduler, one stream per input and per module, captured into a CUDA graph
and replayed (the outputs are cleared between the capture and the replay).

The fp64 oracle computes its own Hessians of all four inputs (bf16 values and
their products are exact in fp64), and everything else from those:
  Hessian  every entry: |ΔH_ij| <= 2e-6 sqrt(T) sqrt(H_ii H_jj), the fp32
           accumulation bound of the small cases.
  U        the oracle's factor of its own Hessian, max |ΔU| <= 2e-4 max |U|.
  REAL-Q   all seven modules (every row) against the full fp64 oracle sweep
           with Block-GD: codes >= 99.9 % equal and none unexplained on the
           CUDA path's branch at rounding ties (tests/parity.py), scales as
           in the small cases, and the surrogate of the CUDA path's output
           (its own value) within 1e-3 of the oracle's token form of the
           oracle's output.
  GPTQ     the sweep without Block-GD on all seven modules: rows are then
           independent, so the oracle sweeps 6 sampled rows of each module.
  all      grid consistency of every module's outputs and the Adam step count.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2609_00049_gb300 as rq
from paper_2609_00049_gb300.block import BlockInput, BlockModule, BlockQuantizer
from parity import OracleSweep, check_codes_and_scales, token_surrogate, unpack

pytestmark = pytest.mark.gpu

WL = "qwen3-0.6b"


@pytest.fixture(scope="module")
def block_run():
    from paper_2609_00049_gb300 import build as b
    b.build()
    rq.lib()
    wl = synth.workloads()[WL]
    dev = torch.device("cuda", 0)
    x_bits = {nm: synth.xhat_full(wl, nm, as_bits=True) for nm in wl.inputs}
    X = {nm: torch.from_numpy(v.view(np.int16)).to(dev).view(torch.bfloat16) for nm, v in x_bits.items()}
    w_bits = {md.name: synth.weights(wl, md) for md in wl.modules}
    W0 = {k: torch.from_numpy(v.view(np.int16)).to(dev).view(torch.bfloat16) for k, v in w_bits.items()}
    F_np = {md.name: synth.fisher(wl, md) for md in wl.modules}
    F = {k: torch.from_numpy(v).to(dev) for k, v in F_np.items()}
    qcfg = rq.quant_cfg(wl.bits, wl.group_size, wl.block_size, wl.symmetric, wl.damp_frac)
    bq = BlockQuantizer([BlockInput(nm, sp.n, sp.T) for nm, sp in wl.inputs.items()],
                        [BlockModule(md.name, md.m, md.n, md.input) for md in wl.modules], qcfg, wl.lr,
                        wl.steps_per_block, sliding_window=wl.sliding_window, device=dev)
    bq.capture(X, W0, F)
    for o in bq.out.values():
        for k in ("codes", "scale", "zero", "W"):
            o[k].fill_(0 if o[k].dtype == torch.uint8 else float("nan"))
    bq.replay()
    torch.cuda.synchronize()
    bq.check_status()
    return wl, bq, x_bits, w_bits, F_np


def _x64(bits):
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


@pytest.fixture(scope="module")
def oracle_H(block_run):
    wl, _, x_bits, _, _ = block_run
    out = {}
    for nm, spec in wl.inputs.items():
        H, T = oracle.hessian_sum(_x64(x_bits[nm][c:c + 8192]) for c in range(0, spec.T, 8192))
        assert T == spec.T
        out[nm] = H
    return out


def test_fullsize_hessians(block_run, oracle_H):
    wl, bq, _, _, _ = block_run
    for nm, spec in wl.inputs.items():
        H = bq.state[nm]["H"].cpu().numpy().astype(np.float64)
        Href = oracle_H[nm]
        scale = np.sqrt(np.outer(np.diag(Href), np.diag(Href)))
        err = np.abs(H - Href) / scale
        print(f"\n{nm}: n={spec.n} max scaled error {err.max():.2e} (bound {2e-6 * np.sqrt(spec.T):.2e})")
        assert err.max() < 2e-6 * np.sqrt(spec.T)


def test_fullsize_factors(block_run, oracle_H):
    wl, bq, _, _, _ = block_run
    for nm, spec in wl.inputs.items():
        s = bq.state[nm]
        ref = oracle.prepare(oracle_H[nm], spec.T, wl.damp_frac)
        Uref = oracle.inverse_upper_cholesky(ref["Hd"])
        U = s["U"].cpu().numpy().astype(np.float64)
        rel = np.abs(U - Uref).max() / np.abs(Uref).max()
        print(f"\n{nm}: n={spec.n} max|dU|/max|U|={rel:.2e}")
        assert rel <= 2e-4
        assert np.all(np.tril(U, -1) == 0)
        assert np.array_equal(s["dead"].cpu().numpy().astype(bool), ref["dead"])


def test_fullsize_sweeps_against_oracle(block_run, oracle_H):
    # every module with Block-GD (Adam at lr 3e-4) against the fp64 oracle's
    # literal sweep on its own Hessian: the codes bar on the CUDA path's
    # branch at rounding ties, scales within 1e-5 apart from the counted
    # Adam-sign groups of reading R18, and the surrogate within 1e-3
    wl, bq, x_bits, w_bits, F_np = block_run
    B = wl.block_size
    qkw = dict(bits=wl.bits, group_size=wl.group_size, block_size=B)
    bstart = 1
    for md in wl.modules:
        spec = wl.inputs[md.input]
        Href, T = oracle_H[md.input], spec.T
        W0 = synth.bf16_bits_to_f32(w_bits[md.name]).astype(np.float64)
        bgd = dict(lr=wl.lr, steps_per_block=wl.steps_per_block, b_global_start=bstart, B_total=1)
        orc = OracleSweep(lambda follow, grad_noise=None: oracle.realq_sweep(
            W0, Href, T, bits=wl.bits, group_size=wl.group_size, block_size=B, symmetric=bool(wl.symmetric),
            damp_frac=wl.damp_frac, bgd=bgd, F=F_np[md.name], record=False, follow=follow, grad_noise=grad_noise))
        nb = -(-md.n // B)
        bstart += nb
        o = bq.out[md.name]
        assert o["adam_t"] == orc["adam_t"] == nb - 1
        codes = unpack(o["codes"].cpu().numpy(), md.n)
        plain, fol, _ = check_codes_and_scales(orc, codes, o["zero"].cpu().numpy(), o["scale"].cpu().numpy(),
                                               md.n, qkw, True, wl.lr, wl.steps_per_block, f"{md.name} {md.m}x{md.n} ")
        # the surrogate of the oracle's result on the CUDA path's branch at
        # rounding ties (the one the codes are compared with; the plain run's
        # is printed: at lr 3e-4 a few ties taken the other way move the loss
        # by about 1e-3)
        L_or = token_surrogate(oracle, fol["deq"], W0, _x64, x_bits[md.input], F_np[md.name])
        L_plain = L_or if fol is plain else token_surrogate(oracle, plain["deq"], W0, _x64, x_bits[md.input],
                                                            F_np[md.name])
        ws = rq.workspace(rq.realq_surrogate_workspace_size(md.m, md.n))
        loss = torch.zeros(1, device="cuda")
        rq.realq_surrogate_loss(o["W"], torch.from_numpy(W0.astype(np.float32)).cuda(), bq.state[md.input]["Hbar"],
                                torch.from_numpy(F_np[md.name]).cuda(), loss, ws)
        L_gpu = float(loss.item())
        print(f"{md.name}: surrogate gpu {L_gpu:.6e} oracle {L_or:.6e} (rel {abs(L_gpu - L_or) / L_or:.2e}); "
              f"plain oracle {L_plain:.6e} (rel {abs(L_gpu - L_plain) / L_plain:.2e})")
        assert abs(L_gpu - L_or) <= 1e-3 * L_or


def test_fullsize_gptq_rows_every_module(block_run, oracle_H):
    wl, _, x_bits, w_bits, _ = block_run
    dev = torch.device("cuda", 0)
    X = {nm: torch.from_numpy(v.view(np.int16)).to(dev).view(torch.bfloat16) for nm, v in x_bits.items()}
    W0 = {k: torch.from_numpy(v.view(np.int16)).to(dev).view(torch.bfloat16) for k, v in w_bits.items()}
    qcfg = rq.quant_cfg(wl.bits, wl.group_size, wl.block_size, wl.symmetric, wl.damp_frac)
    bq = BlockQuantizer([BlockInput(nm, sp.n, sp.T) for nm, sp in wl.inputs.items()],
                        [BlockModule(md.name, md.m, md.n, md.input) for md in wl.modules], qcfg, 0.0, 0,
                        device=dev)
    bq.run(X, W0, {md.name: None for md in wl.modules})
    torch.cuda.synchronize()
    bq.check_status()
    del X
    r = synth.rng(72, "fullsize-gptq-rows")
    B, g = wl.block_size, wl.group_size
    qkw = dict(bits=wl.bits, group_size=g, block_size=B)
    for nm, spec in wl.inputs.items():
        mods = [md for md in wl.modules if md.input == nm]
        rows = {md.name: np.sort(r.choice(md.m, 6, replace=False)) for md in mods}
        W_rows = np.concatenate([synth.bf16_bits_to_f32(w_bits[md.name])[rows[md.name]] for md in mods])
        orc = OracleSweep(lambda follow, grad_noise=None: oracle.realq_sweep(
            W_rows.astype(np.float64), oracle_H[nm], spec.T, bits=wl.bits, group_size=g, block_size=B,
            symmetric=bool(wl.symmetric), damp_frac=wl.damp_frac, follow=follow, grad_noise=grad_noise))
        codes = np.concatenate([unpack(bq.out[md.name]["codes"].cpu().numpy(), md.n)[rows[md.name]]
                                for md in mods])
        scale = np.concatenate([bq.out[md.name]["scale"].cpu().numpy()[rows[md.name]] for md in mods])
        zero = np.concatenate([bq.out[md.name]["zero"].cpu().numpy()[rows[md.name]] for md in mods])
        check_codes_and_scales(orc, codes, zero, scale, spec.n, qkw, False, what=f"{nm} GPTQ rows ")


def test_fullsize_every_module_properties(block_run):
    wl, bq, _, w_bits, F_np = block_run
    B, g, bits = wl.block_size, wl.group_size, wl.bits
    for md in wl.modules:
        o, s_in = bq.out[md.name], bq.state[md.input]
        n = md.n
        codes = unpack(o["codes"].cpu().numpy(), n)
        scale = o["scale"].cpu().numpy()
        zero = o["zero"].cpu().numpy().astype(np.float32)
        assert codes.min() >= 0 and codes.max() <= 2 ** bits - 1
        assert np.all(np.isfinite(scale)) and np.all(scale > 0)
        assert zero.max() <= 2 ** bits - 1
        deq = (scale[:, np.arange(n) // g] * (codes.astype(np.float32) - zero[:, np.arange(n) // g])).astype(np.float32)
        assert np.array_equal(deq, o["W"].cpu().numpy()), md.name
        assert o["adam_t"] == -(-n // B) - 1
        # reported, not asserted: at the paper's learning rate the first Adam
        # step overshoots on these synthetic (nearly diagonal-H) inputs
        W0 = synth.bf16_bits_to_f32(w_bits[md.name])
        rtn = oracle.rtn(W0.astype(np.float64), bits=bits, group_size=g)
        W0d = torch.from_numpy(W0).cuda()
        Fd = torch.from_numpy(F_np[md.name]).cuda()
        ws = rq.workspace(rq.realq_surrogate_workspace_size(md.m, n))
        loss = torch.zeros(1, device="cuda")

        def surrogate(What):
            rq.realq_surrogate_loss(What, W0d, s_in["Hbar"], Fd, loss, ws)
            return float(loss.item())

        L_q = surrogate(o["W"])
        L_rtn = surrogate(torch.from_numpy(np.asarray(rtn[1], np.float32)).cuda())
        print(f"\n{md.name}: surrogate REAL-Q {L_q:.4e} vs RTN {L_rtn:.4e} (ratio {L_q / L_rtn:.3f})")
