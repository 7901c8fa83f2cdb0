"""Concurrent scheduler for one decoder block (Alg. 1, one pass of the inner
loops over every linear module of a transformer block).

The modules of a block share calibration inputs: q/k/v read the attention
input, o the attention output, gate/up the MLP input and down the MLP hidden
state.  Each distinct input needs one Hessian and one preparation; each
module then runs its own column sweep.  Those chains are independent of one
another, so they run concurrently: one host thread per input drives the
input's stream (accumulate, then prepare, which waits on that stream only),
then issues every module fed by that input on a stream of its own.  The
library calls release the interpreter lock, so the threads overlap on the
host as well.  All state (Hessians, factors, optimizer moments, outputs,
workspaces) is allocated once and reused across calls.

No arithmetic happens here; every step is a call through the C ABI.
"""
from __future__ import annotations

from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence

import torch

from . import (REALQ_BF16, QuantCfg, bgd_cfg, realq_hessian_accumulate, realq_hessian_prepare,
               realq_hessian_workspace_size, realq_prepare_workspace_size, realq_quantize_activations,
               realq_quantize_layer, realq_quantize_workspace_size, realq_scale_moment, realq_workspace_status,
               workspace)


@dataclass
class BlockInput:
    """Calibration input X̂ of T tokens and n channels (token-major)."""
    name: str
    n: int
    T: int


@dataclass
class BlockModule:
    """Linear module W (m out x n in) fed by input `input`."""
    name: str
    m: int
    n: int
    input: str


class BlockQuantizer:
    """Quantizes every module of a decoder block with REAL-Q's inner loops.

    modules are given in the block's module order (q, k, v, o, gate, up, down);
    that order numbers the column blocks for the sliding window (b_global runs
    over all modules' blocks).  lr and steps_per_block configure Block-GD (0
    steps disables it); sliding_window=True uses F_eff = alpha F + (1-alpha) F'
    with alpha decaying over the block's B_total column blocks.

    act_quant=(bits, a_clip) selects the activation-aware weight-activation
    variant (Sec. 5): each input is quantized per token first, the Hessian is
    taken over the quantized activations, and the Block-GD surrogate keeps
    the full-precision ones through the cross moment D.
    """

    def __init__(self, inputs: Sequence[BlockInput], modules: Sequence[BlockModule], qcfg: QuantCfg, lr: float,
                 steps_per_block: int = 1, sliding_window: bool = False, device="cuda",
                 host_chunk_tokens: int = 32768, act_quant: Optional[tuple] = None):
        self.inputs: Dict[str, BlockInput] = {i.name: i for i in inputs}
        self.modules: List[BlockModule] = list(modules)
        for md in self.modules:
            if md.input not in self.inputs or self.inputs[md.input].n != md.n:
                raise ValueError(f"module {md.name}: input {md.input!r} missing or of the wrong width")
        self.qcfg = qcfg
        self.device = torch.device(device)
        if self.device.index is None:
            self.device = torch.device(self.device.type, torch.cuda.current_device())
        self.sliding_window = sliding_window
        self.act_quant = act_quant
        self.mods_of = {name: [md for md in self.modules if md.input == name] for name in self.inputs}
        B = qcfg.block_size
        self.B_total = sum(-(-md.n // B) for md in self.modules)
        dev = self.device
        self.state = {}
        for name, spec in self.inputs.items():
            n = spec.n
            self.state[name] = dict(
                H=torch.empty(n, n, device=dev), U=torch.empty(n, n, device=dev), Hbar=torch.empty(n, n, device=dev),
                dead=torch.empty(n, dtype=torch.uint8, device=dev),
                pws=workspace(realq_prepare_workspace_size(n), dev),
                hws=workspace(realq_hessian_workspace_size(n, spec.T, REALQ_BF16, act_quant is not None), dev))
            if act_quant is not None:
                self.state[name].update(Xq=torch.empty(spec.T, n, dtype=torch.bfloat16, device=dev),
                                        D=torch.empty(n, n, device=dev), Dbar=torch.empty(n, n, device=dev))
        self.out = {}
        bstart = 1
        g_eff = qcfg.group_size
        for md in self.modules:
            m, n = md.m, md.n
            g = g_eff or n
            ng = -(-n // g)
            bc = bgd_cfg(lr, steps_per_block, b_global_start=bstart,
                         B_total=self.B_total if sliding_window else 1)
            bstart += -(-n // B)
            bgd = steps_per_block > 0
            self.out[md.name] = dict(
                W=torch.empty(m, n, device=dev),
                codes=torch.empty(m, (n + 1) // 2, dtype=torch.uint8, device=dev),
                scale=torch.empty(m, ng, device=dev), zero=torch.empty(m, ng, dtype=torch.uint8, device=dev),
                am=torch.empty(m, n, device=dev) if bgd else None, av=torch.empty(m, n, device=dev) if bgd else None,
                disp=torch.empty(m, n, device=dev) if bgd else None, bcfg=bc if bgd else None,
                ws=workspace(realq_quantize_workspace_size(m, n, qcfg, bc if bgd else None, sliding_window,
                                                           act_quant is not None and bgd), dev),
                adam_t=0)
        self.in_streams = {name: torch.cuda.Stream(device=dev) for name in self.inputs}
        self.copy_streams = {name: torch.cuda.Stream(device=dev) for name in self.inputs}
        self.mod_streams = {md.name: torch.cuda.Stream(device=dev) for md in self.modules}
        self.pool = ThreadPoolExecutor(len(self.inputs))
        # staging for inputs streamed from host memory (two chunks per input)
        self.host_chunk = host_chunk_tokens
        self._stage = None
        self._chunk_ws = None
        self._w_stage = None

    # ------------------------------------------------------------------ device
    def _quantize_module(self, md: BlockModule, s_in, W0, F, F_next, stream):
        o = self.out[md.name]
        o["adam_t"] = realq_quantize_layer(
            W0, s_in["U"], s_in["Hbar"], self.qcfg, o["W"], o["codes"], o["scale"], o["zero"],
            Dbar=s_in.get("Dbar") if o["bcfg"] is not None else None, dead=s_in["dead"],
            bcfg=o["bcfg"], F=F, F_next=F_next if self.sliding_window else None, adam_m=o["am"], adam_v=o["av"],
            bgd_disp=o["disp"], ws=o["ws"], stream=stream)

    def _input_pipeline(self, name, start, X, W0, F, F_next):
        torch.cuda.set_device(self.device)
        spec, s_in, si = self.inputs[name], self.state[name], self.in_streams[name]
        si.wait_event(start)
        self._hessian(name, X[name], si)
        for md in self.mods_of[name]:
            sm = self.mod_streams[md.name]
            sm.wait_stream(si)
            self._quantize_module(md, s_in, W0[md.name], F[md.name], (F_next or {}).get(md.name), sm)

    def _hessian(self, name, X, stream):
        """H (and, activation-aware, D) of one input, then its preparation."""
        spec, s_in = self.inputs[name], self.state[name]
        with torch.cuda.stream(stream if stream is not None else torch.cuda.current_stream(self.device)):
            s_in["H"].zero_()
            if self.act_quant is not None:
                s_in["D"].zero_()
        if self.act_quant is None:
            realq_hessian_accumulate(X, s_in["H"], ws=s_in["hws"], stream=stream)
        else:
            bits, clip = self.act_quant
            realq_quantize_activations(X, bits, clip, X_q=s_in["Xq"], stream=stream)
            realq_hessian_accumulate(s_in["Xq"], s_in["H"], s_in["D"], X, ws=s_in["hws"], stream=stream)
        realq_hessian_prepare(s_in["H"], spec.T, self.qcfg.damp_frac, s_in["U"], s_in["Hbar"], s_in["dead"],
                              s_in["pws"], stream=stream)
        if self.act_quant is not None:
            realq_scale_moment(s_in["D"], spec.T, s_in["Dbar"], stream=stream)

    def _join(self, start_stream):
        for md in self.modules:
            start_stream.wait_stream(self.mod_streams[md.name])
        for name in self.inputs:
            start_stream.wait_stream(self.in_streams[name])
            start_stream.wait_stream(self.copy_streams[name])

    def run(self, X: Dict[str, torch.Tensor], W0: Dict[str, torch.Tensor], F: Dict[str, torch.Tensor],
            F_next: Optional[Dict[str, torch.Tensor]] = None) -> None:
        """Quantize the block from device-resident inputs (X̂ per input, W0 and
        F per module).  Work is enqueued after everything already on the
        current stream, and the current stream waits for all of it on return."""
        cur = torch.cuda.current_stream(self.device)
        start = torch.cuda.Event()
        start.record(cur)
        futs = [self.pool.submit(self._input_pipeline, name, start, X, W0, F, F_next) for name in self.inputs]
        for f in futs:
            f.result()
        self._join(cur)

    def run_serial(self, X, W0, F, F_next=None) -> None:
        """The same work, one call after another on the current stream."""
        for name, spec in self.inputs.items():
            s_in = self.state[name]
            self._hessian(name, X[name], None)
            for md in self.mods_of[name]:
                self._quantize_module(md, s_in, W0[md.name], F[md.name], (F_next or {}).get(md.name), None)

    def check_status(self) -> None:
        """Raise if any module's sweep recorded a non-finite value or a timeout."""
        for md in self.modules:
            realq_workspace_status(self.out[md.name]["ws"])

    # -------------------------------------------------------------------- host
    def _host_pipeline(self, name, start, X_host, W0_host, F_host, out_host, counts):
        torch.cuda.set_device(self.device)
        spec, s_in = self.inputs[name], self.state[name]
        si, cs = self.in_streams[name], self.copy_streams[name]
        si.wait_event(start)
        cs.wait_event(start)
        with torch.cuda.stream(si):
            s_in["H"].zero_()
        xs = X_host[name]
        C = self.host_chunk
        used = [None, None]
        h2d = d2h = 0
        for c in range(-(-spec.T // C)):
            buf = self._stage[name][c % 2]
            rows = min(C, spec.T - c * C)
            if used[c % 2] is not None:
                cs.wait_event(used[c % 2])
            with torch.cuda.stream(cs):
                buf[:rows].copy_(xs[c * C:c * C + rows], non_blocking=True)
            done = torch.cuda.Event()
            done.record(cs)
            si.wait_event(done)
            realq_hessian_accumulate(buf[:rows], s_in["H"], ws=self._chunk_ws[name], stream=si)
            ev = torch.cuda.Event()
            ev.record(si)
            used[c % 2] = ev
            h2d += rows * spec.n * xs.element_size()
        realq_hessian_prepare(s_in["H"], spec.T, self.qcfg.damp_frac, s_in["U"], s_in["Hbar"], s_in["dead"],
                              s_in["pws"], stream=si)
        for md in self.mods_of[name]:
            sm, o, w = self.mod_streams[md.name], out_host[md.name], self._w_stage[md.name]
            sm.wait_stream(si)
            with torch.cuda.stream(sm):
                w["W0"].copy_(W0_host[md.name], non_blocking=True)
                w["F"].copy_(F_host[md.name], non_blocking=True)
            h2d += W0_host[md.name].numel() * W0_host[md.name].element_size()
            h2d += F_host[md.name].numel() * F_host[md.name].element_size()
            self._quantize_module(md, s_in, w["W0"], w["F"], None, sm)
            with torch.cuda.stream(sm):
                for k in ("codes", "scale", "zero"):
                    o[k].copy_(self.out[md.name][k], non_blocking=True)
                    d2h += o[k].numel() * o[k].element_size()
        counts[name] = (h2d, d2h)

    def run_host(self, X_host, W0_host, F_host, out_host):
        """End to end from pinned host memory: X̂ streams in chunks on a copy
        stream per input (double-buffered, overlapped with accumulation), W0
        and F are copied per module, codes / scale / zero are copied back into
        out_host[module][...] (pinned).  Returns (h2d bytes, d2h bytes).
        The activation-aware variant is not streamed (it runs with run())."""
        if self.act_quant is not None:
            raise NotImplementedError("run_host: the activation-aware variant runs from device-resident inputs")
        dev = self.device
        if self._stage is None:
            self._stage = {name: [torch.empty(self.host_chunk, spec.n, dtype=X_host[name].dtype, device=dev)
                                  for _ in range(2)] for name, spec in self.inputs.items()}
            self._chunk_ws = {name: workspace(realq_hessian_workspace_size(spec.n, self.host_chunk), dev)
                              for name, spec in self.inputs.items()}
            self._w_stage = {md.name: dict(W0=torch.empty(W0_host[md.name].shape, dtype=W0_host[md.name].dtype,
                                                          device=dev),
                                           F=torch.empty(F_host[md.name].shape, dtype=F_host[md.name].dtype,
                                                         device=dev))
                             for md in self.modules}
        cur = torch.cuda.current_stream(dev)
        start = torch.cuda.Event()
        start.record(cur)
        counts = {}
        futs = [self.pool.submit(self._host_pipeline, name, start, X_host, W0_host, F_host, out_host, counts)
                for name in self.inputs]
        for f in futs:
            f.result()
        self._join(cur)
        return sum(v[0] for v in counts.values()), sum(v[1] for v in counts.values())
