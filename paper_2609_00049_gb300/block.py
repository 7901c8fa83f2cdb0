"""Concurrent scheduler for one decoder block (Alg. 1, one pass of the inner
loops over every linear module of a transformer block).

The modules of a block share calibration inputs: q/k/v read the attention
input, o the attention output, gate/up the MLP input and down the MLP hidden
state.  Each distinct input needs one Hessian and one preparation; each
module then runs its own column sweep.  Those chains are independent of one
another, so they run concurrently: one host thread per input drives the
input's stream (accumulate, then prepare), then issues every module fed by
that input on a stream of its own.  The library calls release the
interpreter lock, so the threads overlap on the host as well.  All state
(Hessians, factors, optimizer moments, outputs, workspaces) is allocated once
and reused across calls.

One step enqueues about a thousand kernels, most of them small (the 64-column
steps of the Cholesky factorisation and of the sweeps), so launching them
costs as much host time as they take on the GPU.  capture() records the same
multi-stream step once into a CUDA graph; replay() then launches it whole.
The preparation's factorisation status is therefore never read mid-step:
check_status() reads it, with the sweeps' status words, after the step.

quantize_block_exact runs a block with the exact losses of Sec. 4.4 (the
two-block window, or the KL at the LM head for the last block) instead:
there each module's loss and OBS Hessian depend on the modules quantized
before it, so the modules run one after another on the caller's stream.

No arithmetic happens here; every step is a call through the C ABI.
"""
from __future__ import annotations

from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence

import torch

from . import layer
from . import (BLOCK_MODULES, REALQ_BF16, REALQ_OPT_ADAM, QuantCfg, bgd_cfg, realq_block_forward,
               realq_block_module_inputs, realq_reverse_cosine_lr,
               realq_block_workspace_size, realq_graph_begin, realq_graph_end, realq_hessian_accumulate,
               realq_hessian_accumulate_weighted, realq_hessian_prepare_deferred, realq_hessian_prepare_scaled,
               realq_hessian_weighted_workspace_size, realq_hessian_workspace_size, realq_prepare_status,
               realq_prepare_workspace_size, realq_quantize_activations, realq_quantize_grouped_workspace_size,
               realq_quantize_layer, realq_quantize_layer_grouped, realq_quantize_layer_minibatch,
               realq_quantize_layer_tokens, realq_quantize_minibatch_workspace_size,
               realq_quantize_layer_window, realq_quantize_tokens_workspace_size,
               realq_quantize_window_workspace_size, realq_quantize_workspace_size, realq_saliency_clip,
               realq_scale_moment, realq_workspace_status, workspace)


def _prepare_ws(n: int, dev) -> torch.Tensor:
    """A preparation workspace whose status words read as "no failure" (the
    failing column -1, no timeout) before the first preparation."""
    ws = workspace(realq_prepare_workspace_size(n), dev).zero_()
    ws[:4].fill_(0xFF)
    return ws


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

    minibatch_tokens=T_mb > 0 selects mini-batch Block-GD (Sec. 4.3, 32
    sequences per step in Sec. 5.1): every input's tokens form consecutive
    mini-batches of T_mb tokens, whose second moments the optimizer steps
    rotate through; the OBS keeps the full H.  With a_loss_clip (0.95 in the
    paper's small-model runs) each step's gradient is taken in token form on
    its mini-batch, with the per-token output clipping.

    b_global_start (module name -> 1-based global index of its first column
    block) and B_total override the numbering above, so that a subset of a
    block's modules can run with the indices they have in the whole block.

    saliency_groups=N_g > 0 selects the saliency-weighted grouped Hessians
    (Sec. 3.3, Alg. 1 "for all row-groups g"): every module's rows form N_g
    groups, run() takes a (T x N_g) saliency per module, clipped to its
    saliency_pct percentile, and each group is swept against its own factor;
    Block-GD keeps the input's plain H̄.
    """

    def __init__(self, inputs: Sequence[BlockInput], modules: Sequence[BlockModule], qcfg: QuantCfg, lr: float,
                 steps_per_block: int = 1, sliding_window: bool = False, device="cuda",
                 host_chunk_tokens: int = 32768, act_quant: Optional[tuple] = None, saliency_groups: int = 0,
                 saliency_pct: float = 0.99, minibatch_tokens: int = 0, a_loss_clip: Optional[float] = None,
                 b_global_start: Optional[Dict[str, int]] = None, B_total: Optional[int] = None):
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
        self.sgroups = saliency_groups
        self.spct = saliency_pct
        self.mb_tokens = minibatch_tokens
        self.a_loss_clip = a_loss_clip
        if a_loss_clip is not None and not minibatch_tokens:
            raise ValueError("a_loss_clip takes its gradient on mini-batches: set minibatch_tokens")
        if minibatch_tokens and (saliency_groups or act_quant is not None):
            raise ValueError("mini-batch Block-GD is built for the plain, unperturbed sweep")
        self.mods_of = {name: [md for md in self.modules if md.input == name] for name in self.inputs}
        B = qcfg.block_size
        self.B_total = sum(-(-md.n // B) for md in self.modules) if B_total is None else int(B_total)
        dev = self.device
        self.state = {}
        for name, spec in self.inputs.items():
            n = spec.n
            self.state[name] = dict(
                H=torch.empty(n, n, device=dev), U=torch.empty(n, n, device=dev), Hbar=torch.empty(n, n, device=dev),
                dead=torch.empty(n, dtype=torch.uint8, device=dev),
                pws=_prepare_ws(n, dev),
                hws=workspace(realq_hessian_workspace_size(n, spec.T, REALQ_BF16, act_quant is not None), dev))
            if minibatch_tokens and a_loss_clip is None:
                nmb = -(-spec.T // minibatch_tokens)
                self.state[name].update(Hk=torch.empty(n, n, device=dev), Hmb=torch.empty(nmb, n, n, device=dev),
                                        kws=workspace(realq_hessian_workspace_size(n, minibatch_tokens), dev))
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
            if b_global_start is not None:
                bstart = int(b_global_start[md.name])
            bc = bgd_cfg(lr, steps_per_block, b_global_start=bstart,
                         B_total=self.B_total if sliding_window else 1)
            bstart += -(-n // B)
            bgd = steps_per_block > 0
            if saliency_groups:
                ngs = saliency_groups
                ws_q = workspace(realq_quantize_grouped_workspace_size(m, n, ngs, qcfg, bc if bgd else None,
                                                                       sliding_window, act_quant is not None and bgd),
                                 dev)
                grp = dict(Sc=torch.empty(self.inputs[md.input].T, ngs, device=dev),
                           clip=torch.empty(ngs, device=dev),
                           Hg=torch.empty(ngs, n, n, device=dev), Ug=torch.empty(ngs, n, n, device=dev),
                           Hbg=torch.empty(ngs, n, n, device=dev),
                           dg=torch.empty(ngs, n, dtype=torch.uint8, device=dev),
                           wsum=torch.empty(ngs, dtype=torch.float64, device=dev),
                           wws=workspace(realq_hessian_weighted_workspace_size(n, self.inputs[md.input].T), dev),
                           pws=workspace(realq_prepare_workspace_size(n), dev))
            elif minibatch_tokens and bgd and a_loss_clip is not None:
                ws_q = workspace(realq_quantize_tokens_workspace_size(m, n, minibatch_tokens, qcfg, bc, sliding_window),
                                 dev)
                grp = None
            elif minibatch_tokens and bgd:
                nmb = -(-self.inputs[md.input].T // minibatch_tokens)
                ws_q = workspace(realq_quantize_minibatch_workspace_size(m, n, nmb, qcfg, bc, sliding_window), dev)
                grp = None
            else:
                ws_q = workspace(realq_quantize_workspace_size(m, n, qcfg, bc if bgd else None, sliding_window,
                                                               act_quant is not None and bgd), dev)
                grp = None
            self.out[md.name] = dict(
                grp=grp,
                W=torch.empty(m, n, device=dev),
                codes=torch.empty(m, (n + 1) // 2, dtype=torch.uint8, device=dev),
                scale=torch.empty(m, ng, device=dev), zero=torch.empty(m, ng, dtype=torch.uint8, device=dev),
                am=torch.empty(m, n, device=dev) if bgd else None, av=torch.empty(m, n, device=dev) if bgd else None,
                disp=torch.empty(m, n, device=dev) if bgd else None, bcfg=bc if bgd else None,
                ws=ws_q,
                adam_t=0)
        # Stream priorities follow the length of each input's chain (its
        # preparation and its modules' sweeps are sequences of 64-column
        # steps, so the widest input's chain is the longest): the widest input
        # and its modules get the highest priority, and kernels keep it inside
        # a captured graph.
        lo, hi = torch.cuda.Stream.priority_range()
        widths = sorted({spec.n for spec in self.inputs.values()}, reverse=True)
        self.priority = {name: max(hi, min(lo, hi + widths.index(spec.n))) for name, spec in self.inputs.items()}
        self.in_streams = {name: torch.cuda.Stream(device=dev, priority=self.priority[name]) for name in self.inputs}
        # one host-to-device copy stream shared by all inputs: a single stream
        # already saturates the host link, and in a captured step the inputs
        # arrive in chain order (the longest chain's activations first), so
        # that chain's preparation and sweeps overlap the other copies
        # (equal widths: the input feeding more weights first, so the input
        # whose copy ends the stream has the shortest chain after it)
        load = {name: sum(md.m * md.n for md in self.modules if md.input == name) for name in self.inputs}
        self.chain_order = sorted(self.inputs, key=lambda name: (self.priority[name], -load[name]))
        copy_stream = torch.cuda.Stream(device=dev)
        self.copy_streams = {name: copy_stream for name in self.inputs}

        self.mod_streams = {md.name: torch.cuda.Stream(device=dev, priority=self.priority[md.input])
                            for md in self.modules}
        self.pool = ThreadPoolExecutor(len(self.inputs))
        # staging for inputs streamed from host memory (two chunks per input)
        self.host_chunk = host_chunk_tokens
        self._stage = None
        self._chunk_ws = None
        self._w_stage = None
        self.graph = None

    # ------------------------------------------------------------------ device
    def _quantize_module(self, md: BlockModule, s_in, W0, F, F_next, stream, X=None, sal=None):
        o = self.out[md.name]
        if o["grp"] is not None:
            # saliency-weighted Hessians of this module's row groups, their
            # factors, then the grouped sweep (all on the module's stream)
            gp, T = o["grp"], self.inputs[md.input].T
            realq_saliency_clip(sal, self.spct, S_out=gp["Sc"], clip_out=gp["clip"], stream=stream)
            with torch.cuda.stream(stream if stream is not None else torch.cuda.current_stream(self.device)):
                gp["Hg"].zero_()
                gp["wsum"].zero_()
            realq_hessian_accumulate_weighted(s_in["Xq"] if self.act_quant is not None else X, gp["Sc"], gp["Hg"],
                                              gp["wsum"], gp["wws"], stream=stream)
            wsum = gp["wsum"].cpu() if stream is None else None
            if wsum is None:
                stream.synchronize()
                wsum = gp["wsum"].cpu()
            for g in range(self.sgroups):
                realq_hessian_prepare_scaled(gp["Hg"][g], float(wsum[g]), self.qcfg.damp_frac, gp["Ug"][g],
                                             gp["Hbg"][g], gp["dg"][g], gp["pws"], stream=stream)
            o["adam_t"] = realq_quantize_layer_grouped(
                W0, gp["Ug"], gp["Hbg"], gp["dg"], s_in["Hbar"], self.qcfg, o["W"], o["codes"], o["scale"],
                o["zero"], Dbar=s_in.get("Dbar") if o["bcfg"] is not None else None, bcfg=o["bcfg"], F=F,
                F_next=F_next if self.sliding_window else None, adam_m=o["am"], adam_v=o["av"], bgd_disp=o["disp"],
                ws=o["ws"], stream=stream)
            return
        if self.mb_tokens and o["bcfg"] is not None and self.a_loss_clip is not None:
            o["adam_t"] = realq_quantize_layer_tokens(
                W0, s_in["U"], s_in["Hbar"], X, self.mb_tokens, self.a_loss_clip, self.qcfg, o["W"], o["codes"],
                o["scale"], o["zero"], dead=s_in["dead"], bcfg=o["bcfg"], F=F,
                F_next=F_next if self.sliding_window else None, adam_m=o["am"], adam_v=o["av"], bgd_disp=o["disp"],
                ws=o["ws"], stream=stream)
            return
        if self.mb_tokens and o["bcfg"] is not None:
            o["adam_t"] = realq_quantize_layer_minibatch(
                W0, s_in["U"], s_in["Hbar"], s_in["Hmb"], self.qcfg, o["W"], o["codes"], o["scale"], o["zero"],
                dead=s_in["dead"], bcfg=o["bcfg"], F=F, F_next=F_next if self.sliding_window else None,
                adam_m=o["am"], adam_v=o["av"], bgd_disp=o["disp"], ws=o["ws"], stream=stream)
            return
        o["adam_t"] = realq_quantize_layer(
            W0, s_in["U"], s_in["Hbar"], self.qcfg, o["W"], o["codes"], o["scale"], o["zero"],
            Dbar=s_in.get("Dbar") if o["bcfg"] is not None else None, dead=s_in["dead"],
            bcfg=o["bcfg"], F=F, F_next=F_next if self.sliding_window else None, adam_m=o["am"], adam_v=o["av"],
            bgd_disp=o["disp"], ws=o["ws"], stream=stream)

    def _input_pipeline(self, name, start, X, W0, F, F_next, sal=None):
        torch.cuda.set_device(self.device)
        spec, s_in, si = self.inputs[name], self.state[name], self.in_streams[name]
        si.wait_event(start)
        self._hessian(name, X[name], si)
        for md in self.mods_of[name]:
            sm = self.mod_streams[md.name]
            sm.wait_stream(si)
            self._quantize_module(md, s_in, W0[md.name], F[md.name], (F_next or {}).get(md.name), sm, X=X[name],
                                  sal=(sal or {}).get(md.name))

    def _hessian(self, name, X, stream):
        """H (and, activation-aware, D) of one input, then its preparation."""
        spec, s_in = self.inputs[name], self.state[name]
        with torch.cuda.stream(stream if stream is not None else torch.cuda.current_stream(self.device)):
            s_in["H"].zero_()
            if self.act_quant is not None:
                s_in["D"].zero_()
        if self.act_quant is None and self.sgroups:
            # the groups' factors come per module; the plain H̄ serves Block-GD
            realq_hessian_accumulate(X, s_in["H"], ws=s_in["hws"], stream=stream)
            realq_scale_moment(s_in["H"], spec.T, s_in["Hbar"], stream=stream)
            return
        if self.act_quant is None:
            realq_hessian_accumulate(X, s_in["H"], ws=s_in["hws"], stream=stream)
            if self.mb_tokens and self.a_loss_clip is None:
                # second moments of the consecutive mini-batches
                C = self.mb_tokens
                for k in range(s_in["Hmb"].shape[0]):
                    with torch.cuda.stream(stream if stream is not None else torch.cuda.current_stream(self.device)):
                        s_in["Hk"].zero_()
                    rows = min(C, spec.T - k * C)
                    realq_hessian_accumulate(X[k * C:k * C + rows], s_in["Hk"], ws=s_in["kws"], stream=stream)
                    realq_scale_moment(s_in["Hk"], rows, s_in["Hmb"][k], stream=stream)
        else:
            bits, clip = self.act_quant
            realq_quantize_activations(X, bits, clip, X_q=s_in["Xq"], stream=stream)
            realq_hessian_accumulate(s_in["Xq"], s_in["H"], s_in["D"], X, ws=s_in["hws"], stream=stream)
        realq_hessian_prepare_deferred(s_in["H"], spec.T, self.qcfg.damp_frac, s_in["U"], s_in["Hbar"], s_in["dead"],
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
            F_next: Optional[Dict[str, torch.Tensor]] = None,
            saliency: Optional[Dict[str, torch.Tensor]] = None) -> None:
        """Quantize the block from device-resident inputs (X̂ per input, W0 and
        F per module, and with saliency groups a T x N_g saliency per module).
        Work is enqueued after everything already on the current stream, and
        the current stream waits for all of it on return."""
        if self.sgroups and saliency is None:
            raise ValueError("saliency_groups: run() needs a saliency per module")
        cur = torch.cuda.current_stream(self.device)
        start = torch.cuda.Event()
        start.record(cur)
        futs = [self.pool.submit(self._input_pipeline, name, start, X, W0, F, F_next, saliency)
                for name in self.inputs]
        for f in futs:
            f.result()
        self._join(cur)

    def run_serial(self, X, W0, F, F_next=None, saliency=None) -> None:
        """The same work, one call after another on the current stream."""
        for name, spec in self.inputs.items():
            s_in = self.state[name]
            self._hessian(name, X[name], None)
            for md in self.mods_of[name]:
                self._quantize_module(md, s_in, W0[md.name], F[md.name], (F_next or {}).get(md.name), None,
                                      X=X[name], sal=(saliency or {}).get(md.name))

    def capture(self, X: Dict[str, torch.Tensor], W0: Dict[str, torch.Tensor], F: Dict[str, torch.Tensor],
                F_next: Optional[Dict[str, torch.Tensor]] = None) -> None:
        """Record one step of run() on these tensors into a CUDA graph (every
        input's and module's stream forks from and joins back into the
        capturing stream), after one eager step that creates the library's
        auxiliary streams for the calling thread.  replay() then re-runs the
        whole step, reading the same tensors in place: change their contents,
        not their storage.  The saliency-grouped variant reads its groups'
        token weights on the host mid-step and is not capturable."""
        if self.sgroups:
            raise NotImplementedError("capture: the saliency-grouped variant reads token weights on the host")
        torch.cuda.set_device(self.device)
        self._enqueue(X, W0, F, F_next)
        torch.cuda.synchronize(self.device)
        self.check_status()
        self.graph = self._capture(lambda: self._enqueue(X, W0, F, F_next))

    def _capture(self, enqueue, node_priorities=True):
        cur = torch.cuda.current_stream(self.device)
        cap = torch.cuda.Stream(device=self.device)
        cap.wait_stream(cur)
        with torch.cuda.stream(cap):
            realq_graph_begin(cap)
            try:
                out = enqueue()
            finally:
                g = realq_graph_end(cap, node_priorities)
        cur.wait_stream(cap)
        self.graph_counts = out
        return g

    def replay(self) -> None:
        """Launch the captured step on the current stream."""
        if self.graph is None:
            raise RuntimeError("replay: capture() first")
        self.graph.launch(torch.cuda.current_stream(self.device))

    def _enqueue(self, X, W0, F, F_next) -> None:
        cur = torch.cuda.current_stream(self.device)
        start = torch.cuda.Event()
        start.record(cur)
        for name in self.chain_order:
            self._input_pipeline(name, start, X, W0, F, F_next)
        for md in self.modules:
            cur.wait_stream(self.mod_streams[md.name])
        for name in self.inputs:
            cur.wait_stream(self.in_streams[name])

    def check_status(self) -> None:
        """Synchronizes; raises RealqError(NOT_SPD) if an input's damped Hessian
        was not positive definite, else if any module's sweep recorded a
        non-finite value or a timeout."""
        for name in self.inputs:
            realq_prepare_status(self.state[name]["pws"])
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
        realq_hessian_prepare_deferred(s_in["H"], spec.T, self.qcfg.damp_frac, s_in["U"], s_in["Hbar"], s_in["dead"],
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
        self._host_setup(X_host, W0_host, F_host)
        cur = torch.cuda.current_stream(self.device)
        start = torch.cuda.Event()
        start.record(cur)
        counts = {}
        futs = [self.pool.submit(self._host_pipeline, name, start, X_host, W0_host, F_host, out_host, counts)
                for name in self.inputs]
        for f in futs:
            f.result()
        self._join(cur)
        return sum(v[0] for v in counts.values()), sum(v[1] for v in counts.values())

    def capture_host(self, X_host, W0_host, F_host, out_host):
        """capture() for run_host(): the graph holds the host-to-device copies
        of every step's inputs and the copies of the outputs back into
        out_host, so replay() is the whole step end to end from the same
        pinned host buffers.  Returns (h2d bytes, d2h bytes) per step."""
        self._host_setup(X_host, W0_host, F_host)
        torch.cuda.set_device(self.device)
        self._enqueue_host(X_host, W0_host, F_host, out_host)
        torch.cuda.synchronize(self.device)
        self.check_status()
        # without kernel priorities: a prioritised sweep would delay another
        # input's chunk accumulation, whose staging buffer then holds up the
        # shared copy stream (measured: 24 ms per step without, 27 with)
        self.graph = self._capture(lambda: self._enqueue_host(X_host, W0_host, F_host, out_host),
                                   node_priorities=False)
        return self.graph_counts

    def _enqueue_host(self, X_host, W0_host, F_host, out_host):
        cur = torch.cuda.current_stream(self.device)
        start = torch.cuda.Event()
        start.record(cur)
        counts = {}
        for name in self.chain_order:
            self._host_pipeline(name, start, X_host, W0_host, F_host, out_host, counts)
        self._join(cur)
        return sum(v[0] for v in counts.values()), sum(v[1] for v in counts.values())

    def _host_setup(self, X_host, W0_host, F_host):
        if self.act_quant is not None or self.sgroups:
            raise NotImplementedError("run_host: this variant runs from device-resident inputs")
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


# ---------------------------------------------------------------------------
# The block with the exact losses (Sec. 4.4 Eq. slide_window; Eq. kl_loss for
# the last block): Alg. 1's loop over the linear modules, one after another,
# each module's current pass seeing the modules quantized before it.

_MODULE_KEY = {"q_proj": "Wq", "k_proj": "Wk", "v_proj": "Wv", "o_proj": "Wo", "gate_proj": "Wg", "up_proj": "Wu",
               "down_proj": "Wd"}


@dataclass
class ExactModule:
    """One module's result: packed codes, scale, zero, the dequantized fp32
    weights, the optimizer step count and the per-block losses (before and
    after each block's steps; -1 where a block took none)."""
    codes: torch.Tensor
    scale: torch.Tensor
    zero: torch.Tensor
    W: torch.Tensor
    adam_t: int
    block_loss: torch.Tensor


def quantize_block_exact(dims, W_this: Dict[str, torch.Tensor], x: torch.Tensor, qcfg: QuantCfg, lr: float, *,
                         x_hat: Optional[torch.Tensor] = None, W_next: Optional[Dict[str, torch.Tensor]] = None,
                         F_this: Optional[torch.Tensor] = None, F_next: Optional[torch.Tensor] = None,
                         head_gf: Optional[torch.Tensor] = None, head_Wh: Optional[torch.Tensor] = None,
                         steps_per_block: int = 1, optimizer: int = REALQ_OPT_ADAM,
                         modules: Sequence[str] = BLOCK_MODULES, n_minibatch: int = 1, stream=None):
    """Quantizes the linear modules of decoder block l in order, each with
    Block-GD on the exact two-block window (W_next, F_this, F_next given) or,
    for the last block, on the KL at the LM head (head_gf, head_Wh given).

    W_this: block l's full-precision weights (the reference); x its
    full-precision input (S, L, d) and x_hat its input in the model quantized
    so far (default x).  For each module: its inputs in the current pass
    (realq_block_module_inputs with the weights quantized so far, on x_hat),
    their Hessian and factor, then realq_quantize_layer_window with b_global
    running over the column blocks of all the modules; its dequantized
    weights then replace it in the current weights.  With n_minibatch > 1
    the sequences of x form that many calibration mini-batches: the Hessians
    take all of them, each Block-GD step one in rotation.  Returns each
    module's ExactModule and the final current weights."""
    S_all, L, d = x.shape
    S = S_all // n_minibatch
    dev = x.device
    nb = {md: -(-W_this[_MODULE_KEY[md]].shape[1] // qcfg.block_size) for md in modules}
    B_total = sum(nb.values())
    vocab = int(head_Wh.shape[0]) if head_Wh is not None else 0
    W_hat = dict(W_this)
    bws = workspace(realq_block_workspace_size(dims, S_all, L), dev)
    g = qcfg.group_size
    out = {}
    b_start = 1
    for md in modules:
        key = _MODULE_KEY[md]
        m, n = W_this[key].shape
        X = torch.empty((S_all * L, n), dtype=torch.float32, device=dev)
        realq_block_module_inputs(dims, W_hat, x if x_hat is None else x_hat, md, X, bws, stream=stream)
        H, _, T = layer.accumulate([X], n, device=dev, stream=stream)
        prep = layer.prepare(H, T, qcfg.damp_frac, stream=stream)
        ngroups = -(-n // g) if g > 0 else 1
        W = torch.empty((m, n), dtype=torch.float32, device=dev)
        codes = torch.empty((m, (n + 1) // 2), dtype=torch.uint8, device=dev)
        scale = torch.empty((m, ngroups), dtype=torch.float32, device=dev)
        zero = torch.empty((m, ngroups), dtype=torch.uint8, device=dev)
        am = torch.empty((m, n), dtype=torch.float32, device=dev)
        av = torch.empty((m, n), dtype=torch.float32, device=dev)
        loss = torch.full((nb[md], 2), -1.0, dtype=torch.float32, device=dev)
        ws = workspace(realq_quantize_window_workspace_size(dims, S, L, md, qcfg, vocab), dev)
        b = bgd_cfg(lr, steps_per_block=steps_per_block, optimizer=optimizer, b_global_start=b_start,
                    B_total=B_total)
        t = realq_quantize_layer_window(dims, W_this, W_next if head_Wh is None else None, x, md, prep.U, qcfg, b,
                                        W, codes, scale, zero, F_this=F_this, F_next=F_next, head_gf=head_gf,
                                        head_Wh=head_Wh, dead=prep.dead, adam_m=am, adam_v=av, block_loss=loss,
                                        ws=ws, this_block_hat=W_hat, x_hat=x_hat, n_minibatch=n_minibatch,
                                        stream=stream)
        realq_workspace_status(ws, stream=stream)
        W_hat = dict(W_hat)
        W_hat[key] = W
        out[md] = ExactModule(codes, scale, zero, W, t, loss)
        b_start += nb[md]
    return out, W_hat


def quantize_model_exact(dims, blocks: Sequence[Dict[str, torch.Tensor]], x: torch.Tensor,
                         fishers: Sequence[torch.Tensor], head_gf: torch.Tensor, head_Wh: torch.Tensor,
                         qcfg: QuantCfg, lr_final: float, **kw):
    """Alg. 1's outer loop over a stack of decoder blocks with the exact
    losses: block l with quantize_block_exact against the two-block window
    with block l+1 (fishers[l], fishers[l+1]: the blocks' aggregated
    Fishers, d x d) or, for the last block, the KL at the LM head (head_gf,
    head_Wh), at the reverse-cosine learning rate of block l.  Block l+1's
    full-precision input is block l's full-precision output, and its input in
    the quantized model is block l's output with its quantized weights on its
    own such input (realq_block_forward).  kw go to quantize_block_exact.
    Returns [(modules, quantized weights)] per block."""
    Lb = len(blocks)
    S, L, d = x.shape
    ws = workspace(realq_block_workspace_size(dims, S, L), x.device)
    stream = kw.get("stream")
    x_ref, x_hat = x, x
    out = []
    for l, W in enumerate(blocks):
        last = l == Lb - 1
        lr = realq_reverse_cosine_lr(l + 1, Lb, lr_final)
        if last:
            res, W_hat = quantize_block_exact(dims, W, x_ref, qcfg, lr, x_hat=x_hat, head_gf=head_gf,
                                              head_Wh=head_Wh, **kw)
        else:
            res, W_hat = quantize_block_exact(dims, W, x_ref, qcfg, lr, x_hat=x_hat, W_next=blocks[l + 1],
                                              F_this=fishers[l], F_next=fishers[l + 1], **kw)
        out.append((res, W_hat))
        y_ref, y_hat = torch.empty_like(x), torch.empty_like(x)
        realq_block_forward(dims, W, x_ref, y_ref, ws, stream=stream)
        realq_block_forward(dims, W_hat, x_hat, y_hat, ws, stream=stream)
        x_ref, x_hat = y_ref, y_hat
    return out
