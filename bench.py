"""Throughput of the REAL-Q per-layer quantization sweep on GB300.

One step = the whole sweep of one synthetic decoder block (default: the
LLaMA-3.1-70B-shaped block, 256 x 2048 calibration tokens, the largest
block shape; --workload qwen3-0.6b | llama3.1-8b | qwen3-32b for the others):
for each of its four distinct inputs the Hessian over all tokens and its
preparation, then the column sweep with Block-GD of its seven linear modules.
Metric: quantized weight-columns per second (whole job; N GPUs run N
independent replicas).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gpu|reference]

Prints one JSON line (rank 0).  --impl reference times the fp64 CPU oracle on
a bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "quantized weight-columns/sec per layer on 1 GB300; % tensor-core peak / % HBM BW"
UNIT = "columns/s"

# dram bytes per launch from ncu captures (profiles/), keyed by (workload, kernel); None
# when the kernel changed after its capture.
NCU_TRAFFIC = {
    # the G product of the LLaMA-3.1-70B block (the persistent f16x3 kernel
    # with the fused Adam step): three down_proj launches captured in the
    # bench step with one-pass DRAM counters (14.29-14.51 GB each, 4.64 GB
    # per TFLOP), scaled to the family's average launch (1.128 TFLOP)
    ("llama3.1-70b", "bgd_g_gemm_adam"): 5234000000,
    # the gradient-factor product P of the same block: three down_proj
    # launches (28.4-30.7 GB each, 3.30 GB per TFLOP), scaled to the family's
    # average launch (1.995 TFLOP)
    ("llama3.1-70b", "bgd_p_gemm"): 6584000000,
    # the four Hessians of one step of the same block, one-pass counters:
    # down_in (n = 28,672) 1010 GB, the three n = 8192 inputs 58-66 GB each;
    # averaged per launch
    ("llama3.1-70b", "hessian_syrk_tc"): 299400000000,
}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                "sm_max_mhz": d.get("sm_max_mhz", 2070.0), "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "sm_max_mhz": 2070.0,
                "source": "fallback"}


# --------------------------------------------------------------------------
# clocks sampled during the timed region
# --------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid, log_dir=None):
        self.uuid = uuid
        self.proc = None
        self.path = os.path.join(log_dir or tempfile.gettempdir(), f"clocks_{os.getpid()}.csv")

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "100"], stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            if self.uuid and self.uuid not in parts[1]:
                continue
            try:
                sm.append(float(parts[2]))
                mx = float(parts[3])
            except ValueError:
                continue
            for nm, v in zip(names, parts[6:10]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------------
# the GPU arm
# --------------------------------------------------------------------------
def max_over_ranks(x: float, dist=None, device="cpu") -> float:
    """The largest of every rank's x (each rank's replica timed on its own
    clock; the job takes as long as its slowest rank); x itself on one rank."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([float(x)], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(columns_per_step: int, steps: int, world: int, ms: float) -> float:
    """Whole-job columns/s: every rank quantizes its own replica of the block."""
    return columns_per_step * steps * world / (ms / 1e3)


def gpu_arm(args, wl, rank, world):
    import torch
    import paper_2609_00049_gb300 as rq
    from paper_2609_00049_gb300 import build as rqbuild
    from paper_2609_00049_gb300.block import BlockInput, BlockModule, BlockQuantizer

    rqbuild.build()
    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    rq.lib()
    rq.realq_set_bgd_products(args.bgd_products)
    rq.realq_set_tensor_overlap(args.tensor_overlap)
    stream = torch.cuda.current_stream()
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    def barrier():
        if dist is not None:
            dist.barrier()

    t_gen = time.time()
    # ---- inputs: generated on the host (seeded) straight into page-locked
    # memory, then resident on the device
    host_x, dev_x = {}, {}
    for name, spec in wl.inputs.items():
        t = torch.empty((spec.T, spec.n), dtype=torch.int16, pin_memory=True)
        synth.xhat_full(wl, name, as_bits=True, threads=os.cpu_count() or 8, out=t.numpy())
        t = t.view(torch.bfloat16)
        host_x[name] = t
        dev_x[name] = t.to(dev, non_blocking=True)
    host_w, dev_w, host_f, dev_f = {}, {}, {}, {}
    for mod in wl.modules:
        t = torch.from_numpy(synth.weights(wl, mod).view(np.int16)).view(torch.bfloat16).pin_memory()
        host_w[mod.name] = t
        dev_w[mod.name] = t.to(dev, non_blocking=True)
        f = torch.from_numpy(synth.fisher(wl, mod)).pin_memory()
        host_f[mod.name] = f
        dev_f[mod.name] = f.to(dev, non_blocking=True)
    torch.cuda.synchronize()
    t_gen = time.time() - t_gen

    qcfg = rq.quant_cfg(wl.bits, wl.group_size, wl.block_size, wl.symmetric, wl.damp_frac)
    dev_fn = None
    if wl.sliding_window:
        dev_fn = {mod.name: torch.from_numpy(synth.fisher(wl, mod, "F_next")).to(dev) for mod in wl.modules}
    # the block's modules, scheduled concurrently by the library's block scheduler
    bq = BlockQuantizer([BlockInput(nm, sp.n, sp.T) for nm, sp in wl.inputs.items()],
                        [BlockModule(md.name, md.m, md.n, md.input) for md in wl.modules], qcfg, wl.lr,
                        wl.steps_per_block, sliding_window=wl.sliding_window, device=dev,
                        act_quant=(args.act_bits, args.a_clip) if args.act_bits else None,
                        saliency_groups=args.saliency_groups, minibatch_tokens=2048 * args.minibatch_seqs,
                        a_loss_clip=args.a_loss_clip)
    dev_sal = None
    if args.saliency_groups:
        dev_sal = {mod.name: torch.from_numpy(synth.saliency(wl, mod, args.saliency_groups)).to(dev)
                   for mod in wl.modules}
    host_out = {mod.name: {k: torch.empty_like(bq.out[mod.name][k], device="cpu").pin_memory()
                           for k in ("codes", "scale", "zero")} for mod in wl.modules}
    e2e_bytes = {"h2d": 0, "d2h": 0}

    # One step enqueues about a thousand small kernels over eleven streams;
    # by default it is captured once into a CUDA graph and replayed (every
    # kernel still runs every step, on the same resident inputs).  The
    # saliency-grouped variant reads token weights on the host mid-step and
    # always runs eagerly.
    use_graph = not args.no_graph and not args.saliency_groups
    if use_graph:
        bq.capture(dev_x, dev_w, dev_f, dev_fn)

    def step_device():
        if use_graph:
            bq.replay()
        else:
            bq.run(dev_x, dev_w, dev_f, dev_fn, saliency=dev_sal)
        bq.check_status()

    def step_serial():
        bq.run_serial(dev_x, dev_w, dev_f, dev_fn, saliency=dev_sal)

    def step_e2e():
        if use_graph:
            bq.replay()
        else:
            e2e_bytes["h2d"], e2e_bytes["d2h"] = bq.run_host(host_x, host_w, host_f, host_out)
        bq.check_status()
        torch.cuda.current_stream().synchronize()

    # ---- warm-up
    for _ in range(args.warmup):
        step_device()
    torch.cuda.synchronize()
    barrier()

    # ---- timed region (device-resident inputs)
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    clocks = ClockSampler(uuid, args.clock_log)
    launches0 = rq.realq_launch_count()
    clocks.start()
    torch.cuda.synchronize()
    barrier()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        step_device()
    t1.record(stream)
    torch.cuda.synchronize()
    barrier()
    ms_total = t0.elapsed_time(t1)
    clk = clocks.stop()
    launches = rq.realq_launch_count() - launches0   # a graph launch adds the library kernels it holds

    # The same K steps again, serialized on one stream, with every library
    # launch bracketed by CUDA events on that stream: per-kernel device time for
    # the breakdown and the roofline (in the concurrent timed run the event
    # intervals of overlapping kernels would include each other's time).
    # (at most two steps: the per-launch averages settle after one)
    prof = {}
    prof_steps = min(args.steps, 2)
    if not args.no_profile:
        rq.realq_profile_collect()          # drop anything pending
        rq.realq_profile_enable(True)
        for _ in range(prof_steps):
            step_serial()
        torch.cuda.synchronize()
        rq.realq_profile_enable(False)
        prof = rq.realq_profile_collect(256)
    ms_total = max_over_ranks(ms_total, dist, dev)
    cols = wl.total_columns * args.steps * world
    value = job_throughput(wl.total_columns, args.steps, world, ms_total)

    # ---- end to end through host buffers (at most three steps: each moves
    # every input across the host link again)
    e2e = None
    e_steps = min(args.steps, 3)
    if not args.no_e2e and not args.act_bits and not args.saliency_groups and not args.minibatch_seqs:
        if use_graph:
            e2e_bytes["h2d"], e2e_bytes["d2h"] = bq.capture_host(host_x, host_w, host_f, host_out)
        step_e2e()
        torch.cuda.synchronize()
        barrier()
        e0 = time.perf_counter()
        a0 = torch.cuda.Event(enable_timing=True)
        a1 = torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for _ in range(e_steps):
            step_e2e()
        a1.record(stream)
        torch.cuda.synchronize()
        barrier()
        e_ms = (time.perf_counter() - e0) * 1e3
        e_ms = max_over_ranks(e_ms, dist, dev)
        e_cols = wl.total_columns * e_steps * world
        # the host link's rate right after the timed steps (one pinned copy of
        # the largest input): the end-to-end step is bound by it, and the
        # link is shared with the host's other GPUs
        big = max(host_x.values(), key=lambda t: t.numel())
        dst = dev_x[max(dev_x, key=lambda k: dev_x[k].numel())]
        torch.cuda.synchronize()
        l0 = time.perf_counter()
        dst.copy_(big, non_blocking=True)
        torch.cuda.synchronize()
        link_gbs = big.numel() * big.element_size() / (time.perf_counter() - l0) / 1e9
        e2e = {"value": e_cols / (e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": e2e_bytes["h2d"],
               "d2h_bytes_per_step": e2e_bytes["d2h"], "ms_per_step": e_ms / e_steps, "steps": e_steps,
               "h2d_link_gbs": round(link_gbs, 1)}

    result = None
    if rank == 0:
        peaks = load_peaks()
        roof = roofline(wl, prof, prof_steps, peaks, args)
        # a side measurement outside the timed region: one Block-GD gradient
        # of the exact two-block window on a decoder-block shape (the sweep
        # variant whose loss runs through the block ops)
        window = None if args.no_window else window_measure(args, peaks, 3, 1)
        result = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_total / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": f"synthetic (seeded; {wl.description}; bf16 weights, random init)",
            "config": {"workload": wl.name, "description": wl.description, "modules": len(wl.modules),
                       "calibration_tokens": wl.inputs[wl.modules[0].input].T,
                       "columns_per_step": wl.total_columns, "column_blocks_per_step": wl.total_column_blocks,
                       "quantizer": f"W{wl.bits}" + (f"A{args.act_bits} (activation-aware, a_clip {args.a_clip})"
                                                     if args.act_bits else "") +
                                    f" {'sym' if wl.symmetric else 'asym'} g{wl.group_size} B{wl.block_size}" +
                                    (f", saliency-weighted grouped Hessians (N_g={args.saliency_groups}, clip p99)"
                                     if args.saliency_groups else ""),
                       "bgd": f"Adam lr={wl.lr} steps_per_block={wl.steps_per_block}" +
                              (f", mini-batches of {args.minibatch_seqs} x 2048 tokens" if args.minibatch_seqs else "") +
                              (f", token-form gradient with a_loss_clip {args.a_loss_clip}" if args.a_loss_clip
                               else ""),
                       "parallelism": f"replicas x{world}",
                       "launch": "one CUDA graph per step (11 streams)" if use_graph else
                                 "eager, one host thread per input",
                       "l2": "inputs larger than L2: %.2f GB of calibration activations streamed per step" %
                             (sum(s.T * s.n * 2 for s in wl.inputs.values()) / 1e9),
                       "input_generation_s": round(t_gen, 1)},
            "roofline": roof,
            "roofline_by_kernel": roofline_table(wl, prof, prof_steps, peaks, args),
            "profile_steps": prof_steps if prof else 0,
            "kernels": {k: {"launches": v[0], "ms": round(v[1], 3)} for k, v in
                                           sorted(prof.items(), key=lambda kv: -kv[1][1])},
            "gpu_launches": int(launches), "clocks": clk, "e2e": e2e, "window": window,
        }
    if dist is not None:
        dist.destroy_process_group()
    return result


def work_models(wl, args=None):
    """Algorithmic work per step of each kernel family: (bound, work, unit)."""
    per_step = {}
    # algorithmic work per step of each kernel family
    hess_flops = sum(s.T * s.n * (s.n + 1) for s in wl.inputs.values())       # symmetric X^T X
    per_step["hessian_syrk_simt"] = ("tensor", hess_flops, "TFLOP/s")
    per_step["hessian_syrk_tc"] = ("tensor", hess_flops, "TFLOP/s")
    ng = getattr(args, "saliency_groups", 0) or 0
    if ng:
        # per module and row group: X̂ᵀ (s X̂) as two bf16 passes (high and low
        # part of s x) over the lower tiles
        wflops = sum(2 * wl.inputs[md.input].T * md.n * (md.n + 1) * ng for md in wl.modules)
        per_step["hessian_weighted_tc"] = ("tensor", wflops, "TFLOP/s")
        per_step["saliency_scale"] = ("hbm", sum(wl.inputs[md.input].T * md.n * 6 * ng for md in wl.modules),
                                      "GB/s")
    if getattr(args, "act_bits", 0):
        # D = X̂ᵀX̂ - XᵀX̂: the full non-symmetric product XᵀX̂ per input
        per_step["hessian_cross_tc"] = ("tensor", sum(2 * s.T * s.n * s.n for s in wl.inputs.values()), "TFLOP/s")
        per_step["act_quant"] = ("hbm", sum(s.T * s.n * 2 * 3 for s in wl.inputs.values()), "GB/s")
    bgd_p = bgd_g = trail = trail_planes = 0
    serial_bytes = 0
    for md in wl.modules:
        m, n, B = md.m, md.n, wl.block_size
        for b in range(-(-n // B)):
            be = min((b + 1) * B, n)
            r = n - be
            # M = A H̄ is kept current: the product takes the previous step's
            # free columns (K = n - b B; none before the first step)
            bgd_p += 2 * m * (n - b * B) * r if b > 0 else 0
            bgd_g += 2 * m * m * r
            trail += 2 * m * (be - b * B) * r
            if r > 0:
                # the update's operands as tf32 planes: read E_b and the U
                # panel once, write both planes of each
                trail_planes += 12 * (be - b * B) * (m + r)
            serial_bytes += m * (be - b * B) * (4 + 4 + 4) + m * (be - b * B) // 2
    if getattr(args, "a_loss_clip", None) and getattr(args, "minibatch_seqs", 0):
        # token-form gradient per optimizer step (every block but the last):
        # Δ = X̂_k ΔWᵀ, Z = (κ ⊙ Δ) F, G = gᵀ X̂_k[:, free] on T_k tokens
        tr = tf = tg = clip_b = conv_b = gt_b = 0
        for md in wl.modules:
            m, n, B = md.m, md.n, wl.block_size
            Tk = min(2048 * args.minibatch_seqs, wl.inputs[md.input].T)
            for b in range(-(-n // B) - 1):
                r = n - min((b + 1) * B, n)
                tr += 2 * Tk * m * n
                tf += 2 * Tk * m * m
                tg += 2 * m * r * Tk
                clip_b += Tk * m * 16          # read Δ, write κ and Y's two planes
                conv_b += Tk * n * 10          # read bf16, write fp32 both ways
                gt_b += Tk * m * 16            # read κ and Z, write two planes
        per_step["tok_residual_gemm"] = ("tf32x3", tr, "TFLOP/s")
        per_step["tok_fisher_gemm"] = ("tf32x3", tf, "TFLOP/s")
        per_step["tok_grad_gemm"] = ("tf32x3", tg, "TFLOP/s")
        per_step["tok_clip"] = ("hbm", clip_b, "GB/s")
        per_step["tok_xconv"] = ("hbm", conv_b, "GB/s")
        per_step["tok_grad_t"] = ("hbm", gt_b, "GB/s")
    # the plain Block-GD products run as f16x3 where m, n and the block are
    # multiples of 8 (and the precision switch is on); the row-grouped,
    # mini-batch and token forms as tf32x3
    plain = not (ng or getattr(args, "minibatch_seqs", 0))
    f16 = plain and getattr(args, "bgd_products", 1) == 1 and wl.block_size % 8 == 0 and all(
        md.m % 8 == 0 and md.n % 8 == 0 for md in wl.modules)
    per_step["bgd_p_gemm"] = ("f16x3" if f16 else "tf32x3", bgd_p, "TFLOP/s")
    per_step["bgd_g_gemm_adam"] = ("f16x3" if f16 else "tf32x3", bgd_g, "TFLOP/s")
    if f16:
        # the step's and P^T's fp16 planes, per block: read the fp32 values
        # twice (row maximum, then split) and write two 2-byte planes
        f16_split = 0
        for md in wl.modules:
            m, n, B = md.m, md.n, wl.block_size
            for b in range(-(-n // B)):
                r = n - min((b + 1) * B, n)
                f16_split += 12 * m * (n - b * B) * (b > 0) + 12 * m * r
        per_step["f16_split"] = ("hbm", f16_split, "GB/s")
    per_step["trailing_update"] = ("tf32x3", trail, "TFLOP/s")
    per_step["trailing_planes"] = ("hbm", trail_planes, "GB/s")
    per_step["quant_block"] = ("hbm", serial_bytes, "GB/s")
    prep_flops = sum(2 * s.n ** 3 // 3 for s in wl.inputs.values())
    per_step["chol_diag"] = ("alu", sum(s.n * 64 * 64 for s in wl.inputs.values()), "TFLOP/s")
    # the rank-64 updates: the look-ahead column on fp32 tiles (2 k0 64^2 flop
    # per step, about 64 n^2 in all), the rest on the tensor cores; the
    # triangular inverse's product on the tensor cores, or on fp32 tiles
    # where the workspace lacks the planes of U^T
    tc_prep = [s for s in wl.inputs.values() if s.n > 512 and s.n % 4 == 0]
    per_step["chol_update"] = ("alu", sum(64 * s.n ** 2 for s in wl.inputs.values()) +
                               sum(s.n ** 3 // 3 for s in wl.inputs.values() if s not in tc_prep), "TFLOP/s")
    per_step["chol_update_tc"] = ("tf32x3", sum(s.n ** 3 // 3 - 64 * s.n ** 2 for s in tc_prep), "TFLOP/s")
    per_step["trtri_trmm_tc"] = ("tf32x3", sum(s.n ** 3 // 3 for s in tc_prep), "TFLOP/s")
    per_step["trtri_trmm"] = ("alu", sum(s.n ** 3 // 3 for s in wl.inputs.values() if s not in tc_prep), "TFLOP/s")
    return per_step


def roofline_entry(wl, name, launches, ms, steps, peaks, per_step):
    """Achieved against peak for one kernel family from its summed event time."""
    if name not in per_step:
        return {"kernel": name, "bound": None, "achieved": None, "peak": None, "unit": None, "frac": None,
                "traffic": None, "note": "no algorithmic model for this kernel"}
    bound, work, unit = per_step[name]
    secs = ms / 1e3
    total = work * steps
    fp32_alu_tflops = 152 * 128 * 2 * peaks["sm_max_mhz"] * 1e6 / 1e12
    if bound == "tensor":
        achieved = total / secs / 1e12
        peak = peaks["bf16_tflops_sustained"]
        peak_note = f"bf16 dense, sustained, {peaks['source']}"
    elif bound == "tf32x3":
        # fp32-accurate contraction as three tf32 tensor passes: the peak for
        # this dtype is the tf32 rate (measured bf16 x nominal 1.1/2.25) over 3
        bound = "tensor"
        achieved = total / secs / 1e12
        peak = peaks["bf16_tflops_sustained"] * (1.1 / 2.25) / 3.0
        peak_note = f"fp32 via 3 tf32 passes: sustained bf16 x 1.1/2.25 / 3, {peaks['source']}"
    elif bound == "f16x3":
        # fp32-accurate contraction as three fp16 tensor passes over
        # power-of-two row-scaled planes: fp16 runs at the bf16 rate
        bound = "tensor"
        achieved = total / secs / 1e12
        peak = peaks["bf16_tflops_sustained"] / 3.0
        peak_note = f"fp32 via 3 fp16 passes: sustained bf16 / 3, {peaks['source']}"
    elif bound == "alu":
        achieved = total / secs / 1e12
        peak = fp32_alu_tflops
        peak_note = "fp32 FFMA: 152 SMs x 128 lanes x 2 flop x max SM clock"
    else:
        achieved = total / secs / 1e9
        peak = peaks["hbm_gbs"]
        peak_note = f"HBM copy, {peaks['source']}"
    traffic = NCU_TRAFFIC.get((wl.name, name))
    return {"kernel": name, "bound": bound, "achieved": achieved, "peak": peak, "unit": unit,
            "frac": achieved / peak, "traffic": traffic, "peak_source": peak_note,
            "launches": launches, "avg_launch_ms": ms / launches,
            "work_per_step": work}


def roofline(wl, prof, steps, peaks, args=None):
    """Roofline entry for the kernel with the largest share of device time."""
    if not prof:
        return None
    name, (launches, ms) = max(prof.items(), key=lambda kv: kv[1][1])
    return roofline_entry(wl, name, launches, ms, steps, peaks, work_models(wl, args))


def roofline_table(wl, prof, steps, peaks, args=None, top=8):
    """The same entry for every kernel family with a work model, by device time."""
    if not prof:
        return []
    models = work_models(wl, args)
    rows = sorted(((n, v) for n, v in prof.items() if n in models and models[n][1] > 0 and v[1] > 0 and v[0] > 0),
                  key=lambda kv: -kv[1][1])[:top]
    out = []
    for n, (launches, ms) in rows:
        e = roofline_entry(wl, n, launches, ms, steps, peaks, models)
        out.append({k: e[k] for k in ("kernel", "bound", "achieved", "peak", "unit", "frac")})
    return out


# --------------------------------------------------------------------------
# the CPU oracle (cpu_baseline leg and the reference arm)
# --------------------------------------------------------------------------
def oracle_sample(wl, token_sample=4096, max_columns=128):
    """Times the fp64 oracle, as it stands, on one bounded sample of the
    workload: the k_proj module (or the first), its Hessian over the first
    token_sample calibration tokens, then preparation (H̄, damping, the
    inverse) and the literal column sweep with Block-GD over the module's
    first max_columns columns (the whole module when n <= 2048), each
    column's compensation and Schur downdate applied to every remaining
    column of the full n x n inverse.  Returns (columns swept per second of
    the whole sample, description, seconds).  Nothing is extrapolated: the
    sample's Hessian is cheaper than the full one (fewer tokens) and its
    preparation is whole, so the rate is of this sample, not of the module."""
    import oracle
    mod = next((md for md in wl.modules if md.name == "k_proj"), wl.modules[0])
    spec = wl.inputs[mod.input]
    cols = mod.n if mod.n <= 2048 else min(max_columns, mod.n)
    X = synth.xhat_full(wl, mod.input, as_bits=False, max_tokens=min(token_sample, spec.T))
    W0 = synth.weights(wl, mod, as_bits=False)
    F = synth.fisher(wl, mod)
    Fn = synth.fisher(wl, mod, "F_next") if wl.sliding_window else None
    t0 = time.perf_counter()
    Hs, T = oracle.hessian_sum([X])
    t_h = time.perf_counter() - t0
    t1 = time.perf_counter()
    oracle.realq_sweep(W0, Hs, T, bits=wl.bits, group_size=wl.group_size, block_size=wl.block_size,
                       symmetric=bool(wl.symmetric), damp_frac=wl.damp_frac,
                       bgd={"lr": wl.lr, "steps_per_block": wl.steps_per_block}, F=F, F_next=Fn, record=False,
                       columns=cols)
    t_s = time.perf_counter() - t1
    total = t_h + t_s
    desc = (f"{mod.name} ({mod.n}->{mod.m}) of {wl.name}: Hessian over the first {T} of {spec.T} tokens "
            f"({t_h:.2f} s), prepare + literal sweep with Block-GD of columns 0..{cols - 1} of {mod.n} "
            f"({t_s:.2f} s); rate = {cols} columns / {total:.2f} s")
    return cols / total, desc, total


def cpu_cores():
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS"):
        if os.environ.get(k):
            return int(os.environ[k])
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads") for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(n[0])
    except Exception:
        pass
    return os.cpu_count()


def reference_arm(args, wl, rank, world):
    """The fp64 oracle on the host cores, one bounded sample per step
    (oracle_sample), rank 0 only."""
    if rank != 0:
        return None
    vals, descs, secs = [], None, []
    for _ in range(args.warmup):
        oracle_sample(wl)
    for _ in range(args.steps):
        v, descs, s = oracle_sample(wl)
        vals.append(v)
        secs.append(s)
    value = statistics.mean(vals)
    cb = {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle", "sample": descs}
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * statistics.mean(secs),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": f"synthetic (seeded; {wl.description})",
            "config": {"workload": wl.name, "description": wl.description, "sample": descs}, "cpu_baseline": cb,
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def kernel_bench(args):
    """Times one kernel family alone on a synthetic case sized by --n / --tokens
    (the small-case target of ncu captures).  Prints one JSON line."""
    import torch
    import paper_2609_00049_gb300 as rq
    from paper_2609_00049_gb300 import build as rqbuild
    rqbuild.build()
    rq.lib()
    rq.realq_set_bgd_products(args.bgd_products)
    rq.realq_set_tensor_overlap(args.tensor_overlap)
    from paper_2609_00049_gb300 import layer
    peaks = load_peaks()
    if args.kernel == "window":
        return window_bench(args, peaks)
    n, T = args.n, args.tokens
    wl = synth.Workload("kernel", {"x": synth.InputSpec("x", n, T, "gauss", outlier_frac=0.01, outlier_scale=20.0)},
                        [synth.ModuleSpec("w", args.m, n, "x")], seed=1, lr=3e-4)
    X = torch.from_numpy(synth.xhat_full(wl, "x").view(np.int16)).view(torch.bfloat16).cuda()
    stream = torch.cuda.current_stream()
    H = torch.zeros(n, n, device="cuda")
    ws = rq.workspace(rq.realq_hessian_workspace_size(n, T))
    if args.kernel == "hessian":
        def run():
            rq.realq_hessian_accumulate(X, H, ws=ws)
    else:
        rq.realq_hessian_accumulate(X, H, ws=ws)
        prep = layer.prepare(H, T)
        if args.kernel == "prepare":
            def run():
                layer.prepare(H, T)
        else:
            mod = wl.modules[0]
            W0 = torch.from_numpy(synth.weights(wl, mod).view(np.int16)).view(torch.bfloat16).cuda()
            F = torch.from_numpy(synth.fisher(wl, mod)).cuda()
            q = rq.quant_cfg()
            b = rq.bgd_cfg(wl.lr)
            qws = rq.workspace(rq.realq_quantize_workspace_size(mod.m, n, q, b))

            def run():
                layer.quantize(W0, prep, q, b, F=F, ws=qws)
    for _ in range(args.warmup):
        run()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        run()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    if args.kernel != "hessian":
        print(json.dumps({"kernel": args.kernel, "m": args.m, "n": n, "ms_per_call": ms}))
        return
    flops = T * n * (n + 1)
    tf = flops / (ms / 1e3) / 1e12
    print(json.dumps({"kernel": "hessian_syrk_tc", "n": n, "tokens": T, "ms_per_launch": ms, "achieved": tf,
                      "unit": "TFLOP/s", "peak": peaks["bf16_tflops"], "frac": tf / peaks["bf16_tflops"],
                      "peak_source": f"bf16 dense burst, {peaks['source']}",
                      "input_bytes": T * n * 2}))


def window_bench(args, peaks):
    """Prints window_measure's JSON line (--kernel window)."""
    print(json.dumps(window_measure(args, peaks, args.steps, args.warmup)))


def window_measure(args, peaks, steps, warmup):
    """Times one Block-GD gradient of the exact two-block window
    (realq_block_module_window for down_proj: block l's reference and
    current passes, the next block's two passes and its backward, block l's
    backward to the module) on one decoder-block shape, with seeded random
    weights and inputs.  Returns a dict."""
    import torch
    import paper_2609_00049_gb300 as rq
    d, H, Hkv, dh, f = args.d, args.heads, args.kv_heads, args.head_dim, args.ffn
    S, L = args.seqs, args.seq_len
    T = S * L
    g = torch.Generator().manual_seed(5)

    def w(rows, cols):
        return (torch.randn(rows, cols, generator=g) * 0.8 / cols ** 0.5).cuda()

    def block():
        return {"g1": (1 + 0.1 * torch.randn(d, generator=g)).cuda(), "Wq": w(H * dh, d), "Wk": w(Hkv * dh, d),
                "Wv": w(Hkv * dh, d), "Wo": w(d, H * dh), "g2": (1 + 0.1 * torch.randn(d, generator=g)).cuda(),
                "Wg": w(f, d), "Wu": w(f, d), "Wd": w(d, f)}

    rq.realq_set_block_products(args.block_products)
    Wl, Wn = block(), block()
    x = torch.randn(S, L, d, generator=g).cuda()
    x_hat = x + 0.05 * torch.randn(S, L, d, generator=g).cuda()
    Z = torch.randn(d, 16, generator=g)
    F = (0.5 * torch.eye(d) + Z @ Z.T / 32).cuda()
    Wm = Wl["Wd"] + 0.01 * torch.randn(d, f, generator=g).cuda()
    dims = rq.block_dims(d, H, Hkv, dh, f)
    ws = rq.workspace(rq.realq_block_module_workspace_size(dims, S, L))
    grad = torch.empty(d, f, device="cuda")
    loss = torch.zeros(1, device="cuda")
    stream = torch.cuda.current_stream()

    def run():
        rq.realq_block_module_window(dims, Wl, Wn, x, "down_proj", Wm, 0.5, F, F, grad, ws, loss=loss,
                                     x_hat=x_hat)
    for _ in range(warmup):
        run()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        run()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    rq.realq_workspace_status(ws)
    # one forward pass: the seven projections and the causal attention
    # (q.k and p.v over half the sequence on average); a backward is about
    # two forwards; a call runs four forwards and two backwards
    fwd = 2 * T * (2 * d * H * dh + 2 * d * Hkv * dh + 3 * d * f) + 2 * T * L * H * dh
    flop = 8 * fwd
    tf = flop / (ms / 1e3) / 1e12
    if args.block_products:
        # the projections as tf32x3 tensor-core products (the attention stays
        # on the CUDA cores)
        peak = peaks["bf16_tflops_sustained"] * (1.1 / 2.25) / 3.0
        src, bound = f"fp32 via 3 tf32 passes: sustained bf16 x 1.1/2.25 / 3, {peaks['source']}", "tensor"
    else:
        peak = 152 * 128 * 2 * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12
        src, bound = "fp32 ALU: 152 SMs x 128 lanes x 2 x max clock", "alu"
    return {"kernel": "block_module_window", "d": d, "heads": H, "kv_heads": Hkv, "head_dim": dh, "ffn": f,
            "seqs": S, "seq_len": L, "block_products": args.block_products, "steps": steps, "ms_per_call": ms,
            "achieved": tf, "unit": "TFLOP/s", "peak": peak, "frac": tf / peak, "peak_source": src, "bound": bound}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gpu", choices=["gpu", "reference"])
    ap.add_argument("--workload", default="llama3.1-70b")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--act-bits", type=int, default=0,
                    help="activation-aware weight-activation variant: per-token activation bits (0: weights only)")
    ap.add_argument("--a-clip", type=float, default=0.9, help="activation clipping ratio for --act-bits")
    ap.add_argument("--minibatch-seqs", type=int, default=0,
                    help="mini-batch Block-GD with this many 2048-token sequences per step (0: full batch)")
    ap.add_argument("--saliency-groups", type=int, default=0,
                    help="saliency-weighted grouped Hessians with this many row groups (0: one Hessian per input)")
    ap.add_argument("--bgd-products", type=int, choices=[0, 1], default=1,
                    help="the plain Block-GD products as f16x3 (1, where the shapes allow) or tf32x3 (0)")
    ap.add_argument("--tensor-overlap", type=int, choices=[0, 1, 2], default=1,
                    help="wide-tile f16x3 products as persistent kernels with the epilogue overlapped: 1 the G "
                         "product, 2 G and P, 0 none (one tile per CTA)")
    ap.add_argument("--a-loss-clip", type=float, default=None,
                    help="with --minibatch-seqs: token-form Block-GD gradient with per-token output clipping")
    ap.add_argument("--clock-log", default=None, help="directory for the raw clock samples (default: temp dir)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-window", action="store_true", help="skip the window gradient's side measurement")
    ap.add_argument("--no-profile", action="store_true", help="skip the event-profiled pass")
    ap.add_argument("--no-graph", action="store_true", help="launch the block step eagerly instead of as a CUDA graph")
    ap.add_argument("--kernel", choices=["hessian", "prepare", "sweep", "window"], default=None,
                    help="time one stage alone on a small synthetic case (window: the exact two-block window's "
                         "gradient on the decoder-block shape below)")
    ap.add_argument("--d", type=int, default=1024)
    ap.add_argument("--heads", type=int, default=16)
    ap.add_argument("--kv-heads", type=int, default=8)
    ap.add_argument("--head-dim", type=int, default=128)
    ap.add_argument("--ffn", type=int, default=3072)
    ap.add_argument("--seqs", type=int, default=2)
    ap.add_argument("--seq-len", type=int, default=2048)
    ap.add_argument("--block-products", type=int, choices=[0, 1], default=0,
                    help="window: the block ops' products on tf32x3 tensor cores (1) or fp32 CUDA cores (0)")
    ap.add_argument("--n", type=int, default=2048)
    ap.add_argument("--m", type=int, default=1024)
    ap.add_argument("--tokens", type=int, default=65536)
    args = ap.parse_args()
    if args.kernel:
        kernel_bench(args)
        return
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    wl = synth.workloads()[args.workload]
    if args.impl == "reference":
        res = reference_arm(args, wl, rank, world)
    else:
        res = gpu_arm(args, wl, rank, world)
        if res is not None and rank == 0 and world == 1 and not args.no_cpu_baseline:
            v, desc, _ = oracle_sample(wl)
            res["cpu_baseline"] = {"value": v, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle", "sample": desc}
        elif res is not None:
            res["cpu_baseline"] = None
    if rank == 0 and res is not None:
        print(json.dumps(res))


if __name__ == "__main__":
    main()
