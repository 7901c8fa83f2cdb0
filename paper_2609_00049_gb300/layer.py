"""One linear module through the C ABI: allocate outputs and workspaces with
torch, then call accumulate -> prepare -> quantize_layer.  No arithmetic here."""
from __future__ import annotations

from dataclasses import dataclass
from typing import Iterable, Optional

import torch

from . import (BgdCfg, QuantCfg, realq_hessian_accumulate, realq_hessian_prepare, realq_hessian_workspace_size,
               realq_prepare_workspace_size, realq_quantize_layer, realq_quantize_workspace_size,
               realq_scale_moment, workspace, REALQ_BF16, REALQ_F32)


@dataclass
class Prepared:
    U: torch.Tensor
    Hbar: torch.Tensor
    dead: torch.Tensor
    T: int
    Dbar: Optional[torch.Tensor] = None


@dataclass
class Quantized:
    codes: torch.Tensor
    scale: torch.Tensor
    zero: torch.Tensor
    W: torch.Tensor          # fp32 dequantized weights
    adam_t: int


def accumulate(chunks: Iterable[torch.Tensor], n: int, x_fp_chunks: Optional[Iterable[torch.Tensor]] = None,
               device="cuda", stream=None):
    """H_sum (and D_sum) over device chunks of calibration tokens; returns (H_sum, D_sum, T)."""
    H = torch.zeros((n, n), dtype=torch.float32, device=device)
    D = torch.zeros((n, n), dtype=torch.float32, device=device) if x_fp_chunks is not None else None
    T = 0
    xf_iter = iter(x_fp_chunks) if x_fp_chunks is not None else None
    ws, ws_cap = None, 0
    for c in chunks:
        xf = next(xf_iter) if xf_iter is not None else None
        dt = REALQ_BF16 if c.dtype == torch.bfloat16 else REALQ_F32
        need = realq_hessian_workspace_size(n, c.shape[0], dt, xf is not None)
        if need > ws_cap:
            ws, ws_cap = workspace(need, device), need
        realq_hessian_accumulate(c, H, D, xf, ws=ws if need else None, stream=stream)
        T += c.shape[0]
    return H, D, T


def prepare(H_sum: torch.Tensor, T: int, damp_frac: float = 0.01, D_sum: Optional[torch.Tensor] = None,
            stream=None) -> Prepared:
    n = H_sum.shape[0]
    U = torch.empty_like(H_sum)
    Hbar = torch.empty_like(H_sum)
    dead = torch.empty(n, dtype=torch.uint8, device=H_sum.device)
    ws = workspace(realq_prepare_workspace_size(n), H_sum.device)
    realq_hessian_prepare(H_sum, T, damp_frac, U, Hbar, dead, ws, stream=stream)
    Dbar = None
    if D_sum is not None:
        Dbar = torch.empty_like(D_sum)
        realq_scale_moment(D_sum, T, Dbar, stream=stream)
    return Prepared(U, Hbar, dead, T, Dbar)


def quantize(W0: torch.Tensor, prep: Prepared, qcfg: QuantCfg, bcfg: Optional[BgdCfg] = None,
             F: Optional[torch.Tensor] = None, F_next: Optional[torch.Tensor] = None, use_dbar: bool = True,
             stream=None, ws: Optional[torch.Tensor] = None) -> Quantized:
    m, n = W0.shape
    dev = W0.device
    g = qcfg.group_size if qcfg.group_size > 0 else n
    ngroups = -(-n // g)
    bgd = bcfg is not None and bcfg.steps_per_block > 0
    Dbar = prep.Dbar if (use_dbar and bgd) else None
    W = torch.empty((m, n), dtype=torch.float32, device=dev)
    codes = torch.empty((m, (n + 1) // 2), dtype=torch.uint8, device=dev)
    scale = torch.empty((m, ngroups), dtype=torch.float32, device=dev)
    zero = torch.empty((m, ngroups), dtype=torch.uint8, device=dev)
    am = torch.empty((m, n), dtype=torch.float32, device=dev) if bgd else None
    av = torch.empty((m, n), dtype=torch.float32, device=dev) if bgd else None
    disp = torch.empty((m, n), dtype=torch.float32, device=dev) if bgd else None
    if ws is None:
        ws = workspace(realq_quantize_workspace_size(m, n, qcfg, bcfg, F_next is not None, Dbar is not None), dev)
    t = realq_quantize_layer(W0, prep.U, prep.Hbar, qcfg, W, codes, scale, zero, Dbar=Dbar, dead=prep.dead,
                             bcfg=bcfg, F=F, F_next=F_next, adam_m=am, adam_v=av, bgd_disp=disp, ws=ws,
                             stream=stream)
    return Quantized(codes, scale, zero, W, t)


def unpack_codes(codes: torch.Tensor, n: int) -> torch.Tensor:
    """m x ceil(n/2) packed bytes -> m x n int codes (even column in the low nibble)."""
    lo = (codes & 15).to(torch.int64)
    hi = (codes >> 4).to(torch.int64)
    out = torch.stack([lo, hi], dim=2).reshape(codes.shape[0], -1)
    return out[:, :n]
