"""Seeded synthetic inputs for the per-layer quantization sweep.

This module is the only code shared by the CUDA path's callers (tests, bench)
and the fp64 oracle.  It draws inputs and nothing else: it holds none of the
method's arithmetic (no Hessian, no quantizer, no inverse, no gradient).

Every tensor is a pure function of (workload seed, tensor name, chunk index),
drawn from numpy's SFC64 bit generator keyed through ``SeedSequence``, so any
chunk of any tensor can be regenerated independently and in parallel.

Workloads mirror the layer shapes of the paper's evaluated models (Sec. 5.1,
"Setup"; LLaMA-3.1 and Qwen3 families) with synthetic values standing in for
the real weights and for the WikiText-2 calibration activations, which are not
available here.  The distributions (Gaussian with scaled outlier channels,
unit-variance Student-t) follow the workload descriptions of the build's
configurations.
"""
from __future__ import annotations

import zlib
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field
from typing import Dict, List, Optional

import numpy as np

CHUNK_TOKENS = 8192


# --------------------------------------------------------------------------
# bf16 bit helpers (storage format only; round-to-nearest-even on the cast)
# --------------------------------------------------------------------------
def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (nearest-even) and return the raw uint16 bits."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    rounding = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + rounding) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp32."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _key(name: str) -> int:
    return zlib.crc32(name.encode("utf-8")) & 0xFFFFFFFF


def rng(seed: int, *names) -> np.random.Generator:
    """Independent generator for (seed, names...)."""
    keys = [int(seed)] + [(_key(n) if isinstance(n, str) else int(n)) for n in names]
    return np.random.Generator(np.random.SFC64(np.random.SeedSequence(keys)))


# --------------------------------------------------------------------------
# workload descriptions
# --------------------------------------------------------------------------
@dataclass
class InputSpec:
    """Calibration activations X̂ (T tokens x n channels, token-major)."""
    name: str
    n: int
    T: int
    dist: str = "gauss"            # "gauss" | "student_t"
    nu: float = 4.0                # Student-t degrees of freedom
    outlier_frac: float = 0.0      # fraction of channels scaled by outlier_scale
    outlier_count: int = 0         # or an absolute count of outlier channels
    outlier_scale: float = 1.0
    dtype: str = "bf16"            # "bf16" | "f32"


@dataclass
class ModuleSpec:
    """One linear module W (m out x n in) fed by input `input`."""
    name: str
    m: int
    n: int
    input: str
    w_std: float = 0.02
    w_dtype: str = "bf16"


@dataclass
class Workload:
    name: str
    inputs: Dict[str, InputSpec]
    modules: List[ModuleSpec]
    seed: int = 0
    bits: int = 4
    group_size: int = 128
    block_size: int = 128
    symmetric: int = 0
    damp_frac: float = 0.01
    lr: float = 1e-4
    steps_per_block: int = 1
    fisher_rows: str = "uniform"   # per-row surrogate weights: "uniform" U(0.5,2) | "lognormal" LN(0,1)
    fisher_rank: int = 16          # rank of the cross-channel coupling term
    sliding_window: bool = False   # blend F of this block with F of the next block
    description: str = ""

    def input_of(self, mod: ModuleSpec) -> InputSpec:
        return self.inputs[mod.input]

    @property
    def total_columns(self) -> int:
        return sum(md.n for md in self.modules)

    @property
    def total_column_blocks(self) -> int:
        return sum(-(-md.n // self.block_size) for md in self.modules)


def _block(name, hidden, q_out, kv_out, inter, T, x_kwargs, w_std, lr, seed=0, **kw) -> Workload:
    inputs = {
        "attn_in": InputSpec("attn_in", hidden, T, **x_kwargs),
        "o_in": InputSpec("o_in", q_out, T, **x_kwargs),
        "mlp_in": InputSpec("mlp_in", hidden, T, **x_kwargs),
        "down_in": InputSpec("down_in", inter, T, **x_kwargs),
    }
    mods = [
        ModuleSpec("q_proj", q_out, hidden, "attn_in", w_std),
        ModuleSpec("k_proj", kv_out, hidden, "attn_in", w_std),
        ModuleSpec("v_proj", kv_out, hidden, "attn_in", w_std),
        ModuleSpec("o_proj", hidden, q_out, "o_in", w_std),
        ModuleSpec("gate_proj", inter, hidden, "mlp_in", w_std),
        ModuleSpec("up_proj", inter, hidden, "mlp_in", w_std),
        ModuleSpec("down_proj", hidden, inter, "down_in", w_std),
    ]
    return Workload(name, inputs, mods, seed=seed, lr=lr, **kw)


def workloads() -> Dict[str, Workload]:
    """The five layer workloads: one small fp32 layer, four decoder-block shapes.

    Learning rates follow the paper's per-model table of REAL-Q learning rates
    (App. "REAL-Q Learning Rates", W4A16 rows), used as a constant for the block.
    """
    w = {}
    w["fc256x512"] = Workload(
        "fc256x512",
        {"x": InputSpec("x", 512, 2048, "gauss", outlier_count=4, outlier_scale=10.0, dtype="f32")},
        [ModuleSpec("fc", 256, 512, "x", 0.02, "f32")],
        lr=1e-4, description="single fp32 linear layer 512->256, 2048 tokens, 4 outlier channels x10")
    w["qwen3-0.6b"] = _block(
        "qwen3-0.6b", 1024, 2048, 1024, 3072, 128 * 2048,
        dict(dist="gauss", outlier_frac=0.01, outlier_scale=20.0), 0.02, 3e-4,
        description="Qwen3-0.6B-shaped decoder block, 128x2048 tokens, 1% outlier channels x20")
    w["llama3.1-8b"] = _block(
        "llama3.1-8b", 4096, 4096, 1024, 14336, 128 * 2048,
        dict(dist="student_t", nu=4.0), 0.02, 1e-5, sliding_window=True,
        description="LLaMA-3.1-8B-shaped decoder block, Student-t(4) activations, sliding window")
    w["qwen3-32b"] = _block(
        "qwen3-32b", 5120, 8192, 1024, 25600, 128 * 2048,
        dict(dist="gauss", outlier_frac=0.005, outlier_scale=50.0), 0.02, 2e-6,
        description="Qwen3-32B-shaped decoder block, 0.5% outlier channels x50")
    w["llama3.1-70b"] = _block(
        "llama3.1-70b", 8192, 8192, 1024, 28672, 256 * 2048,
        dict(dist="student_t", nu=3.0), 0.015, 3e-6, fisher_rows="lognormal",
        description="LLaMA-3.1-70B-shaped decoder block, Student-t(3) activations, log-normal row weights")
    return w


# --------------------------------------------------------------------------
# tensor generators
# --------------------------------------------------------------------------
def outlier_channels(wl: Workload, spec: InputSpec) -> np.ndarray:
    cnt = spec.outlier_count or int(round(spec.outlier_frac * spec.n))
    if cnt <= 0:
        return np.zeros(0, dtype=np.int64)
    r = rng(wl.seed, "outliers", spec.name)
    return np.sort(r.choice(spec.n, size=cnt, replace=False))


def _draw_x(wl: Workload, spec: InputSpec, chunk: int, rows: int, salt: str = "") -> np.ndarray:
    r = rng(wl.seed, "xhat" + salt, spec.name, chunk)
    if spec.dist == "gauss":
        x = r.standard_normal((rows, spec.n), dtype=np.float32)
    elif spec.dist == "student_t":
        x = r.standard_t(spec.nu, size=(rows, spec.n)).astype(np.float32)
        x *= np.float32(1.0 / np.sqrt(spec.nu / (spec.nu - 2.0)))
    else:
        raise ValueError(spec.dist)
    oc = outlier_channels(wl, spec)
    if oc.size:
        x[:, oc] *= np.float32(spec.outlier_scale)
    return x


def xhat_chunk(wl: Workload, input_name: str, chunk: int, chunk_tokens: int = CHUNK_TOKENS,
               as_bits: bool = True) -> np.ndarray:
    """Tokens [chunk*chunk_tokens, ...) of input `input_name`.

    Returns uint16 bf16 bits for bf16 inputs (as_bits=True), else fp32 values
    (bf16-rounded when the input dtype is bf16).
    """
    spec = wl.inputs[input_name]
    t0 = chunk * chunk_tokens
    rows = min(chunk_tokens, spec.T - t0)
    if rows <= 0:
        raise IndexError("chunk out of range")
    x = _draw_x(wl, spec, chunk, rows) if chunk_tokens == CHUNK_TOKENS else None
    if x is None:
        # arbitrary chunking: assemble from canonical chunks
        parts, t = [], t0
        while t < t0 + rows:
            c, off = divmod(t, CHUNK_TOKENS)
            base = _draw_x(wl, spec, c, min(CHUNK_TOKENS, spec.T - c * CHUNK_TOKENS))
            take = min(base.shape[0] - off, t0 + rows - t)
            parts.append(base[off:off + take])
            t += take
        x = np.concatenate(parts, axis=0)
    if spec.dtype == "bf16":
        b = f32_to_bf16_bits(x)
        return b if as_bits else bf16_bits_to_f32(b)
    return x


def xhat_full(wl: Workload, input_name: str, as_bits: bool = True, max_tokens: Optional[int] = None,
              threads: int = 8, out: Optional[np.ndarray] = None) -> np.ndarray:
    """All (or the first max_tokens) calibration tokens of an input, generated in
    parallel, into `out` if given (T x n, uint16 for bf16 bits, else fp32;
    e.g. a view of page-locked memory)."""
    spec = wl.inputs[input_name]
    T = spec.T if max_tokens is None else min(spec.T, max_tokens)
    nch = -(-T // CHUNK_TOKENS)
    dt = np.uint16 if (spec.dtype == "bf16" and as_bits) else np.float32
    if out is None:
        out = np.empty((T, spec.n), dtype=dt)
    elif out.shape != (T, spec.n) or out.dtype.itemsize != np.dtype(dt).itemsize:
        raise ValueError(f"out must be {T} x {spec.n} of {np.dtype(dt).itemsize}-byte elements")
    else:
        out = out.view(dt)

    def work(c):
        a = xhat_chunk(wl, input_name, c, CHUNK_TOKENS, as_bits)
        t0 = c * CHUNK_TOKENS
        k = min(a.shape[0], T - t0)
        out[t0:t0 + k] = a[:k]

    with ThreadPoolExecutor(threads) as ex:
        list(ex.map(work, range(nch)))
    return out


def weights(wl: Workload, mod: ModuleSpec, as_bits: bool = True) -> np.ndarray:
    """W0 (m x n, row-major); bf16 bits or fp32 values."""
    r = rng(wl.seed, "weight", mod.name)
    w = (r.standard_normal((mod.m, mod.n), dtype=np.float32) * np.float32(mod.w_std))
    if mod.w_dtype == "bf16":
        b = f32_to_bf16_bits(w)
        return b if as_bits else bf16_bits_to_f32(b)
    return w


def fisher(wl: Workload, mod: ModuleSpec, which: str = "F") -> np.ndarray:
    """Synthetic aggregated Fisher on the module-output space (m x m, fp32, SPD).

    F = D^1/2 (I/2 + Z Z^T / (2k)) D^1/2 with per-row weights D (Uniform(0.5, 2)
    or log-normal(0, 1)) and a rank-k Gaussian coupling Z, so that F is full
    (cross-channel coupled) with diag(F) close to the per-row weights.
    `which` = "F" for this block's Fisher, "F_next" for the next block's.
    """
    r = rng(wl.seed, "fisher", which, mod.name)
    m = mod.m
    if wl.fisher_rows == "lognormal":
        d = r.lognormal(0.0, 1.0, size=m)
    else:
        d = r.uniform(0.5, 2.0, size=m)
    k = wl.fisher_rank
    z = r.standard_normal((m, k)) * np.sqrt(d)[:, None]
    F = (z @ z.T) / (2.0 * k)
    F[np.diag_indices(m)] += 0.5 * d
    return F.astype(np.float32)


def fisher_diag(wl: Workload, mod: ModuleSpec) -> np.ndarray:
    """Diagonal variant: F = diag(per-row weights)."""
    r = rng(wl.seed, "fisher", "F", mod.name)
    d = r.lognormal(0.0, 1.0, size=mod.m) if wl.fisher_rows == "lognormal" else r.uniform(0.5, 2.0, size=mod.m)
    return np.diag(d).astype(np.float32)


def saliency(wl: Workload, mod: ModuleSpec, n_groups: int = 4) -> np.ndarray:
    """Synthetic per-token saliency of a module's row groups (T x n_groups fp32).

    Stands in for the squared output-gradient norms of Stage 0: log-normal(0, 1)
    per token and group, with 0.1 % of the tokens 10^6 x larger (the gradient
    outliers the paper clips at the 99th percentile)."""
    T = wl.inputs[mod.input].T
    r = rng(wl.seed, "saliency", mod.name)
    s = r.lognormal(0.0, 1.0, size=(T, n_groups))
    hot = r.random(T) < 1e-3
    s[hot] *= 1e6
    return s.astype(np.float32)


# --------------------------------------------------------------------------
# small free-form cases for tests
# --------------------------------------------------------------------------
@dataclass
class LayerCase:
    W0: np.ndarray          # m x n fp32 values
    Xhat: np.ndarray        # T x n fp32 values
    X: Optional[np.ndarray]  # T x n fp32 values of the unperturbed input, or None (X = X̂)
    F: np.ndarray           # m x m fp32
    F_next: Optional[np.ndarray] = None
    extra: dict = field(default_factory=dict)


def layer_case(seed: int, m: int, n: int, T: int, *, outliers: int = 0, outlier_scale: float = 10.0,
               w_std: float = 0.02, perturbed: bool = False, perturb_std: float = 0.05,
               dead_cols=(), fisher_kind: str = "full", with_next: bool = False,
               integer_x: bool = False, bf16: bool = False) -> LayerCase:
    """A small seeded layer for parity tests.

    integer_x draws X̂ from {-2,...,2} so that X̂^T X̂ is exact in fp32 and fp64.
    dead_cols are input channels that are identically zero.  perturbed adds an
    unperturbed X with X̂ = X + noise.  bf16 rounds W0 and X̂ to bf16 values.
    """
    r = rng(seed, "case", m, n, T)
    W0 = r.standard_normal((m, n), dtype=np.float32) * np.float32(w_std)
    if integer_x:
        Xh = r.integers(-2, 3, size=(T, n)).astype(np.float32)
    else:
        Xh = r.standard_normal((T, n), dtype=np.float32)
    if outliers:
        oc = r.choice(n, size=outliers, replace=False)
        Xh[:, oc] *= np.float32(outlier_scale)
    X = None
    if perturbed:
        X = Xh.copy()
        Xh = X + r.standard_normal((T, n), dtype=np.float32) * np.float32(perturb_std) * X.std(axis=0, keepdims=True)
    for c in dead_cols:
        Xh[:, c] = 0.0
        if X is not None:
            X[:, c] = 0.0
    if bf16:
        W0 = bf16_bits_to_f32(f32_to_bf16_bits(W0))
        Xh = bf16_bits_to_f32(f32_to_bf16_bits(Xh))
        if X is not None:
            X = bf16_bits_to_f32(f32_to_bf16_bits(X))

    def mk_f(tag):
        rf = rng(seed, "caseF", tag, m)
        d = rf.uniform(0.5, 2.0, size=m)
        if fisher_kind == "diag":
            return np.diag(d).astype(np.float32)
        if fisher_kind == "identity":
            return np.eye(m, dtype=np.float32)
        k = min(16, m)
        z = rf.standard_normal((m, k)) * np.sqrt(d)[:, None]
        F = (z @ z.T) / (2.0 * k)
        F[np.diag_indices(m)] += 0.5 * d
        return F.astype(np.float32)

    return LayerCase(W0=W0, Xhat=Xh, X=X, F=mk_f("F"), F_next=mk_f("F_next") if with_next else None)
