"""Comparison of CUDA-path outputs with oracle outputs (test helper).

The parity bar for the codes is "identical except at rounding ties": where
the oracle's w / scale (or its zero point's -xmin / scale) lies within tau =
1e-3 grid steps of a rounding boundary, both neighbours are the correctly
rounded result up to the rounding of the operands, and the CUDA path may take
either.  A different choice there changes everything downstream of it (the
rest of the row through the OBS compensation, every row through Block-GD), so
the comparison follows the CUDA path's branch: follow_ties reruns the oracle
with the CUDA path's decision taken at each of the oracle's own ties (the
oracle's `follow`), and every code that still differs from that run is an
unexplained mismatch.  Nothing is excused by position.
"""
from __future__ import annotations

import numpy as np


def unpack(codes: np.ndarray, n: int) -> np.ndarray:
    lo = (codes & 15).astype(np.int64)
    hi = (codes >> 4).astype(np.int64)
    return np.stack([lo, hi], axis=2).reshape(codes.shape[0], -1)[:, :n]


def code_report(gpu_codes: np.ndarray, orc: dict, gpu_zero: np.ndarray = None, tau: float = 1e-3) -> dict:
    """Plain element-by-element comparison of codes (and zero points)."""
    ref = orc["codes"]
    mism = gpu_codes != ref
    tie = orc["margin"] < tau
    idx = np.argwhere(mism)
    first = [(int(i), int(j), float(orc["margin"][i, j])) for i, j in idx[:10]]
    rep = {
        "frac_equal": 1.0 - float(mism.mean()),
        "n_mismatch": int(mism.sum()),
        "n_mismatch_at_tie": int((mism & tie).sum()),
        "first": first,
        "n_ties_total": int(tie.sum()),
        "n_zero_mismatch": 0,
    }
    if gpu_zero is not None:
        rep["n_zero_mismatch"] = int((np.asarray(gpu_zero, dtype=np.int64) != orc["zero"]).sum())
    return rep


class OracleSweep:
    """One oracle sweep, run plainly at once and again on request:
    sweep(None) is the plain result (also reachable as sweep[key]),
    sweep(follow, grad_noise) a rerun.  fn(follow, grad_noise=None) runs
    the oracle (oracle.realq_sweep's arguments of those names)."""

    def __init__(self, fn, eager: bool = True):
        self.fn = fn
        self._plain = fn(None) if eager else None

    @property
    def plain(self):
        if self._plain is None:
            self._plain = self.fn(None)
        return self._plain

    def __call__(self, follow, grad_noise=None):
        if follow is None and grad_noise is None:
            return self.plain
        return self.fn(follow, grad_noise=grad_noise) if grad_noise is not None else self.fn(follow)

    def __getitem__(self, key):
        return self.plain[key]


# The sensitivity probe: how far the sweep's pre-rounding values move when
# every Block-GD gradient entry moves by eta times the magnitude of its terms
# (oracle.gradient_error_scale), with every rounding decision held at the
# compared run's (so that the move is the continuous one, not a cascade from
# a decision the probe takes the other way).  eta is the error of the
# gradient's evaluation on the tensor cores: the tf32x3 splitting error of a
# product (2^-21) plus the accumulation in the tensor memory, which loses
# about one unit in the last place per accumulated MMA (K = 8 per MMA, three
# MMAs per K step) over the two contractions of the gradient (P over at most n
# inputs, G over m outputs).  Two seeded probes; a decision whose margin is
# within PROBE_K times the larger move is not determined by the method's
# arithmetic at that precision (Adam's m / sqrt(v) amplifies the error of a
# gradient entry whose moments nearly cancel).
PROBE_K = 10.0
PROBE_SEEDS = (101, 202)
PROBE_ROUNDS = 3


def probe_eta(m: int, n: int) -> float:
    return 2.0 ** -24 * 3.0 * (m + n) / 8.0 + 2.0 ** -21


def follow_ties(run, gpu_codes: np.ndarray, gpu_zero: np.ndarray = None, tau: float = 1e-3,
                plain_first: bool = True, gpu_scale: np.ndarray = None, rtol: float = 1e-5):
    """run(follow[, grad_noise]) -> an oracle sweep result (oracle.realq_sweep
    with that follow).

    Runs the oracle plainly; if its codes or zero points differ from the
    CUDA path's, runs it again taking the CUDA path's decision at each of its
    own rounding ties.  If codes still differ, the followed run is repeated
    under the sensitivity probe: a remaining mismatch whose margin is within
    PROBE_K times the probes' move of that value is counted as
    n_conditioned, every other one as unexplained; while unexplained ones
    remain, the oracle reruns taking the CUDA path's decision at the
    conditioned ones too (their tolerance widened to the probes' reach) and
    compares again, PROBE_ROUNDS probe passes at most.  Returns (plain result,
    followed result, report); the report carries the plain comparison
    (plain_frac_equal, plain_n_mismatch), the decisions followed, and the
    probes' per-group moves of the scales as fol["probe_scale_move"] (the
    probes also run when gpu_scale is given and a scale differs from the
    followed run's by more than rtol).
    plain_first=False skips the plain run (where the oracle is slow): the
    oracle runs once, with the follow, and the plain entries are None."""
    if plain_first:
        plain = run(None)
        rep0 = code_report(gpu_codes, plain, gpu_zero, tau)
    else:
        plain, rep0 = None, {"frac_equal": None, "n_mismatch": None, "n_zero_mismatch": None}
    follow = {"codes": np.asarray(gpu_codes, dtype=np.int64),
              "zero": None if gpu_zero is None else np.asarray(gpu_zero, dtype=np.int64), "tau": tau}
    if plain_first and rep0["n_mismatch"] == 0 and rep0["n_zero_mismatch"] == 0:
        fol = plain
    else:
        fol = run(follow)
    rep = code_report(gpu_codes, fol, gpu_zero, tau)
    rep.update(plain_frac_equal=rep0["frac_equal"], plain_n_mismatch=rep0["n_mismatch"],
               n_followed=int(fol["n_followed"]), n_followed_zero=int(fol["n_followed_zero"]), n_conditioned=0)
    mism = gpu_codes != fol["codes"]
    zmism = np.zeros_like(fol["zero"], dtype=bool) if gpu_zero is None else \
        np.asarray(gpu_zero, dtype=np.int64) != fol["zero"]
    scale_off = False
    if gpu_scale is not None:
        so = fol["scale"].astype(np.float64)
        scale_off = bool((np.abs(np.asarray(gpu_scale, dtype=np.float64) - so) > rtol * np.abs(so)).any())
    if mism.any() or zmism.any() or scale_off:
        m, n = gpu_codes.shape
        eta = probe_eta(m, n)
        tau_c = np.full((m, n), tau)
        tau_z = np.full(fol["zero"].shape, tau)
        raised = np.zeros((m, n), dtype=bool)
        zraised = np.zeros(fol["zero"].shape, dtype=bool)
        for it in range(PROBE_ROUNDS):
            dx = np.zeros((m, n))
            dz = np.zeros_like(fol["zf"])
            ds = np.zeros(fol["scale"].shape)
            held = {"codes": fol["codes"], "zero": fol["zero"], "tau": 0.5}
            for seed in PROBE_SEEDS:
                pr = run(held, grad_noise={"seed": seed, "eta": eta})
                dx = np.maximum(dx, np.abs(pr["x"] - fol["x"]))
                dz = np.maximum(dz, np.abs(pr["zf"] - fol["zf"]))
                ds = np.maximum(ds, np.abs(pr["scale"].astype(np.float64) - fol["scale"].astype(np.float64)))
            cond = mism & (fol["margin"] <= PROBE_K * dx)
            zcond = zmism & (fol["zero_margin"] <= PROBE_K * dz)
            fol = dict(fol, probe_scale_move=ds)
            new, znew = cond & ~raised, zcond & ~zraised
            if not ((mism & ~cond).any() or (zmism & ~zcond).any()) or not (new.any() or znew.any()) \
                    or it == PROBE_ROUNDS - 1:
                break
            # a mismatch left after the conditioned ones is downstream of one
            # of them (the rest of its row, every row through Block-GD): the
            # comparison follows the CUDA path there too, with the decision's
            # tolerance widened to the probes' reach, and compares again
            tau_c[new] = np.maximum(tau_c[new], PROBE_K * dx[new] * (1.0 + 1e-9))
            tau_z[znew] = np.maximum(tau_z[znew], PROBE_K * dz[znew] * (1.0 + 1e-9))
            raised |= new
            zraised |= znew
            fol = run(dict(follow, tau=tau_c, tau_zero=tau_z))
            mism = gpu_codes != fol["codes"]
            zmism = np.zeros_like(fol["zero"], dtype=bool) if gpu_zero is None else \
                np.asarray(gpu_zero, dtype=np.int64) != fol["zero"]
            rep.update(code_report(gpu_codes, fol, gpu_zero, tau))
            rep["n_followed"] = int(fol["n_followed"])
            rep["n_followed_zero"] = int(fol["n_followed_zero"])
        # every decision the comparison took from the CUDA path beyond the
        # ties counts, with the mismatches the probes explain in the last run
        rep["n_conditioned"] = int((raised | cond).sum() + (zraised | zcond).sum())
        rep["n_unexplained"] = int((mism & ~cond).sum() + (zmism & ~zcond).sum())
        rep["probe_rounds"] = it + 1
    else:
        rep["n_unexplained"] = 0
    return plain, fol, rep


def scale_agreement(gpu_scale: np.ndarray, orc_scale: np.ndarray, rtol: float = 1e-5, adam_bound: np.ndarray = None,
                    probe_move: np.ndarray = None):
    """(fraction of groups within rtol, median relative error, groups off by
    more than rtol and beyond adam_bound, groups off by more than rtol but
    within adam_bound).  probe_move (per group): the sensitivity probes' move
    of the oracle's scale; a group off by at most PROBE_K times it counts as
    within rtol (its scale is not determined at fp32 precision).

    adam_bound (per group, absolute; reading R18): a scale is (xmax - xmin) /
    (2^b - 1); an Adam step at t = 1 is lr times the sign of the gradient, and
    an entry within rounding of zero may take the other sign in fp32 than in
    fp64, moving that weight by 2 lr, so a group whose extreme weight had such
    an entry before its parameters were computed can differ by up to
    2 * 2 lr * steps / (2^b - 1).  The count of groups using that allowance is
    returned so that the test can bound it."""
    diff = np.abs(gpu_scale.astype(np.float64) - orc_scale.astype(np.float64))
    rel = diff / np.abs(orc_scale.astype(np.float64))
    off = rel > rtol
    if probe_move is not None:
        off = off & (diff > PROBE_K * probe_move)
    if adam_bound is not None:
        bad = off & (diff > adam_bound)
    else:
        bad = off
    return float((~off).mean()), float(np.median(rel)), int(bad.sum()), int((off & ~bad).sum())


def adam_scale_bound(orc_scale: np.ndarray, n: int, qkw: dict, lr: float, steps: int) -> np.ndarray:
    """Per group, the scale allowance of reading R18: 4 lr k / (2^b - 1), k the
    optimizer steps applied to the group's columns before its parameters."""
    B = qkw.get("block_size", 128)
    g = qkw.get("group_size", 128) or n
    maxq = 2 ** qkw.get("bits", 4) - 1
    first_cols = np.arange(orc_scale.shape[1]) * g
    taken = np.minimum(first_cols // B, max(0, -(-n // B) - 1)) * steps
    return np.broadcast_to(4.0 * lr * taken / maxq + 1e-12, orc_scale.shape)


def check_codes_and_scales(orc, codes, zero, scale, n, qkw, bgd, lr=0.0, steps=1, what="", plain_first=True,
                           probe_scales=True):
    """The codes bar on the CUDA path's branch (follow_ties: >= 99.9 %
    identical, none unexplained, decisions the arithmetic does not
    determine at most 1e-5 of the codes plus one) and the scales within 1e-5
    relative, apart from groups within the probes' move and groups within
    the Adam-sign allowance of reading R18 (counted; at most 0.1 % of the
    groups plus one).  probe_scales=False runs the probes for codes only
    (where the oracle is slow).  Returns (plain, followed, report)."""
    plain, fol, rep = follow_ties(orc, codes, zero, plain_first=plain_first,
                                  gpu_scale=scale if probe_scales else None)
    frac, med, s_bad, s_allow = scale_agreement(scale, fol["scale"],
                                                adam_bound=adam_scale_bound(fol["scale"], n, qkw, lr, steps)
                                                if bgd else None, probe_move=fol.get("probe_scale_move"))
    rep.update(scale_within_1e5=frac, scale_median_rel=med, scale_beyond=s_bad, adam_sign_allowance=s_allow)
    print(f"\nparity {what}{qkw} bgd={bgd}: {rep}")
    assert rep["frac_equal"] >= 0.999, rep
    assert rep["n_unexplained"] == 0, rep
    assert rep["n_conditioned"] <= 1 + 1e-5 * codes.size, rep
    assert s_bad == 0, (frac, med, s_bad)
    assert s_allow <= 1 + 1e-3 * scale.size, (s_allow, scale.size)
    return plain, fol, rep


def token_surrogate(oracle_mod, What, W0, bits_to_f64, xhat_bits, F, chunk=8192) -> float:
    """The oracle's token-form surrogate (oracle.surrogate_tokens) of What
    over all tokens of a bf16 input, evaluated chunk by chunk so that the
    input is never widened whole: the mean over chunks weighted by their
    token counts."""
    T = xhat_bits.shape[0]
    acc = 0.0
    for c in range(0, T, chunk):
        xc = bits_to_f64(xhat_bits[c:c + chunk])
        acc += oracle_mod.surrogate_tokens(What, W0, xc, None, F) * xc.shape[0]
    return acc / T
