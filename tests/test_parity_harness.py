"""The comparison that the GPU parity tests apply (tests/parity.py), checked on
the CPU with the oracle standing in for the CUDA path.

A stand-in run is the oracle's sweep with its Block-GD gradient perturbed by
twice the evaluation error that the comparison's sensitivity probe models
(a seed the probe does not use).  Its codes differ from the plain oracle's
at a handful of decisions and, through the compensation, at later columns of
the same rows.  The comparison must explain every difference (following the
ties and the decisions the probes reach, then the rows downstream of them),
and must still flag a code planted one level off at a decision that is not
close to a rounding boundary."""
import numpy as np

import oracle
import parity
import synth
from parity import OracleSweep, follow_ties, probe_eta


def _case():
    m, n = 64, 384
    c = synth.layer_case(23, m, n, 800, outliers=2, perturbed=True)
    H, T = oracle.hessian_sum([c.Xhat])
    D = oracle.cross_moment_sum([c.Xhat], [c.X])
    kw = dict(group_size=64, block_size=64, bgd={"lr": 3e-3}, F=c.F, D_sum=D)
    run = OracleSweep(lambda follow, grad_noise=None: oracle.realq_sweep(c.W0, H, T, follow=follow,
                                                                         grad_noise=grad_noise, **kw))
    stand_in = oracle.realq_sweep(c.W0, H, T, grad_noise={"seed": 7, "eta": 2 * probe_eta(m, n)}, **kw)
    return run, stand_in


def test_a_perturbed_run_is_explained_and_a_planted_code_is_not(monkeypatch):
    run, emu = _case()
    _, _, rep = follow_ties(run, emu["codes"], emu["zero"])
    print(f"\nstand-in: {rep}")
    assert rep["plain_n_mismatch"] > 0 and rep["n_conditioned"] > 0
    assert rep["n_mismatch"] == 0 and rep["n_unexplained"] == 0 and rep["probe_rounds"] >= 2
    # one probe pass without the follow-up leaves the conditioned decisions'
    # downstream columns unexplained
    monkeypatch.setattr(parity, "PROBE_ROUNDS", 1)
    _, _, rep1 = follow_ties(run, emu["codes"], emu["zero"])
    assert rep1["n_unexplained"] > 0
    monkeypatch.undo()
    # a code one level off where the oracle's value is far from a boundary
    bad = emu["codes"].copy()
    i, j = np.argwhere(run.plain["margin"][:, :64] > 0.3)[5]
    bad[i, j] += 1 if bad[i, j] < 15 else -1
    _, _, repb = follow_ties(run, bad, emu["zero"])
    assert repb["n_unexplained"] >= 1, repb
