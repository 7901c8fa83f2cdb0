"""The allocation-free prepare entry point, for callers that cannot allocate
device memory (a plugin inside a host application that owns all device
memory, or a service that reserves everything up front).  Its results must
match the workspace entry point's on the same input, call after call.

Kept in a file of its own that pytest collects last."""
import numpy as np
import pytest
import torch

import synth
import paper_2609_00049_gb300 as rq

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_00049_gb300 import build as b
    b.build()
    rq.lib()


def _hessian(seed, n, T, dead=()):
    case = synth.layer_case(seed, 4, n, T, outliers=3, dead_cols=dead)
    x = case.Xhat.astype(np.float64)
    return torch.from_numpy((x.T @ x).astype(np.float32)).cuda(), T


def _with_workspace(H, T):
    n = H.shape[0]
    U, Hbar = torch.empty_like(H), torch.empty_like(H)
    dead = torch.empty(n, dtype=torch.uint8, device="cuda")
    ws = rq.workspace(rq.realq_prepare_workspace_size(n))
    rq.realq_hessian_prepare(H, T, 0.01, U, Hbar, dead, ws)
    return U, Hbar, dead


def _no_alloc(H, T):
    n = H.shape[0]
    U, Hbar = torch.empty_like(H), torch.empty_like(H)
    dead = torch.empty(n, dtype=torch.uint8, device="cuda")
    assert rq.realq_hessian_prepare_noalloc(H, T, 0.01, U, Hbar, dead) == -1
    return U, Hbar, dead


def test_no_alloc_prepare_matches_workspace_entry_point_on_consecutive_calls():
    # two calls in a row on different inputs (the second sees the first's leftovers)
    for seed, n, T, dead in ((40, 300, 1500, (5, 77)), (41, 1024, 4096, ())):
        H, T = _hessian(seed, n, T, dead)
        U0, Hbar0, dead0 = _with_workspace(H, T)
        U1, Hbar1, dead1 = _no_alloc(H, T)
        torch.cuda.synchronize()
        # the U tolerance used by the parity tests (fp32 blocked factorisation)
        assert (U1 - U0).abs().max().item() <= 2e-4 * U0.abs().max().item()
        assert torch.equal(Hbar1, Hbar0)
        assert torch.equal(dead1, dead0)


def test_no_alloc_prepare_rejects_too_large_and_reports_not_spd():
    n = rq.PREPARE_NOALLOC_MAX_N + 8
    big = torch.empty(1, device="cuda")
    fc = rq.ctypes.c_int64(0)
    st = rq.lib().realq_hessian_prepare_noalloc(None, n, 10, 0.01, rq.ctypes.c_void_p(big.data_ptr()),
                                                rq.ctypes.c_void_p(big.data_ptr() + 256),
                                                None, rq.ctypes.c_void_p(big.data_ptr() + 512), rq.ctypes.byref(fc))
    assert st == rq.REALQ_ERR_INVALID_ARG
    assert "maximum" in rq.realq_last_error()
    H = -10.0 * torch.eye(64, device="cuda")
    with pytest.raises(rq.RealqError) as ei:
        _no_alloc(H, 10)
    assert ei.value.status == rq.REALQ_ERR_NOT_SPD and ei.value.fail_col == 63
