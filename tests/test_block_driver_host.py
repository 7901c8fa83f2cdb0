"""Host logic of the block-level driver with the exact losses
(paper_2609_00049_gb300.block.quantize_block_exact), with the library's
device calls replaced by recorders: the modules run in the paper's order,
b_global runs over the column blocks of all of them with B_total their sum,
each module sees the modules quantized before it (the current weights and
the perturbed input), and the final current weights are every module's
dequantized weights.  No GPU is used."""
import pytest
import torch

import paper_2609_00049_gb300 as rq
from paper_2609_00049_gb300 import block as pb
from paper_2609_00049_gb300 import layer

KEYS = ("g1", "Wq", "Wk", "Wv", "Wo", "g2", "Wg", "Wu", "Wd")


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_00049_gb300 import build as b
    b.build()
    rq.lib()


def _weights(d, H, Hkv, dh, f):
    shapes = {"g1": (d,), "Wq": (H * dh, d), "Wk": (Hkv * dh, d), "Wv": (Hkv * dh, d), "Wo": (d, H * dh),
              "g2": (d,), "Wg": (f, d), "Wu": (f, d), "Wd": (d, f)}
    return {k: torch.zeros(shapes[k]) for k in KEYS}


@pytest.mark.parametrize("kl,nmb", [(False, 1), (True, 1), (False, 2)])
def test_driver_order_global_block_index_and_current_weights(monkeypatch, kl, nmb):
    d, H, Hkv, dh, f, S, L = 128, 4, 2, 32, 320, 2, 8
    dims = rq.block_dims(d, H, Hkv, dh, f)
    W_this, W_next = _weights(d, H, Hkv, dh, f), _weights(d, H, Hkv, dh, f)
    x, x_hat = torch.zeros(S, L, d), torch.ones(S, L, d)
    calls = []

    def module_inputs(dims_, weights, xin, module, X_out, ws, stream=None):
        calls.append(("inputs", module, dict(weights), xin))

    def accumulate(chunks, n, x_fp_chunks=None, device="cuda", stream=None):
        (X,) = list(chunks)
        assert X.shape == (S * L, n)                                   # the Hessian takes every mini-batch
        return torch.zeros(n, n), None, X.shape[0]

    def prepare(H_, T, damp_frac=0.01, D_sum=None, stream=None):
        n = H_.shape[0]
        return layer.Prepared(torch.zeros(n, n), torch.zeros(n, n), torch.zeros(n, dtype=torch.uint8), T)

    def sweep(dims_, this_block, next_block, xin, module, U, qcfg, bcfg, W, codes, scale, zero, **kw):
        calls.append(("sweep", module, bcfg.b_global_start, bcfg.B_total, dict(kw["this_block_hat"]), kw["x_hat"],
                      next_block is None, kw["head_Wh"] is not None))
        assert kw["n_minibatch"] == nmb
        assert this_block is W_this and xin is x
        W.fill_(float(len(calls)))
        return 7

    monkeypatch.setattr(pb, "realq_block_module_inputs", module_inputs)
    monkeypatch.setattr(pb.layer, "accumulate", accumulate)
    monkeypatch.setattr(pb.layer, "prepare", prepare)
    monkeypatch.setattr(pb, "realq_quantize_layer_window", sweep)
    monkeypatch.setattr(pb, "realq_workspace_status", lambda ws, stream=None: 0)
    monkeypatch.setattr(pb, "workspace", lambda nbytes, device=None: torch.zeros(8, dtype=torch.uint8))
    q = rq.quant_cfg(group_size=64, block_size=64)
    if kl:
        out, W_hat = pb.quantize_block_exact(dims, W_this, x, q, 1e-3, x_hat=x_hat, head_gf=torch.zeros(d),
                                             head_Wh=torch.zeros(50, d), n_minibatch=nmb)
    else:
        out, W_hat = pb.quantize_block_exact(dims, W_this, x, q, 1e-3, x_hat=x_hat, W_next=W_next,
                                             F_this=torch.zeros(d, d), F_next=torch.zeros(d, d), n_minibatch=nmb)
    sweeps = [c for c in calls if c[0] == "sweep"]
    inputs = [c for c in calls if c[0] == "inputs"]
    order = ["q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj"]
    assert [c[1] for c in sweeps] == order and [c[1] for c in inputs] == order
    # column blocks: six modules of 128 inputs (2 blocks each), o_proj 128, down 320 (5 blocks)
    nb = [2, 2, 2, 2, 2, 2, 5]
    starts = [1 + sum(nb[:i]) for i in range(7)]
    assert [c[2] for c in sweeps] == starts
    assert all(c[3] == sum(nb) for c in sweeps)
    key = {"q_proj": "Wq", "k_proj": "Wk", "v_proj": "Wv", "o_proj": "Wo", "gate_proj": "Wg", "up_proj": "Wu",
           "down_proj": "Wd"}
    for i, (inp, sw) in enumerate(zip(inputs, sweeps)):
        assert inp[3] is x_hat and sw[5] is x_hat                  # the current pass runs on x̂
        for j, prev in enumerate(order):
            # modules before this one are their dequantized weights; the rest the reference
            want = out[prev].W if j < i else W_this[key[prev]]
            assert inp[2][key[prev]] is want and sw[4][key[prev]] is want
        assert sw[6] == kl and sw[7] == kl                          # the next block or the LM head
    for md in order:
        assert W_hat[key[md]] is out[md].W and out[md].adam_t == 7
        assert out[md].block_loss.shape == (nb[order.index(md)], 2)


def test_model_loop_schedule_windows_and_inputs(monkeypatch):
    # Alg. 1's outer loop: the reverse-cosine rate per block, the window to
    # the next block (the KL head for the last), and each block's inputs are
    # the previous block's outputs (full precision and quantized)
    import oracle
    d, H, Hkv, dh, f, S, L = 64, 4, 2, 16, 96, 2, 8
    dims = rq.block_dims(d, H, Hkv, dh, f)
    blocks = [_weights(d, H, Hkv, dh, f) for _ in range(4)]
    fishers = [torch.zeros(d, d) for _ in range(4)]
    gf, Wh = torch.zeros(d), torch.zeros(30, d)
    x = torch.zeros(S, L, d)
    calls, fwd = [], []

    def block_exact(dims_, W, x_ref, qcfg, lr, x_hat=None, W_next=None, F_this=None, F_next=None, head_gf=None,
                    head_Wh=None, **kw):
        calls.append((W, x_ref, x_hat, lr, W_next, F_this, F_next, head_gf, head_Wh))
        return {}, {"hat": len(calls)}

    def forward(dims_, weights, xin, y, ws, stream=None):
        fwd.append((weights, xin, y))

    monkeypatch.setattr(pb, "quantize_block_exact", block_exact)
    monkeypatch.setattr(pb, "realq_block_forward", forward)
    monkeypatch.setattr(pb, "workspace", lambda nbytes, device=None: torch.zeros(8, dtype=torch.uint8))
    out = pb.quantize_model_exact(dims, blocks, x, fishers, gf, Wh, rq.quant_cfg(), 1e-3)
    assert len(out) == 4 and [o[1]["hat"] for o in out] == [1, 2, 3, 4]
    for l, c in enumerate(calls):
        W, x_ref, x_hat, lr, W_next, F_this, F_next, hgf, hWh = c
        assert W is blocks[l]
        assert lr == pytest.approx(oracle.reverse_cosine_lr(l + 1, 4, 1e-3), rel=1e-15)
        if l < 3:
            assert W_next is blocks[l + 1] and F_this is fishers[l] and F_next is fishers[l + 1] and hWh is None
        else:
            assert W_next is None and hgf is gf and hWh is Wh
        if l == 0:
            assert x_ref is x and x_hat is x
        else:
            # block l-1's two forward passes: reference weights on the
            # reference input, quantized weights on the quantized input
            (w_ref, in_ref, y_ref), (w_hat, in_hat, y_hat) = fwd[2 * (l - 1)], fwd[2 * (l - 1) + 1]
            assert w_ref is blocks[l - 1] and w_hat == {"hat": l}
            assert in_ref is calls[l - 1][1] and in_hat is calls[l - 1][2]
            assert x_ref is y_ref and x_hat is y_hat
