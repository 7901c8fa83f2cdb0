"""Host-side checks of the C ABI: the library builds, loads, exports every
declared entry point, and rejects bad arguments before touching the GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    from paper_2609_00049_gb300 import build as b
    b.build()
    import paper_2609_00049_gb300 as rq
    return rq.lib()


def _declared():
    src = open(os.path.join(ROOT, "include", "realq.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(realq_\w+)\s*\(", src)))


def test_exports_every_declared_symbol(L):
    names = _declared()
    assert len(names) >= 15
    for n in names:
        assert hasattr(L, n), n


def test_every_symbol_resolves_at_load(L):
    # immediate binding: a symbol the library uses but does not define (e.g.
    # a helper declared in one namespace and defined in another) fails here
    # instead of at its first call on a GPU
    from paper_2609_00049_gb300 import library_path
    ctypes.CDLL(library_path, mode=os.RTLD_NOW)


def test_status_strings(L):
    import paper_2609_00049_gb300 as rq
    for s in range(8):
        assert rq.realq_status_string(s)
    assert rq.realq_status_string(3) == "damped Hessian not positive definite"


def test_workspace_sizes(L):
    import paper_2609_00049_gb300 as rq
    q = rq.quant_cfg()
    b = rq.bgd_cfg(1e-4)
    w0 = rq.realq_quantize_workspace_size(256, 512, q, None)
    w1 = rq.realq_quantize_workspace_size(256, 512, q, b)
    w2 = rq.realq_quantize_workspace_size(256, 512, q, b, has_F_next=True, has_Dbar=True)
    assert 0 < w0 < w1 < w2
    assert w1 >= 2 * 256 * 512 * 4
    assert rq.realq_prepare_workspace_size(1000) >= 1000 * 64 * 4
    assert rq.realq_quantize_workspace_size(0, 512, q, None) == 0
    # a small Hessian on many tokens splits the token range; a large one does not
    assert rq.realq_hessian_workspace_size(128, 65536) > 0
    assert rq.realq_hessian_workspace_size(8192, 8192) == 256


FAKE = ctypes.c_void_p(0x10000)   # never dereferenced: every call below fails validation first


def _ql(L, m=256, n=512, qcfg=None, bcfg=None, F=FAKE, W0=FAKE, ws=FAKE, ws_bytes=1 << 30, blocks=(0, 4)):
    import paper_2609_00049_gb300 as rq
    q = qcfg or rq.quant_cfg()
    t = ctypes.c_int64(0)
    return L.realq_quantize_layer(None, m, n, W0, 0, FAKE, FAKE, None, None, ctypes.byref(q),
                                  ctypes.byref(bcfg) if bcfg is not None else None, F, None, FAKE, FAKE, FAKE,
                                  FAKE, ctypes.byref(t), FAKE, FAKE, FAKE, None, 0, blocks[0], blocks[1], ws,
                                  ws_bytes)


def test_argument_validation(L):
    import paper_2609_00049_gb300 as rq
    assert _ql(L, m=0) == rq.REALQ_ERR_INVALID_ARG
    assert "m, n" in rq.realq_last_error()
    assert _ql(L, W0=None) == rq.REALQ_ERR_INVALID_ARG
    assert _ql(L, qcfg=rq.quant_cfg(bits=5)) == rq.REALQ_ERR_INVALID_ARG
    assert _ql(L, qcfg=rq.quant_cfg(block_size=96)) == rq.REALQ_ERR_INVALID_ARG
    assert _ql(L, qcfg=rq.quant_cfg(group_size=16)) == rq.REALQ_ERR_UNSUPPORTED
    assert _ql(L, qcfg=rq.quant_cfg(group_size=192)) == rq.REALQ_ERR_INVALID_ARG
    assert _ql(L, bcfg=rq.bgd_cfg(1e-4), F=None) == rq.REALQ_ERR_INVALID_ARG
    assert _ql(L, bcfg=rq.bgd_cfg(1e-4, beta1=1.0)) == rq.REALQ_ERR_INVALID_ARG
    assert _ql(L, bcfg=rq.bgd_cfg(float("nan"))) == rq.REALQ_ERR_INVALID_ARG
    assert _ql(L, blocks=(0, 5)) == rq.REALQ_ERR_INVALID_ARG
    assert _ql(L, blocks=(3, 2)) == rq.REALQ_ERR_INVALID_ARG
    assert _ql(L, ws=None) == rq.REALQ_ERR_WORKSPACE
    assert _ql(L, ws=ctypes.c_void_p(0x10010)) == rq.REALQ_ERR_WORKSPACE
    assert _ql(L, ws_bytes=100) == rq.REALQ_ERR_WORKSPACE
    fc = ctypes.c_int64(7)
    assert L.realq_hessian_prepare(None, 0, 10, 0.01, FAKE, FAKE, FAKE, FAKE, ctypes.byref(fc), FAKE, 1 << 20) == 1
    assert L.realq_hessian_prepare(None, 64, 10, 0.01, FAKE, ctypes.c_void_p(0x20000), FAKE, FAKE, ctypes.byref(fc),
                                   None, 0) == 2
    assert L.realq_hessian_prepare(None, 64, 10, 0.01, FAKE, FAKE, FAKE, FAKE, ctypes.byref(fc), FAKE, 1 << 20) == 1
    assert L.realq_hessian_prepare(None, 64, 10, -1.0, FAKE, ctypes.c_void_p(0x20000), FAKE, FAKE,
                                   ctypes.byref(fc), FAKE, 1 << 20) == 1
    assert L.realq_hessian_accumulate(None, 64, 100, FAKE, FAKE, 1, FAKE, None, None, 0) == 1
    assert L.realq_hessian_accumulate(None, 64, 100, FAKE, None, 9, FAKE, None, None, 0) == 1
    assert L.realq_hessian_accumulate(None, 64, 0, None, None, 1, FAKE, None, None, 0) == 0  # empty chunk
    assert L.realq_bgd_refine(None, 4, 4, 5, FAKE, FAKE, 0, FAKE, None, FAKE, None, 1.0, FAKE, FAKE,
                              ctypes.byref(ctypes.c_int64(0)), ctypes.byref(rq.bgd_cfg(1e-3)), FAKE, 1 << 20) == 1
    assert L.realq_bgd_refine(None, 4, 4, 0, FAKE, FAKE, 0, FAKE, None, FAKE, None, 1.5, FAKE, FAKE,
                              ctypes.byref(ctypes.c_int64(0)), ctypes.byref(rq.bgd_cfg(1e-3)), FAKE, 1 << 20) == 1


def test_binding_fails_loudly_without_library(tmp_path, monkeypatch):
    import paper_2609_00049_gb300 as rq
    monkeypatch.setattr(rq, "_lib", None)
    monkeypatch.setattr(rq, "library_path", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        rq.lib()


def _qt(L, T=8000, T_mb=2048, clip=0.95, X=FAKE, n=512):
    import paper_2609_00049_gb300 as rq
    q = rq.quant_cfg()
    b = rq.bgd_cfg(1e-4)
    t = ctypes.c_int64(0)
    return L.realq_quantize_layer_tokens(None, 256, n, FAKE, 0, FAKE, FAKE, None, X, T, T_mb, clip, ctypes.byref(q),
                                         ctypes.byref(b), FAKE, None, FAKE, FAKE, FAKE, FAKE, ctypes.byref(t), FAKE,
                                         FAKE, FAKE, None, 0, 0, 4, FAKE, 1 << 40)


def test_token_path_argument_validation(L):
    import paper_2609_00049_gb300 as rq
    assert _qt(L, T_mb=2046) == rq.REALQ_ERR_INVALID_ARG                 # not a multiple of 4
    assert _qt(L, T_mb=65535 * 32 + 4) == rq.REALQ_ERR_INVALID_ARG       # beyond the layout kernels' grid
    assert _qt(L, T=0) == rq.REALQ_ERR_INVALID_ARG
    assert _qt(L, clip=0.0) == rq.REALQ_ERR_INVALID_ARG
    assert _qt(L, clip=1.5) == rq.REALQ_ERR_INVALID_ARG
    assert _qt(L, clip=float("nan")) == rq.REALQ_ERR_INVALID_ARG
    assert _qt(L, X=ctypes.c_void_p(0x10008)) == rq.REALQ_ERR_INVALID_ARG  # not 16-byte aligned
    assert rq.realq_last_error().endswith("16-byte aligned with n % 8 == 0")
    assert _qt(L, X=None) == rq.REALQ_ERR_INVALID_ARG
    assert rq.realq_quantize_tokens_workspace_size(256, 512, 2048, rq.quant_cfg(), rq.bgd_cfg(1e-4)) > \
        rq.realq_quantize_workspace_size(256, 512, rq.quant_cfg(), rq.bgd_cfg(1e-4))


def test_trace_and_graph_argument_validation(L):
    import paper_2609_00049_gb300 as rq
    q = rq.quant_cfg()
    b = rq.bgd_cfg(1e-4)
    t = ctypes.c_int64(0)
    # a NULL block_loss, and a trace workspace too small
    assert L.realq_quantize_layer_traced(None, 256, 512, FAKE, 0, FAKE, FAKE, None, ctypes.byref(q), ctypes.byref(b),
                                         FAKE, None, FAKE, FAKE, FAKE, FAKE, ctypes.byref(t), FAKE, FAKE, FAKE, None,
                                         0, 0, 4, FAKE, 1 << 40, None, FAKE, 1 << 30) == rq.REALQ_ERR_INVALID_ARG
    assert L.realq_quantize_layer_traced(None, 256, 512, FAKE, 0, FAKE, FAKE, None, ctypes.byref(q), ctypes.byref(b),
                                         FAKE, None, FAKE, FAKE, FAKE, FAKE, ctypes.byref(t), FAKE, FAKE, FAKE, None,
                                         0, 0, 4, FAKE, 1 << 40, FAKE, FAKE, 16) == rq.REALQ_ERR_WORKSPACE
    assert rq.realq_quantize_trace_workspace_size(256, 512) > 3 * 256 * 512 * 4
    # graphs: the legacy default stream cannot be captured; no graph to launch
    assert L.realq_graph_begin(None) == rq.REALQ_ERR_INVALID_ARG
    assert L.realq_graph_launch(None, None) == rq.REALQ_ERR_INVALID_ARG
    assert L.realq_graph_kernels(None) == 0
    L.realq_graph_destroy(None)                                          # a no-op
    # the deferred preparation and its status
    fc = ctypes.c_int64(7)
    assert L.realq_hessian_prepare_deferred(None, 0, 10, 0.01, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20) == 1
    assert L.realq_hessian_prepare_deferred(None, 64, 10, 0.01, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20) == 1  # U == H
    assert L.realq_hessian_prepare_deferred(None, 64, 10, 0.01, FAKE, ctypes.c_void_p(0x20000), FAKE, FAKE, None,
                                            0) == rq.REALQ_ERR_WORKSPACE
    assert L.realq_prepare_status(None, None, 0, ctypes.byref(fc)) == rq.REALQ_ERR_INVALID_ARG


def test_block_entry_points_reject_bad_arguments(L):
    # the decoder block of the exact sliding window: every check is on the
    # host, before any launch (fake device addresses are never dereferenced)
    import paper_2609_00049_gb300 as rq
    fake = ctypes.c_void_p(1 << 20)
    w = rq.BlockWeights(*([fake.value] * 9))

    def fwd(dims, S=2, L=8, ws=fake, nbytes=1 << 40):
        return L_.realq_block_forward(None, ctypes.byref(dims), ctypes.byref(w), S, L, fake, fake, ws, nbytes)

    L_ = L
    ok = rq.block_dims(64, 4, 2, 16, 96)
    assert rq.realq_block_workspace_size(ok, 2, 8) > (2 * 8) * (8 * 64 + 3 * 96) * 4
    assert fwd(rq.block_dims(64, 4, 3, 16, 96)) == rq.REALQ_ERR_INVALID_ARG      # n_heads % n_kv
    assert rq.realq_last_error() == "block_forward: n_heads % n_kv != 0"
    assert fwd(rq.block_dims(64, 4, 2, 15, 96)) == rq.REALQ_ERR_INVALID_ARG      # odd head_dim
    assert fwd(rq.block_dims(64, 4, 2, 512, 96)) == rq.REALQ_ERR_INVALID_ARG     # head_dim > 256
    assert fwd(rq.block_dims(64, 4, 2, 16, 96, rms_eps=0.0)) == rq.REALQ_ERR_INVALID_ARG
    assert fwd(rq.block_dims(64, 4, 2, 16, 96, rope_base=1.0)) == rq.REALQ_ERR_INVALID_ARG
    assert fwd(ok, S=0) == rq.REALQ_ERR_INVALID_ARG
    assert fwd(ok, S=4096, L=4096) == rq.REALQ_ERR_UNSUPPORTED                   # over 4194240 tokens
    assert fwd(ok, nbytes=16) == rq.REALQ_ERR_WORKSPACE
    assert fwd(ok, ws=ctypes.c_void_p((1 << 20) + 4)) == rq.REALQ_ERR_WORKSPACE  # misaligned
    w.Wd = None
    assert fwd(ok) == rq.REALQ_ERR_INVALID_ARG
    w.Wd = fake.value
    # the window: a NULL F_next
    assert L_.realq_block_window(None, ctypes.byref(ok), ctypes.byref(w), 2, 8, fake, fake, None, fake, None, fake,
                                 1 << 40) == rq.REALQ_ERR_INVALID_ARG
    assert "block_window" in rq.realq_last_error()


def test_block_module_and_head_entry_points_reject_bad_arguments(L):
    import paper_2609_00049_gb300 as rq
    fake = ctypes.c_void_p(1 << 20)
    w = rq.BlockWeights(*([fake.value] * 9))
    ok = rq.block_dims(64, 4, 2, 16, 96)
    big = 1 << 40

    def win(module=0, alpha=0.5, F=fake, nbytes=big, hat=None):
        return L.realq_block_module_window(None, ctypes.byref(ok), ctypes.byref(w), hat, ctypes.byref(w), 2, 8, fake,
                                           None, module, fake, alpha, F, fake, fake, None, fake, nbytes)

    # every block workspace starts with a status word and four tensor-core
    # operand planes of max(T, d) max(d, H dh, f) floats (T = 16, d = 64, f = 96)
    planes = 256 + 4 * max(16, 64) * max(64, 4 * 16, 96) * 4
    assert rq.realq_block_workspace_size(ok, 2, 8) > planes
    assert rq.realq_block_module_workspace_size(ok, 2, 8) > 2 * rq.realq_block_workspace_size(ok, 2, 8) - planes
    assert rq.realq_block_module_workspace_size(ok, 2, 8, 1000) > 2 * 8 * 1000 * 8
    assert rq.realq_block_head_workspace_size(64, 2, 8, 1000) > 2 * 8 * 1000 * 8
    assert win(module=7) == rq.REALQ_ERR_INVALID_ARG
    assert win(module=-1) == rq.REALQ_ERR_INVALID_ARG
    assert win(alpha=1.5) == rq.REALQ_ERR_INVALID_ARG
    assert win(F=None) == rq.REALQ_ERR_INVALID_ARG
    assert win(nbytes=1024) == rq.REALQ_ERR_WORKSPACE
    assert "block_module_window" in rq.realq_last_error()
    bad = rq.BlockWeights(*([fake.value] * 8 + [None]))                 # the current pass's weights are checked too
    assert win(hat=ctypes.byref(bad)) == rq.REALQ_ERR_INVALID_ARG
    # the head: vocab, eps and the token limit
    kl = L.realq_block_head_kl
    assert kl(None, 64, 2, 8, fake, fake, 0, 1e-6, fake, fake, fake, None, fake, big) == rq.REALQ_ERR_INVALID_ARG
    assert kl(None, 64, 2, 8, fake, fake, 100, 0.0, fake, fake, fake, None, fake, big) == rq.REALQ_ERR_INVALID_ARG
    assert kl(None, 64, 4096, 4096, fake, fake, 100, 1e-6, fake, fake, fake, None, fake, big) == \
        rq.REALQ_ERR_INVALID_ARG
    assert kl(None, 64, 2, 8, fake, fake, 100, 1e-6, fake, fake, fake, None, fake, 64) == rq.REALQ_ERR_WORKSPACE
    assert L.realq_block_module_kl(None, ctypes.byref(ok), ctypes.byref(w), None, 2, 8, fake, None, 3, fake, fake,
                                   None, 100, fake, None, fake, big) == rq.REALQ_ERR_INVALID_ARG     # NULL Wh


def test_window_sweep_entry_point_rejects_bad_arguments(L):
    # the sweep with Block-GD on the block ops' loss: every check is on the
    # host, before any launch or memset
    import paper_2609_00049_gb300 as rq
    fake = ctypes.c_void_p(1 << 20)
    w = rq.BlockWeights(*([fake.value] * 9))
    ok = rq.block_dims(64, 4, 2, 16, 96)
    q = rq.quant_cfg(group_size=64, block_size=64)
    big = 1 << 40
    t = ctypes.c_int64(0)

    def sweep(module=6, nxt=True, F=fake, vocab=0, head=fake, bcfg=None, qcfg=q, blocks=(0, 2), nbytes=big,
              deq_dtype=0, adam=fake, nmb=1):
        b = bcfg if bcfg is not None else rq.bgd_cfg(1e-3)
        return L.realq_quantize_layer_window(None, ctypes.byref(ok), ctypes.byref(w), None,
                                             ctypes.byref(w) if nxt else None, 2, 8, nmb, fake, None, module, F, fake,
                                             head, head,
                                             vocab, fake, None, ctypes.byref(qcfg), ctypes.byref(b), fake, adam, adam,
                                             ctypes.byref(t), fake, fake, fake, None, deq_dtype, None, blocks[0],
                                             blocks[1], fake, nbytes)

    n_win = rq.realq_quantize_window_workspace_size(ok, 2, 8, "down_proj", q)
    n_kl = rq.realq_quantize_window_workspace_size(ok, 2, 8, "down_proj", q, vocab=1000)
    assert n_win > rq.realq_block_module_workspace_size(ok, 2, 8) + 64 * 96 * 4
    assert n_kl > rq.realq_block_module_workspace_size(ok, 2, 8, 1000)
    assert rq.realq_quantize_window_workspace_size(ok, 2, 8, "q_proj", q) < n_win   # 64 x 64 against 64 x 96
    assert sweep(module=7) == rq.REALQ_ERR_INVALID_ARG
    assert sweep(F=None) == rq.REALQ_ERR_INVALID_ARG                               # the window needs F, F'
    assert sweep(nxt=False, vocab=0) == rq.REALQ_ERR_INVALID_ARG                   # the final block needs a head
    assert sweep(nxt=False, vocab=100, head=None) == rq.REALQ_ERR_INVALID_ARG
    assert sweep(bcfg=rq.bgd_cfg(1e-3, steps_per_block=0)) == rq.REALQ_ERR_INVALID_ARG
    assert "steps_per_block >= 1" in rq.realq_last_error()
    assert sweep(bcfg=rq.bgd_cfg(-1.0)) == rq.REALQ_ERR_INVALID_ARG
    assert sweep(adam=None) == rq.REALQ_ERR_INVALID_ARG                             # Adam needs its moments
    assert sweep(qcfg=rq.quant_cfg(block_size=96)) == rq.REALQ_ERR_INVALID_ARG
    assert sweep(blocks=(0, 3)) == rq.REALQ_ERR_INVALID_ARG                         # down_proj: 96 columns, 2 blocks
    assert sweep(deq_dtype=5) == rq.REALQ_ERR_INVALID_ARG
    assert sweep(nmb=0) == rq.REALQ_ERR_INVALID_ARG
    assert "n_minibatch" in rq.realq_last_error()
    assert sweep(nbytes=n_win - 1) == rq.REALQ_ERR_WORKSPACE
    assert "quantize_layer_window" in rq.realq_last_error()
    assert t.value == 0


def test_module_inputs_entry_point_rejects_bad_arguments(L):
    import paper_2609_00049_gb300 as rq
    fake = ctypes.c_void_p(1 << 20)
    w = rq.BlockWeights(*([fake.value] * 9))
    ok = rq.block_dims(64, 4, 2, 16, 96)

    def mi(module=0, X=fake, nbytes=1 << 40):
        return L.realq_block_module_inputs(None, ctypes.byref(ok), ctypes.byref(w), 2, 8, fake, module, X, fake,
                                           nbytes)

    assert mi(module=7) == rq.REALQ_ERR_INVALID_ARG
    assert mi(X=None) == rq.REALQ_ERR_INVALID_ARG
    assert mi(nbytes=rq.realq_block_workspace_size(ok, 2, 8) - 1) == rq.REALQ_ERR_WORKSPACE
    assert "block_module_inputs" in rq.realq_last_error()


def test_block_bindings_check_shapes_before_any_call(L):
    # the binding checks every shape the library will read against dims
    # (the C ABI takes plain pointers and cannot)
    import torch
    import paper_2609_00049_gb300 as rq
    d, H, Hkv, dh, f = 64, 4, 2, 16, 96
    dims = rq.block_dims(d, H, Hkv, dh, f)
    shapes = {"g1": (d,), "Wq": (H * dh, d), "Wk": (Hkv * dh, d), "Wv": (Hkv * dh, d), "Wo": (d, H * dh),
              "g2": (d,), "Wg": (f, d), "Wu": (f, d), "Wd": (d, f)}
    W = {k: torch.zeros(v) for k, v in shapes.items()}
    x, F = torch.zeros(2, 8, d), torch.zeros(d, d)
    grad = torch.zeros(d, f)
    with pytest.raises(ValueError, match="x"):
        rq.realq_block_module_window(dims, W, W, torch.zeros(2, 8, d + 1), "down_proj", W["Wd"], 0.5, F, F, grad,
                                     None)
    with pytest.raises(ValueError, match="x_hat"):
        rq.realq_block_module_window(dims, W, W, x, "down_proj", W["Wd"], 0.5, F, F, grad, None,
                                     x_hat=torch.zeros(3, 8, d))
    with pytest.raises(ValueError, match="W_module"):
        rq.realq_block_module_window(dims, W, W, x, "down_proj", torch.zeros(f, d), 0.5, F, F, torch.zeros(f, d),
                                     None)
    with pytest.raises(ValueError, match="F_next"):
        rq.realq_block_module_window(dims, W, W, x, "down_proj", W["Wd"], 0.5, F, torch.zeros(d, d + 1), grad, None)
    bad = dict(W, Wk=torch.zeros(H * dh, d))                     # n_kv heads' worth of rows expected
    with pytest.raises(ValueError, match="Wk"):
        rq.realq_block_forward(dims, bad, x, torch.zeros_like(x), None)
    with pytest.raises(ValueError, match="X_out"):
        rq.realq_block_module_inputs(dims, W, x, "o_proj", torch.zeros(16, d + 1), None)


def test_reverse_cosine_schedule_is_the_oracles(L):
    # host arithmetic behind the ABI (Eq. reverse_cosine): the same rates as
    # the oracle's schedule, and invalid indices refused
    import oracle
    import paper_2609_00049_gb300 as rq
    for Lb in (1, 2, 28, 80):
        for i in range(1, Lb + 1):
            got = rq.realq_reverse_cosine_lr(i, Lb, 3e-6)
            assert abs(got - oracle.reverse_cosine_lr(i, Lb, 3e-6)) <= 1e-15 * 3e-6
    out = ctypes.c_double(0.0)
    for i, Lb in ((0, 4), (5, 4), (1, 0)):
        assert L.realq_reverse_cosine_lr(i, Lb, ctypes.c_double(1e-3), ctypes.byref(out)) == 1
