"""The seeded input generators that both the oracle and the CUDA path draw
from: deterministic, chunk-consistent, and with the distributions the input
recipe states (outlier channels, unit-variance Student-t, SPD Fisher with
the stated row weights, heavy-tailed saliency)."""
import numpy as np

import synth


def test_chunks_are_deterministic_and_consistent():
    wl = synth.workloads()["qwen3-0.6b"]
    a = synth.xhat_full(wl, "attn_in", max_tokens=20000, threads=1)
    b = synth.xhat_full(wl, "attn_in", max_tokens=20000, threads=8)
    assert np.array_equal(a, b)
    c0 = synth.xhat_chunk(wl, "attn_in", 0)
    c1 = synth.xhat_chunk(wl, "attn_in", 1)
    assert np.array_equal(a[:8192], c0) and np.array_equal(a[8192:16384], c1)
    # arbitrary chunk sizes assemble from the canonical chunks
    odd = synth.xhat_chunk(wl, "attn_in", 2, chunk_tokens=5000)
    assert np.array_equal(odd, a[10000:15000])
    # other inputs and weights draw from other streams
    assert not np.array_equal(synth.xhat_chunk(wl, "mlp_in", 0), c0)
    md = wl.modules
    assert not np.array_equal(synth.weights(wl, md[1]), synth.weights(wl, md[2]))


def test_bf16_inputs_are_rounded_to_nearest_even():
    x = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5, 3.14159], dtype=np.float32)
    y = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(x))
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7: even mantissa (1.0);
    # 1 + 3 2^-8 ties between 1 + 2^-7 and 1 + 2^-6: even (1 + 2^-6)
    assert list(y[:3]) == [1.0, 1.0, 1.0 + 2 ** -6]
    assert y[3] == -2.5 and abs(y[4] - 3.140625) == 0


def test_outlier_channels_and_scales():
    wl = synth.workloads()["qwen3-0.6b"]
    spec = wl.inputs["down_in"]
    oc = synth.outlier_channels(wl, spec)
    assert oc.size == round(0.01 * spec.n)
    x = synth.xhat_full(wl, "down_in", as_bits=False, max_tokens=8192)
    sd = x.std(axis=0)
    normal = np.setdiff1d(np.arange(spec.n), oc)
    assert abs(np.median(sd[normal]) - 1.0) < 0.03
    assert abs(np.median(sd[oc]) - 20.0) < 0.6


def test_student_t_is_unit_variance_and_heavy_tailed():
    wl = synth.workloads()["llama3.1-8b"]
    x = synth.xhat_full(wl, "attn_in", as_bits=False, max_tokens=8192).astype(np.float64)
    assert abs(x.var() - 1.0) < 0.05
    kurt = ((x - x.mean()) ** 4).mean() / x.var() ** 2
    assert kurt > 4.0            # a Gaussian has 3


def test_fisher_is_spd_with_the_stated_row_weights():
    wl = synth.workloads()["qwen3-0.6b"]
    md = next(m for m in wl.modules if m.name == "k_proj")
    F = synth.fisher(wl, md).astype(np.float64)
    assert np.allclose(F, F.T)
    assert np.linalg.eigvalsh(F).min() > 0
    d = np.diag(synth.fisher_diag(wl, md))
    assert d.min() >= 0.5 and d.max() <= 2.0
    # diag(F) = d (1 + chi2_k / k) / 2 with k = 16: mean d, relative spread
    # sqrt(2 / k) / 2 = 0.18 against the row weights' 0.35, so a correlation
    # of about 0.88 with d
    assert np.corrcoef(np.diag(F), d)[0, 1] > 0.8
    assert abs(np.mean(np.diag(F) / d) - 1.0) < 0.1
    assert not np.array_equal(F, synth.fisher(wl, md, "F_next"))


def test_saliency_is_heavy_tailed():
    wl = synth.workloads()["qwen3-0.6b"]
    md = next(m for m in wl.modules if m.name == "k_proj")
    S = synth.saliency(wl, md, 4)
    assert S.shape == (wl.inputs[md.input].T, 4) and S.min() > 0
    assert (S.max(axis=0) / np.median(S, axis=0)).min() > 1e5
