"""The hyper-parameters the paper prints (tests/golden/paper_settings.txt,
each with its citation) against the defaults of the library's bindings, the
oracle and the scheduler, and against the learning rates of the workloads."""
import inspect
import math
import os

import oracle
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _settings():
    out = {}
    for line in open(os.path.join(ROOT, "tests", "golden", "paper_settings.txt")):
        line = line.split("#", 1)[0].strip()
        if line:
            k, v = (x.strip() for x in line.split("=", 1))
            out[k] = float(v)
    return out


def _default(fn, name):
    return inspect.signature(fn).parameters[name].default


def test_optimizer_defaults():
    import paper_2609_00049_gb300 as rq
    s = _settings()
    b = rq.bgd_cfg(1e-4)
    assert math.isclose(b.beta1, s["adam_beta1"], rel_tol=1e-7)
    assert math.isclose(b.beta2, s["adam_beta2"], rel_tol=1e-7)
    assert math.isclose(b.eps, s["adam_eps"], rel_tol=1e-6)
    assert b.steps_per_block == 1
    opt = oracle.Adam((1, 1), 1e-4)
    assert (opt.beta1, opt.beta2, opt.eps) == (s["adam_beta1"], s["adam_beta2"], s["adam_eps"])


def test_block_size_and_clipping_defaults():
    import paper_2609_00049_gb300 as rq
    from paper_2609_00049_gb300.block import BlockQuantizer
    s = _settings()
    assert rq.quant_cfg().block_size == s["block_size"]
    assert _default(BlockQuantizer.__init__, "saliency_pct") == s["saliency_clip_percentile"]
    assert _default(oracle.saliency_clip, "pct") == s["saliency_clip_percentile"]
    assert _default(oracle.quantize_activations, "a_clip") == s["a_clip"]


def test_bench_options_follow_the_paper():
    src = open(os.path.join(ROOT, "bench.py")).read()
    s = _settings()
    assert f'"--a-clip", type=float, default={s["a_clip"]}' in src
    # the mini-batch option counts 2048-token sequences, as the paper does
    assert "minibatch_tokens=2048 * args.minibatch_seqs" in src


def test_workload_learning_rates():
    s = _settings()
    wl = synth.workloads()
    for name in ("llama3.1-8b", "llama3.1-70b", "qwen3-0.6b", "qwen3-32b"):
        assert wl[name].lr == s["lr_w4a16_" + name], name


def test_reverse_cosine_base():
    s = _settings()
    eta = 3e-4
    assert math.isclose(oracle.reverse_cosine_lr(1, 28, eta), s["reverse_cosine_base_over_final"] * eta)
    assert math.isclose(oracle.reverse_cosine_lr(28, 28, eta), eta)
