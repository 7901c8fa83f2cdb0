"""Host logic of bench.py on CPU: the roofline entries computed from a
per-kernel profile (the one a 40-step run of the Qwen3-0.6B block recorded),
for the bench line's `roofline` and `roofline_by_kernel`."""
import argparse
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import synth  # noqa: E402

# {kernel family: (launches, total ms)} over 40 steps
PROF = {"bgd_g_gemm_adam": (5560, 194.618), "chol_diag": (4480, 145.768), "hessian_syrk_tc": (160, 125.379),
        "trtri_trmm_tc": (4320, 116.026), "chol_update": (8480, 114.924), "bgd_p_gemm": (2920, 111.765),
        "quant_block": (3200, 97.391), "trtri_panel": (4320, 80.342), "trailing_update": (2920, 67.88),
        "chol_update_tc": (4320, 44.897), "bgd_g_gsum_adam": (2920, 26.335), "hessian_reduce": (160, 17.334),
        "trtri_trmm": (10, 0.5)}
# (the profile was recorded with the Block-GD products as tf32x3)
ARGS = argparse.Namespace(saliency_groups=0, act_bits=0, a_loss_clip=None, minibatch_seqs=0, bgd_products=0)
PEAKS = {"hbm_gbs": 6764.0, "bf16_tflops": 1888.7, "bf16_tflops_sustained": 1708.1, "sm_max_mhz": 2070.0,
         "source": "measured"}


def test_dominant_entry():
    wl = synth.workloads()["qwen3-0.6b"]
    r = bench.roofline(wl, PROF, 40, PEAKS, ARGS)
    assert r["kernel"] == "bgd_g_gemm_adam" and r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    # the G product's work: sum over modules and blocks of 2 m^2 r_b
    work = sum(2 * md.m * md.m * (md.n - min((b + 1) * 128, md.n)) for md in wl.modules
               for b in range(-(-md.n // 128)))
    assert r["work_per_step"] == work
    assert r["achieved"] == pytest.approx(work * 40 / 0.194618 / 1e12)
    assert r["peak"] == pytest.approx(1708.1 * 1.1 / 2.25 / 3)
    assert r["frac"] == pytest.approx(r["achieved"] / r["peak"])
    # (no counters of the current G kernel for this workload)
    assert r["traffic"] is bench.NCU_TRAFFIC.get(("qwen3-0.6b", "bgd_g_gemm_adam"))


def test_f16x3_products_take_the_fp16_peak():
    # with the products as f16x3 the peak is the fp16 (= bf16) tensor rate
    # over three passes, and the planes' split pass is modelled; the
    # row-grouped variant keeps tf32x3
    wl = synth.workloads()["qwen3-0.6b"]
    a = argparse.Namespace(**{**vars(ARGS), "bgd_products": 1})
    r = bench.roofline(wl, PROF, 40, PEAKS, a)
    assert r["kernel"] == "bgd_g_gemm_adam" and r["peak"] == pytest.approx(1708.1 / 3)
    models = bench.work_models(wl, a)
    assert models["bgd_p_gemm"][0] == "f16x3" and models["f16_split"][0] == "hbm"
    g = argparse.Namespace(**{**vars(a), "saliency_groups": 4})
    assert bench.work_models(wl, g)["bgd_g_gemm_adam"][0] == "tf32x3" and "f16_split" not in bench.work_models(wl, g)


def test_table_by_device_time():
    wl = synth.workloads()["qwen3-0.6b"]
    t = bench.roofline_table(wl, PROF, 40, PEAKS, ARGS)
    names = [e["kernel"] for e in t]
    assert names[0] == "bgd_g_gemm_adam" and len(t) == 8
    assert "bgd_g_gsum_adam" not in names and "hessian_reduce" not in names    # no work model
    assert "trtri_trmm" not in names     # no work on the fp32 tiles at these widths
    ms = [PROF[n][1] for n in names]
    assert ms == sorted(ms, reverse=True)
    for e in t:
        assert 0.0 < e["frac"] < 1.2, e
    hess = next(e for e in t if e["kernel"] == "hessian_syrk_tc")
    flops = sum(s.T * s.n * (s.n + 1) for s in wl.inputs.values())
    assert hess["achieved"] == pytest.approx(flops * 40 / 0.125379 / 1e12)


def test_empty_profile():
    wl = synth.workloads()["qwen3-0.6b"]
    assert bench.roofline(wl, {}, 40, PEAKS, ARGS) is None
    assert bench.roofline_table(wl, {}, 40, PEAKS, ARGS) == []


def test_table_skips_empty_rows():
    wl = synth.workloads()["qwen3-0.6b"]
    t = bench.roofline_table(wl, {"quant_block": (10, 0.0), "chol_diag": (0, 0.0), "bgd_p_gemm": (73, 2.7)}, 1,
                             PEAKS, ARGS)
    assert [e["kernel"] for e in t] == ["bgd_p_gemm"]
