"""bench.py's roofline arithmetic on the CPU: the algorithmic bytes and FLOPs per kernel launch and
the layer roofline, written out by hand for the DeiT-B layer (T = 50,432, d = 768, H = 3,072,
E = 8, r = 128, bf16), the whole-job rate, and the fp32 layer's tensor peak (three TF32 products
per fp32 product)."""
import importlib.util
import os

import pytest

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_stage_work_deit_base(bench):
    s = synth.DEIT_BASE_BF16
    w = bench.stage_work(s)
    T = 50432
    # routing: every token row once (bf16), W_g and b_g once, idx + tinfo per token, counts + offsets
    assert w["route"]["bytes"] == T * 768 * 2 + (8 * 768 + 8) * 2 + 8 * T + 8 * 8 == 77_879_376
    assert w["fc1_gelu"]["flops"] == 2 * T * 768 * 3072  # 237.97 GFLOP
    assert w["basis"]["flops"] == 2 * T * 3072 * 128  # 39.66 GFLOP
    assert w["grouped"]["flops"] == 2 * T * 768 * 128 + 2 * T * 768 * 3072  # 247.9 GFLOP
    assert w["fc1_gelu"]["flops"] == 237_968_031_744


def test_layer_roofline_deit_base(bench):
    s = synth.DEIT_BASE_BF16
    pk = {"bf16_tflops_sustained": 1732.6, "hbm_gbs": 6682.5}
    flops = 50432 * (2 * 768 * 3072 + 2 * 128 * (3072 + 768) + 2 * 768 * 3072 + 2 * 768 * 8)
    assert flops == 526_132_445_184
    t = bench.layer_roofline_s(s, pk)
    assert t == pytest.approx(flops / 1732.6e12)  # tensor-bound: 303.7 us
    assert 303e-6 < t < 304.5e-6
    # at a tiny HBM figure the same layer is bandwidth-bound: tokens in and out plus the weights
    weights = (3072 * 768 + 3072 + 768 * 128 + 128 + 128 * 3072 + 8 * 768 * 3072 + 8 * 768 + 8) * 2
    assert bench.layer_roofline_s(s, {"bf16_tflops_sustained": 1e9, "hbm_gbs": 1.0}) == pytest.approx(
        (2 * 50432 * 768 * 2 + weights) / 1e9)


def test_whole_job_rate(bench):
    assert bench.whole_job_rate(50432, 1, 10, 4.07) == pytest.approx(50432 * 10 / 4.07e-3)
    assert bench.whole_job_rate(50432, 8, 1, 1.0) == pytest.approx(8 * 50432 / 1e-3)  # weak scaling


def test_fp32_layer_peak_is_tf32_over_three(bench):
    """The fp32 layer's GEMMs run as three TF32 products per fp32 product: their peak in fp32
    FLOP/s is the measured bf16 peak x 1.1 / 2.25 (nominal dense TF32 / bf16) / 3."""
    assert bench.TF32X3_OF_BF16 == pytest.approx(1.1 / 2.25 / 3)
    pk = {"bf16_tflops": 1916.0, "bf16_tflops_sustained": 1732.6, "hbm_gbs": 6682.5}
    s = synth.DEIT_TINY_FP32
    stages = {"route": [0.010], "fc1_gelu": [0.010], "basis": [0.010], "grouped": [0.010]}
    out = bench.stage_summary(s, stages, pk)
    tf = 2 * 788 * 192 * 768 / 10e-6 / 1e12  # fc1 in 10 us
    assert out["fc1_gelu"]["TFLOP_s"] == pytest.approx(tf)
    assert out["fc1_gelu"]["tensor_frac"] == pytest.approx(tf / (1916.0 * 1.1 / 2.25 / 3))
    assert "alu_frac" not in out["fc1_gelu"]
