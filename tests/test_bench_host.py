"""Host-side pieces of bench.py's JSON line: the workload table and the roofline object of the
dominant kernel (gate/up), for decode batches (HBM) and the prefill-shaped batch (tensor cores)."""
import pytest

import bench

PEAKS = {"hbm_gbs": 6790.3, "bf16_tflops": 1904.5, "bf16_tflops_sustained": 1717.4}


def test_default_workload_is_the_headline():
    """The 480B-shaped FP8 layer at 64 tokens: the largest single-GPU decode
    layer of the two served models."""
    wl = bench.workload(bench.parse([]))
    assert (wl["name"], wl["fmt"], wl["H"], wl["E"], wl["k"], wl["I"], wl["T"]) == \
        ("qwen3_480b_fp8_T64", 1, 6144, 160, 8, 2560, 64)
    assert not wl["prefill"] and wl["layers"] == 1


def test_sweep_covers_both_served_models_at_small_batches():
    names = {n for n, _ in bench.SWEEP}
    assert names == {"qwen3_235b_nvfp4", "qwen3_480b_fp8_zipf", "qwen3_235b_nvfp4_prefill"}
    batches = dict(bench.SWEEP)
    assert set(batches["qwen3_235b_nvfp4"]) == {1, 8, 32, 64}
    assert {1, 8, 32}.issubset(batches["qwen3_480b_fp8_zipf"])
    assert batches["qwen3_235b_nvfp4_prefill"] == (2048,)
    assert not bench.parse([]).no_sweep and bench.parse(["--no-sweep"]).no_sweep


def test_decode_roofline_is_hbm():
    wl = bench.workload(bench.parse([]))
    r = bench.gateup_roofline(wl, 2, 64, 8, 4096, 1536, 0.147, 6100.0, PEAKS, 926321408)
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["peak"] == 6790.3
    assert r["frac"] == pytest.approx(6100.0 / 6790.3)
    assert r["traffic"] == 926321408 and r["peak_source"] == "measured"
    r = bench.gateup_roofline(wl, 2, 64, 8, 4096, 1536, 0.147, 6100.0, {}, None)
    assert r["peak"] == 6800.0 and r["peak_source"] == "fallback"


def test_prefill_roofline_is_the_tensor_cores():
    wl = bench.workload(bench.parse(["--workload", "qwen3_235b_nvfp4_prefill"]))
    assert wl["prefill"] and wl["T"] == 2048
    gu_ms = 1.12
    r = bench.gateup_roofline(wl, 2, 2048, 8, 4096, 1536, gu_ms, 800.0, PEAKS, None)
    flops = 2048 * 8 * 2 * 2 * 4096 * 1536  # assignments x (gate, up) x 2 flops x H x I
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["achieved"] == pytest.approx(flops / (gu_ms * 1e-3) / 1e12)
    assert r["peak"] == pytest.approx(6 * 1717.4)  # NVFP4 dense = bf16 x 13.5 / 2.25
    assert r["frac"] == pytest.approx(r["achieved"] / r["peak"])
    assert r["hbm"]["frac"] == pytest.approx(800.0 / 6790.3)
    fp8 = bench.gateup_roofline(wl, 1, 2048, 8, 4096, 1536, gu_ms, 800.0, PEAKS, None)
    assert fp8["peak"] == pytest.approx(2 * 1717.4)  # FP8 dense = bf16 x 4.5 / 2.25
    fb = bench.gateup_roofline(wl, 2, 2048, 8, 4096, 1536, gu_ms, 800.0, {}, None)
    assert fb["peak"] == pytest.approx(6 * 1700.0) and fb["peak_source"].startswith("fallback")


def test_every_workload_parses():
    for name in bench.WORKLOADS:
        wl = bench.workload(bench.parse(["--workload", name]))
        assert wl["name"].startswith(name) and wl["T"] >= 1


def test_both_arms_name_the_same_metric():
    names = {n: bench.metric_name(bench.workload(bench.parse(["--workload", n])))
             for n in bench.WORKLOADS}
    assert names["qwen3_235b_nvfp4"] == "MoE decode-layer tokens/s"
    assert names["qwen3_235b_nvfp4_prefill"] == "MoE prefill-shaped layer tokens/s"
    assert names["qwen3_235b_nvfp4_x94"] == "MoE 94-layer decode-step tokens/s"
