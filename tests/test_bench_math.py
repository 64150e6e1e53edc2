"""The bench's roofline arithmetic on the CPU: the algorithmic work per step of
each kernel kind, checked against the workloads' closed forms written out by
hand (routed rows T*k; W13 is [2I, H], W2 is [H, I]; bf16 weights 2 bytes,
4-bit weights 0.5625 bytes with their group-32 fp16 scales), and the choice of
bound, peak and fraction for the dominant kernel."""
import pytest

import bench
import synth

PEAKS = {"hbm_gbs": 6785.2, "bf16_tflops": 1932.4, "bf16_tflops_sustained": 1709.1}


def test_gateup_and_down_work_qwen_4k():
    cfg = synth.config("qwen3next_4k")
    flops, nbytes = bench.algorithmic(cfg, "gateup", {})
    # 40,960 routed rows x 2 x 2048 x 1024
    assert flops == 171_798_691_840
    # all 512 W13 (4 MiB each) + each token's row once (4 KiB each) + h written (1 KiB a routed row)
    assert nbytes == 2_147_483_648 + 16_777_216 + 41_943_040
    flops, nbytes = bench.algorithmic(cfg, "down", {})
    assert flops == 85_899_345_920
    assert nbytes == 1_073_741_824 + 41_943_040 + 167_772_160


def test_gateup_work_32k_bf16_and_q4():
    cfg = synth.config("prefill32k_lru64")
    flops, nbytes = bench.algorithmic(cfg, "gateup", {})
    assert flops == 1_374_389_534_720          # 16 launches of ~85.9 GFLOP
    assert nbytes == 2_147_483_648 + 134_217_728 + 335_544_320
    q4 = synth.config("prefill32k_q4_lru64")
    f4, b4 = bench.algorithmic(q4, "gateup", {})
    assert f4 == flops
    assert b4 == 603_979_776 + 134_217_728 + 335_544_320   # W13 at 0.5625 B a weight


def test_roofline_of_the_routed_gemm_pair():
    """4K: the gate-up and down pair is HBM-bound (intensity ~88 flop/byte,
    below the burst ridge of ~285); 32K: tensor-bound against the burst peak."""
    cfg = synth.config("qwen3next_4k")
    kt = {"gateup": (3.5, 10), "down": (1.9, 10), "combine": (0.3, 10)}
    r = bench.roofline(cfg, kt, 10, PEAKS, {"sm_mhz": 2070.0}, "no-such-workload")
    assert r["kernel"] == "gateup+down" and r["bound"] == "hbm" and r["unit"] == "GB/s"
    pair_bytes = (2_147_483_648 + 16_777_216 + 41_943_040) + (1_073_741_824 + 41_943_040 + 167_772_160)
    achieved = pair_bytes / 0.54e-3 / 1e9
    assert r["achieved"] == pytest.approx(achieved)
    assert r["peak"] == 6785.2 and r["frac"] == pytest.approx(achieved / 6785.2)
    assert r["parts"]["gateup"]["achieved"] == pytest.approx(
        (2_147_483_648 + 16_777_216 + 41_943_040) / 0.35e-3 / 1e9)
    assert r["traffic"] is None
    # 32K, 16 waves: 2.06 TFLOP in 1.41 + 0.85 ms per step
    cfg = synth.config("prefill32k_lru64")
    kt = {"gateup": (1.41 * 4, 64), "down": (0.85 * 4, 64)}
    r = bench.roofline(cfg, kt, 4, PEAKS, {"sm_mhz": 2070.0}, "no-such-workload")
    assert r["bound"] == "tensor" and r["peak"] == 1932.4
    flops_step = 1_374_389_534_720 + 687_194_767_360
    assert r["achieved"] == pytest.approx(flops_step / 2.26e-3 / 1e12)
    assert r["frac"] == pytest.approx(flops_step / 2.26e-3 / 1e12 / 1932.4)
    assert r["launches_per_step"] == 16
    assert r["parts"]["down"]["achieved"] == pytest.approx(687_194_767_360 / 0.85e-3 / 1e12)


def test_single_kernel_fallback_when_no_routed_gemms():
    cfg = synth.config("qwen3next_4k")
    r = bench.roofline(cfg, {"combine": (0.4, 10)}, 10, PEAKS, {}, "x")
    assert r["kernel"] == "combine" and r["bound"] == "hbm"


def test_router_roof_is_the_fp32_alu_rate():
    cfg = synth.config("qwen3next_4k")
    r = bench.roofline(cfg, {"router": (1.0, 10)}, 10, PEAKS, {"sm_mhz": 2000.0}, "x")
    assert r["bound"] == "alu"
    assert r["peak"] == pytest.approx(82.6 * 2000.0 / 2070.0)


def test_roofline_of_fused_wave_launches():
    """Fused wave launches (one kernel per wave for both projections) carry
    the pair's flops over their own time."""
    cfg = synth.config("prefill32k_lru64")
    kt = {"ffn": (2.0 * 4, 64)}
    r = bench.roofline(cfg, kt, 4, PEAKS, {}, "no-such-workload")
    flops_step = 1_374_389_534_720 + 687_194_767_360
    assert r["bound"] == "tensor" and r["fused_waves"]
    assert r["achieved"] == pytest.approx(flops_step / 2.0e-3 / 1e12)
    assert r["launches_per_step"] == 16
