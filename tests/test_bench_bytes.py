"""The roofline's algorithmic bytes against the bytes of the arrays the
generator actually produces for one expert (weights and scales)."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402
import synth  # noqa: E402


@pytest.mark.parametrize("wq", ["f32", "bf16", "fp8_b128", "int4_g128", "mxfp4"])
@pytest.mark.parametrize("H,I", [(256, 128), (512, 384)])
def test_expert_bytes_match_generated_arrays(wq, H, I):
    wl = synth.WORKLOADS[1].replace(H=H, I=I, E=2, top_k=1, wq=wq, act="f32" if wq == "f32" else "bf16")
    one = synth.expert_weights(wl, wl.E, I, e0=1, ne=1)
    assert bench.expert_bytes(wq, H, I) == sum(a.nbytes for a in one.values())


def test_layer_bytes_count_active_and_shared_experts():
    wl = synth.WORKLOADS[4]
    routed = bench.expert_bytes(wl.wq, wl.H, wl.I)
    shared = bench.expert_bytes(wl.wq, wl.H, wl.I_shared)
    assert bench.algorithmic_weight_bytes(wl, 200) == 200 * routed + shared
    wl2 = synth.WORKLOADS[2]
    assert bench.algorithmic_weight_bytes(wl2, 110) == 110 * 3 * wl2.H * wl2.I * 2


PK = {"hbm_gbs": 6780.0, "bf16_tflops": 1908.6, "bf16_tflops_sustained": 1705.1}


def test_roofline_takes_the_slower_bound():
    # 4 GB in 0.7 ms with 10 GFLOP: HBM-bound
    r = bench.roofline_entry(4.0e9, 1.0e10, 0.7, PK, "measured", {"kernel": "k"})
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert r["achieved"] == pytest.approx(4.0e9 / 0.7e-3 / 1e9)
    assert r["frac"] == pytest.approx(r["achieved"] / 6780.0)
    assert r["roofline_ms"] == pytest.approx(4.0e9 / 6780e9 * 1e3) and r["kernel"] == "k"
    # 5 GB and 2.5 TFLOP in 2 ms: tensor-bound, burst and sustained fractions
    r = bench.roofline_entry(5.0e9, 2.5e12, 2.0, PK, "measured", {})
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["achieved"] == pytest.approx(1250.0)
    assert r["frac"] == pytest.approx(1250.0 / 1908.6)
    assert r["frac_sustained"] == pytest.approx(1250.0 / 1705.1)


def test_fallback_peaks_have_every_key_the_roofline_reads():
    assert set(PK) <= set(bench.FALLBACK_PEAKS)


def test_roofline_without_a_sustained_peak():
    r = bench.roofline_entry(5.0e9, 2.5e12, 2.0, {"hbm_gbs": 6780.0, "bf16_tflops": 1908.6}, "measured", {})
    assert r["bound"] == "tensor" and "frac_sustained" not in r
