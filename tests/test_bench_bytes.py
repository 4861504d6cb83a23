"""The roofline's algorithmic bytes against the bytes of the arrays the
generator actually produces for one expert (weights and scales)."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402
import synth  # noqa: E402


@pytest.mark.parametrize("wq", ["f32", "bf16", "fp8_b128", "int4_g128"])
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
