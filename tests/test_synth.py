"""Checks of the seeded input generator (not of the layer): determinism,
counter addressing, moments, and that its storage forms are the RNE roundings
torch's own dtype conversions produce."""
import numpy as np
import torch

import synth


def test_streams_are_deterministic_and_counter_addressed():
    a = synth.normal_f32(7, 3, 0.5, (10000,))
    b = synth.normal_f32(7, 3, 0.5, (10000,))
    assert np.array_equal(a, b)
    c = synth.normal_f32(7, 3, 0.5, (100,), offset=1234)
    assert np.array_equal(c, a[1234:1334])
    assert not np.array_equal(a, synth.normal_f32(7, 4, 0.5, (10000,)))
    assert not np.array_equal(a, synth.normal_f32(8, 3, 0.5, (10000,)))


def test_normal_moments():
    a = synth.normal_f32(1, 1, 0.02, (1 << 21,)).astype(np.float64)
    assert abs(a.mean()) < 0.02 * 5 / np.sqrt(a.size)
    assert abs(a.std() / 0.02 - 1) < 0.01
    kurt = ((a - a.mean()) ** 4).mean() / a.var() ** 2
    assert 2.7 < kurt < 3.0  # Irwin-Hall(8): 3 - 6/40 = 2.85


def test_bf16_is_rne_of_the_f32_stream():
    f = synth.normal_f32(2, 5, 1.0, (50000,))
    b = synth.normal_bf16(2, 5, 1.0, (50000,))
    ref = torch.from_numpy(f).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(b, ref)


def test_fp8_blocks_are_rne_e4m3_of_w_over_blockscale():
    N, K, e0, ne = 256, 384, 1, 2
    q, s = synth.fp8_b128(3, 3, 0.02, N, K, e0, ne)
    w = synth.normal_f32(3, 3, 0.02, (ne, N, K), offset=e0 * N * K)
    blocks = w.reshape(ne, N // 128, 128, K // 128, 128)
    amax = np.abs(blocks).max(axis=(2, 4)).astype(np.float32)
    assert np.array_equal(s, (amax / np.float32(448.0)).astype(np.float32))
    ratio = (blocks / s[:, :, None, :, None]).astype(np.float32).reshape(ne, N, K)
    ratio = np.clip(ratio, -448.0, 448.0)  # torch's conversion does not saturate
    ref = torch.from_numpy(ratio).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    assert np.array_equal(q, ref)


def test_int4_groups_are_rne_of_w_over_bf16_scale():
    N, K = 5, 512
    q, s = synth.int4_g128(4, 4, 0.02, N, K, 3, 1)
    w = synth.normal_f32(4, 4, 0.02, (N, K), offset=3 * N * K)
    g = w.reshape(N, K // 128, 128)
    sc = torch.from_numpy((np.abs(g).max(axis=2) / np.float32(7.0)).astype(np.float32)).to(torch.bfloat16)
    assert np.array_equal(s[0], sc.view(torch.int16).numpy().view(np.uint16))
    sf = sc.to(torch.float32).numpy()
    vals = np.clip(np.rint((g / sf[:, :, None]).astype(np.float32)), -8, 7).astype(np.int64).reshape(N, K)
    lo, hi = q[0] & 0xf, q[0] >> 4
    dec = np.empty((N, K), np.int64)
    dec[:, 0::2] = np.where(lo >= 8, lo.astype(np.int64) - 16, lo)
    dec[:, 1::2] = np.where(hi >= 8, hi.astype(np.int64) - 16, hi)
    assert np.array_equal(dec, vals)


def test_zipf_offsets_shape_and_order():
    b = synth.zipf_logit_bias(64)
    assert b.shape == (64,) and b[0] == 0.0 and np.all(np.diff(b) < 0)
