"""Pins for the oracle's number formats against independent library conversions.

bf16 rounding is checked against torch's conversion, binary16 decoding against
numpy's float16 for every bit pattern, and binary16 round-up against numpy's
round-to-nearest plus one step (numpy.nextafter in float16).
"""
import numpy as np
import torch


def _rand_f32(n, seed):
    rng = np.random.default_rng(seed)
    a = rng.standard_normal(n).astype(np.float32) * np.exp2(rng.integers(-30, 20, n)).astype(np.float32)
    # exact bf16 ties and near-ties
    base = rng.integers(0, 1 << 15, n // 4).astype(np.uint32) << 16
    ties = (base | 0x8000).view(np.float32)
    near = (base | 0x7FFF).view(np.float32)
    return np.concatenate([a, ties, near, np.array([0.0, -0.0, 1.0, -1.0, 65504.0, 1e-40], np.float32)])


def test_bf16_round_nearest_even_matches_torch(orc):
    x = _rand_f32(4000, 1)
    x = x[np.isfinite(x)]
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = orc.f32_to_bf16(x)
    assert np.array_equal(got, ref)


def test_bf16_decode_is_upper_half(orc):
    b = np.arange(0, 1 << 16, 97, dtype=np.uint16)
    f = orc.bf16_to_f32(b)
    ref = torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).float().numpy()
    fin = np.isfinite(ref)
    assert np.array_equal(f[fin], ref[fin])


def test_f16_decode_all_bit_patterns(orc):
    b = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16)
    got = orc.f16_to_f32(b)
    ref = b.view(np.float16).astype(np.float32)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan], ref[~nan])


def test_f16_round_up_is_smallest_not_below(orc):
    rng = np.random.default_rng(2)
    x = np.abs(rng.standard_normal(3000).astype(np.float32)) * np.exp2(rng.integers(-26, 16, 3000)).astype(np.float32)
    exact = np.abs(rng.standard_normal(500)).astype(np.float16).astype(np.float32)  # already on the grid
    x = np.concatenate([x, exact, np.array([0.0, 65504.0, 2.0**-24, 2.0**-25, 6.1e-5], np.float32)])
    got = orc.f32_to_f16_ru(x).view(np.float16)
    near = x.astype(np.float16)  # round to nearest (numpy)
    ref = np.where(near.astype(np.float32) >= x, near, np.nextafter(near, np.float16(np.inf)))
    assert np.array_equal(got.astype(np.float32), ref.astype(np.float32))
    assert np.all(got.astype(np.float32) >= x)
