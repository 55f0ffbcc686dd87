"""Pins for the element-wise add's reference (oracle/ewise.py): the bf16
rounding against an independent library routine (torch's float32 -> bfloat16
conversion, round to nearest even) including exact ties, exactness on small
integers, the identity x + 0 = x, commutativity, and the widening being the
exact inverse of truncation for every bf16 pattern."""
import numpy as np
import torch

from oracle import ewise as ew


def test_widening_is_exact_for_every_pattern():
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    f = ew.bf16_bits_to_f32(bits)
    ref = torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).float().numpy()
    finite = np.isfinite(ref)
    assert np.array_equal(f[finite], ref[finite])
    assert np.array_equal(np.isnan(f), np.isnan(ref))


def test_rounding_matches_torch_including_ties():
    rng = np.random.default_rng(0)
    x = rng.standard_normal(200000).astype(np.float32) * np.float32(1e3)
    # exact ties: a bf16 value plus half of its last place, both parities
    base = (rng.integers(0x3F00, 0x4700, 5000).astype(np.uint32) << 16)
    ties = (base | 0x8000).view(np.float32)
    for v in (x, ties):
        ours = ew.f32_to_bf16_bits(v)
        ref = torch.from_numpy(v).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
        assert np.array_equal(ours, ref)


def test_small_integers_exact_and_identities():
    a = np.arange(-200, 200, dtype=np.float32)
    ab = ew.f32_to_bf16_bits(a)
    s = ew.add_bf16(ab, ab[::-1])
    assert np.array_equal(ew.bf16_bits_to_f32(s), a + a[::-1])
    zero = ew.f32_to_bf16_bits(np.zeros_like(a))
    assert np.array_equal(ew.add_bf16(ab, zero), ab)
    rng = np.random.default_rng(1)
    x = ew.f32_to_bf16_bits(rng.standard_normal(1000).astype(np.float32))
    y = ew.f32_to_bf16_bits(rng.standard_normal(1000).astype(np.float32))
    assert np.array_equal(ew.add_bf16(x, y), ew.add_bf16(y, x))


def test_bf16_add_matches_library_composition():
    rng = np.random.default_rng(2)
    xb = torch.from_numpy(rng.standard_normal(50000).astype(np.float32)).to(torch.bfloat16)
    yb = torch.from_numpy((rng.standard_normal(50000) * 1e-3).astype(np.float32)).to(torch.bfloat16)
    ref = (xb.float() + yb.float()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    ours = ew.add_bf16(xb.view(torch.int16).numpy().view(np.uint16), yb.view(torch.int16).numpy().view(np.uint16))
    assert np.array_equal(ours, ref)


def test_f32_add_is_ieee_single():
    x = np.array([1.0, 1e-8, 3.0, -2.5], dtype=np.float32)
    y = np.array([2 ** -24, 1.0, -3.0, 0.5], dtype=np.float32)
    z = ew.add_f32(x, y)
    assert z.dtype == np.float32
    assert z[0] == np.float32(1.0)          # 1 + 2^-24 ties to even -> 1
    assert z[1] == np.float32(1.0) and z[2] == 0.0 and z[3] == np.float32(-2.0)
