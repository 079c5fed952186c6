"""32-bit metadata (Sec. 5.4 storage model; reading R13): the oracle's
binary16 conversion and the quantizer that computes codes against the stored
binary16 scale and zero."""
import numpy as np

import oracle


def test_f16_conversion_hand_values():
    f = oracle.f32_to_f16_bits
    assert f(1.0) == 0x3C00
    assert f(-2.0) == 0xC000
    assert f(65504.0) == 0x7BFF
    assert f(1.0e5) == 0x7BFF            # saturates instead of inf
    assert f(-7.0e4) == 0xFBFF
    assert f(2.0 ** -24) == 0x0001       # smallest subnormal
    assert f(2.0 ** -25) == 0x0000       # tie between 0 and 2^-24: even
    assert f(3 * 2.0 ** -25) == 0x0002   # tie between 1 and 2 units: even
    assert f(2.0 ** -14) == 0x0400       # smallest normal
    assert f(1.0 + 2.0 ** -11) == 0x3C00          # tie: even mantissa
    assert f(1.0 + 3 * 2.0 ** -11) == 0x3C02      # tie: even mantissa (up)
    assert f(1.0 + 2.0 ** -11 + 2.0 ** -20) == 0x3C01  # just above the tie
    assert oracle.f16_bits_to_f32(0x0001) == np.float32(2.0 ** -24)
    assert oracle.f16_bits_to_f32(0x7BFF) == np.float32(65504.0)


def test_f16_conversion_matches_ieee_round_to_nearest():
    # within the finite range the rule is plain IEEE round-to-nearest-even,
    # which numpy's float16 cast also implements
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.uniform(-9, 4.8, 20000),
                        np.float32(2.0) ** rng.integers(-26, 15, 2000) * (1 + 2.0 ** -11)])
    x = x.astype(np.float32)
    x = x[np.abs(x) < 65504]
    got = np.array([oracle.f32_to_f16_bits(v) for v in x], np.uint16)
    want = x.astype(np.float16).view(np.uint16)
    assert np.array_equal(got, want)
    back = np.array([oracle.f16_bits_to_f32(h) for h in got], np.float32)
    assert np.array_equal(back, want.view(np.float16).astype(np.float32))


def test_meta16_quantizer_hand_example():
    # [-1, 0, 0.5, 2], 2-bit: scale 1 and zero -1 are exact in binary16, so the
    # 32-bit-metadata codes equal the 64-bit ones: [0, 1, 2, 3] (1.5 -> 2)
    c16, s16, z16 = oracle.quantize_group([-1.0, 0.0, 0.5, 2.0], 2, meta16=True)
    c32, s32, z32 = oracle.quantize_group([-1.0, 0.0, 0.5, 2.0], 2)
    assert c16.tolist() == c32.tolist() == [0, 1, 2, 3]
    assert (s16, z16) == (s32, z32) == (np.float32(1.0), np.float32(-1.0))
    # a zero that binary16 cannot hold: min 0.1 is stored as 0.0999755859375,
    # and the codes are computed against the stored values
    x = np.array([0.1, 0.4, 0.7, 1.0], np.float32)
    c, s, z = oracle.quantize_group(x, 2, meta16=True)
    assert z == np.float32(np.float16(0.1)) and s == np.float32(np.float16(np.float32(0.9) / np.float32(3)))
    want = np.clip(np.rint((x - z) / s), 0, 3).astype(np.uint8)
    assert c.tolist() == want.tolist() == [0, 1, 2, 3]


def test_meta16_quantizer_properties():
    rng = np.random.default_rng(2)
    for bits in (2, 4):
        L = (1 << bits) - 1
        for _ in range(300):
            x = (rng.standard_normal(128) * 10.0 ** rng.uniform(-3, 3)).astype(np.float32)
            c, s, z = oracle.quantize_group(x, bits, meta16=True)
            # stored values are binary16 values
            assert np.float32(np.float16(s)) == s and np.float32(np.float16(z)) == z
            assert c.min() >= 0 and c.max() <= L
            # reconstruction from the stored values stays within half a step
            # (plus the offset of the rounded zero at the ends of the range)
            xr = np.float32(c.astype(np.float32) * s) + z
            assert np.all(np.abs(xr - x) <= s / 2 + abs(float(z) - float(x.min())) + 4e-6 * np.abs(x).max())
