"""Pins of the oracle's group quantizer and bit packing (paper Sec. 1, Sec. 4).

Every check here compares the oracle with something other than itself: hand
-worked examples, exact rational arithmetic, or invariants the definition
implies.
"""
import os
from fractions import Fraction

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _hand_examples():
    rows = []
    with open(os.path.join(GOLDEN, "quantizer_hand_examples.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            bits, vals, codes, scale, zero, rec = [p.strip() for p in line.split("|")]
            rows.append((int(bits), [float(x) for x in vals.split()], [int(c) for c in codes.split()],
                         float(scale), float(zero), [float(x) for x in rec.split()]))
    return rows


@pytest.mark.parametrize("bits,vals,codes,scale,zero,rec", _hand_examples())
def test_hand_examples(oracle, bits, vals, codes, scale, zero, rec):
    c, s, z = oracle.quantize_group(np.array(vals, np.float32), bits)
    assert list(c) == codes
    assert s == np.float32(scale) and z == np.float32(zero)
    got = [oracle.dequant(ci, s, z) for ci in c]
    assert got == [np.float32(r) for r in rec]


def _groups(rng, n, count):
    out = []
    for i in range(count):
        kind = i % 5
        if kind == 0:
            x = rng.standard_normal(n)
        elif kind == 1:
            x = rng.standard_normal(n) * 8 + 3           # outlier-channel law
        elif kind == 2:
            x = rng.standard_normal(n) * 1e-30           # tiny magnitudes (near subnormal)
        elif kind == 3:
            x = rng.integers(-4, 5, n).astype(np.float64) / 4   # many exact ties
        else:
            x = rng.standard_normal(n) * 1e4
        out.append(x.astype(np.float32))
    return out


@pytest.mark.parametrize("bits", [2, 3, 4])
@pytest.mark.parametrize("n", [4, 32, 128])
def test_invariants_and_nearest_level(oracle, bits, n):
    """codes in [0, L]; min -> 0, max -> L; each code is a nearest level in exact arithmetic."""
    rng = np.random.default_rng(1234 + bits * 10 + n)
    L = (1 << bits) - 1
    for x in _groups(rng, n, 40):
        c, s, z = oracle.quantize_group(x, bits)
        assert c.min() >= 0 and c.max() <= L
        mn, mx = x.min(), x.max()
        assert z == mn + np.float32(0.0)
        if mx == mn:
            assert s == 0 and (c == 0).all()
            continue
        assert c[np.argmin(x)] == 0 and c[np.argmax(x)] == L
        # exact rationals: the chosen level is within half a step (plus the two
        # fp32 roundings of d and d/scale) of the exact position d/scale.
        S = Fraction(float(s))
        for xi, ci in zip(x, c):
            pos = (Fraction(float(xi)) - Fraction(float(mn))) / S
            dist = abs(pos - ci)
            assert dist <= Fraction(1, 2) + Fraction(1, 1 << 18), (xi, ci, float(pos))
            # and no other level is strictly nearer by more than the rounding slack
            best = min(abs(pos - k) for k in range(L + 1))
            assert dist - best <= Fraction(1, 1 << 18)


@pytest.mark.parametrize("bits", [2, 4])
def test_reconstruction_error_bound(oracle, bits):
    """|x - x^| <= scale / 2 + a few ulps of the group magnitude (Sec. 4 reconstruction)."""
    rng = np.random.default_rng(99 + bits)
    for x in _groups(rng, 128, 50):
        c, s, z = oracle.quantize_group(x, bits)
        rec = np.array([oracle.dequant(ci, s, z) for ci in c], np.float32)
        slack = 8 * np.spacing(np.float32(np.abs(x).max()))
        assert np.all(np.abs(rec.astype(np.float64) - x) <= float(s) / 2 + slack)


def test_constant_and_signed_zero_groups(oracle):
    for v in [0.0, -0.0, 3.5, -7.25, 1e-40]:
        x = np.full(128, v, np.float32)
        c, s, z = oracle.quantize_group(x, 2)
        assert s == 0 and (c == 0).all()
        assert oracle.dequant(0, s, z) == np.float32(v)
    # a group whose minimum is -0 stores zero = +0 (one bit pattern)
    x = np.array([-0.0, 1.0, 2.0, 3.0], np.float32)
    _, _, z = oracle.quantize_group(x, 2)
    assert np.signbit(z) == False  # noqa: E712


def test_pack_hand_examples(oracle):
    # 2-bit codes 1, 2, 3 in elements 0, 1, 2: 1 | 2<<2 | 3<<4 = 0x39
    c = np.zeros(16, np.uint8)
    c[:3] = [1, 2, 3]
    assert list(oracle.pack(c, 2)) == [0x39]
    # element 15 of a 2-bit word sits in bits 30..31
    c = np.zeros(32, np.uint8)
    c[15] = 3
    c[16] = 1
    assert list(oracle.pack(c, 2)) == [0xC0000000, 0x1]
    # 4-bit: 15 then 1 -> 0x1F; element 7 in bits 28..31
    c = np.zeros(8, np.uint8)
    c[0], c[1], c[7] = 15, 1, 9
    assert list(oracle.pack(c, 4)) == [0x9000001F]


@pytest.mark.parametrize("bits", [2, 4])
def test_pack_roundtrip(oracle, bits):
    rng = np.random.default_rng(bits)
    c = rng.integers(0, 1 << bits, 128).astype(np.uint8)
    w = oracle.pack(c, bits)
    assert w.size == 128 * bits // 32
    assert (oracle.unpack(w, 128, bits) == c).all()
    # independent extraction through numpy's bit view (little-endian words)
    bitsarr = np.unpackbits(w.view(np.uint8), bitorder="little").reshape(-1, bits)
    vals = (bitsarr * (1 << np.arange(bits))).sum(1)
    assert (vals == c).all()


def test_pack3_hand_examples(oracle):
    """R16: bits 0-1 in the 2-bit packing, then a bit-2 plane whose element e
    sits at e mod 32 with index bits 3 and 4 exchanged."""
    c = np.zeros(32, np.uint8)
    assert list(oracle.pack(c, 3)) == [0, 0, 0]
    c[:] = 4
    assert list(oracle.pack(c, 3)) == [0, 0, 0xFFFFFFFF]
    c[:] = 0
    c[8] = 7    # low bits 3 at word 0 bits 16-17; plane position 16
    c[16] = 4   # low bits 0; plane position 8
    c[23] = 5   # low bits 1 at word 1 bits 14-15; plane position 15
    c[31] = 6   # low bits 2 at word 1 bits 30-31; plane position 31
    assert list(oracle.pack(c, 3)) == [0x00030000, 0x80004000, 0x80018100]
    assert [oracle.lib().hgo_plane_pos(e) for e in (0, 7, 8, 15, 16, 23, 24, 31, 40)] == \
        [0, 7, 16, 23, 8, 15, 24, 31, 16]


def test_pack3_roundtrip_and_pairing(oracle):
    rng = np.random.default_rng(33)
    for n in (32, 128):
        c = rng.integers(0, 8, n).astype(np.uint8)
        w = oracle.pack(c, 3)
        assert w.size == n * 3 // 32
        assert (oracle.unpack(w, n, 3) == c).all()
        # low part: numpy's bit view of the first n/16 words as 2-bit fields
        lo = np.unpackbits(w[:n // 16].view(np.uint8), bitorder="little").reshape(-1, 2)
        assert ((lo * [1, 2]).sum(1) == (c & 3)).all()
        # plane: each code's bit 2 exactly once
        hi = np.unpackbits(w[n // 16:].view(np.uint8), bitorder="little")
        assert hi.sum() == int((c >> 2).sum())
    # codes e and e + 8 of one 16-code word: low bits 16 apart, and so are their plane bits
    for e in range(128):
        if e % 16 < 8:
            pe, pf = oracle.lib().hgo_plane_pos(e), oracle.lib().hgo_plane_pos(e + 8)
            assert pf - pe == 16 and (e // 32) == ((e + 8) // 32)
