"""Pins of the oracle's layer quantization: protection mask bypass (paper Sec. 3),
the three bases (Sec. 1, Sec. 4) and the KIVI-style grouping rules.

Each base is reduced to the group quantizer (pinned by hand examples in
test_oracle_quantizer.py) applied to slices assembled independently here,
so a wrong index, a transposed operand or a dropped rotation fails.
"""
import numpy as np
import pytest
from scipy.linalg import hadamard

HAD = hadamard(128).astype(np.float64) / np.sqrt(128.0)


def _bf16_bits(rng, shape, outliers=()):
    x = rng.standard_normal(shape).astype(np.float32)
    for c in outliers:
        x[..., c] = x[..., c] * 8 + 3
    u = x.view(np.uint32)
    # round to nearest even into the upper 16 bits
    r = ((u.astype(np.uint64) + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    return r


def _f32(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32)


@pytest.mark.parametrize("T,s,n,R,expect", [
    (100, 10, 75, 32, 32),    # end = min(85, 68) = 68 -> 58 tokens -> one group
    (100, 10, 50, 32, 32),    # end = min(60, 68) -> 50 -> one group
    (100, 10, 50, 0, 32),
    (64, 0, 64, 0, 64),
    (64, 0, 64, 1, 32),       # residual takes the last token -> 63 -> one group
    (64, 0, 31, 0, 0),        # shorter than a group
    (40, 8, 32, 0, 32),
    (40, 8, 32, 1, 0),        # the window reaches into the image
])
def test_kivi_quantized_count(oracle, T, s, n, R, expect):
    assert oracle.quantized_count(T, s, n, oracle.BASE_KIVI, 32, R) == expect
    # the per-token bases code the whole image span
    assert oracle.quantized_count(T, s, n, oracle.BASE_MINMAX, 32, R) == n
    assert oracle.quantized_count(T, s, n, oracle.BASE_AKVQ, 32, R) == n


def _layer(oracle, base, bits, mask, keys_only, B=2, H=4, T=90, s=10, n=64, R=8, seed=0):
    rng = np.random.default_rng(seed)
    k = _bf16_bits(rng, (B, H, T, 128), outliers=(7, 63, 101))
    v = _bf16_bits(rng, (B, H, T, 128))
    out = oracle.quantize_layer(k, v, s, n, base, bits, np.array(mask, np.uint8), keys_only,
                                residual=R)
    return k, v, out


@pytest.mark.parametrize("base", [0, 1, 2])
@pytest.mark.parametrize("keys_only", [0, 1])
def test_text_and_protected_entries_are_exact(oracle, base, keys_only):
    mask = [0, 1, 0, 1]
    k, v, o = _layer(oracle, base, 2, mask, keys_only)
    B, H, T, _ = k.shape
    s, nq = 10, o["nq"]
    text = np.ones(T, bool)
    text[s:s + nq] = False
    for h in range(H):
        # text (and uncoded image) entries: BF16 values exactly
        assert np.array_equal(o["k_deq"][:, h, text], _f32(k[:, h, text]))
        assert np.array_equal(o["v_deq"][:, h, text], _f32(v[:, h, text]))
        assert not o["kq"][:, h, text].any() and not o["vq"][:, h, text].any()
        if mask[h]:
            assert np.array_equal(o["k_deq"][:, h], _f32(k[:, h]))
            assert not o["kq"][:, h].any()
            if not keys_only:
                assert np.array_equal(o["v_deq"][:, h], _f32(v[:, h]))
                assert not o["vq"][:, h].any()
            else:
                assert o["vq"][:, h, s:s + nq].all()
        else:
            assert o["kq"][:, h, s:s + nq].all() and o["vq"][:, h, s:s + nq].all()


@pytest.mark.parametrize("bits", [2, 3])
def test_minmax_is_per_token_group(oracle, bits):
    k, v, o = _layer(oracle, 0, bits, [0, 0, 0, 0], 0)
    s, nq = 10, o["nq"]
    W = 4 * bits
    for b in range(k.shape[0]):
        for h in range(k.shape[1]):
            kw = o["k_words"][b, h].reshape(nq, W)
            km = o["k_meta"][b, h].reshape(nq, 2)
            vw = o["v_words"][b, h].reshape(nq, W)
            for i in (0, 1, nq // 2, nq - 1):
                c, sc, z = oracle.quantize_group(_f32(k[b, h, s + i]), bits)
                assert np.array_equal(kw[i], oracle.pack(c, bits)) and km[i, 0] == sc and km[i, 1] == z
                c, sc, z = oracle.quantize_group(_f32(v[b, h, s + i]), bits)
                assert np.array_equal(vw[i], oracle.pack(c, bits))


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_kivi_key_groups_are_channel_slices(oracle, bits):
    k, v, o = _layer(oracle, 1, bits, [0, 1, 0, 0], 1, T=130, s=5, n=100, R=20)
    s, nq = 5, o["nq"]
    assert nq == 96
    per = 32 * bits // 32
    for b in range(2):
        for h in (0, 2):
            kw = o["k_words"][b, h].reshape(nq // 32, 128, per)
            km = o["k_meta"][b, h].reshape(nq // 32, 128, 2)
            vw = o["v_words"][b, h].reshape(nq, 128 * bits // 32)
            vm = o["v_meta"][b, h].reshape(nq, 4, 2)
            for g in range(nq // 32):
                for c in (0, 7, 63, 127):
                    col = _f32(k[b, h, s + 32 * g: s + 32 * g + 32, c])   # 32 tokens of channel c
                    codes, sc, z = oracle.quantize_group(col, bits)
                    assert np.array_equal(kw[g, c], oracle.pack(codes, bits))
                    assert km[g, c, 0] == sc and km[g, c, 1] == z
            for i in (0, 31, 95):
                row = _f32(v[b, h, s + i])
                allc = []
                for j in range(4):
                    codes, sc, z = oracle.quantize_group(row[32 * j: 32 * j + 32], bits)
                    assert vm[i, j, 0] == sc and vm[i, j, 1] == z
                    allc.append(codes)
                assert np.array_equal(vw[i], oracle.pack(np.concatenate(allc), bits))
    # keys-only protected head 1: keys exact everywhere, values coded on the groups
    assert np.array_equal(o["k_deq"][:, 1], _f32(k[:, 1]))
    assert o["vq"][:, 1, s:s + nq].all() and not o["vq"][:, 1, s + nq:].any()


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_akvq_rotates_keys_only(oracle, bits):
    k, v, o = _layer(oracle, 2, bits, [0, 0, 1, 0], 0)
    s, nq = 10, o["nq"]
    W = 128 * bits // 32
    for b in range(2):
        h = 0
        kw = o["k_words"][b, h].reshape(nq, W)
        km = o["k_meta"][b, h].reshape(nq, 2)
        for i in (0, 17, nq - 1):
            x = _f32(k[b, h, s + i])
            rot = (HAD @ x.astype(np.float64))
            r32 = oracle.fwht128(x)
            assert np.max(np.abs(r32 - rot)) < 1e-4 * np.abs(x).max()
            codes, sc, z = oracle.quantize_group(r32, bits)
            assert np.array_equal(kw[i], oracle.pack(codes, bits)) and km[i, 0] == sc
            # reconstruction: inverse rotation of the coded rotated key
            rec_rot = np.array([oracle.dequant(c, sc, z) for c in codes], np.float32)
            assert np.allclose(o["k_att"][b, h, s + i], HAD @ rec_rot.astype(np.float64), atol=1e-12)
            assert np.array_equal(o["k_deq"][b, h, s + i], oracle.fwht128(rec_rot))
            # values are not rotated: per-token group of the raw value
            codes_v, sv, zv = oracle.quantize_group(_f32(v[b, h, s + i]), bits)
            assert np.array_equal(o["v_words"][b, h].reshape(nq, W)[i], oracle.pack(codes_v, bits))


def test_empty_mask_equals_base_and_full_mask_is_bf16(oracle):
    k, v, o0 = _layer(oracle, 0, 2, [0, 0, 0, 0], 0, seed=3)
    _, _, o1 = _layer(oracle, 0, 2, [1, 1, 1, 1], 0, seed=3)
    # full K+V mask: the reconstruction is the BF16 cache itself
    assert np.array_equal(o1["k_deq"], _f32(k)) and np.array_equal(o1["v_deq"], _f32(v))
    assert not o1["kq"].any() and not o1["vq"].any()
    # empty mask: every image entry is coded
    assert o0["kq"][:, :, 10:74].all() and o0["vq"][:, :, 10:74].all()
