"""Pins of the oracle's AKVQ-style salient tokens (Sec. 4 "Quantization setup":
in each KV head the keys and values of a nominal 2% of the image tokens, those
with the largest key norms, stay BF16; reading R15).

The selection is checked against a brute-force ranking on keys whose squared
norms are exact small integers, and the quantized tokens against the base
quantizer run by the oracle on the compacted sequence (the image span with the
salient tokens cut out), so a token left in place, an uncompacted index or a
swapped K/V slot fails.
"""
import numpy as np
import pytest


def _bf16_of_int(x):
    """Exact BF16 bits of small integers (|x| < 256)."""
    f = np.asarray(x, np.float32)
    return (f.view(np.uint32) >> 16).astype(np.uint16)


def _f32(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32)


def _bf16_bits(rng, shape):
    x = rng.standard_normal(shape).astype(np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


@pytest.mark.parametrize("n,permille,expect", [
    (1296, 20, 26),   # 25.92 rounds up
    (3328, 20, 67),   # 66.56
    (1000, 20, 20),   # exact
    (50, 20, 1),
    (49, 20, 1),
    (64, 0, 0),
    (64, 1000, 64),
    (0, 20, 0),
])
def test_salient_count(oracle, n, permille, expect):
    assert oracle.salient_count(n, permille) == expect


def test_select_hand_examples(oracle):
    assert list(oracle.select_salient(np.array([1, 5, 5, 2, 9, 0], np.float32), 3)) == [1, 2, 4]
    # ties keep the lower index
    assert list(oracle.select_salient(np.array([3, 3, 3, 3], np.float32), 2)) == [0, 1]
    assert list(oracle.select_salient(np.array([0, 7, 7, 1], np.float32), 1)) == [1]
    assert list(oracle.select_salient(np.array([2, 1], np.float32), 0)) == []
    assert list(oracle.select_salient(np.array([2, 1, 4], np.float32), 3)) == [0, 1, 2]


def test_select_matches_brute_force(oracle):
    rng = np.random.default_rng(4)
    for trial in range(20):
        n = int(rng.integers(1, 300))
        ns = int(rng.integers(0, n + 1))
        score = rng.integers(0, 12, n).astype(np.float32)  # many ties
        order = sorted(range(n), key=lambda i: (-score[i], i))
        want = sorted(order[:ns])
        assert list(oracle.select_salient(score, ns)) == want


def test_key_norm_is_the_sum_of_squares(oracle):
    rng = np.random.default_rng(5)
    for trial in range(50):
        x = rng.integers(-15, 16, 128)
        assert float(oracle.key_norm2(_bf16_of_int(x))) == float(np.sum(x.astype(np.int64) ** 2))
    one = np.zeros(128, np.int64)
    for c in (0, 1, 63, 127):
        one[:] = 0
        one[c] = 11
        assert float(oracle.key_norm2(_bf16_of_int(one))) == 121.0


def _layer(oracle, base, bits, mask, permille, B=2, H=4, T=120, s=9, n=96, seed=0, integer=False,
           meta16=False):
    rng = np.random.default_rng(seed)
    if integer:
        k = _bf16_of_int(rng.integers(-7, 8, (B, H, T, 128)))
    else:
        k = _bf16_bits(rng, (B, H, T, 128))
    v = _bf16_bits(rng, (B, H, T, 128))
    ns = oracle.salient_count(n, permille)
    o = oracle.quantize_layer(k, v, s, n, base, bits, np.array(mask, np.uint8), 0,
                              meta16=meta16, n_salient=ns)
    return k, v, ns, o


@pytest.mark.parametrize("base", [0, 2])
def test_selection_is_the_largest_exact_norms(oracle, base):
    mask = [0, 1, 0, 0]
    k, v, ns, o = _layer(oracle, base, 2, mask, 50, integer=True)
    B, H, T, _ = k.shape
    s, n = 9, 96
    assert ns == 5
    for b in range(B):
        for h in range(H):
            if mask[h]:
                assert not o["salient"][b, h].any()
                continue
            norms = (_f32(k[b, h, s:s + n]).astype(np.int64) ** 2).sum(axis=1)
            order = sorted(range(n), key=lambda i: (-norms[i], i))
            assert list(o["salient"][b, h]) == sorted(order[:ns])


@pytest.mark.parametrize("base,bits,meta16", [(2, 4, False), (2, 2, False), (0, 2, False),
                                              (2, 4, True)])
def test_salient_tokens_stay_bf16_and_the_rest_is_the_compacted_base(oracle, base, bits, meta16):
    mask = [0, 1, 0, 0]
    k, v, ns, o = _layer(oracle, base, bits, mask, 20, seed=3, meta16=meta16, n=150, T=170)
    B, H, T, _ = k.shape
    s, n = 9, 150
    assert ns == 3
    W = 128 * bits // 32
    for b in range(B):
        for h in range(H):
            if mask[h]:
                continue
            sal = o["salient"][b, h]
            assert len(set(sal)) == ns and np.all(np.diff(sal) > 0)
            keep = np.setdiff1d(np.arange(n), sal)
            # salient tokens: exact, not quantized
            for i in sal:
                t = s + i
                assert o["kq"][b, h, t] == 0 and o["vq"][b, h, t] == 0
                assert np.array_equal(o["k_deq"][b, h, t], _f32(k[b, h, t]))
                assert np.array_equal(o["v_deq"][b, h, t], _f32(v[b, h, t]))
                assert np.array_equal(o["k_att"][b, h, t], _f32(k[b, h, t]).astype(np.float64))
            assert np.all(o["kq"][b, h, s + keep] == 1) and np.all(o["vq"][b, h, s + keep] == 1)
            # the other image tokens: the base on the compacted sequence
            toks = np.concatenate([np.arange(s), s + keep, np.arange(s + n, T)])
            kc = k[b:b + 1, h:h + 1][:, :, toks]
            vc = v[b:b + 1, h:h + 1][:, :, toks]
            r = oracle.quantize_layer(kc, vc, s, n - ns, base, bits, np.zeros(1, np.uint8), 0,
                                      meta16=meta16)
            nc = n - ns
            assert np.array_equal(o["k_words"][b, h][:nc * W], r["k_words"][0, 0][:nc * W])
            assert np.array_equal(o["v_words"][b, h][:nc * W], r["v_words"][0, 0][:nc * W])
            assert np.array_equal(o["k_meta"][b, h][:nc * 2], r["k_meta"][0, 0][:nc * 2])
            assert np.array_equal(o["v_meta"][b, h][:nc * 2], r["v_meta"][0, 0][:nc * 2])
            assert np.array_equal(o["k_deq"][b, h][toks], r["k_deq"][0, 0])
            assert np.array_equal(o["v_deq"][b, h][toks], r["v_deq"][0, 0])
            assert np.array_equal(o["k_att"][b, h][toks], r["k_att"][0, 0])


def test_zero_rate_is_the_plain_base(oracle):
    rng = np.random.default_rng(8)
    k = _bf16_bits(rng, (1, 2, 60, 128))
    v = _bf16_bits(rng, (1, 2, 60, 128))
    a = oracle.quantize_layer(k, v, 5, 40, 2, 4, np.array([0, 1], np.uint8), 0)
    b = oracle.quantize_layer(k, v, 5, 40, 2, 4, np.array([0, 1], np.uint8), 0, n_salient=0)
    for key in ("k_words", "k_meta", "v_words", "v_meta", "k_deq", "v_deq", "k_att", "kq", "vq"):
        assert np.array_equal(a[key], b[key])


def test_every_token_salient_is_bf16_attention(oracle):
    rng = np.random.default_rng(9)
    k = _bf16_bits(rng, (1, 2, 40, 128))
    v = _bf16_bits(rng, (1, 2, 40, 128))
    o = oracle.quantize_layer(k, v, 4, 30, 2, 2, np.array([0, 0], np.uint8), 0, n_salient=30)
    assert not o["kq"].any() and not o["vq"].any()
    assert np.array_equal(o["k_deq"], _f32(k)) and np.array_equal(o["v_deq"], _f32(v))


def test_unsupported_combinations_are_rejected(oracle):
    rng = np.random.default_rng(1)
    k = _bf16_bits(rng, (1, 2, 80, 128))
    v = _bf16_bits(rng, (1, 2, 80, 128))
    with pytest.raises(ValueError):  # KIVI-style groups
        oracle.quantize_layer(k, v, 4, 64, 1, 2, np.array([0, 1], np.uint8), 0, residual=0,
                              n_salient=2)


# --------------------------------------------------------------------------
# K-only protection (Sec. 4 keeps salient tokens whether or not a head is
# protected; a K-only protected head keeps its image keys BF16, so only its
# salient tokens' values are kept BF16 -- reading R15)
# --------------------------------------------------------------------------

def test_keys_only_hand_example(oracle):
    """One K-only protected head, 8 text + 64 image + 8 text tokens, 4 salient
    tokens (permille 50: ceil(3.2)).  Image keys are zero except tokens 3, 17,
    40, 41 (image-relative), whose channel 5 holds 6, 9, 7, 8: those four are
    the salient ones.  Their values stay BF16; image token 4 is the fourth
    coded value (slot 3), token 18 slot 16, token 42 slot 38."""
    T, s, n = 80, 8, 64
    k = np.zeros((1, 1, T, 128), np.int64)
    for i, x in ((3, 6), (17, 9), (40, 7), (41, 8)):
        k[0, 0, s + i, 5] = x
    k[0, 0, :s, :] = 50  # text keys are not ranked: only image tokens are candidates
    kb = _bf16_of_int(k)
    rng = np.random.default_rng(12)
    v = _bf16_bits(rng, (1, 1, T, 128))
    ns = oracle.salient_count(n, 50)
    assert ns == 4
    o = oracle.quantize_layer(kb, v, s, n, 2, 4, np.array([1], np.uint8), 1, n_salient=ns)
    assert list(o["salient"][0, 0]) == [3, 17, 40, 41]
    assert not o["kq"].any()                                   # every key BF16
    assert np.array_equal(o["k_deq"][0, 0], _f32(kb[0, 0]))
    for i in (3, 17, 40, 41):
        assert o["vq"][0, 0, s + i] == 0
        assert np.array_equal(o["v_deq"][0, 0, s + i], _f32(v[0, 0, s + i]))
    W = 16  # 4-bit words per 128-channel token
    for i, slot in ((0, 0), (4, 3), (18, 16), (42, 38), (63, 59)):
        assert o["vq"][0, 0, s + i] == 1
        codes, sc, z = oracle.quantize_group(_f32(v[0, 0, s + i]), 4)
        assert np.array_equal(o["v_words"][0, 0][slot * W:(slot + 1) * W], oracle.pack(codes, 4))
        assert o["v_meta"][0, 0][2 * slot] == sc and o["v_meta"][0, 0][2 * slot + 1] == z


@pytest.mark.parametrize("base,bits", [(2, 4), (2, 2), (0, 2), (2, 3)])
def test_keys_only_selection_and_compacted_values(oracle, base, bits):
    """Every head with coded values (quantized heads and K-only protected heads)
    ranks its image tokens by exact integer key norms; the salient tokens keep
    BF16 keys and values and the rest is the base on the compacted sequence
    (for a K-only protected head: values only, every key BF16)."""
    mask = np.array([0, 1, 0, 1], np.uint8)
    B, H, T, s, n = 2, 4, 150, 11, 128
    rng = np.random.default_rng(20 + bits)
    k = _bf16_of_int(rng.integers(-7, 8, (B, H, T, 128)))
    v = _bf16_bits(rng, (B, H, T, 128))
    ns = oracle.salient_count(n, 40)
    assert ns == 6
    o = oracle.quantize_layer(k, v, s, n, base, bits, mask, 1, n_salient=ns)
    W = 128 * bits // 32
    nc = n - ns
    for b in range(B):
        for h in range(H):
            norms = (_f32(k[b, h, s:s + n]).astype(np.int64) ** 2).sum(axis=1)
            order = sorted(range(n), key=lambda i: (-norms[i], i))
            sal = o["salient"][b, h]
            assert list(sal) == sorted(order[:ns])
            keep = np.setdiff1d(np.arange(n), sal)
            for i in sal:
                assert o["vq"][b, h, s + i] == 0 and o["kq"][b, h, s + i] == 0
                assert np.array_equal(o["v_deq"][b, h, s + i], _f32(v[b, h, s + i]))
                assert np.array_equal(o["k_deq"][b, h, s + i], _f32(k[b, h, s + i]))
            toks = np.concatenate([np.arange(s), s + keep, np.arange(s + n, T)])
            r = oracle.quantize_layer(k[b:b + 1, h:h + 1][:, :, toks], v[b:b + 1, h:h + 1][:, :, toks],
                                      s, nc, base, bits, mask[h:h + 1], 1)
            assert np.array_equal(o["v_words"][b, h][:nc * W], r["v_words"][0, 0][:nc * W])
            assert np.array_equal(o["v_meta"][b, h][:nc * 2], r["v_meta"][0, 0][:nc * 2])
            assert np.array_equal(o["v_deq"][b, h][toks], r["v_deq"][0, 0])
            assert np.array_equal(o["k_deq"][b, h][toks], r["k_deq"][0, 0])
            if mask[h]:
                assert not o["kq"][b, h].any()
                assert np.array_equal(o["k_deq"][b, h], _f32(k[b, h]))
            else:
                assert np.array_equal(o["k_words"][b, h][:nc * W], r["k_words"][0, 0][:nc * W])
                assert np.array_equal(o["k_meta"][b, h][:nc * 2], r["k_meta"][0, 0][:nc * 2])
                assert np.all(o["kq"][b, h, s + keep] == 1)


def test_keys_only_all_protected_matches_k_plus_v_values(oracle):
    """With every head K-only protected, the values (and their salient tokens)
    are exactly those of the quantized heads of a K+V-free mask: the selection
    depends on the keys only, never on the protection of the keys."""
    rng = np.random.default_rng(31)
    B, H, T, s, n = 1, 3, 90, 5, 70
    k = _bf16_bits(rng, (B, H, T, 128))
    v = _bf16_bits(rng, (B, H, T, 128))
    ns = oracle.salient_count(n, 20)
    a = oracle.quantize_layer(k, v, s, n, 2, 4, np.ones(H, np.uint8), 1, n_salient=ns)
    q = oracle.quantize_layer(k, v, s, n, 2, 4, np.zeros(H, np.uint8), 0, n_salient=ns)
    for key in ("salient", "v_words", "v_meta", "v_deq", "vq"):
        assert np.array_equal(a[key], q[key]), key
