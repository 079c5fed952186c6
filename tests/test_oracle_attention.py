"""Pins of the oracle's binary64 decode attention (paper Sec. 4: attention over the
reconstructed cache) by closed forms, invariants and special cases."""
import math
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _bits(x):
    x = np.asarray(x, np.float32)
    u = x.view(np.uint32)
    return ((u.astype(np.uint64) + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def _f32(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32)


def test_zero_query_gives_mean_of_values(oracle):
    rng = np.random.default_rng(0)
    V = rng.standard_normal((1, 2, 9, 128))
    K = rng.standard_normal((1, 2, 9, 128))
    q = np.zeros((1, 4, 128), np.uint16)
    out = oracle.attention_layer(q, K, V, 0.0883883476)
    for qh in range(4):
        assert np.allclose(out[0, qh], V[0, qh // 2].mean(0), atol=1e-14)


def test_identical_keys_give_mean(oracle):
    rng = np.random.default_rng(1)
    V = rng.standard_normal((1, 1, 6, 128))
    K = np.repeat(rng.standard_normal((1, 1, 1, 128)), 6, axis=2)
    q = _bits(rng.standard_normal((1, 3, 128)))
    out = oracle.attention_layer(q, K, V, 0.1)
    for qh in range(3):
        assert np.allclose(out[0, qh], V[0, 0].mean(0), atol=1e-13)


def test_two_token_closed_form(oracle):
    # q = e_0, keys differ only in channel 0: scores sigma*a, sigma*b; the output
    # is the logistic mix sigmoid(sigma (a - b)) v1 + (1 - .) v2.
    q = np.zeros((1, 1, 128), np.float32)
    q[0, 0, 0] = 1.0
    K = np.zeros((1, 1, 2, 128))
    K[0, 0, 0, 0], K[0, 0, 1, 0] = 2.5, -1.0
    V = np.zeros((1, 1, 2, 128))
    V[0, 0, 0, :], V[0, 0, 1, :] = 1.0, 3.0
    sigma = 0.75
    out = oracle.attention_layer(_bits(q), K, V, sigma)
    w = 1.0 / (1.0 + math.exp(-sigma * (2.5 - -1.0)))
    assert np.allclose(out[0, 0], w * 1.0 + (1 - w) * 3.0, atol=1e-15)


def test_dominant_key_selects_its_value(oracle):
    rng = np.random.default_rng(2)
    K = rng.standard_normal((1, 1, 5, 128)) * 0.01
    K[0, 0, 3, :] = 50.0
    V = rng.standard_normal((1, 1, 5, 128))
    q = _bits(np.ones((1, 1, 128)))
    out = oracle.attention_layer(q, K, V, 1.0)
    assert np.allclose(out[0, 0], V[0, 0, 3], atol=1e-12)


def test_token_permutation_invariance(oracle):
    rng = np.random.default_rng(3)
    K = rng.standard_normal((2, 2, 17, 128))
    V = rng.standard_normal((2, 2, 17, 128))
    q = _bits(rng.standard_normal((2, 6, 128)))
    perm = rng.permutation(17)
    a = oracle.attention_layer(q, K, V, 0.09)
    b = oracle.attention_layer(q, K[:, :, perm], V[:, :, perm], 0.09)
    assert np.allclose(a, b, atol=1e-13)


def test_grouped_query_mapping(oracle):
    # KV head 0 values are all 1, KV head 1 values all 2: query heads 0,1 read
    # head 0 and 2,3 read head 1 (contiguous groups), whatever the scores.
    rng = np.random.default_rng(4)
    K = rng.standard_normal((1, 2, 8, 128))
    V = np.stack([np.full((8, 128), 1.0), np.full((8, 128), 2.0)])[None]
    q = _bits(rng.standard_normal((1, 4, 128)))
    out = oracle.attention_layer(q, K, V, 0.09)
    assert np.allclose(out[0, :, 0], [1, 1, 2, 2], atol=1e-14)


def test_softmax_weights_sum_to_one(oracle):
    # with V = 1 everywhere the output is exactly the sum of the weights
    rng = np.random.default_rng(5)
    K = rng.standard_normal((1, 1, 300, 128)) * 4
    V = np.ones((1, 1, 300, 128))
    q = _bits(rng.standard_normal((1, 2, 128)) * 3)
    out = oracle.attention_layer(q, K, V, 0.0883883476)
    assert np.allclose(out, 1.0, atol=1e-13)


def _storage_rows():
    rows = []
    with open(os.path.join(GOLDEN, "storage_model.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                name, frac, ko, printed = [p.strip() for p in line.split("|")]
                rows.append((name, float(frac), int(ko), float(printed)))
    return rows


@pytest.mark.parametrize("name,frac,keys_only,printed", _storage_rows())
def test_storage_model_matches_paper(oracle, name, frac, keys_only, printed):
    got = oracle.image_bits_per_elem(2, 32, frac, keys_only)
    assert round(got, 2) == printed


def test_storage_k_only_saving_about_22_percent(oracle):
    kv = oracle.image_bits_per_elem(2, 32, 0.125, 0)
    ko = oracle.image_bits_per_elem(2, 32, 0.125, 1)
    assert round(100 * (kv - ko) / kv) == 22


def _brute_attention(q, K, V, sigma):
    """Scalar double-precision decode attention written out term by term for tiny
    shapes: softmax over every token of sigma * <q, k_t>, then the weighted sum of
    the values; query head qh reads KV head qh // G."""
    B, Hq, D = len(q), len(q[0]), len(q[0][0])
    H, T = len(K[0]), len(K[0][0])
    G = Hq // H
    out = [[[0.0] * D for _ in range(Hq)] for _ in range(B)]
    for b in range(B):
        for qh in range(Hq):
            h = qh // G
            scores = []
            for t in range(T):
                acc = 0.0
                for d in range(D):
                    acc += q[b][qh][d] * K[b][h][t][d]
                scores.append(sigma * acc)
            top = max(scores)
            w = [math.exp(x - top) for x in scores]
            z = math.fsum(w)
            for d in range(D):
                out[b][qh][d] = math.fsum(w[t] * V[b][h][t][d] for t in range(T)) / z
    return out


@pytest.mark.parametrize("B,Hq,H,T,sigma,scale", [
    (1, 1, 1, 1, 0.0883883476, 1.0),    # one token: the output is its value
    (2, 4, 2, 3, 0.0883883476, 1.0),
    (1, 6, 2, 8, 0.2, 3.0),             # G = 3, sharp softmax
    (2, 2, 2, 5, 1.0, 0.5),             # MHA
    (1, 8, 1, 7, 0.05, 40.0),           # scores far beyond exp's range without the shift
])
def test_matches_brute_force_on_tiny_shapes(oracle, B, Hq, H, T, sigma, scale):
    rng = np.random.default_rng(100 + T * 7 + Hq)
    qb = _bits(rng.standard_normal((B, Hq, 128)) * scale)
    K = rng.standard_normal((B, H, T, 128)) * scale
    V = rng.standard_normal((B, H, T, 128))
    got = oracle.attention_layer(qb, K, V, sigma)
    want = np.array(_brute_attention(_f32(qb).astype(np.float64).tolist(), K.tolist(),
                                      V.tolist(), sigma))
    assert np.allclose(got, want, rtol=1e-12, atol=1e-13)
    if T == 1:
        for qh in range(Hq):
            assert np.allclose(got[:, qh], V[:, qh * H // Hq, 0], atol=1e-15)


def test_common_key_shift_leaves_the_output(oracle):
    # adding one vector u to every key of a head adds sigma * <q, u> to every
    # score of that head, which the softmax cancels
    rng = np.random.default_rng(11)
    K = rng.standard_normal((2, 2, 23, 128))
    V = rng.standard_normal((2, 2, 23, 128))
    q = _bits(rng.standard_normal((2, 6, 128)))
    u = rng.standard_normal((2, 2, 1, 128)) * 5
    a = oracle.attention_layer(q, K, V, 0.09)
    b = oracle.attention_layer(q, K + u, V, 0.09)
    assert np.allclose(a, b, atol=1e-12)


def test_affine_in_the_values(oracle):
    rng = np.random.default_rng(12)
    K = rng.standard_normal((1, 2, 19, 128))
    V = rng.standard_normal((1, 2, 19, 128))
    q = _bits(rng.standard_normal((1, 4, 128)))
    a = oracle.attention_layer(q, K, V, 0.1)
    b = oracle.attention_layer(q, K, 2.5 * V - 0.75, 0.1)
    assert np.allclose(b, 2.5 * a - 0.75, atol=1e-12)


def test_query_scale_equals_softmax_scale(oracle):
    # doubling q (exact in BF16) is the same as doubling sigma
    rng = np.random.default_rng(13)
    K = rng.standard_normal((1, 1, 31, 128))
    V = rng.standard_normal((1, 1, 31, 128))
    q = rng.standard_normal((1, 3, 128))
    a = oracle.attention_layer(_bits(2 * _f32(_bits(q))), K, V, 0.07)
    b = oracle.attention_layer(_bits(q), K, V, 0.14)
    assert np.allclose(a, b, atol=1e-13)


def test_replicated_heads_equal_grouped_heads(oracle):
    # G = 1 with each KV head copied to the query heads of its group equals the
    # grouped-query layout
    rng = np.random.default_rng(14)
    B, H, G, T = 2, 3, 4, 11
    K = rng.standard_normal((B, H, T, 128))
    V = rng.standard_normal((B, H, T, 128))
    q = _bits(rng.standard_normal((B, H * G, 128)))
    gqa = oracle.attention_layer(q, K, V, 0.09)
    mha = oracle.attention_layer(q, np.repeat(K, G, axis=1), np.repeat(V, G, axis=1), 0.09)
    assert np.array_equal(gqa, mha)
