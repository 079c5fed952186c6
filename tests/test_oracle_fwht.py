"""Pins of the oracle's Hadamard-128 rotation (paper Sec. 4, AKVQ-style base).

The reference is the Sylvester-ordered Hadamard matrix built by
scipy.linalg.hadamard (textbook construction), scaled by 1/sqrt(128).
"""
import numpy as np
import pytest
from scipy.linalg import hadamard

H = hadamard(128).astype(np.float64) / np.sqrt(128.0)


def test_matrix_is_orthonormal_and_symmetric():
    assert np.allclose(H @ H.T, np.eye(128), atol=1e-14)
    assert np.array_equal(H, H.T)


def test_unit_vectors(oracle):
    c = np.float32(1.0 / np.sqrt(128.0))
    e0 = np.zeros(128, np.float32)
    e0[0] = 1
    assert np.all(oracle.fwht128(e0) == c)
    e1 = np.zeros(128, np.float32)
    e1[1] = 1
    expect = np.where(np.arange(128) % 2 == 0, c, -c).astype(np.float32)
    assert np.array_equal(oracle.fwht128(e1), expect)
    # column j of H is the transform of e_j
    for j in (2, 5, 64, 127):
        e = np.zeros(128, np.float32)
        e[j] = 1
        assert np.array_equal(oracle.fwht128(e), H[:, j].astype(np.float32))


@pytest.mark.parametrize("seed", range(6))
def test_matches_dense_product(oracle, seed):
    rng = np.random.default_rng(seed)
    x = (rng.standard_normal(128) * (8 if seed % 2 else 1)).astype(np.float32)
    ref = H @ x.astype(np.float64)
    got32 = oracle.fwht128(x).astype(np.float64)
    assert np.max(np.abs(got32 - ref)) <= 1e-6 * np.linalg.norm(x) * 4
    got64 = oracle.fwht128_f64(x.astype(np.float64))
    assert np.allclose(got64, ref, rtol=0, atol=1e-13 * np.linalg.norm(x))


def test_involution_and_norm(oracle):
    rng = np.random.default_rng(7)
    x = rng.standard_normal(128).astype(np.float32)
    y = oracle.fwht128(x)
    assert abs(np.linalg.norm(y.astype(np.float64)) - np.linalg.norm(x.astype(np.float64))) < 1e-5
    assert np.allclose(oracle.fwht128(y), x, atol=2e-6)
