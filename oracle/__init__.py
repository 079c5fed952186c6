"""HeadGuard CPU oracle -- TEST INFRASTRUCTURE ONLY.

A thin numpy/ctypes wrapper over ``hg_oracle.c``: the plain C statement of
the mixed-precision KV-cache path (base quantizers, protection mask, bit
packing, Hadamard rotation, binary64 decode attention).  Only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may
import this package; the product library never does.

Every function cites the paper passage it follows (section numbers of
"HeadGuard: Selective Head Protection for Low-Bit VLM KV-Cache
Quantization"); the readings R1-R16 are stated in ``hg_oracle.c``.
"""
import ctypes
import os

import numpy as np

from . import build as _build

BASE_MINMAX = 0   # Sec. 1: per-token min-max RTN
BASE_KIVI = 1     # Sec. 4: KIVI-style per-channel keys / per-token values
BASE_AKVQ = 2     # Sec. 4: AKVQ-style Hadamard rotation + per-token RTN
D = 128

_lib = None


def lib():
    """Load (building first if needed) the oracle library."""
    global _lib
    if _lib is None:
        path = _build.build()
        L = ctypes.CDLL(path)
        P = ctypes.c_void_p
        i = ctypes.c_int
        L.hgo_bf16_to_f32.argtypes = [ctypes.c_uint16]
        L.hgo_bf16_to_f32.restype = ctypes.c_float
        L.hgo_quantize_group.argtypes = [P, i, i, i, P, P, P]
        L.hgo_quantize_group.restype = None
        L.hgo_quantize_group_m.argtypes = [P, i, i, i, i, P, P, P]
        L.hgo_quantize_group_m.restype = None
        L.hgo_f32_to_f16.argtypes = [ctypes.c_float]
        L.hgo_f32_to_f16.restype = ctypes.c_uint16
        L.hgo_f16_to_f32.argtypes = [ctypes.c_uint16]
        L.hgo_f16_to_f32.restype = ctypes.c_float
        L.hgo_dequant.argtypes = [ctypes.c_uint8, ctypes.c_float, ctypes.c_float]
        L.hgo_dequant.restype = ctypes.c_float
        L.hgo_pack.argtypes = [P, i, i, P]
        L.hgo_pack.restype = None
        L.hgo_unpack.argtypes = [P, i, i]
        L.hgo_unpack.restype = ctypes.c_uint8
        L.hgo_unpack_group.argtypes = [P, i, i, i]
        L.hgo_unpack_group.restype = ctypes.c_uint8
        L.hgo_plane_pos.argtypes = [i]
        L.hgo_plane_pos.restype = i
        L.hgo_fwht128.argtypes = [P]
        L.hgo_fwht128.restype = None
        L.hgo_fwht128_f64.argtypes = [P]
        L.hgo_fwht128_f64.restype = None
        L.hgo_quantized_count.argtypes = [i, i, i, i, i, i]
        L.hgo_quantized_count.restype = i
        L.hgo_quantize_head.argtypes = [P, P, i, i, i, i, i, i, i, i, i, i] + [P] * 9
        L.hgo_quantize_head.restype = i
        L.hgo_quantize_layer.argtypes = [P, P, i, i, i, i, i, i, i, P, i, i, i, i] + [P] * 9
        L.hgo_quantize_layer.restype = i
        L.hgo_quantize_layer_m.argtypes = [P, P, i, i, i, i, i, i, i, i, P, i, i, i, i] + [P] * 9
        L.hgo_quantize_layer_m.restype = i
        L.hgo_quantize_layer_s.argtypes = [P, P, i, i, i, i, i, i, i, i, P, i, i, i, i, i] + [P] * 10
        L.hgo_quantize_layer_s.restype = i
        L.hgo_key_norm2.argtypes = [P]
        L.hgo_key_norm2.restype = ctypes.c_float
        L.hgo_salient_count.argtypes = [i, i]
        L.hgo_salient_count.restype = i
        L.hgo_select_salient.argtypes = [P, i, i, P]
        L.hgo_select_salient.restype = None
        L.hgo_attention_layer.argtypes = [P, P, P, i, i, i, i, ctypes.c_double, P]
        L.hgo_attention_layer.restype = i
        L.hgo_image_bits_per_elem.argtypes = [i, i, i, ctypes.c_double, i]
        L.hgo_image_bits_per_elem.restype = ctypes.c_double
        _lib = L
    return _lib


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p) if a is not None else None


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


# --------------------------------------------------------------------------
# Elementwise helpers
# --------------------------------------------------------------------------

def bf16_bits_to_f32(bits):
    """Exact BF16 -> fp32 widening of uint16 bit patterns (vectorised)."""
    b = np.asarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def quantize_group(x, bits, meta16=False):
    """Sec. 1 group quantizer: (codes uint8[n], scale f32, zero f32).  With
    meta16 (Sec. 5.4 32-bit metadata, reading R13) scale and zero are the
    stored binary16 values and the codes are computed against them."""
    x = _c(x, np.float32)
    codes = np.zeros(x.size, np.uint8)
    sc = np.zeros(1, np.float32)
    ze = np.zeros(1, np.float32)
    if meta16:
        lib().hgo_quantize_group_m(_ptr(x), x.size, 1, bits, 1, _ptr(codes), _ptr(sc), _ptr(ze))
    else:
        lib().hgo_quantize_group(_ptr(x), x.size, 1, bits, _ptr(codes), _ptr(sc), _ptr(ze))
    return codes, np.float32(sc[0]), np.float32(ze[0])


def f32_to_f16_bits(x):
    """binary32 -> binary16 bits, round to nearest even, |x| >= 65504 saturating (R13)."""
    return np.uint16(lib().hgo_f32_to_f16(float(np.float32(x))))


def f16_bits_to_f32(h):
    return np.float32(lib().hgo_f16_to_f32(int(h)))


def dequant(code, scale, zero):
    """Sec. 4 reconstruction fl32(fl32(code*scale) + zero)."""
    return np.float32(lib().hgo_dequant(int(code), float(scale), float(zero)))


def pack(codes, bits):
    """Canonical packing (R16 for 3 bits: a 2-bit low part, then a bit-2 plane)."""
    codes = _c(codes, np.uint8)
    if bits == 3:
        assert codes.size % 32 == 0
        words = np.zeros(codes.size * 3 // 32, np.uint32)
    else:
        per = 32 // bits
        words = np.zeros((codes.size + per - 1) // per, np.uint32)
    lib().hgo_pack(_ptr(codes), codes.size, bits, _ptr(words))
    return words


def unpack(words, n, bits):
    words = _c(words, np.uint32)
    return np.array([lib().hgo_unpack_group(_ptr(words), n, e, bits) for e in range(n)], np.uint8)


def fwht128(x):
    """Sec. 4 AKVQ-style rotation (fp32, normalised, self-inverse)."""
    y = np.array(x, dtype=np.float32, copy=True)
    assert y.size == D
    lib().hgo_fwht128(_ptr(y))
    return y


def fwht128_f64(x):
    y = np.array(x, dtype=np.float64, copy=True)
    assert y.size == D
    lib().hgo_fwht128_f64(_ptr(y))
    return y


def quantized_count(T, s, n, base, group_tokens=32, residual=32):
    """Sec. 4 / reading R7: number of image tokens eligible for low precision."""
    return lib().hgo_quantized_count(T, s, n, base, group_tokens, residual)


def image_bits_per_elem(bits, meta_bits, frac_protected, keys_only, head_dim=D):
    """Sec. 5.4 storage model."""
    return lib().hgo_image_bits_per_elem(bits, meta_bits, head_dim, float(frac_protected),
                                         int(keys_only))


# --------------------------------------------------------------------------
# Layer-level quantization (Sec. 3 protection over a Sec. 4 base)
# --------------------------------------------------------------------------

def key_norm2(k_row_bits):
    """R15: squared norm of one BF16 key row, binary32 in the fixed order."""
    return np.float32(lib().hgo_key_norm2(_ptr(_c(k_row_bits, np.uint16))))


def salient_count(n, permille):
    """R15: salient tokens per head, ceil(n * permille / 1000)."""
    return lib().hgo_salient_count(int(n), int(permille))


def select_salient(score, ns):
    """R15: indices of the ns largest scores (ties to the lower index), ascending."""
    score = _c(score, np.float32)
    idx = np.zeros(max(ns, 1), np.int32)
    lib().hgo_select_salient(_ptr(score), score.size, int(ns), _ptr(idx))
    return idx[:ns]


def quantize_layer(k_bits, v_bits, s, n, base, bits, head_mask, keys_only,
                   group_tokens=32, group_channels=32, residual=32, want_att=True, meta16=False,
                   n_salient=0):
    """Quantize one layer.

    k_bits, v_bits: uint16 [B][H][T][128] BF16 bit patterns.
    head_mask: uint8 [H] (1 = protected).
    Returns a dict with per-(b,h) arrays:
      nq, kq, vq [B,H,T], k_words [B,H,...], k_meta, v_words, v_meta (shapes as
      documented in hg_oracle.c), k_deq, v_deq [B,H,T,128] fp32, k_att fp64.
    n_salient > 0 (R15): every head that is not protected K+V keeps that many
    image tokens' keys and values BF16 (indices in salient [B,H,n_salient]; a
    K-only protected head's image keys are BF16 anyway); their codes and
    metadata fill the first nq - n_salient token slots.
    """
    k_bits = _c(k_bits, np.uint16)
    v_bits = _c(v_bits, np.uint16)
    B, H, T, Dd = k_bits.shape
    assert Dd == D and v_bits.shape == k_bits.shape
    head_mask = _c(head_mask, np.uint8)
    assert head_mask.size == H
    nq = quantized_count(T, s, n, base, group_tokens, residual)
    kw = nq * D * bits // 32
    if base == BASE_KIVI:
        km = (nq // group_tokens) * D * 2
        vm = nq * (D // group_channels) * 2
    else:
        km = nq * 2
        vm = nq * 2
    out = dict(
        nq=nq,
        kq=np.zeros((B, H, T), np.uint8), vq=np.zeros((B, H, T), np.uint8),
        k_words=np.zeros((B, H, kw), np.uint32), k_meta=np.zeros((B, H, km), np.float32),
        v_words=np.zeros((B, H, kw), np.uint32), v_meta=np.zeros((B, H, vm), np.float32),
        k_deq=np.zeros((B, H, T, D), np.float32), v_deq=np.zeros((B, H, T, D), np.float32),
        k_att=np.zeros((B, H, T, D), np.float64) if want_att else None,
        salient=np.zeros((B, H, max(n_salient, 0)), np.int32), n_salient=n_salient,
    )
    rc = lib().hgo_quantize_layer_s(_ptr(k_bits), _ptr(v_bits), B, H, T, s, n, base, bits,
                                    int(meta16), _ptr(head_mask), int(keys_only), group_tokens,
                                    group_channels, residual, int(n_salient), _ptr(out["kq"]),
                                    _ptr(out["vq"]), _ptr(out["k_words"]), _ptr(out["k_meta"]),
                                    _ptr(out["v_words"]), _ptr(out["v_meta"]), _ptr(out["k_deq"]),
                                    _ptr(out["v_deq"]), _ptr(out["k_att"]),
                                    _ptr(out["salient"]) if n_salient > 0 else None)
    if rc < 0:
        raise ValueError("hgo_quantize_layer_s: unsupported salient configuration")
    return out


def attention_layer(q_bits, K, V, sigma):
    """Binary64 grouped-query decode attention (Sec. 4 simulated quantization).

    q_bits: uint16 [B][Hq][128]; K, V: float64 [B][H][Tt][128]; returns [B][Hq][128].
    """
    q_bits = _c(q_bits, np.uint16)
    K = _c(K, np.float64)
    V = _c(V, np.float64)
    B, Hq, _ = q_bits.shape
    _, H, Tt, _ = K.shape
    out = np.zeros((B, Hq, D), np.float64)
    rc = lib().hgo_attention_layer(_ptr(q_bits), _ptr(K), _ptr(V), B, Hq, H, Tt, float(sigma),
                                   _ptr(out))
    if rc != 0:
        raise ValueError("hgo_attention_layer failed (%d)" % rc)
    return out

