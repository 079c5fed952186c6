"""Host-only tests of the C ABI: the library loads, exports every declared entry
point, validates arguments before touching the GPU, and lays the arena out as
the storage model says.  No CUDA call is made here."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2609_35800_gb300 as hg
from paper_2609_35800_gb300 import build, workloads as wl
from paper_2609_35800_gb300.runner import config_of, shape_of

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return hg.library()


def _declared():
    txt = open(os.path.join(ROOT, "include", "headguard.h")).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(hg_[a-z0-9_]+)\s*\(", txt)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 14
    for n in names:
        assert hasattr(lib, n), n


def _shape(**kw):
    d = dict(batch=2, num_layers=3, num_kv_heads=4, num_q_heads=28, head_dim=128, seq_len=300,
             img_start=20, img_len=256, max_new_tokens=8)
    d.update(kw)
    return hg.Shape(**d)


def _cfg(**kw):
    d = dict(base=0, bits=2, keys_only=0, kivi_group_tokens=32, kivi_group_channels=32,
             kivi_residual=32)
    d.update(kw)
    return hg.QuantConfig(**d)


def _status(f, *a):
    return f(*a)


@pytest.mark.parametrize("shape_kw,cfg_kw,status", [
    (dict(head_dim=64), {}, 3),
    (dict(num_q_heads=30), {}, 1),
    (dict(img_start=100, img_len=256), {}, 1),
    (dict(num_kv_heads=65, num_q_heads=65), {}, 3),
    (dict(num_kv_heads=1, num_q_heads=17), {}, 3),
    (dict(seq_len=0, img_len=0, img_start=0), {}, 1),
    (dict(batch=0), {}, 1),
    ({}, dict(bits=5), 3),
    ({}, dict(bits=1), 3),
    ({}, dict(base=7), 1),
    ({}, dict(base=1, kivi_group_tokens=16), 3),
    ({}, dict(base=1, kivi_residual=-1), 1),
    ({}, dict(keys_only=2), 1),
    ({}, dict(meta_bits=16), 1),
    ({}, dict(meta_bits=48), 1),
    ({}, dict(base=2, salient_permille=-1), 1),
    ({}, dict(base=2, salient_permille=1001), 1),
    ({}, dict(base=0, salient_permille=20), 3),
    ({}, dict(base=1, salient_permille=20), 3),
    (dict(max_new_tokens=-1), {}, 1),
    (dict(img_start=-1), {}, 1),
    (dict(num_layers=0), {}, 1),
    (dict(img_len=-1), {}, 1),
    (dict(seq_len=1 << 28, img_start=0), {}, 3),          # token index range
    (dict(batch=20000), {}, 3),                            # batch x KV heads > grid.y
    ({}, dict(base=1, kivi_group_channels=16), 3),
    (dict(seq_len=60100, img_start=50, img_len=60000), dict(base=2, salient_permille=20), 3),
])
def test_layout_validation(lib, shape_kw, cfg_kw, status):
    mask = np.zeros((3, max(4, shape_kw.get("num_kv_heads", 4))), np.uint8)
    with pytest.raises(hg.HGError) as e:
        hg.hg_cache_layout(_shape(**shape_kw), _cfg(**cfg_kw), mask)
    assert e.value.status == status


def _fake_cache(w, arena_addr=1 << 40):
    mask = wl.protection_mask(w).numpy()
    sh, cf = shape_of(w), config_of(w)
    n = hg.hg_cache_layout(sh, cf, mask)
    return hg.hg_cache_create(sh, cf, mask, arena_addr, n), n, mask


def test_create_checks_arena(lib):
    w = wl.WORKLOADS["tiny"]
    mask = wl.protection_mask(w).numpy()
    sh, cf = shape_of(w), config_of(w)
    n = hg.hg_cache_layout(sh, cf, mask)
    with pytest.raises(hg.HGError) as e:
        hg.hg_cache_create(sh, cf, mask, 1 << 40, n - 1)
    assert e.value.status == 7
    with pytest.raises(hg.HGError) as e:
        hg.hg_cache_create(sh, cf, mask, (1 << 40) + 16, n)
    assert e.value.status == 2


ODD = {"odd_nq_minmax": wl.custom("odd", 3, 3, 16, 4, 64, 333, 17, wl.BASE_MINMAX, 4, 0),
       "odd_nq_konly": wl.custom("odd2", 2, 5, 8, 8, 7, 77, 3, wl.BASE_AKVQ, 2, 1),
       "kivi_odd_rows": wl.custom("odd3", 2, 3, 8, 8, 5, 131, 40, wl.BASE_KIVI, 2, 1),
       "meta16_minmax": wl.custom("m16a", 2, 3, 16, 4, 9, 333, 17, wl.BASE_MINMAX, 2, 0,
                                  meta_bits=32),
       "meta16_kivi_konly": wl.custom("m16b", 2, 3, 8, 8, 5, 131, 40, wl.BASE_KIVI, 4, 1,
                                      meta_bits=32),
       "three_bit_minmax": wl.custom("b3", 2, 3, 16, 4, 9, 333, 17, wl.BASE_MINMAX, 3, 0),
       "three_bit_kivi_konly": wl.custom("b3k", 2, 2, 8, 8, 5, 131, 40, wl.BASE_KIVI, 3, 1),
       "salient_akvq": wl.custom("sal", 3, 2, 16, 4, 9, 333, 17, wl.BASE_AKVQ, 4, 0,
                                 salient_permille=20),
       "salient_all": wl.custom("sal2", 2, 3, 8, 8, 5, 70, 9, wl.BASE_AKVQ, 2, 0,
                                salient_permille=1000),
       "salient_akvq_konly": wl.custom("salk", 3, 2, 16, 4, 9, 333, 17, wl.BASE_AKVQ, 4, 1,
                                       salient_permille=20),
       "salient_akvq3_konly": wl.custom("salk3", 2, 3, 8, 8, 5, 131, 40, wl.BASE_AKVQ, 3, 1,
                                        salient_permille=40)}


@pytest.mark.parametrize("name", list(wl.WORKLOADS) + list(ODD))
def test_regions_tile_the_arena_without_overlap(lib, name):
    w = wl.WORKLOADS[name] if name in wl.WORKLOADS else ODD[name]
    cache, n, mask = _fake_cache(w)
    base = 1 << 40
    spans = []
    W = 128 * w.bits // 8
    for l in range(w.layers):
        for h in range(w.kv_heads):
            r = hg.hg_cache_head_regions(cache, l, h)
            B = w.batch
            assert r.head_class == (0 if not mask[l, h] else (1 if w.keys_only else 2))
            spans.append((r.kb, B * r.kb_bstride))
            spans.append((r.vb, B * r.kb_bstride))
            assert r.kb_bstride == r.bf16_capacity * 256
            if r.kq != hg.NONE_OFFSET:
                assert r.kq_bstride == r.n_coded * W
                spans.append((r.kq, B * r.kq_bstride))
                spans.append((r.kqm, B * r.kqm_bstride))
            if r.vq != hg.NONE_OFFSET:
                spans.append((r.vq, B * r.vq_bstride))
                spans.append((r.vqm, B * r.vqm_bstride))
            if r.kimg != hg.NONE_OFFSET:
                spans.append((r.kimg, B * r.kimg_bstride))
            if r.sal != hg.NONE_OFFSET:
                assert r.n_salient > 0 and r.sal_bstride >= (r.nq + 31) // 32 * 8
                spans.append((r.sal, B * r.sal_bstride))
            for off in (r.kb, r.vb, r.kq, r.kqm, r.vq, r.vqm, r.kimg, r.sal):
                if off != hg.NONE_OFFSET:
                    assert off % 16 == 0
            for st in (r.kb_bstride, r.kq_bstride, r.kqm_bstride, r.vq_bstride, r.vqm_bstride,
                       r.kimg_bstride):
                assert st % 16 == 0
    spans = sorted(s for s in spans if s[1] > 0)
    for (a, la), (b, _) in zip(spans, spans[1:]):
        assert a + la <= b, (a, la, b)
    assert spans[-1][0] + spans[-1][1] <= n


def test_image_storage_matches_paper_storage_model(lib, oracle):
    # exactly 1/8 of the heads protected, 2-bit min-max, no text outside the image:
    # the arena's image bits/elem equals the Sec. 5.4 model with 64-bit metadata.
    for keys_only in (0, 1):
        w = wl.custom("st", 2, 1, 8, 8, 0, 64, 0, wl.BASE_MINMAX, 2, keys_only,
                      protected=[(0, 3), (1, 6)])
        cache, _, _ = _fake_cache(w)
        got = hg.hg_cache_image_bits_per_elem(cache)
        want = oracle.image_bits_per_elem(2, 64, 0.125, keys_only)
        assert got == pytest.approx(want, rel=1e-12)
    w = wl.custom("st", 1, 1, 8, 8, 0, 64, 0, wl.BASE_MINMAX, 2, 0, protected=[])
    cache, _, _ = _fake_cache(w)
    assert hg.hg_cache_image_bits_per_elem(cache) == pytest.approx(2.5)
    assert oracle.image_bits_per_elem(2, 64, 0.0, 0) == pytest.approx(2.5)


def test_meta16_storage_model(lib, oracle):
    # 32-bit metadata (binary16 scale and zero): 2-bit codes cost 2.25 bits per
    # image element (Sec. 5.4), and protection adds what the model says.
    w = wl.custom("st16", 1, 1, 8, 8, 0, 64, 0, wl.BASE_MINMAX, 2, 0, protected=[], meta_bits=32)
    cache, _, _ = _fake_cache(w)
    assert hg.hg_cache_image_bits_per_elem(cache) == pytest.approx(2.25)
    for keys_only in (0, 1):
        w = wl.custom("st16", 2, 1, 8, 8, 0, 64, 0, wl.BASE_MINMAX, 2, keys_only,
                      protected=[(0, 3), (1, 6)], meta_bits=32)
        cache, _, _ = _fake_cache(w)
        want = oracle.image_bits_per_elem(2, 32, 0.125, keys_only)
        assert hg.hg_cache_image_bits_per_elem(cache) == pytest.approx(want, rel=1e-12)


@pytest.mark.parametrize("base", [wl.BASE_MINMAX, wl.BASE_KIVI, wl.BASE_AKVQ])
def test_meta16_halves_metadata_regions(lib, base):
    # binary16 pairs: 4 bytes per group instead of 8; row strides stay 16-byte padded
    kw = dict(protected=[(0, 1)])
    w64 = wl.custom("m64", 1, 2, 8, 4, 16, 256, 8, base, 2, 0, **kw)
    w32 = wl.custom("m32", 1, 2, 8, 4, 16, 256, 8, base, 2, 0, meta_bits=32, **kw)
    c64, n64, _ = _fake_cache(w64)
    c32, n32, _ = _fake_cache(w32)
    assert n32 < n64
    r64 = hg.hg_cache_head_regions(c64, 0, 0)
    r32 = hg.hg_cache_head_regions(c32, 0, 0)
    assert r64.nq == r32.nq > 0
    groups_k = (r64.nq // 32) * 128 if base == wl.BASE_KIVI else r64.nq
    groups_v = r64.nq * (4 if base == wl.BASE_KIVI else 1)
    pad = lambda x: (x + 15) // 16 * 16
    assert (r64.kqm_bstride, r32.kqm_bstride) == (pad(8 * groups_k), pad(4 * groups_k))
    assert (r64.vqm_bstride, r32.vqm_bstride) == (pad(8 * groups_v), pad(4 * groups_v))


def test_salient_layout(lib):
    # AKVQ-style salient tokens (Sec. 4): quantized heads hold ceil(2% of n) image
    # tokens in BF16 and the rest coded; protected heads are unchanged
    w = wl.custom("s", 1, 2, 8, 4, 16, 1296, 8, wl.BASE_AKVQ, 2, 0, protected=[(0, 1)],
                  salient_permille=20)
    w0 = wl.custom("s0", 1, 2, 8, 4, 16, 1296, 8, wl.BASE_AKVQ, 2, 0, protected=[(0, 1)])
    c, _, _ = _fake_cache(w)
    c0, _, _ = _fake_cache(w0)
    for h in range(4):
        r, r0 = hg.hg_cache_head_regions(c, 0, h), hg.hg_cache_head_regions(c0, 0, h)
        if h == 1:
            assert (r.n_salient, r.n_coded, r.bf16_prefill) == (0, 0, r0.bf16_prefill)
            assert r.sal == hg.NONE_OFFSET
        else:
            assert (r.n_salient, r.n_coded) == (26, 1270)
            assert r.bf16_prefill == r0.bf16_prefill + 26
            assert r.bf16_capacity == r0.bf16_capacity + 26
            assert r.kq_bstride == 1270 * 32 and r.kqm_bstride == 1270 * 8
    # stored bits: 26 of 1296 image tokens of each quantized head in BF16
    got = hg.hg_cache_image_bits_per_elem(c)
    q = (1270 * (2 * 128 + 64) + 26 * 16 * 128) / (1296 * 128)
    want = (3 * q + 1 * 16) / 4
    assert got == pytest.approx(want, rel=1e-12)


def test_calls_validate_before_any_launch(lib):
    w = wl.custom("v", 2, 1, 8, 2, 8, 64, 8, wl.BASE_MINMAX, 2, 0, decode_steps=0,
                  protected=[(0, 0)])
    cache, n, _ = _fake_cache(w)
    base = 1 << 40
    # null / misaligned inputs
    with pytest.raises(hg.HGError) as e:
        hg.hg_quantize_kv(cache, 0, [0, 0], [base, base], stream=0)
    assert e.value.status == 1
    with pytest.raises(hg.HGError) as e:
        hg.hg_quantize_kv(cache, 0, [base + 8], [base], stream=0)
    assert e.value.status == 2
    with pytest.raises(hg.HGError) as e:
        hg.hg_quantize_kv(cache, 1, [base, base], [base, base], stream=0)  # layers 1..2 of 2
    assert e.value.status == 1
    # capacity 0: appending fails before launching
    with pytest.raises(hg.HGError) as e:
        hg.hg_append_kv(cache, 0, 1, base, base, stream=0)
    assert e.value.status == 5
    # workspace too small
    need = hg.hg_decode_workspace_size(cache, 2)
    assert need > 0
    with pytest.raises(hg.HGError) as e:
        hg.hg_decode_attention(cache, 0, 2, base, base, 0.0, base, need - 1, stream=0)
    assert e.value.status == 4
    with pytest.raises(hg.HGError) as e:
        hg.hg_decode_attention(cache, 0, 2, base, base, float("nan"), base, need, stream=0)
    assert e.value.status == 1
    with pytest.raises(hg.HGError) as e:
        hg.hg_dequantize_kv(cache, 2, 1, base, base, 1, stream=0)
    assert e.value.status == 1
    assert hg.hg_cache_appended(cache, 0) == 0
    assert hg.hg_cache_appended(cache, 5) == -1


def test_workspace_size_grows_with_layers(lib):
    w = wl.WORKLOADS["qwen25vl7b"]
    cache, _, _ = _fake_cache(w)
    one = hg.hg_decode_workspace_size(cache, 1)
    allw = hg.hg_decode_workspace_size(cache, w.layers)
    assert 0 < one < allw


def test_status_strings(lib):
    for s in range(8):
        assert isinstance(hg.hg_status_string(s), str) and hg.hg_status_string(s)


def test_salient_selection_size_limit(lib):
    # one score per image token in the selection kernel's shared memory: 40000
    # image tokens fit, 60000 do not (the case above)
    mask = np.zeros((3, 4), np.uint8)
    n = hg.hg_cache_layout(_shape(seq_len=40100, img_start=50, img_len=40000),
                           _cfg(base=2, salient_permille=20), mask)
    assert n > 0
