"""The Python binding's own argument checks, on CPU: a tensor argument must be
dense and hold the bytes the call reads or writes through it, and live on a
CUDA device; the check fires before the library is entered, so no kernel can
be handed a buffer shorter than its extent.  Raw integer addresses pass through
to the library's own validation."""
import pytest
import torch

import paper_2609_35800_gb300 as hg
from paper_2609_35800_gb300 import build, workloads as wl
from paper_2609_35800_gb300.runner import config_of, shape_of

B, L, HQ, H, PRE, IMG, SUF = 2, 3, 8, 2, 8, 64, 8
T = PRE + IMG + SUF


@pytest.fixture(scope="module")
def cache():
    build.build()
    w = wl.custom("chk", L, B, HQ, H, PRE, IMG, SUF, wl.BASE_MINMAX, 2, 0, decode_steps=2,
                  protected=[(0, 0)])
    mask = wl.protection_mask(w).numpy()
    sh, cf = shape_of(w), config_of(w)
    n = hg.hg_cache_layout(sh, cf, mask)
    return hg.hg_cache_create(sh, cf, mask, 1 << 40, n)


def _bf16(*shape):
    return torch.zeros(shape, dtype=torch.bfloat16)


def _raises(fn, what):
    with pytest.raises(ValueError) as e:
        fn()
    assert what in str(e.value), str(e.value)


def test_quantize_inputs(cache):
    ok = _bf16(B, H, T, 128)
    _raises(lambda: hg.hg_quantize_kv(cache, 0, [ok], [ok]), "must be a CUDA tensor")
    _raises(lambda: hg.hg_quantize_kv(cache, 0, [_bf16(B, H, T - 1, 128)], [ok]), "k[0] holds")
    _raises(lambda: hg.hg_quantize_kv(cache, 0, [ok, ok], [ok, _bf16(B, H, T, 127)]), "v[1] holds")
    _raises(lambda: hg.hg_quantize_kv(cache, 0, [_bf16(B, H, 128, T).transpose(2, 3)], [ok]),
            "contiguous")
    _raises(lambda: hg.hg_quantize_kv(cache, 0, [ok, ok], [ok]), "2 key and 1 value")


def test_decode_inputs(cache):
    q, kv = _bf16(L, B, HQ, 128), _bf16(L, B, H, 128)
    ws = torch.zeros(hg.hg_decode_workspace_size(cache, L), dtype=torch.uint8)
    _raises(lambda: hg.hg_decode_step(cache, 0, L, q, kv, kv, q, 0.0, ws), "must be a CUDA tensor")
    _raises(lambda: hg.hg_decode_step(cache, 0, L, q[:2], kv, kv, q, 0.0, ws), "q holds")
    _raises(lambda: hg.hg_decode_step(cache, 0, L, q, kv[:1], kv, q, 0.0, ws), "k_new holds")
    _raises(lambda: hg.hg_decode_step(cache, 0, L, q, kv, kv, _bf16(L, B, H, 128), 0.0, ws),
            "out holds")
    _raises(lambda: hg.hg_decode_step(cache, 0, L, q, kv, kv, q, 0.0, ws, ws.numel() + 1),
            "workspace holds")
    # one layer of a multi-layer buffer is enough for a one-layer call
    _raises(lambda: hg.hg_decode_attention(cache, 1, 1, q[1], q[1], 0.0, ws), "must be a CUDA")
    _raises(lambda: hg.hg_decode_attention(cache, 0, 2, q[1], q, 0.0, ws), "q holds")
    _raises(lambda: hg.hg_decode_attention_noalloc(cache, 0, L, q, q[:1], 0.0), "out holds")
    _raises(lambda: hg.hg_append_kv(cache, 0, L, kv, kv[:2]), "v_new holds")


def test_dequantize_outputs(cache):
    # fp32 output needs 4 bytes per entry; nothing appended yet: T tokens
    _raises(lambda: hg.hg_dequantize_kv(cache, 0, 1, _bf16(B, H, T, 128), _bf16(B, H, T, 128), True),
            "k_out holds")
    k32 = torch.zeros((B, H, T, 128), dtype=torch.float32)
    _raises(lambda: hg.hg_dequantize_kv(cache, 0, 1, k32, k32, True), "must be a CUDA tensor")
    _raises(lambda: hg.hg_dequantize_kv(cache, 0, 1, _bf16(B, H, T, 128), _bf16(B, H, T, 128), False),
            "must be a CUDA tensor")


def test_workspace_and_arena(cache):
    small = torch.zeros(8, dtype=torch.uint8)
    _raises(lambda: hg.hg_workspace_clear(small, 16), "workspace holds")
    _raises(lambda: hg.hg_workspace_clear(small), "must be a CUDA tensor")
    _raises(lambda: hg.hg_workspace_status(torch.zeros(3, dtype=torch.uint8)), "workspace holds")
    _raises(lambda: hg.hg_check_bounded_wait(torch.zeros(1, dtype=torch.int16), 10), "word holds")
    sh, cf = cache.shape, cache.config
    n = hg.hg_cache_layout(sh, cf, cache.mask)
    _raises(lambda: hg.hg_cache_create(sh, cf, cache.mask, torch.zeros(16, dtype=torch.uint8), n),
            "arena holds")


def test_raw_addresses_reach_the_library(cache):
    # ints are not checked here: the library's own validation answers
    with pytest.raises(hg.HGError) as e:
        hg.hg_quantize_kv(cache, 0, [(1 << 40) + 8], [1 << 40], stream=0)
    assert e.value.status == 2


@pytest.mark.parametrize("name", ["tiny", "qwen25vl7b"])
def test_generated_inputs_pass_the_extent_checks(name):
    """The inputs the runner, the tests and the bench hand to the binding (the
    workload generators' shapes, whole or one layer at a time) pass every
    extent check: on CPU the only complaint left is the device."""
    build.build()
    w = wl.WORKLOADS[name]
    mask = wl.protection_mask(w).numpy()
    sh, cf = shape_of(w), config_of(w)
    c = hg.hg_cache_create(sh, cf, mask, 1 << 40, hg.hg_cache_layout(sh, cf, mask))
    k, v = wl.layer_kv(w, 0, "cpu")
    q = wl.step_query(w, 0, "cpu")
    kn, vn = wl.step_new_kv(w, 0, "cpu")
    out = torch.empty_like(q)
    ws = torch.zeros(hg.hg_decode_workspace_size(c, w.layers), dtype=torch.uint8)
    k32 = torch.empty(w.batch, w.kv_heads, w.seq_len, 128, dtype=torch.float32)
    cuda = "must be a CUDA tensor"
    _raises(lambda: hg.hg_quantize_kv(c, 0, [k] * w.layers, [v] * w.layers), cuda)
    _raises(lambda: hg.hg_append_kv(c, 0, w.layers, kn, vn), cuda)
    _raises(lambda: hg.hg_decode_attention(c, 0, w.layers, q, out, 0.0, ws), cuda)
    _raises(lambda: hg.hg_decode_step(c, 0, w.layers, q, kn, vn, out, 0.0, ws), cuda)
    _raises(lambda: hg.hg_decode_attention_noalloc(c, 0, w.layers, q, out, 0.0), cuda)
    last = w.layers - 1
    _raises(lambda: hg.hg_decode_step(c, last, 1, q[last], kn[last], vn[last], out[last], 0.0, ws),
            cuda)
    _raises(lambda: hg.hg_dequantize_kv(c, 0, 1, k32, k32, True), cuda)
    _raises(lambda: hg.hg_dequantize_kv(c, 0, 1, k, v, False), cuda)
    _raises(lambda: hg.hg_workspace_clear(ws), cuda)
