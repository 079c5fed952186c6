"""GPU parity of the CUDA path against the CPU oracle, through the C ABI.

Packed codes, metadata (fp32 pairs, or binary16 pairs with 32-bit metadata)
and BF16 copies must be bit-identical; the fp32
reconstruction (hg_dequantize_kv) must be bit-identical; decode attention
must match the fp64 oracle within |g - r| <= 2e-3 + 1e-2 |r| element-wise.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_35800_gb300 as hg
from paper_2609_35800_gb300 import workloads as wl
from paper_2609_35800_gb300.runner import CacheRunner

from parity import (assert_close, attention_reference, bf16_rne, bits16, check_arena_layer,
                    oracle_layer)

pytestmark = pytest.mark.gpu

SIGMA = float(np.float32(1.0 / np.sqrt(128.0)))


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_35800_gb300 import build
    build.build()
    hg.library()


M, K, A = wl.BASE_MINMAX, wl.BASE_KIVI, wl.BASE_AKVQ

# name, layers, batch, q_heads, kv_heads, prefix, image, suffix, base, bits, keys_only, steps, protected, residual
CASES = [
    ("minmax2_gqa7", 2, 1, 28, 4, 32, 256, 32, M, 2, 0, 3, [(0, 1), (1, 3)], 32),
    ("minmax4_g2_b2", 1, 2, 4, 2, 10, 70, 5, M, 4, 0, 3, [(0, 0)], 32),
    ("minmax2_konly", 2, 2, 8, 4, 7, 200, 9, M, 2, 1, 2, [(0, 2), (1, 0), (1, 1)], 32),
    ("kivi2_konly_mha", 1, 2, 4, 4, 3, 100, 40, K, 2, 1, 3, [(0, 1)], 32),
    ("kivi4_residual_in_image", 1, 1, 8, 2, 5, 80, 10, K, 4, 0, 2, [(0, 1)], 32),
    ("kivi2_unaligned_start", 2, 1, 4, 4, 13, 130, 45, K, 2, 0, 2, [(1, 2)], 32),
    ("akvq4_g4_b3", 1, 3, 16, 4, 64, 333, 17, A, 4, 0, 3, [(0, 3)], 32),
    ("akvq2_konly", 1, 2, 8, 4, 20, 150, 30, A, 2, 1, 2, [(0, 0), (0, 2)], 32),
    ("no_image", 1, 1, 8, 2, 40, 0, 30, M, 2, 0, 2, [(0, 0)], 32),
    ("image_at_start_and_end", 1, 2, 8, 4, 0, 300, 0, M, 2, 0, 2, [(0, 2)], 32),
    ("all_protected", 1, 1, 8, 2, 16, 100, 16, A, 4, 0, 2, [(0, 0), (0, 1)], 32),
    ("none_protected", 1, 1, 8, 2, 16, 100, 16, K, 2, 0, 2, [], 0),
    ("g16", 1, 1, 32, 2, 16, 200, 16, M, 4, 0, 2, [(0, 1)], 32),
    ("long_multisplit", 1, 1, 28, 4, 50, 3000, 50, M, 2, 0, 2, [(0, 0)], 32),
]


def _workload(case, meta_bits=64, salient_permille=0):
    (name, L, B, Hq, H, pre, img, suf, base, bits, ko, steps, prot, R) = case
    return wl.custom(name, L, B, Hq, H, pre, img, suf, base, bits, ko, decode_steps=steps,
                     seed=7, protected=prot, residual=R, meta_bits=meta_bits,
                     salient_permille=salient_permille)


def _run_and_check(w, layer_batched=True, fused=False):
    runner = CacheRunner(w)
    kept = runner.quantize_all(keep=True)
    torch.cuda.synchronize()
    arena = runner.arena.cpu().numpy()
    outs = []
    for l, (k, v) in enumerate(kept):
        kb, vb = bits16(k), bits16(v)
        o = oracle_layer(runner, l, kb, vb)
        check_arena_layer(runner, l, kb, vb, o, arena=arena)
        outs.append(o)
    # decode steps (append + attention, or the fused step), compared after every step
    app_k = [[] for _ in range(w.layers)]
    app_v = [[] for _ in range(w.layers)]
    for step in range(w.decode_steps):
        k_new, v_new = wl.step_new_kv(w, step, "cuda")
        q = wl.step_query(w, step, "cuda")
        out = torch.empty_like(q)
        if fused:
            hg.hg_decode_step(runner.cache, 0, w.layers, q, k_new, v_new, out, SIGMA, runner.ws,
                              runner.ws_bytes)
        elif layer_batched:
            hg.hg_append_kv(runner.cache, 0, w.layers, k_new, v_new)
            hg.hg_decode_attention(runner.cache, 0, w.layers, q, out, SIGMA, runner.ws,
                                   runner.ws_bytes)
        else:
            hg.hg_append_kv(runner.cache, 0, w.layers, k_new, v_new)
            for l in range(w.layers):
                hg.hg_decode_attention(runner.cache, l, 1, q[l], out[l], SIGMA, runner.ws,
                                       runner.ws_bytes)
        torch.cuda.synchronize()
        kn, vn, qb, ob = bits16(k_new), bits16(v_new), bits16(q), bits16(out)
        for l in range(w.layers):
            app_k[l].append(kn[l])
            app_v[l].append(vn[l])
            ref = attention_reference(runner, outs[l], qb[l], app_k[l], app_v[l], SIGMA)
            assert_close(ob[l], ref, "%s layer %d step %d" % (w.name, l, step))
    return runner, kept, outs


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_quantize_and_decode_parity(case):
    _run_and_check(_workload(case))


def test_tiny_workload_parity():
    _run_and_check(wl.WORKLOADS["tiny"])


@pytest.mark.parametrize("case", [CASES[0], CASES[3], CASES[6]], ids=["minmax", "kivi", "akvq"])
def test_per_layer_launches(case):
    _run_and_check(_workload(case), layer_batched=False)


@pytest.mark.parametrize("case", [CASES[0], CASES[2], CASES[3], CASES[6], CASES[12], CASES[13]],
                         ids=["minmax", "minmax_konly", "kivi", "akvq", "g16", "long"])
def test_fused_decode_step(case):
    """hg_decode_step appends and attends in one launch: same attention as the
    oracle after every step, and the new tokens end up in the cache."""
    w = _workload(case)
    runner, kept, outs = _run_and_check(w, fused=True)
    assert hg.hg_cache_appended(runner.cache, 0) == w.decode_steps
    Tt = w.seq_len + w.decode_steps
    # every layer in one reconstruction launch
    k32 = torch.empty(w.layers, w.batch, w.kv_heads, Tt, 128, dtype=torch.float32, device="cuda")
    v32 = torch.empty_like(k32)
    hg.hg_dequantize_kv(runner.cache, 0, w.layers, k32, v32, True)
    torch.cuda.synchronize()
    for l in range(w.layers):
        for step in range(w.decode_steps):
            k_new, v_new = wl.step_new_kv(w, step, "cuda")
            assert np.array_equal(k32[l, :, :, w.seq_len + step].cpu().numpy(),
                                  k_new[l].float().cpu().numpy())
            assert np.array_equal(v32[l, :, :, w.seq_len + step].cpu().numpy(),
                                  v_new[l].float().cpu().numpy())


def test_decode_step_capacity_and_rollback():
    w = _workload(CASES[1])
    runner = CacheRunner(w)
    runner.quantize_all()
    q = wl.step_query(w, 0, "cuda")
    out = torch.empty_like(q)
    k_new, v_new = wl.step_new_kv(w, 0, "cuda")
    for _ in range(w.decode_steps):
        hg.hg_decode_step(runner.cache, 0, w.layers, q, k_new, v_new, out, SIGMA, runner.ws,
                          runner.ws_bytes)
    with pytest.raises(hg.HGError) as e:
        hg.hg_decode_step(runner.cache, 0, w.layers, q, k_new, v_new, out, SIGMA, runner.ws,
                          runner.ws_bytes)
    assert e.value.status == 5
    assert hg.hg_cache_appended(runner.cache, 0) == w.decode_steps


META16 = [CASES[i] for i in (0, 1, 2, 3, 4, 6, 7, 12, 13)]


@pytest.mark.parametrize("case", META16, ids=[c[0] for c in META16])
def test_meta16_quantize_and_decode_parity(case):
    """32-bit metadata (binary16 scale and zero): codes, metadata bits and
    attention against the oracle with the same storage model."""
    _run_and_check(_workload(case, meta_bits=32))


@pytest.mark.parametrize("case", [CASES[0], CASES[3], CASES[6]], ids=["minmax", "kivi", "akvq"])
def test_meta16_fused_decode_step(case):
    _run_and_check(_workload(case, meta_bits=32), fused=True)


# 3-bit codes (reading R16: a 2-bit low part and a bit-2 plane)
CASES3 = [
    ("minmax3_gqa7", 2, 1, 28, 4, 32, 256, 32, M, 3, 0, 2, [(0, 1), (1, 3)], 32),
    ("minmax3_konly_b2", 2, 2, 8, 4, 7, 200, 9, M, 3, 1, 2, [(0, 2), (1, 0), (1, 1)], 32),
    ("kivi3_konly_mha", 1, 2, 4, 4, 3, 100, 40, K, 3, 1, 2, [(0, 1)], 32),
    ("kivi3_unaligned", 2, 1, 4, 4, 13, 130, 45, K, 3, 0, 2, [(1, 2)], 32),
    ("akvq3_g4_b3", 1, 3, 16, 4, 64, 333, 17, A, 3, 0, 2, [(0, 3)], 32),
    ("akvq3_konly", 1, 2, 8, 4, 20, 150, 30, A, 3, 1, 2, [(0, 0), (0, 2)], 32),
    ("minmax3_g16", 1, 1, 32, 2, 16, 200, 16, M, 3, 0, 2, [(0, 1)], 32),
    ("minmax3_long", 1, 1, 28, 4, 50, 3000, 50, M, 3, 0, 2, [(0, 0)], 32),
]


@pytest.mark.parametrize("case", CASES3, ids=[c[0] for c in CASES3])
def test_three_bit_parity(case):
    _run_and_check(_workload(case))


@pytest.mark.parametrize("case", [CASES3[0], CASES3[2], CASES3[4]], ids=["minmax", "kivi", "akvq"])
def test_three_bit_fused_meta16_salient(case):
    """3-bit codes with the fused decode step, binary16 metadata, and (AKVQ)
    salient tokens."""
    _run_and_check(_workload(case, meta_bits=32), fused=True)
    if case[8] == A:
        _run_and_check(_workload(case, salient_permille=20), fused=True)


@pytest.mark.parametrize("case", [CASES3[1], CASES3[2], CASES3[3], CASES3[5]],
                         ids=["minmax_konly", "kivi_konly", "kivi", "akvq_konly"])
def test_three_bit_dequantize_bit_exact(case):
    _dequantize_bit_exact(_workload(case))


# AKVQ-style salient tokens (Sec. 4): (case, permille)
SALIENT = [
    (("akvq4_sal", 2, 2, 16, 4, 64, 333, 17, A, 4, 0, 3, [(0, 3), (1, 0)], 32), 20),
    (("akvq2_sal_unaligned", 1, 3, 8, 4, 13, 250, 30, A, 2, 0, 2, [(0, 1)], 32), 20),
    (("akvq2_sal_heavy", 1, 1, 28, 4, 20, 300, 10, A, 2, 0, 2, [(0, 0)], 32), 150),
    (("akvq4_sal_all", 1, 2, 8, 2, 5, 70, 9, A, 4, 0, 2, [], 32), 1000),
    (("akvq2_sal_g16", 1, 1, 32, 2, 16, 200, 16, A, 2, 0, 2, [(0, 1)], 32), 20),
    (("akvq2_sal_long", 1, 1, 28, 4, 50, 3000, 50, A, 2, 0, 2, [(0, 0)], 32), 20),
    # K-only protection: a protected head keeps its salient tokens' values BF16
    (("akvq4_konly_sal", 2, 2, 16, 4, 64, 333, 17, A, 4, 1, 3, [(0, 3), (1, 0), (1, 2)], 32), 20),
    (("akvq2_konly_sal_unaligned", 1, 3, 8, 4, 13, 250, 30, A, 2, 1, 2, [(0, 1)], 32), 40),
    (("akvq3_konly_sal", 1, 2, 8, 4, 20, 150, 30, A, 3, 1, 2, [(0, 0), (0, 2)], 32), 100),
    (("akvq4_konly_sal_all_protected", 1, 1, 8, 2, 5, 300, 9, A, 4, 1, 2, [(0, 0), (0, 1)], 32), 20),
]


@pytest.mark.parametrize("case,permille", SALIENT, ids=[c[0][0] for c in SALIENT])
def test_salient_quantize_and_decode_parity(case, permille):
    """Salient tokens: maps, BF16 rows, compacted codes bit-exact; attention
    within tolerance (plain and fused decode)."""
    _run_and_check(_workload(case, salient_permille=permille))
    _run_and_check(_workload(case, salient_permille=permille), fused=True)


def test_salient_ties_and_meta16():
    """Integer-valued keys give many equal norms: the selection must keep the
    lower token index on ties, exactly as the oracle; with binary16 metadata."""
    w = wl.custom("sal_ties", 1, 2, 8, 4, 7, 160, 9, A, 4, 0, decode_steps=1, seed=3,
                  protected=[(0, 2)], meta_bits=32, salient_permille=50)
    runner = CacheRunner(w)
    B, H, T = w.batch, w.kv_heads, w.seq_len
    gen = torch.Generator().manual_seed(21)
    k = torch.randint(-2, 3, (B, H, T, 128), generator=gen).float().to(torch.bfloat16)
    v = torch.randn((B, H, T, 128), generator=gen).to(torch.bfloat16)
    k, v = k.contiguous().cuda(), v.contiguous().cuda()
    hg.hg_quantize_kv(runner.cache, 0, [k], [v])
    torch.cuda.synchronize()
    kb, vb = bits16(k), bits16(v)
    o = oracle_layer(runner, 0, kb, vb)
    check_arena_layer(runner, 0, kb, vb, o)


@pytest.mark.parametrize("mode", ["all_equal", "one_salient", "overflow"])
def test_salient_select_extremes(mode):
    """The selection's edge cases against the oracle: every image key the same
    (all scores tie: the first ns tokens by index), a single salient token per
    head, and keys whose squared norm overflows to +inf (they rank above every
    finite score, ties among them to the lower index)."""
    permille = 1 if mode == "one_salient" else 20
    w = wl.custom("sal_x_" + mode, 1, 2, 8, 4, 7, 160, 9, A, 4, 0, decode_steps=1, seed=5,
                  protected=[(0, 2)], salient_permille=permille)
    runner = CacheRunner(w)
    B, H, T = w.batch, w.kv_heads, w.seq_len
    gen = torch.Generator().manual_seed(31)
    k = torch.randn((B, H, T, 128), generator=gen)
    v = torch.randn((B, H, T, 128), generator=gen)
    s0 = w.img_start
    if mode == "all_equal":
        k[:, :, s0:s0 + w.image] = k[:, :, s0:s0 + 1]
    elif mode == "overflow":
        ns = oracle.salient_count(w.image, permille)
        rows = torch.tensor([3, 17, 17 + 64, 150])[:ns - 1]  # fewer than ns, so all are taken
        k[:, :, s0 + rows, 5] = 1e20  # squared in binary32: +inf
    kb16 = k.to(torch.bfloat16).contiguous().cuda()
    vb16 = v.to(torch.bfloat16).contiguous().cuda()
    hg.hg_quantize_kv(runner.cache, 0, [kb16], [vb16])
    torch.cuda.synchronize()
    kb, vb = bits16(kb16), bits16(vb16)
    o = oracle_layer(runner, 0, kb, vb)
    check_arena_layer(runner, 0, kb, vb, o)


@pytest.mark.parametrize("meta_bits", [64, 32])
@pytest.mark.parametrize("case", [CASES[1], CASES[2], CASES[4], CASES[5], CASES[7]],
                         ids=["minmax4", "minmax2_konly", "kivi4", "kivi2", "akvq2"])
def test_dequantize_bit_exact(case, meta_bits):
    _dequantize_bit_exact(_workload(case, meta_bits))


@pytest.mark.parametrize("case,permille", [SALIENT[0], SALIENT[1], SALIENT[3], SALIENT[6], SALIENT[7],
                                          SALIENT[9]],
                         ids=["akvq4", "akvq2_unaligned", "all", "konly4", "konly2_unaligned",
                              "konly_all_protected"])
def test_salient_dequantize_bit_exact(case, permille):
    _dequantize_bit_exact(_workload(case, salient_permille=permille))


def _dequantize_bit_exact(w):
    runner = CacheRunner(w)
    kept = runner.quantize_all(keep=True)
    # append one step so the appended tail is reconstructed too
    k_new, v_new = wl.step_new_kv(w, 0, "cuda")
    hg.hg_append_kv(runner.cache, 0, w.layers, k_new, v_new)
    Tt = w.seq_len + 1
    # all layers in one launch (fp32 and BF16 outputs), and each layer alone (fp32)
    K32 = torch.empty(w.layers, w.batch, w.kv_heads, Tt, 128, dtype=torch.float32, device="cuda")
    V32 = torch.empty_like(K32)
    hg.hg_dequantize_kv(runner.cache, 0, w.layers, K32, V32, True)
    K16 = torch.empty(w.layers, w.batch, w.kv_heads, Tt, 128, dtype=torch.bfloat16, device="cuda")
    V16 = torch.empty_like(K16)
    hg.hg_dequantize_kv(runner.cache, 0, w.layers, K16, V16, False)
    for l, (k, v) in enumerate(kept):
        o = oracle_layer(runner, l, bits16(k), bits16(v))
        k32 = torch.empty(w.batch, w.kv_heads, Tt, 128, dtype=torch.float32, device="cuda")
        v32 = torch.empty_like(k32)
        hg.hg_dequantize_kv(runner.cache, l, 1, k32, v32, True)
        torch.cuda.synchronize()
        assert torch.equal(k32, K32[l]) and torch.equal(v32, V32[l])
        k16, v16 = K16[l], V16[l]
        kd = np.concatenate([o["k_deq"], (bits16(k_new[l]).astype(np.uint32) << 16)
                             .view(np.float32)[:, :, None]], axis=2)
        vd = np.concatenate([o["v_deq"], (bits16(v_new[l]).astype(np.uint32) << 16)
                             .view(np.float32)[:, :, None]], axis=2)
        assert np.array_equal(k32.cpu().numpy().view(np.uint32), kd.view(np.uint32))
        assert np.array_equal(v32.cpu().numpy().view(np.uint32), vd.view(np.uint32))
        assert np.array_equal(bits16(k16), bf16_rne(kd))
        assert np.array_equal(bits16(v16), bf16_rne(vd))


def test_quantize_is_idempotent_and_resets_appended():
    w = _workload(CASES[0])
    runner = CacheRunner(w)
    kept = runner.quantize_all(keep=True)
    runner.decode_step(0)
    assert hg.hg_cache_appended(runner.cache, 0) == 1
    a1 = runner.arena.clone()
    hg.hg_quantize_kv(runner.cache, 0, [k for k, _ in kept], [v for _, v in kept])
    torch.cuda.synchronize()
    assert hg.hg_cache_appended(runner.cache, 0) == 0
    # every prefill region is rewritten identically
    l = 0
    r = hg.hg_cache_head_regions(runner.cache, l, 0)
    span = slice(r.kq, r.kq + r.kq_bstride)
    assert torch.equal(a1[span], runner.arena[span])


def test_capacity_error_leaves_state():
    w = _workload(CASES[1])
    runner = CacheRunner(w)
    runner.quantize_all()
    for s in range(w.decode_steps):
        runner.decode_step(s)
    k_new, v_new = wl.step_new_kv(w, 0, "cuda")
    with pytest.raises(hg.HGError) as e:
        hg.hg_append_kv(runner.cache, 0, w.layers, k_new, v_new)
    assert e.value.status == 5
    assert hg.hg_cache_appended(runner.cache, 0) == w.decode_steps


@pytest.mark.parametrize("meta_bits", [64, 32])
@pytest.mark.parametrize("bits", [2, 3, 4])
def test_minmax_quantize_exact_ties(bits, meta_bits):
    """Vectors built so that (x - min) / scale lands exactly on half-integers:
    every such element must round half to even, as the oracle does (the
    kernel's fast multiply-by-reciprocal path has to hand these to the exact
    division rule)."""
    w = wl.custom("ties%d" % bits, 1, 2, 8, 4, 5, 96, 7, M, bits, 0, decode_steps=1, seed=3,
                  protected=[(0, 1)], residual=32, meta_bits=meta_bits)
    runner = CacheRunner(w)
    B, H, T = w.batch, w.kv_heads, w.seq_len
    gen = torch.Generator().manual_seed(11)
    L = (1 << bits) - 1
    # x = (g / 2 + m) * 2^e with g in [0, 2L]: min m 2^e and max (L + m) 2^e are
    # pinned, so scale = 2^e exactly and (x - min) / scale = g / 2 -- exact in BF16
    g = torch.randint(0, 2 * L + 1, (2, B, H, T, 128), generator=gen).float()
    g[..., 0] = 0.0
    g[..., 1] = 2.0 * L
    m = torch.randint(-8, 8, (2, B, H, T, 1), generator=gen).float()
    e = torch.randint(-6, 6, (2, B, H, T, 1), generator=gen).float()
    x = (g * 0.5 + m) * torch.pow(2.0, e)
    # a quarter of the vectors random instead (ordinary, tie-free values)
    rnd = torch.rand((2, B, H, T, 1), generator=gen) < 0.25
    x = torch.where(rnd, torch.randn((2, B, H, T, 128), generator=gen) * 3.0, x)
    xb = x.to(torch.bfloat16)
    assert torch.equal(xb[~rnd.expand_as(x)].float(), x[~rnd.expand_as(x)])  # exact in BF16
    k = xb[0].contiguous().cuda()
    v = xb[1].contiguous().cuda()
    hg.hg_quantize_kv(runner.cache, 0, [k], [v])
    torch.cuda.synchronize()
    kb, vb = bits16(k), bits16(v)
    o = oracle_layer(runner, 0, kb, vb)
    check_arena_layer(runner, 0, kb, vb, o)


@pytest.mark.parametrize("base,bits,lo,hi", [(M, 2, -1.0, 1.375), (M, 2, -1.0, 5.25), (M, 3, -0.3125, 2.75),
                                             (M, 3, -1.0, 1.375), (M, 4, 0.5, 7.5), (M, 4, 1.375, 9.5),
                                             (K, 2, -2.5, 0.8125), (K, 2, -2.5, 12.0), (K, 3, -1.0, 1.375),
                                             (K, 4, -0.3125, 7.5), (A, 4, -1.0, 1.375), (A, 2, -1.0, 5.25)],
                         ids=["minmax2", "minmax2n", "minmax3", "minmax3n", "minmax4", "minmax4n", "kivi2",
                              "kivi2n", "kivi3n", "kivi4n", "akvq4", "akvq2n"])
@pytest.mark.parametrize("meta_bits", [64, 32])
def test_quantize_near_ties(base, bits, lo, hi, meta_bits):
    """Every group (per-token rows, 32-channel value groups, 32-token key
    groups) holds the same minimum lo and maximum hi, and the other entries
    are the BF16 roundings of lo + (g + 1/2) * scale, scale = (hi - lo) /
    levels not a power of two: a few per cent of the elements land within
    2^-13 of a half-integer quotient, some of them exactly on it, which the
    kernel decides without a division and the oracle by the IEEE quotient.
    With binary16 metadata the codes are taken against the rounded pair.
    Arena bits must equal the oracle's."""
    w = wl.custom("near%d" % bits, 1, 2, 8, 4, 7, 160, 9, base, bits, 0, decode_steps=1, seed=4,
                  protected=[(0, 1)], residual=32, meta_bits=meta_bits)
    runner = CacheRunner(w)
    B, H, T = w.batch, w.kv_heads, w.seq_len
    gen = torch.Generator().manual_seed(23 + bits)
    L = (1 << bits) - 1
    scale = np.float32((np.float32(hi) - np.float32(lo)) / np.float32(L))
    g = torch.randint(0, L, (2, B, H, T, 128), generator=gen).double()
    x = float(lo) + (g + 0.5) * float(scale)
    x[..., 0::32] = lo   # every 32-channel group and every token row: lo and hi
    x[..., 1::32] = hi
    off = (torch.arange(T) - w.img_start) % 32  # every 32-token key group of the image
    x[:, :, :, off == 0, :] = lo
    x[:, :, :, off == 1, :] = hi
    xb = x.float().to(torch.bfloat16)
    assert float(xb.float().min()) == lo and float(xb.float().max()) == hi
    k = xb[0].contiguous().cuda()
    v = xb[1].contiguous().cuda()
    hg.hg_quantize_kv(runner.cache, 0, [k], [v])
    torch.cuda.synchronize()
    kb, vb = bits16(k), bits16(v)
    o = oracle_layer(runner, 0, kb, vb)
    check_arena_layer(runner, 0, kb, vb, o)


@pytest.mark.parametrize("base,bits", [(M, 2), (M, 4), (K, 2), (A, 4)],
                         ids=["minmax2", "minmax4", "kivi2", "akvq4"])
def test_meta16_extreme_ranges(base, bits):
    """Binary16 metadata at the edges of its range: magnitudes past 65504
    (the zero saturates), steps below the smallest subnormal (the stored scale
    is 0), and subnormal offsets whose rounded zero lies above the group
    minimum (codes clamp at 0 and at the top level).  Arena bits and the fp32 reconstruction
    must equal the oracle's."""
    w = wl.custom("x16", 1, 2, 8, 4, 5, 96, 7, base, bits, 0, decode_steps=1, seed=5,
                  protected=[(0, 1)], residual=32, meta_bits=32)
    runner = CacheRunner(w)
    B, H, T = w.batch, w.kv_heads, w.seq_len
    gen = torch.Generator().manual_seed(17)
    shape = (2, B, H, T, 128)
    kind = torch.randint(0, 5, (2, B, H, T, 1), generator=gen)
    z = torch.randn(shape, generator=gen)
    x = torch.where(kind == 0, z * 3e4 - 6e4, z)                       # past -65504
    x = torch.where(kind == 1, z * 2e4 + 7e4, x)                       # past +65504
    x = torch.where(kind == 2, z * 1e-8, x)                            # step below 2^-24
    # tiny offset: a BF16 minimum below 2^-14 rounds to a binary16 subnormal,
    # which can lie above it (BF16 values in the normal binary16 range convert exactly)
    x = torch.where(kind == 3, 1e-6 + torch.rand(shape, generator=gen) * 9e-6, x)
    xb = x.to(torch.bfloat16)
    k = xb[0].contiguous().cuda()
    v = xb[1].contiguous().cuda()
    hg.hg_quantize_kv(runner.cache, 0, [k], [v])
    k32 = torch.empty(B, H, T, 128, dtype=torch.float32, device="cuda")
    v32 = torch.empty_like(k32)
    hg.hg_dequantize_kv(runner.cache, 0, 1, k32, v32, True)
    torch.cuda.synchronize()
    kb, vb = bits16(k), bits16(v)
    o = oracle_layer(runner, 0, kb, vb)
    check_arena_layer(runner, 0, kb, vb, o)
    assert np.array_equal(k32.cpu().numpy().view(np.uint32), o["k_deq"].view(np.uint32))
    assert np.array_equal(v32.cpu().numpy().view(np.uint32), o["v_deq"].view(np.uint32))


def test_bounded_wait_gives_up_and_flags():
    """Failure detection without a fault: the decode kernel's tile wait, run on
    an mbarrier phase that nothing completes, returns after its bound and sets
    the timeout bit; on a completed phase it succeeds.  The context stays usable."""
    import time
    word = torch.zeros(4, dtype=torch.int32, device="cuda")
    t0 = time.time()
    hg.hg_check_bounded_wait(word, 200)  # at most 200 x 50 us
    torch.cuda.synchronize()
    assert time.time() - t0 < 30.0
    assert int(word[0].item()) == 3
    # the device still works: an ordinary decode afterwards is correct
    _run_and_check(_workload(CASES[1]))


def test_decode_step_reads_and_writes_pinned_host_memory():
    """The decode step's query, new K/V and output may live in pinned host
    memory (addressable from the device): the result is bit-identical to the
    same step on device buffers, and the new tokens land in the cache."""
    w = _workload(CASES[0])
    ra, rb = CacheRunner(w), CacheRunner(w)
    ra.quantize_all()
    rb.quantize_all()
    for step in range(w.decode_steps):
        k_new, v_new = wl.step_new_kv(w, step, "cuda")
        q = wl.step_query(w, step, "cuda")
        out = torch.empty_like(q)
        hg.hg_decode_step(ra.cache, 0, w.layers, q, k_new, v_new, out, SIGMA, ra.ws, ra.ws_bytes)
        hq, hk, hv = q.cpu().pin_memory(), k_new.cpu().pin_memory(), v_new.cpu().pin_memory()
        hout = torch.full(q.shape, float("nan"), dtype=q.dtype).pin_memory()
        hg.hg_decode_step(rb.cache, 0, w.layers, hq.data_ptr(), hk.data_ptr(), hv.data_ptr(),
                          hout.data_ptr(), SIGMA, rb.ws, rb.ws_bytes)
        torch.cuda.synchronize()
        assert torch.equal(hout.view(torch.int16), out.cpu().view(torch.int16)), "step %d" % step
