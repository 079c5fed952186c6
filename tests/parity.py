"""Parity helpers: compare the library's arena, reconstruction and attention with
the CPU oracle on the same seeded inputs (test infrastructure)."""
import numpy as np
import torch

import oracle
import paper_2609_35800_gb300 as hg

ATOL, RTOL = 2e-3, 1e-2   # attention tolerance (allclose form) on BF16 outputs


def bits16(t):
    """BF16 tensor -> host uint16 numpy bit patterns."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def f32_from_bits(b):
    return (b.astype(np.uint32) << 16).view(np.float32)


def bf16_rne(x):
    """fp32 -> BF16 bits, round to nearest even (numpy, independent of the GPU)."""
    u = np.ascontiguousarray(x, np.float32).view(np.uint32).astype(np.uint64)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def n_salient(w):
    """Salient tokens per quantized head (Sec. 4, reading R15) of a workload."""
    return oracle.salient_count(w.image, w.salient_permille) if w.salient_permille else 0


def oracle_layer(runner, layer, k_bits, v_bits):
    w = runner.w
    return oracle.quantize_layer(k_bits, v_bits, w.img_start, w.image, w.base, w.bits,
                                 runner.mask[layer], int(w.keys_only), w.kivi_group_tokens,
                                 w.kivi_group_channels, w.kivi_residual,
                                 meta16=w.meta_bits == 32, n_salient=n_salient(w))


def _slice(arena, off, nbytes, dtype):
    return arena[off: off + nbytes].view(dtype)


def _meta_words(meta, meta16):
    """Expected arena words of a metadata array: fp32 pairs as stored, or with
    32-bit metadata the binary16 bits of each value (scale in the low half)."""
    if meta16:
        h = meta.astype(np.float16)  # exact: the oracle's values are binary16 values
        assert np.array_equal(h.astype(np.float32).view(np.uint32), meta.view(np.uint32))
        return h.view(np.uint16).view(np.uint32)
    return meta.view(np.uint32)


def check_arena_layer(runner, layer, k_bits, v_bits, o, arena=None, heads=None, rows=None,
                      local=False):
    """Bit-exact comparison of every region of one layer (or the given heads / rows).

    local: k_bits, v_bits and the oracle output o hold only the given rows and
    heads (index [i][j] for rows[i], heads[j]), and the arena is read region
    by region from the device (caches too large to copy whole)."""
    w = runner.w
    m16 = w.meta_bits == 32
    if local:
        def rd(off, nbytes, dtype):
            return runner.arena[off: off + nbytes].cpu().numpy().view(dtype)
    else:
        if arena is None:
            arena = runner.arena.cpu().numpy()

        def rd(off, nbytes, dtype):
            return _slice(arena, off, nbytes, dtype)
    B, H, T = w.batch, w.kv_heads, w.seq_len
    s, nq = w.img_start, o["nq"]
    W = 128 * w.bits // 32
    heads = range(H) if heads is None else heads
    rows = range(B) if rows is None else rows
    ns = o["n_salient"]
    for hi, h in enumerate(heads):
        r = hg.hg_cache_head_regions(runner.cache, layer, h)
        assert r.nq == nq
        cls = r.head_class
        assert r.n_salient == (0 if cls == hg.HG_HEAD_PROTECTED else ns)
        nc = 0 if cls == hg.HG_HEAD_PROTECTED else nq - r.n_salient
        assert r.n_coded == nc
        for bi, b in enumerate(rows):
            ob, oh = (bi, hi) if local else (b, h)  # oracle / input index of (b, h)
            if cls == hg.HG_HEAD_PROTECTED:
                toks = np.arange(T)
            elif r.n_salient:
                # leading text, salient image tokens in order, trailing text
                sal = o["salient"][ob, oh]
                toks = np.concatenate([np.arange(0, s), s + sal, np.arange(s + nq, T)])
                nblk = (nq + 31) // 32
                words = rd(r.sal + b * r.sal_bstride, nblk * 8, np.uint32)
                want = np.zeros(nblk, np.uint32)
                for i in sal:
                    want[i >> 5] |= np.uint32(1 << (i & 31))
                ranks = np.concatenate([[0], np.cumsum([bin(int(x)).count("1") for x in want])[:-1]])
                assert np.array_equal(words[:nblk], want), (layer, h, b, "salient bits")
                assert np.array_equal(words[nblk:].view(np.int32), ranks), (layer, h, b, "ranks")
            else:
                toks = np.concatenate([np.arange(0, s), np.arange(s + nq, T)])
            assert r.bf16_prefill == toks.size
            kb = rd(r.kb + b * r.kb_bstride, toks.size * 256, np.uint16).reshape(-1, 128)
            vb = rd(r.vb + b * r.kb_bstride, toks.size * 256, np.uint16).reshape(-1, 128)
            assert np.array_equal(kb, k_bits[ob, oh, toks]), (layer, h, b, "kb")
            assert np.array_equal(vb, v_bits[ob, oh, toks]), (layer, h, b, "vb")
            kmeta_n = o["k_meta"][ob, oh].size if w.base == 1 else 2 * nc
            vmeta_n = o["v_meta"][ob, oh].size * nc // max(nq, 1)
            if cls == hg.HG_HEAD_QUANTIZED and nc:
                kw = rd(r.kq + b * r.kq_bstride, nc * W * 4, np.uint32)
                ek = _meta_words(o["k_meta"][ob, oh][:kmeta_n], m16)
                km = rd(r.kqm + b * r.kqm_bstride, ek.nbytes, np.uint32)
                assert np.array_equal(kw, o["k_words"][ob, oh][:nc * W]), (layer, h, b, "kq")
                assert np.array_equal(km, ek), (layer, h, b, "kqm")
            if cls != hg.HG_HEAD_PROTECTED and nc:
                vw = rd(r.vq + b * r.vq_bstride, nc * W * 4, np.uint32)
                ev = _meta_words(o["v_meta"][ob, oh][:vmeta_n], m16)
                vm = rd(r.vqm + b * r.vqm_bstride, ev.nbytes, np.uint32)
                assert np.array_equal(vw, o["v_words"][ob, oh][:nc * W]), (layer, h, b, "vq")
                assert np.array_equal(vm, ev), (layer, h, b, "vqm")
            if cls == hg.HG_HEAD_KEYS_ONLY and nc:
                # image keys of the coded tokens (the salient ones are in kb), compacted
                coded = np.setdiff1d(np.arange(nq), o["salient"][ob, oh]) if r.n_salient else np.arange(nq)
                ki = rd(r.kimg + b * r.kimg_bstride, nc * 256, np.uint16).reshape(-1, 128)
                assert np.array_equal(ki, k_bits[ob, oh, s + coded]), (layer, h, b, "kimg")


def attention_reference(runner, o, q_bits, appended_k, appended_v, sigma):
    """fp64 oracle attention of one layer over the reconstruction + appended tokens.

    appended_k/v: list of uint16 [B][H][128] (one per appended step)."""
    K = o["k_att"]
    V = o["v_deq"].astype(np.float64)
    if appended_k:
        ak = np.stack([f32_from_bits(a) for a in appended_k], axis=2).astype(np.float64)
        av = np.stack([f32_from_bits(a) for a in appended_v], axis=2).astype(np.float64)
        K = np.concatenate([K, ak], axis=2)
        V = np.concatenate([V, av], axis=2)
    return oracle.attention_layer(q_bits, K, V, sigma)


def assert_close(got_bf16_bits, ref, where=""):
    g = f32_from_bits(got_bf16_bits).astype(np.float64)
    err = np.abs(g - ref)
    bad = err > ATOL + RTOL * np.abs(ref)
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError("%s: %d / %d outside tolerance; first at %s got %r ref %r "
                             "(max abs err %.3g)" % (where, bad.sum(), bad.size, tuple(i),
                                                     g[tuple(i)], ref[tuple(i)], err.max()))
    return float(err.max())


def layer_block(runner, layer):
    """Host copy of one layer's block of the arena: (numpy bytes, base offset)."""
    w = runner.w
    lo, hi = None, 0
    for h in range(w.kv_heads):
        r = hg.hg_cache_head_regions(runner.cache, layer, h)
        for off, stride in ((r.kb, r.kb_bstride), (r.vb, r.kb_bstride), (r.kq, r.kq_bstride),
                            (r.kqm, r.kqm_bstride), (r.vq, r.vq_bstride), (r.vqm, r.vqm_bstride),
                            (r.kimg, r.kimg_bstride), (r.sal, r.sal_bstride)):
            if off == hg.NONE_OFFSET:
                continue
            lo = off if lo is None else min(lo, off)
            hi = max(hi, off + w.batch * stride)
    return runner.arena[lo:hi].cpu().numpy(), lo


def check_arena_layer_blocks(runner, layer, k_bits, v_bits, o, block=None):
    """Bit-exact comparison of every region of one layer, all batch rows of a
    head at once (caches without salient tokens).  k_bits, v_bits: uint16
    [B][H][T][128]; o: the oracle's quantize_layer output for the same layer."""
    w = runner.w
    assert not o["n_salient"]
    m16 = w.meta_bits == 32
    arena, base = block if block is not None else layer_block(runner, layer)
    B, H, T = w.batch, w.kv_heads, w.seq_len
    s, nq = w.img_start, o["nq"]
    W = 128 * w.bits // 32

    def rows(off, stride, n, dtype):
        a = arena[off - base: off - base + B * stride].reshape(B, stride)
        return a[:, :n * np.dtype(dtype).itemsize].view(dtype)

    for h in range(H):
        r = hg.hg_cache_head_regions(runner.cache, layer, h)
        cls = r.head_class
        assert r.nq == nq and r.n_salient == 0
        toks = np.arange(T) if cls == hg.HG_HEAD_PROTECTED else np.concatenate([np.arange(s), np.arange(s + nq, T)])
        assert r.bf16_prefill == toks.size
        kb = rows(r.kb, r.kb_bstride, toks.size * 128, np.uint16)
        vb = rows(r.vb, r.kb_bstride, toks.size * 128, np.uint16)
        assert np.array_equal(kb, k_bits[:, h][:, toks].reshape(B, -1)), (layer, h, "kb")
        assert np.array_equal(vb, v_bits[:, h][:, toks].reshape(B, -1)), (layer, h, "vb")
        if cls == hg.HG_HEAD_PROTECTED or not nq:
            continue
        if cls == hg.HG_HEAD_QUANTIZED:
            kw = rows(r.kq, r.kq_bstride, nq * W, np.uint32)
            assert np.array_equal(kw, o["k_words"][:, h, :nq * W]), (layer, h, "kq")
            ek = _meta_words(o["k_meta"][:, h], m16)
            km = rows(r.kqm, r.kqm_bstride, ek.shape[1], np.uint32)
            assert np.array_equal(km, ek), (layer, h, "kqm")
        else:
            ki = rows(r.kimg, r.kimg_bstride, nq * 128, np.uint16)
            assert np.array_equal(ki, k_bits[:, h, s:s + nq].reshape(B, -1)), (layer, h, "kimg")
        vw = rows(r.vq, r.vq_bstride, nq * W, np.uint32)
        assert np.array_equal(vw, o["v_words"][:, h, :nq * W]), (layer, h, "vq")
        ev = _meta_words(o["v_meta"][:, h], m16)
        vm = rows(r.vqm, r.vqm_bstride, ev.shape[1], np.uint32)
        assert np.array_equal(vm, ev), (layer, h, "vqm")
