"""Parity at the benchmark's full cache shapes, in the launch configuration
bench.py times: one quantize call over all layers, then fused decode steps
(append + attention over all layers, one launch each).

- Qwen2.5-VL-7B shape (the one the benchmark times): the whole arena of every
  layer bit for bit against the oracle, and the attention output of every
  layer, batch row and query head after every one of the 32 decode steps
  within the tolerance of the parity tests.
- LLaVA-NeXT-7B, InternVL2.5-8B and Qwen2.5-VL-72B shapes: every layer's arena
  bit for bit (layer by layer through device-to-host copies of its block),
  and attention on a seeded sample of 4 layers x 4 batch rows x every query
  head after the first and the last decode step.
- Options of the later rows (salient tokens, 3-bit codes, binary16 metadata)
  at full size: sampled (layer, row, head) triples, arena and attention.
"""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from paper_2609_35800_gb300 import workloads as wl
from paper_2609_35800_gb300.runner import CacheRunner

from parity import (assert_close, bits16, check_arena_layer, check_arena_layer_blocks, f32_from_bits,
                    layer_block, n_salient)

pytestmark = pytest.mark.gpu

SIGMA = float(np.float32(1.0 / np.sqrt(128.0)))
STEPS = 2


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_35800_gb300 import build
    build.build()


def _oracle_layer(w, mask_row, kb, vb, want_att=True):
    return oracle.quantize_layer(kb, vb, w.img_start, w.image, w.base, w.bits, mask_row,
                                 int(w.keys_only), w.kivi_group_tokens, w.kivi_group_channels,
                                 w.kivi_residual, want_att=want_att, meta16=w.meta_bits == 32,
                                 n_salient=n_salient(w))


def _appended(news, l, rows, heads, upto):
    """fp64 [len(rows)][len(heads)][upto][128] appended K and V of steps < upto."""
    ak = np.stack([f32_from_bits(news[s][0][l][np.ix_(rows, heads)]) for s in range(upto)], axis=2)
    av = np.stack([f32_from_bits(news[s][1][l][np.ix_(rows, heads)]) for s in range(upto)], axis=2)
    return ak.astype(np.float64), av.astype(np.float64)


def test_full_size_qwen25vl7b_complete():
    """Every arena byte of all 28 layers; every attention output of every step."""
    w = wl.WORKLOADS["qwen25vl7b"]
    runner = CacheRunner(w)
    kept = runner.quantize_all(keep=True)
    S = w.decode_steps
    outs, qs, news = [], [], []
    for step in range(S):
        k_new, v_new = wl.step_new_kv(w, step, "cuda")
        q = wl.step_query(w, step, "cuda")
        out = runner.decode_step(step, q=q, k_new=k_new, v_new=v_new)
        outs.append(bits16(out))
        qs.append(bits16(q))
        news.append((bits16(k_new), bits16(v_new)))
    torch.cuda.synchronize()
    rows, heads = np.arange(w.batch), np.arange(w.kv_heads)
    for l, (k, v) in enumerate(kept):
        kb, vb = bits16(k), bits16(v)
        o = _oracle_layer(w, runner.mask[l], kb, vb)
        check_arena_layer_blocks(runner, l, kb, vb, o)
        ak, av = _appended(news, l, rows, heads, S)
        K = np.concatenate([o["k_att"], ak], axis=2)
        V = np.concatenate([o["v_deq"].astype(np.float64), av], axis=2)
        for step in range(S):
            Tt = w.seq_len + step + 1
            ref = oracle.attention_layer(qs[step][l], K[:, :, :Tt], V[:, :, :Tt], SIGMA)
            assert_close(outs[step][l], ref, "qwen25vl7b layer %d step %d" % (l, step))


@pytest.mark.parametrize("name", ["llavanext7b", "internvl25_8b", "qwen25vl72b"])
def test_full_size_every_layer_bit_exact(name):
    """Every layer's arena regions bit for bit; attention on 4 layers x 4 rows
    x every query head after the first and the last decode step."""
    w = wl.WORKLOADS[name]
    runner = CacheRunner(w)
    runner.quantize_all()
    S = w.decode_steps
    rng = np.random.default_rng(17)
    sample_layers = sorted(set([0, w.layers - 1] + [int(x) for x in rng.choice(w.layers, 2, replace=False)]))
    while len(sample_layers) < 4:
        sample_layers = sorted(set(sample_layers + [int(rng.integers(w.layers))]))
    sample_rows = np.array(sorted(set([0, w.batch - 1] + [int(x) for x in rng.choice(w.batch, 2, replace=False)])))
    picked = {}  # step -> (outputs, queries) of the sampled layers and rows
    news = []
    for step in range(S):
        k_new, v_new = wl.step_new_kv(w, step, "cuda")
        q = wl.step_query(w, step, "cuda")
        out = runner.decode_step(step, q=q, k_new=k_new, v_new=v_new)
        news.append((bits16(k_new[sample_layers]), bits16(v_new[sample_layers])))
        if step in (0, S - 1):
            torch.cuda.synchronize()
            picked[step] = (bits16(out[sample_layers][:, sample_rows]), bits16(q[sample_layers][:, sample_rows]))
        del out, q, k_new, v_new
    torch.cuda.synchronize()
    heads = np.arange(w.kv_heads)
    for l in range(w.layers):
        k, v = wl.layer_kv(w, l, "cuda")
        kb, vb = bits16(k), bits16(v)
        del k, v
        o = _oracle_layer(w, runner.mask[l], kb, vb, want_att=False)
        check_arena_layer_blocks(runner, l, kb, vb, o, layer_block(runner, l))
        if l in sample_layers:
            i = sample_layers.index(l)
            os_ = _oracle_layer(w, runner.mask[l], kb[sample_rows], vb[sample_rows])
            ak, av = _appended([(n[0], n[1]) for n in news], i, sample_rows, heads, S)
            K = np.concatenate([os_["k_att"], ak], axis=2)
            V = np.concatenate([os_["v_deq"].astype(np.float64), av], axis=2)
            for step in (0, S - 1):
                Tt = w.seq_len + step + 1
                out_b, q_b = picked[step]
                ref = oracle.attention_layer(q_b[i], K[:, :, :Tt], V[:, :, :Tt], SIGMA)
                assert_close(out_b[i], ref, "%s layer %d step %d" % (name, l, step))
        del kb, vb, o


def _samples(w, mask, seed):
    """First and last layer, a protected head, the rest seeded at random."""
    rng = np.random.default_rng(seed)
    picks = [(0, 0, 0), (w.layers - 1, w.batch - 1, w.kv_heads - 1)]
    prot = np.argwhere(mask)
    if len(prot):
        l, h = prot[rng.integers(len(prot))]
        picks.append((int(l), int(rng.integers(w.batch)), int(h)))
    picks.append((int(rng.integers(w.layers)), int(rng.integers(w.batch)), int(rng.integers(w.kv_heads))))
    return picks


# options of the later rows at full size
VARIANTS = [("internvl25_8b", {"salient_permille": 20}),
            ("internvl25_8b", {"salient_permille": 20, "keys_only": True}),
            ("llavanext7b", {"base": wl.BASE_AKVQ, "salient_permille": 20}),  # K-only, MHA
            ("qwen25vl7b", {"bits": 3}), ("llavanext7b", {"bits": 3}),
            ("qwen25vl72b", {"meta_bits": 32})]


@pytest.mark.parametrize("name,opts", VARIANTS,
                         ids=[n + "".join("-%s%s" % kv for kv in o.items()) for n, o in VARIANTS])
def test_full_size_sampled_parity(name, opts):
    w = dataclasses.replace(wl.WORKLOADS[name], **opts)
    runner = CacheRunner(w)
    runner.quantize_all()
    G = w.q_heads // w.kv_heads
    picks = _samples(w, runner.mask, 5)
    outs, qs, news = [], [], []
    for step in range(STEPS):
        k_new, v_new = wl.step_new_kv(w, step, "cuda")
        q = wl.step_query(w, step, "cuda")
        out = runner.decode_step(step, q=q, k_new=k_new, v_new=v_new)
        torch.cuda.synchronize()
        outs.append([bits16(out[l, b, h * G:(h + 1) * G]) for l, b, h in picks])
        qs.append([bits16(q[l, b, h * G:(h + 1) * G]) for l, b, h in picks])
        news.append([(bits16(k_new[l, b, h]), bits16(v_new[l, b, h])) for l, b, h in picks])
    for i, (l, b, h) in enumerate(picks):
        k, v = wl.layer_kv(w, l, "cuda")
        kb = bits16(k[b:b + 1, h:h + 1])
        vb = bits16(v[b:b + 1, h:h + 1])
        del k, v
        o = _oracle_layer(w, runner.mask[l][h:h + 1], kb, vb)
        check_arena_layer(runner, l, kb, vb, o, heads=[h], rows=[b], local=True)
        K = o["k_att"][0, 0]
        V = o["v_deq"][0, 0].astype(np.float64)
        for step in range(STEPS):
            ak = np.stack([f32_from_bits(news[s][i][0]) for s in range(step + 1)]).astype(np.float64)
            av = np.stack([f32_from_bits(news[s][i][1]) for s in range(step + 1)]).astype(np.float64)
            Kt = np.concatenate([K, ak])[None, None]
            Vt = np.concatenate([V, av])[None, None]
            ref = oracle.attention_layer(qs[step][i][None], Kt, Vt, SIGMA)[0]
            assert_close(outs[step][i], ref, "%s layer %d row %d head %d step %d" % (name, l, b, h, step))
