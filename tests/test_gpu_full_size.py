"""Parity at the benchmark's full cache shapes, in the launch configuration
bench.py times: one quantize call over all layers, then fused decode steps
(append + attention over all layers, one launch each).  The oracle recomputes
sampled (layer, batch row, KV head) triples one by one: the head's arena
regions bit for bit, and its G query heads' attention outputs after every
step within the tolerance of the parity tests."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from paper_2609_35800_gb300 import workloads as wl
from paper_2609_35800_gb300.runner import CacheRunner

from parity import assert_close, bits16, check_arena_layer, f32_from_bits, n_salient

pytestmark = pytest.mark.gpu

SIGMA = float(np.float32(1.0 / np.sqrt(128.0)))
STEPS = 2


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_35800_gb300 import build
    build.build()


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


# the four benchmark shapes, then options of the next rows at full size
VARIANTS = [("qwen25vl7b", {}), ("llavanext7b", {}), ("internvl25_8b", {}), ("qwen25vl72b", {}),
            ("internvl25_8b", {"salient_permille": 20}), ("qwen25vl7b", {"bits": 3}),
            ("llavanext7b", {"bits": 3}), ("qwen25vl72b", {"meta_bits": 32})]


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
        o = oracle.quantize_layer(kb, vb, w.img_start, w.image, w.base, w.bits,
                                  runner.mask[l][h:h + 1], int(w.keys_only), w.kivi_group_tokens,
                                  w.kivi_group_channels, w.kivi_residual,
                                  meta16=w.meta_bits == 32, n_salient=n_salient(w))
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
