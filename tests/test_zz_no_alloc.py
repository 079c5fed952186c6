"""The allocation-free decode entry point against the workspace entry point.

hg_decode_attention_noalloc serves callers that may not allocate device
memory (plugin interfaces that pass only inputs and outputs, a device pool
owned by another framework, loops that cannot take cudaMalloc's implicit
synchronisation): it runs decode attention with the library's own static
scratch array instead of a caller-provided workspace.  Both entry points run
the same kernel with the same work plan and a fixed merge order, so their
outputs must be bit-identical -- on consecutive calls (each sees the scratch
the previous one left), after a call over a different layer range (other
counters, other partial slots), on a non-default stream, and at a full
benchmark shape.  A launch whose workspace exceeds the 32 MiB scratch is
refused before anything is enqueued.  The file is named to be collected last.
"""
import numpy as np
import pytest
import torch

import paper_2609_35800_gb300 as hg
from paper_2609_35800_gb300 import workloads as wl
from paper_2609_35800_gb300.runner import CacheRunner

pytestmark = pytest.mark.gpu

SIGMA = float(np.float32(1.0 / np.sqrt(128.0)))
SCRATCH_BYTES = 32 << 20


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_35800_gb300 import build
    build.build()
    hg.library()


def _same(got, ref, where):
    g = got.view(torch.int16).cpu().numpy()
    r = ref.view(torch.int16).cpu().numpy()
    assert np.array_equal(g, r), "%s: %d of %d outputs differ" % (where, int((g != r).sum()), g.size)


def _both(runner, layer_begin, layer_count, q, stream=None):
    ref = torch.empty_like(q)
    hg.hg_decode_attention(runner.cache, layer_begin, layer_count, q, ref, SIGMA, runner.ws,
                           runner.ws_bytes, stream)
    got = torch.full_like(q, float("nan"))
    hg.hg_decode_attention_noalloc(runner.cache, layer_begin, layer_count, q, got, SIGMA, stream)
    return got, ref


@pytest.mark.parametrize("base,bits,keys_only", [(wl.BASE_MINMAX, 2, 0), (wl.BASE_KIVI, 2, 1),
                                                 (wl.BASE_AKVQ, 4, 0)])
def test_noalloc_matches_workspace_entry_point(base, bits, keys_only):
    w = wl.custom("noalloc", 3, 2, 16, 4, 24, 700, 40, base, bits, keys_only, decode_steps=2,
                  seed=11, protected=[(0, 1), (2, 3)])
    runner = CacheRunner(w)
    runner.quantize_all()
    hg.hg_workspace_clear(None)
    for step in range(2):
        k_new, v_new = wl.step_new_kv(w, step, "cuda")
        q = wl.step_query(w, step, "cuda")
        hg.hg_append_kv(runner.cache, 0, w.layers, k_new, v_new)
        got, ref = _both(runner, 0, w.layers, q)
        torch.cuda.synchronize()
        _same(got, ref, "step %d, all layers" % step)
        # a differently sized launch right after: one layer, then two
        got1, ref1 = _both(runner, 2, 1, q[2:3].contiguous())
        got2, ref2 = _both(runner, 0, 2, q[0:2].contiguous())
        torch.cuda.synchronize()
        _same(got1, ref1, "step %d, layer 2 alone" % step)
        _same(got2, ref2, "step %d, layers 0-1" % step)
        _same(got2, ref[0:2], "step %d, layers 0-1 against the all-layer launch" % step)
    assert hg.hg_workspace_status(None) == 0


def test_noalloc_full_shape_one_layer_side_stream():
    """One layer of the Qwen2.5-VL-7B-shaped cache on a non-default stream."""
    w = wl.WORKLOADS["qwen25vl7b"]
    runner = CacheRunner(w)
    runner.quantize_all()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    k_new, v_new = wl.step_new_kv(w, 0, "cuda")
    q = wl.step_query(w, 0, "cuda")
    with torch.cuda.stream(side):
        hg.hg_append_kv(runner.cache, 0, w.layers, k_new, v_new, side)
        for l in (0, w.layers - 1):
            got, ref = _both(runner, l, 1, q[l:l + 1].contiguous(), side)
            side.synchronize()
            _same(got, ref, "layer %d" % l)
    assert hg.hg_workspace_status(None, side) == 0


def test_noalloc_refuses_a_workspace_beyond_the_scratch():
    """The InternVL2.5-8B-shaped cache over all 32 layers needs just over 32 MiB
    of workspace; the call is refused and `out` is left as it was."""
    w = wl.WORKLOADS["internvl25_8b"]
    runner = CacheRunner(w, ws_layers=1)
    need = hg.hg_decode_workspace_size(runner.cache, w.layers)
    assert need > SCRATCH_BYTES
    assert hg.hg_decode_workspace_size(runner.cache, 1) <= SCRATCH_BYTES
    q = wl.step_query(w, 0, "cuda")
    out = torch.full_like(q, float("nan"))
    before = out.view(torch.int16).clone()
    with pytest.raises(hg.HGError) as err:
        hg.hg_decode_attention_noalloc(runner.cache, 0, w.layers, q, out, SIGMA)
    assert err.value.status == 4  # HG_ERR_WORKSPACE_TOO_SMALL
    torch.cuda.synchronize()
    assert torch.equal(out.view(torch.int16), before)
