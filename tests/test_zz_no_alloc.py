"""The allocation-free decode entry point against the workspace entry point.

hg_decode_attention_noalloc serves callers that may not allocate device
memory (plugin interfaces that pass only inputs and outputs, a device pool
owned by another framework, loops that cannot take cudaMalloc's implicit
synchronisation): it runs decode attention with the library's own static
scratch array instead of a caller-provided workspace.  Here it must give the
same attention output as hg_decode_attention on the same cache, within the
tolerance of the parity tests, on two consecutive decode steps (the second
call sees the scratch contents the first one left).  The file is named to be
collected last.
"""
import numpy as np
import pytest
import torch

import paper_2609_35800_gb300 as hg
from paper_2609_35800_gb300 import workloads as wl
from paper_2609_35800_gb300.runner import CacheRunner

pytestmark = pytest.mark.gpu

ATOL, RTOL = 2e-3, 1e-2
SIGMA = float(np.float32(1.0 / np.sqrt(128.0)))


def _f32(t):
    return t.float().cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("base,bits,keys_only", [(wl.BASE_MINMAX, 2, 0), (wl.BASE_KIVI, 2, 1),
                                                 (wl.BASE_AKVQ, 4, 0)])
def test_noalloc_matches_workspace_entry_point(base, bits, keys_only):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_35800_gb300 import build
    build.build()
    w = wl.custom("noalloc", 3, 2, 16, 4, 24, 700, 40, base, bits, keys_only, decode_steps=2,
                  seed=11, protected=[(0, 1), (2, 3)])
    runner = CacheRunner(w)
    runner.quantize_all()
    for step in range(2):
        k_new, v_new = wl.step_new_kv(w, step, "cuda")
        q = wl.step_query(w, step, "cuda")
        hg.hg_append_kv(runner.cache, 0, w.layers, k_new, v_new)
        ref = torch.empty_like(q)
        hg.hg_decode_attention(runner.cache, 0, w.layers, q, ref, SIGMA, runner.ws, runner.ws_bytes)
        got = torch.full_like(q, float("nan"))
        hg.hg_decode_attention_noalloc(runner.cache, 0, w.layers, q, got, SIGMA)
        torch.cuda.synchronize()
        g, r = _f32(got), _f32(ref)
        assert np.all(np.isfinite(g))
        assert np.all(np.abs(g - r) <= ATOL + RTOL * np.abs(r)), "step %d" % step
