"""Workload plumbing over the C ABI: allocate the arena and workspace with torch,
create the cache descriptor, quantize the synthetic prefill and drive decode
steps.  Marshalling only -- every step of the path runs in the library."""
import torch

from . import (QuantConfig, Shape, hg_cache_create, hg_cache_layout, hg_decode_step,
               hg_decode_workspace_size, hg_quantize_kv, hg_workspace_clear, workloads)


def shape_of(w):
    return Shape(batch=w.batch, num_layers=w.layers, num_kv_heads=w.kv_heads,
                 num_q_heads=w.q_heads, head_dim=128, seq_len=w.seq_len, img_start=w.img_start,
                 img_len=w.image, max_new_tokens=w.decode_steps)


def config_of(w):
    return QuantConfig(base=w.base, bits=w.bits, keys_only=int(w.keys_only),
                       kivi_group_tokens=w.kivi_group_tokens,
                       kivi_group_channels=w.kivi_group_channels,
                       kivi_residual=w.kivi_residual, meta_bits=w.meta_bits,
                       salient_permille=w.salient_permille)


class CacheRunner:
    """One cache of a workload on one device, with a workspace for `ws_layers` layers."""

    def __init__(self, w, device="cuda", ws_layers=None):
        self.w = w
        self.device = device
        self.mask = workloads.protection_mask(w).numpy()
        self.shape = shape_of(w)
        self.config = config_of(w)
        self.arena_bytes = hg_cache_layout(self.shape, self.config, self.mask)
        self.arena = torch.empty(self.arena_bytes, dtype=torch.uint8, device=device)
        self.cache = hg_cache_create(self.shape, self.config, self.mask, self.arena,
                                     self.arena_bytes)
        # large enough for per-layer launches and for one launch over ws_layers layers
        ws_layers = w.layers if ws_layers is None else ws_layers
        self.ws_bytes = max(hg_decode_workspace_size(self.cache, 1),
                            hg_decode_workspace_size(self.cache, ws_layers))
        self.ws = torch.empty(max(self.ws_bytes, 256), dtype=torch.uint8, device=device)
        hg_workspace_clear(self.ws, self.ws_bytes)

    def quantize_all(self, keep=False, layers_per_call=None):
        """Generate and quantize every layer's prefill; return the inputs if keep."""
        w = self.w
        per = layers_per_call or w.layers
        kept = []
        for l0 in range(0, w.layers, per):
            n = min(per, w.layers - l0)
            ks, vs = [], []
            for l in range(l0, l0 + n):
                k, v = workloads.layer_kv(w, l, self.device)
                ks.append(k)
                vs.append(v)
            hg_quantize_kv(self.cache, l0, ks, vs)
            if keep:
                kept.extend(zip(ks, vs))
        return kept

    def decode_step(self, step, layer_begin=0, layer_count=None, q=None, k_new=None, v_new=None,
                    out=None, softmax_scale=0.0):
        """Append the step's K/V and run decode attention in one launch; returns
        out [layers][B][Hq][128]."""
        w = self.w
        n = w.layers if layer_count is None else layer_count
        if k_new is None:
            k_new, v_new = workloads.step_new_kv(w, step, self.device, n)
        if q is None:
            q = workloads.step_query(w, step, self.device, n)
        if out is None:
            out = torch.empty_like(q)
        hg_decode_step(self.cache, layer_begin, n, q, k_new, v_new, out, softmax_scale, self.ws,
                       self.ws_bytes)
        return out
