"""Seeded synthetic KV-cache workloads (inputs only -- none of the method's arithmetic).

The paper's VLM caches and benchmark data are not available, so every input
is synthetic, shaped like the paper's models, and drawn from a seeded
generator:

  K ~ N(0, 1) except a few outlier channels per (layer, KV head), which are
  8 z + 3 (z ~ N(0, 1)); V ~ N(0, 1); decode queries and appended K/V follow
  the same laws.  Values are drawn in fp32 and rounded to BF16 (nearest even).
  The protection mask keeps round(N_KV / 8) (layer, KV head) pairs, drawn by a
  seeded permutation (Sec. 3, Eq. 2's budget K = round(N_KV / 8)).

Both the CUDA path and the CPU oracle receive the same tensors from here.
"""
import dataclasses

import torch

D = 128

BASE_MINMAX = 0
BASE_KIVI = 1
BASE_AKVQ = 2

# tensor kinds for seed derivation
_K, _V, _OUTLIER, _MASK, _Q, _KNEW, _VNEW = range(7)


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    layers: int
    batch: int
    q_heads: int
    kv_heads: int
    text_prefix: int
    image: int
    text_suffix: int
    base: int
    bits: int
    keys_only: bool
    decode_steps: int
    seed: int
    fixed_outliers: tuple = ()      # same outlier channels in every head (tiny case)
    n_outliers: int = 4             # else this many random channels per (layer, head)
    fixed_protected: tuple = None   # explicit (layer, head) pairs (may be empty); None: round(N_KV / 8)
    kivi_group_tokens: int = 32
    kivi_group_channels: int = 32
    kivi_residual: int = 32
    meta_bits: int = 64             # 64: fp32 {scale, zero}; 32: binary16 pair (Sec. 5.4)
    salient_permille: int = 0       # AKVQ-style salient tokens kept BF16 (Sec. 4; 20 = 2%)

    @property
    def seq_len(self):
        return self.text_prefix + self.image + self.text_suffix

    @property
    def img_start(self):
        return self.text_prefix

    @property
    def group(self):
        return self.q_heads // self.kv_heads

    @property
    def n_kv(self):
        return self.layers * self.kv_heads


# The five cache shapes.
WORKLOADS = {
    # one layer, 28 q / 4 KV heads, 32 text + 256 image + 32 text, min-max 2-bit,
    # KV head 1 protected (K+V), fixed outlier channels {7, 63, 101}, one query.
    "tiny": Workload("tiny", 1, 1, 28, 4, 32, 256, 32, BASE_MINMAX, 2, False, 1, 0,
                     fixed_outliers=(7, 63, 101), fixed_protected=((0, 1),)),
    # Qwen2.5-VL-7B-shaped: 28 layers, 28 q / 4 KV heads, 64 + 1296 + 100 tokens.
    "qwen25vl7b": Workload("qwen25vl7b", 28, 1, 28, 4, 64, 1296, 100, BASE_MINMAX, 2, False,
                           32, 1),
    # LLaVA-NeXT-7B-shaped: 32 layers, MHA 32, batch 16, 40 + 2880 + 200, KIVI-style 2-bit, K-only.
    "llavanext7b": Workload("llavanext7b", 32, 16, 32, 32, 40, 2880, 200, BASE_KIVI, 2, True,
                            64, 2),
    # InternVL2.5-8B-shaped: 32 layers, 32 q / 8 KV, batch 32, 64 + 3328 + 128, AKVQ-style 4-bit.
    "internvl25_8b": Workload("internvl25_8b", 32, 32, 32, 8, 64, 3328, 128, BASE_AKVQ, 4, False,
                              64, 3),
    # Qwen2.5-VL-72B-shaped: 80 layers, 64 q / 8 KV, batch 32, 128 + 8192 + 256, min-max 2-bit.
    "qwen25vl72b": Workload("qwen25vl72b", 80, 32, 64, 8, 128, 8192, 256, BASE_MINMAX, 2, False,
                            128, 4),
}


def _seed(w, layer, kind, step=0):
    return ((w.seed * 1000003 + layer) * 16 + kind) * 100003 + step


def _gen(device, seed):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _randn_bf16(shape, device, seed):
    x = torch.randn(shape, generator=_gen(device, seed), device=device, dtype=torch.float32)
    return x.to(torch.bfloat16)


def protection_mask(w):
    """uint8 [layers][kv_heads] (CPU tensor), 1 = protected."""
    m = torch.zeros(w.layers, w.kv_heads, dtype=torch.uint8)
    if w.fixed_protected is not None:
        for l, h in w.fixed_protected:
            m[l, h] = 1
        return m
    k = int(round(w.n_kv / 8))
    perm = torch.randperm(w.n_kv, generator=_gen("cpu", _seed(w, 0, _MASK)))[:k]
    m.view(-1)[perm] = 1
    return m


def outlier_channels(w, layer):
    """[kv_heads][n] long (CPU): outlier channel indices of each head of a layer."""
    if w.fixed_outliers:
        return torch.tensor([list(w.fixed_outliers)] * w.kv_heads, dtype=torch.long)
    g = _gen("cpu", _seed(w, layer, _OUTLIER))
    return torch.stack([torch.randperm(D, generator=g)[: w.n_outliers] for _ in range(w.kv_heads)])


def layer_kv(w, layer, device):
    """BF16 prefill K, V of one layer: [batch][kv_heads][seq_len][128]."""
    shape = (w.batch, w.kv_heads, w.seq_len, D)
    k = torch.randn(shape, generator=_gen(device, _seed(w, layer, _K)), device=device,
                    dtype=torch.float32)
    ch = outlier_channels(w, layer).to(device)
    for h in range(w.kv_heads):
        idx = ch[h]
        k[:, h, :, idx] = k[:, h, :, idx] * 8.0 + 3.0
    v = torch.randn(shape, generator=_gen(device, _seed(w, layer, _V)), device=device,
                    dtype=torch.float32)
    return k.to(torch.bfloat16), v.to(torch.bfloat16)


def step_query(w, step, device, layers=None):
    """Decode queries of one step: [layers][batch][q_heads][128] BF16."""
    layers = w.layers if layers is None else layers
    return _randn_bf16((layers, w.batch, w.q_heads, D), device, _seed(w, 0, _Q, step))


def step_new_kv(w, step, device, layers=None):
    """Appended K, V of one step: [layers][batch][kv_heads][128] BF16 (K with outliers)."""
    layers = w.layers if layers is None else layers
    k = torch.randn((layers, w.batch, w.kv_heads, D), generator=_gen(device, _seed(w, 0, _KNEW, step)),
                    device=device, dtype=torch.float32)
    for l in range(layers):
        ch = outlier_channels(w, l).to(device)
        for h in range(w.kv_heads):
            k[l, :, h, ch[h]] = k[l, :, h, ch[h]] * 8.0 + 3.0
    v = _randn_bf16((layers, w.batch, w.kv_heads, D), device, _seed(w, 0, _VNEW, step))
    return k.to(torch.bfloat16), v


def custom(name, layers, batch, q_heads, kv_heads, text_prefix, image, text_suffix, base, bits,
           keys_only, decode_steps=2, seed=0, protected=None, residual=32, n_outliers=4,
           meta_bits=64, salient_permille=0):
    """A small workload for tests: `protected` lists (layer, head) pairs (empty = none),
    None draws round(N_KV / 8) of them."""
    return Workload(name, layers, batch, q_heads, kv_heads, text_prefix, image, text_suffix, base,
                    bits, bool(keys_only), decode_steps, seed,
                    fixed_protected=None if protected is None else tuple(protected),
                    n_outliers=n_outliers, kivi_residual=residual, meta_bits=meta_bits,
                    salient_permille=salient_permille)
