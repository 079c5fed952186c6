"""Protected-head selection oracle -- TEST INFRASTRUCTURE ONLY (plain numpy, fp64).

Follows Sec. 3 "Selecting physical KV heads" (Eq. 2) step by step:
  1. average the query-head scores of each GQA group into per-KV-head scores
     g_i and o_i (query head qh belongs to KV head qh // G);
  2. standardise each over all KV heads of the model: z(x) = (x - mean) / std;
  3. s_i = z(g_i) + z(o_i);
  4. protect the K heads with the largest s (TopK).
Readings where the paper is silent: population std (the selection does not
depend on it: both terms scale alike); a constant score has z = 0; ties go to
the lower index i = layer * H_kv + head; K defaults to round(N_KV / 8).
"""
import numpy as np


def select_heads(g_scores, o_scores, num_kv_heads, k=None):
    g = np.asarray(g_scores, dtype=np.float64)
    o = np.asarray(o_scores, dtype=np.float64)
    L, Hq = g.shape
    G = Hq // num_kv_heads
    gb = g.reshape(L, num_kv_heads, G).mean(axis=2).ravel()
    ob = o.reshape(L, num_kv_heads, G).mean(axis=2).ravel()

    def z(x):
        sd = x.std()
        return (x - x.mean()) / sd if sd > 0 else np.zeros_like(x)

    s = z(gb) + z(ob)
    n = s.size
    if k is None:
        k = int(round(n / 8.0))
    k = max(0, min(k, n))
    order = sorted(range(n), key=lambda i: (-s[i], i))
    mask = np.zeros(n, dtype=np.uint8)
    mask[order[:k]] = 1
    return mask.reshape(L, num_kv_heads)
