"""Protected-head selection (Sec. 3, Eq. 2): the numpy oracle pinned by hand
examples and invariants, and the library's host routine hg_select_heads
against it.  CPU only."""
import numpy as np
import pytest

from oracle.selection import select_heads


def test_hand_examples():
    # G = 2: KV head 0 <- query heads 0, 1; KV head 1 <- query heads 2, 3.
    # g means [2, 0] -> z = [1, -1]; o means [0, 5] -> z = [-1, 1]; s = [0, 0]:
    # a tie, the lower index wins
    m = select_heads([[1.0, 3.0, 0.0, 0.0]], [[0.0, 0.0, 5.0, 5.0]], 2, k=1)
    assert m.tolist() == [[1, 0]]
    # constant o contributes nothing (z = 0): the larger g mean wins
    m = select_heads([[0.0, 0.0, 4.0, 2.0]], [[1.0, 1.0, 1.0, 1.0]], 2, k=1)
    assert m.tolist() == [[0, 1]]
    # two layers, MHA (G = 1): s = z(g) + z(o) = [-2.5, ...] worked by hand
    g = [[0.0, 1.0], [2.0, 3.0]]          # z(g) = [-1.342, -0.447, 0.447, 1.342]
    o = [[3.0, 0.0], [0.0, 0.0]]          # z(o) = [1.732, -0.577, -0.577, -0.577]
    assert select_heads(g, o, 2, k=2).tolist() == [[1, 0], [0, 1]]   # s = 0.39, -1.02, -0.13, 0.76


def test_default_budget_is_an_eighth():
    rng = np.random.default_rng(0)
    for L, Hkv, G, want in [(28, 4, 7, 14), (32, 32, 1, 128), (32, 8, 4, 32), (80, 8, 8, 80)]:
        g = rng.standard_normal((L, Hkv * G))
        o = rng.standard_normal((L, Hkv * G))
        assert int(select_heads(g, o, Hkv).sum()) == want


def test_invariants():
    rng = np.random.default_rng(1)
    L, Hkv, G = 6, 4, 3
    g = rng.standard_normal((L, Hkv * G))
    o = rng.exponential(size=(L, Hkv * G))
    base = select_heads(g, o, Hkv, k=5)
    assert int(base.sum()) == 5
    # positive affine maps of either score leave z, hence the selection, unchanged
    assert np.array_equal(select_heads(3.0 * g - 7.0, o, Hkv, k=5), base)
    assert np.array_equal(select_heads(g, 0.25 * o + 2.0, Hkv, k=5), base)
    # the two scores enter symmetrically
    assert np.array_equal(select_heads(o, g, Hkv, k=5), base)
    # query heads inside a GQA group are averaged: their order does not matter
    perm = np.concatenate([h * G + rng.permutation(G) for h in range(Hkv)])
    assert np.array_equal(select_heads(g[:, perm], o[:, perm], Hkv, k=5), base)
    # nested budgets: the top 3 are inside the top 5
    assert np.all(select_heads(g, o, Hkv, k=3) <= base)
    # a head with both scores largest is always chosen first
    g2, o2 = g.copy(), o.copy()
    g2[2, 4:4 + G] = 100.0
    o2[2, 4:4 + G] = 100.0
    assert select_heads(g2, o2, Hkv, k=1)[2, 1] == 1


@pytest.fixture(scope="module")
def hg_lib():
    import paper_2609_35800_gb300 as hg
    from paper_2609_35800_gb300 import build
    build.build()
    hg.library()
    return hg


@pytest.mark.parametrize("L,Hkv,G,k", [(1, 4, 7, -1), (28, 4, 7, -1), (32, 32, 1, -1), (5, 8, 4, 9),
                                       (3, 2, 2, 0), (2, 3, 5, 6)])
def test_library_matches_oracle(hg_lib, L, Hkv, G, k):
    rng = np.random.default_rng(L * 100 + Hkv * 10 + G)
    g = rng.standard_normal((L, Hkv * G)).astype(np.float32)
    o = (rng.standard_normal((L, Hkv * G)) * 0.01 + 3.0).astype(np.float32)
    got = hg_lib.hg_select_heads(g, o, L, Hkv * G, Hkv, k)
    want = select_heads(g, o, Hkv, k=None if k < 0 else k)
    assert np.array_equal(got, want)


def test_library_ties_and_errors(hg_lib):
    # all scores equal: s = 0 everywhere, the k lowest indices are chosen
    m = hg_lib.hg_select_heads(np.ones((2, 8), np.float32), np.ones((2, 8), np.float32), 2, 8, 4, 3)
    assert m.ravel().tolist() == [1, 1, 1, 0, 0, 0, 0, 0]
    bad = np.zeros((2, 8), np.float32)
    bad[1, 3] = np.nan
    with pytest.raises(hg_lib.HGError) as e:
        hg_lib.hg_select_heads(bad, np.zeros((2, 8), np.float32), 2, 8, 4)
    assert e.value.status == 1
    with pytest.raises(hg_lib.HGError) as e:   # 8 query heads over 3 KV heads
        hg_lib.hg_select_heads(np.zeros((2, 8), np.float32), np.zeros((2, 8), np.float32), 2, 8, 3)
    assert e.value.status == 1
