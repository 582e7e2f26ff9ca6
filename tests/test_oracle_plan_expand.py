"""Pins of the oracle's expand-then-prune first pass (EAGLE-2 style, Sec. 3.1 / App. B.3),
CPU only.

The planner is checked against an independent path-enumeration construction of the
layer-wise frontiers (rank tuples sorted with scores from scipy's logsumexp and exact
fractional comparison of same-depth sums), against the max-heap planner once the frontier
can hold the whole budget (App. B.3: a wide enough frontier recovers the heap's tree), and
against the heap's optimality: the i-th kept path is never more probable than the heap's.
"""
import functools
import itertools
from fractions import Fraction

import numpy as np
import pytest
from scipy.special import logsumexp

TREE_KEYS = ("parent", "depth", "rank", "plan_token", "child_off", "child_ids")


def _x(draft, T):
    return draft.astype(np.float32) * np.float32(np.float32(1.0) / np.float32(T))


def _topk(x, K):
    return np.lexsort((np.arange(len(x)), -x.astype(np.float64)))[:K]


def _order(x, K, L):
    """Comparator of rank tuples: log-probability desc, shorter first, then (for equal
    length) exact sum of logits desc, then the parent's order, then rank."""
    lse = [logsumexp(x[d].astype(np.float64)) for d in range(L)]
    top = [_topk(x[d], K) for d in range(L)]

    def xs(p):
        return [float(x[j][top[j][r]]) for j, r in enumerate(p)]

    @functools.lru_cache(maxsize=None)
    def key(p):
        return sum(v - lse[j] for j, v in enumerate(xs(p)))

    def cmp(a, b):
        if a == b:
            return 0
        if len(a) != len(b):
            ka, kb = key(a), key(b)
            assert abs(ka - kb) > 1e-9, "cross-depth near tie: choose another seed"
            return -1 if ka > kb else 1
        sa, sb = sum(Fraction(v) for v in xs(a)), sum(Fraction(v) for v in xs(b))
        if sa != sb:
            return -1 if sa > sb else 1
        c = cmp(a[:-1], b[:-1]) if len(a) > 1 else 0
        return c if c != 0 else (-1 if a[-1] < b[-1] else 1)

    return functools.cmp_to_key(cmp), top, key


def _brute_force(x, K, L, N, W):
    """Layer d+1 = every child of the W best paths of layer d; keep the N best of all layers."""
    sk, top, key = _order(x, K, L)
    layer = [(r,) for r in range(K)]
    generated = []
    for d in range(1, L + 1):
        layer.sort(key=sk)
        generated.extend(layer)
        if d < L:
            layer = [p + (r,) for p in layer[:W] for r in range(K)]
    generated.sort(key=sk)
    return generated[:N], top, key


def _paths(tree, b=0):
    NN = tree["parent"].shape[1]
    path = {0: ()}
    out = []
    for i in range(1, NN):
        p = int(tree["parent"][b, i])
        assert 0 <= p < i
        path[i] = path[p] + (int(tree["rank"][b, i]),)
        out.append(path[i])
    return out


def _check_tree(tree, K, L, b=0):
    par, dep, rk = tree["parent"][b], tree["depth"][b], tree["rank"][b]
    NN = len(par)
    off, ids = tree["child_off"][b], tree["child_ids"][b]
    assert off[0] == 0 and off[-1] == NN - 1
    for u in range(NN):
        ch = list(ids[off[u]:off[u + 1]])
        assert ch == [i for i in range(1, NN) if par[i] == u]
        assert [int(rk[c]) for c in ch] == list(range(len(ch)))
        for c in ch:
            assert dep[c] == dep[u] + 1 and dep[c] <= L
    assert np.all(np.diff(tree["score"][b, 1:]) <= 0.0)


@pytest.mark.parametrize("seed,V,K,L,N,W", [(2000, 32, 4, 4, 8, 1), (2001, 32, 4, 4, 20, 2), (2002, 40, 3, 4, 30, 3),
                                            (2003, 300, 5, 4, 40, 4), (2004, 64, 4, 5, 60, 10)])
def test_expand_matches_path_enumeration(orc, seed, V, K, L, N, W):
    rng = np.random.default_rng(seed)
    draft = (2.0 * rng.standard_normal((1, L, V))).astype(np.float32)
    tree = orc.plan_expand(draft, 1.0, N, K, L, W)
    want, top, _ = _brute_force(_x(draft[0], 1.0), K, L, N, W)
    assert _paths(tree) == want
    _check_tree(tree, K, L)
    for i in range(1, N + 1):
        d, r = tree["depth"][0, i], tree["rank"][0, i]
        assert tree["plan_token"][0, i] == top[d - 1][r]


def test_expand_with_exact_ties(orc):
    """Integer logits tie many same-depth paths exactly; frontiers and the final order follow
    the parent's order, then rank."""
    rng = np.random.default_rng(17)
    V, K, L, N, W = 16, 3, 4, 30, 4
    draft = rng.integers(-3, 4, size=(1, L, V)).astype(np.float32)
    tree = orc.plan_expand(draft, 1.0, N, K, L, W)
    want, _, _ = _brute_force(_x(draft[0], 1.0), K, L, N, W)
    assert _paths(tree) == want


@pytest.mark.parametrize("seed,V,K,L,N", [(2010, 200, 8, 16, 64), (2011, 500, 4, 6, 100), (2012, 64, 2, 10, 40)])
def test_wide_frontier_is_the_heap_tree(orc, seed, V, K, L, N):
    rng = np.random.default_rng(seed)
    draft = (3.0 * rng.standard_normal((3, L, V))).astype(np.float32)
    heap = orc.plan(draft, 1.0, N, K, L)
    for W in (N, N + 7):
        ept = orc.plan_expand(draft, 1.0, N, K, L, W)
        for k in TREE_KEYS:
            assert np.array_equal(heap[k], ept[k]), k
        assert np.array_equal(heap["score"], ept["score"])


@pytest.mark.parametrize("W", [1, 2, 4, 10])
def test_narrow_frontier_never_beats_the_heap(orc, W):
    """The heap keeps the N most probable paths of the whole tree and expand-then-prune the N
    most probable of a subset, so its i-th path probability is at most the heap's."""
    rng = np.random.default_rng(30 + W)
    V, K, L, N = 300, 8, 16, 64
    draft = (3.0 * rng.standard_normal((4, L, V))).astype(np.float32)
    heap = orc.plan(draft, 1.0, N, K, L)
    ept = orc.plan_expand(draft, 1.0, N, K, L, W)
    for b in range(4):
        _check_tree(ept, K, L, b)
        assert np.all(ept["score"][b] <= heap["score"][b] + 1e-12)
        # only frontier members have children: at most W parents per depth
        dep, par = ept["depth"][b], ept["parent"][b]
        for d in range(1, L):
            assert len({int(p) for i, p in enumerate(par) if i > 0 and dep[i] == d + 1}) <= W


def test_expand_k1_is_top1_chain(orc):
    rng = np.random.default_rng(4)
    V, L = 64, 6
    draft = rng.standard_normal((2, L, V)).astype(np.float32)
    tree = orc.plan_expand(draft, 1.0, L, 1, L, 1)
    for b in range(2):
        assert list(tree["parent"][b]) == [-1] + list(range(L))
        assert list(tree["plan_token"][b, 1:]) == [int(np.argmax(draft[b, d])) for d in range(L)]


def test_expand_rejects_budget_above_generated_nodes(orc):
    draft = np.zeros((1, 3, 8), dtype=np.float32)
    # K=2, W=1: 2 + 2 + 2 = 6 candidates
    with pytest.raises(RuntimeError):
        orc.plan_expand(draft, 1.0, 7, 2, 3, 1)
    orc.plan_expand(draft, 1.0, 6, 2, 3, 1)


def test_expand_small_enumeration_is_exhaustive(orc):
    """K=2, L=3, W=1: the generated set is the root's children, the best one's children and the
    best grandchild's children; check against all 14 paths filtered by that rule."""
    rng = np.random.default_rng(8)
    V, K, L = 12, 2, 3
    draft = (1.5 * rng.standard_normal((1, L, V))).astype(np.float32)
    x = _x(draft[0], 1.0)
    sk, _, key = _order(x, K, L)
    all_paths = [p for d in range(1, L + 1) for p in itertools.product(range(K), repeat=d)]
    best1 = max([(0,), (1,)], key=key)
    best2 = max([best1 + (0,), best1 + (1,)], key=key)
    gen = [p for p in all_paths if len(p) == 1 or p[:-1] in (best1, best2)]
    gen.sort(key=sk)
    for N in range(1, 7):
        tree = orc.plan_expand(draft, 1.0, N, K, L, 1)
        assert _paths(tree) == gen[:N]
