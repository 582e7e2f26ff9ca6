"""Pins of the oracle's planner (first pass, Sec. 3.1 / App. B.3), CPU only.

The planner's pop order is checked against a brute-force enumeration of every path of the
(K, L) tree, sorted with scores computed independently (scipy logsumexp) and exact
(fractional) comparison of same-depth candidates. The optimality claim of App. B.3
(max summed path probability under the node budget) is checked by exhaustive search over
prefix-closed node sets.
"""
import functools
import itertools
from fractions import Fraction

import numpy as np
import pytest
from scipy.special import logsumexp


def _x(draft, T):
    return draft.astype(np.float32) * np.float32(np.float32(1.0) / np.float32(T))


def _topk(x, K):
    order = np.lexsort((np.arange(len(x)), -x.astype(np.float64)))  # (x desc, id asc)
    return order[:K]


def _brute_force(draft_row_x, K, L, N):
    """All paths (rank tuples) sorted by the contract's order; the first N."""
    lse = [logsumexp(draft_row_x[d].astype(np.float64)) for d in range(L)]
    top = [_topk(draft_row_x[d], K) for d in range(L)]
    paths = []
    for d in range(1, L + 1):
        paths.extend(itertools.product(range(K), repeat=d))

    def xs(p):
        return [float(draft_row_x[j][top[j][r]]) for j, r in enumerate(p)]

    def logprob(p):
        return sum(x - lse[j] for j, x in enumerate(xs(p)))

    def exact_sum(p):
        return sum(Fraction(v) for v in xs(p))

    @functools.lru_cache(maxsize=None)
    def key(p):
        return logprob(p)

    def cmp(a, b):
        if a == b:
            return 0
        if len(a) != len(b):
            ka, kb = key(a), key(b)
            assert abs(ka - kb) > 1e-9, "cross-depth near tie: choose another seed"
            return -1 if ka > kb else 1
        sa, sb = exact_sum(a), exact_sum(b)
        if sa != sb:
            return -1 if sa > sb else 1
        c = cmp(a[:-1], b[:-1]) if len(a) > 1 else 0
        if c != 0:
            return c
        return -1 if a[-1] < b[-1] else 1

    paths.sort(key=functools.cmp_to_key(cmp))
    return paths[:N], top


def _oracle_paths(tree, b=0):
    NN = tree["parent"].shape[1]
    path = {0: ()}
    out = []
    for i in range(1, NN):
        p = int(tree["parent"][b, i])
        assert p < i
        path[i] = path[p] + (int(tree["rank"][b, i]),)
        out.append(path[i])
    return out


def _check_invariants(tree, K, L, b=0):
    par, dep, rk = tree["parent"][b], tree["depth"][b], tree["rank"][b]
    NN = len(par)
    off, ids = tree["child_off"][b], tree["child_ids"][b]
    assert off[0] == 0 and off[-1] == NN - 1
    for u in range(NN):
        ch = list(ids[off[u]:off[u + 1]])
        assert ch == sorted(ch)
        assert ch == [i for i in range(1, NN) if par[i] == u]
        assert [int(rk[c]) for c in ch] == list(range(len(ch)))  # siblings are ranks 0..m-1
        for c in ch:
            assert dep[c] == dep[u] + 1 and dep[c] <= L
        assert len(ch) <= K
    sc = tree["score"][b]
    assert np.all(np.diff(sc[1:]) <= 0.0)  # pops come out in non-increasing score


@pytest.mark.parametrize("seed,V,K,L,N", [(1000, 32, 4, 4, 8), (1001, 32, 4, 4, 40), (1002, 40, 3, 3, 39),
                                          (1003, 300, 5, 4, 60)])
def test_plan_matches_brute_force(orc, seed, V, K, L, N):
    rng = np.random.default_rng(seed)
    draft = (2.0 * rng.standard_normal((1, L, V))).astype(np.float32)
    tree = orc.plan(draft, 1.0, N, K, L)
    want, top = _brute_force(_x(draft[0], 1.0), K, L, N)
    assert _oracle_paths(tree) == want
    _check_invariants(tree, K, L)
    # planning tokens are the ranked candidates of the depth's row
    for i in range(1, N + 1):
        d, r = tree["depth"][0, i], tree["rank"][0, i]
        assert tree["plan_token"][0, i] == top[d - 1][r]


def test_plan_with_exact_ties(orc):
    """Integer logits make many same-depth paths tie exactly: the order must follow the
    tie rule (parent popped earlier first, then rank)."""
    rng = np.random.default_rng(7)
    V, K, L, N = 16, 3, 4, 60
    draft = rng.integers(-3, 4, size=(1, L, V)).astype(np.float32)
    tree = orc.plan(draft, 1.0, N, K, L)
    want, _ = _brute_force(_x(draft[0], 1.0), K, L, N)
    assert _oracle_paths(tree) == want
    _check_invariants(tree, K, L)


def test_plan_temperature(orc):
    rng = np.random.default_rng(11)
    V, K, L, N = 50, 4, 3, 20
    draft = (2.0 * rng.standard_normal((1, L, V))).astype(np.float32)
    tree = orc.plan(draft, 0.6, N, K, L)
    want, _ = _brute_force(_x(draft[0], 0.6), K, L, N)
    assert _oracle_paths(tree) == want


def test_plan_k1_is_top1_chain(orc):
    rng = np.random.default_rng(3)
    V, L = 64, 6
    draft = rng.standard_normal((2, L, V)).astype(np.float32)
    tree = orc.plan(draft, 1.0, L, 1, L)
    for b in range(2):
        assert list(tree["parent"][b]) == [-1] + list(range(L))
        assert list(tree["plan_token"][b, 1:]) == [int(np.argmax(draft[b, d])) for d in range(L)]


def test_plan_maximises_summed_path_probability(orc):
    """App. B.3: the max-heap set has the largest summed draft path probability among all
    prefix-closed node sets of the same size (exhaustive search)."""
    rng = np.random.default_rng(5)
    V, K, L = 12, 2, 3
    draft = (1.5 * rng.standard_normal((1, L, V))).astype(np.float32)
    x = _x(draft[0], 1.0)
    lse = [logsumexp(x[d].astype(np.float64)) for d in range(L)]
    top = [_topk(x[d], K) for d in range(L)]
    paths = [p for d in range(1, L + 1) for p in itertools.product(range(K), repeat=d)]

    def prob(p):
        return float(np.exp(sum(float(x[j][top[j][r]]) - lse[j] for j, r in enumerate(p))))

    for N in range(1, 8):
        best = 0.0
        for subset in itertools.combinations(paths, N):
            s = set(subset)
            if all(p[:-1] in s or len(p) == 1 for p in subset):
                best = max(best, sum(prob(p) for p in subset))
        tree = orc.plan(draft, 1.0, N, K, L)
        got = sum(prob(p) for p in _oracle_paths(tree))
        assert got == pytest.approx(best, rel=1e-12)


def test_plan_rejects_oversized_budget(orc):
    draft = np.zeros((1, 2, 8), dtype=np.float32)
    with pytest.raises(RuntimeError):
        orc.plan(draft, 1.0, 7, 2, 2)  # 2 + 4 = 6 nodes at most
    orc.plan(draft, 1.0, 6, 2, 2)


def test_plan_bf16_input(orc):
    """bf16 bit patterns are widened exactly: same plan as the same values in fp32."""
    rng = np.random.default_rng(9)
    f = (3.0 * rng.standard_normal((2, 4, 500))).astype(np.float32)
    bits = (f.view(np.uint32) >> 16).astype(np.uint16)  # truncation to a bf16 value
    f_exact = (bits.astype(np.uint32) << 16).view(np.float32)
    t1 = orc.plan(bits, 1.0, 30, 4, 4)
    t2 = orc.plan(np.ascontiguousarray(f_exact), 1.0, 30, 4, 4)
    for k in ("parent", "rank", "plan_token"):
        assert np.array_equal(t1[k], t2[k])
