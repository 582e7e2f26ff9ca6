"""Pins of the oracle's pooled draft laws (Sec. 3.1 and 3.2: the draft law of a position is
restricted to its P most probable tokens and normalised within them; Sec. 3.3: verification
uses those pooled probabilities, the residual stays full-vocabulary), CPU only.

Planner: brute-force path enumeration with pooled normalisers (scipy logsumexp over the top-P
logits), and P = V reduces to the full-vocabulary planner. Replay: chi-square of ordered draws
against the closed-form WoR law of the pooled q, tokens stay in the pool, and P = V is the flat
Gumbel-top-k sampler token for token. Verification: chi-square of the emitted token against the
target law (losslessness with pooled q), single-child acceptance sum min(p, q_pool), and P = V
is the full-vocabulary verifier.
"""
import functools
import itertools

import numpy as np
import pytest
from scipy.special import logsumexp

import helpers

TRIALS = 100_000
P_MIN = 1e-4


def _x(a, T=1.0):
    return a.astype(np.float32) * np.float32(np.float32(1.0) / np.float32(T))


def _top(x, k):
    return np.lexsort((np.arange(len(x)), -x.astype(np.float64)))[:k]


def _pooled_q(x, pool):
    q = np.zeros(len(x))
    xp = x[pool].astype(np.float64)
    q[pool] = np.exp(xp - logsumexp(xp))
    return q


def _tree_paths(tree, b=0):
    NN = tree["parent"].shape[1]
    path = {0: ()}
    out = []
    for i in range(1, NN):
        path[i] = path[int(tree["parent"][b, i])] + (int(tree["rank"][b, i]),)
        out.append(path[i])
    return out


@pytest.mark.parametrize("seed,V,K,L,N,P", [(3000, 32, 4, 4, 20, 6), (3001, 300, 3, 4, 30, 16), (3002, 64, 4, 3, 40, 4)])
def test_pooled_plan_matches_brute_force(orc, seed, V, K, L, N, P):
    rng = np.random.default_rng(seed)
    draft = (2.0 * rng.standard_normal((1, L, V))).astype(np.float32)
    tree = orc.plan(draft, 1.0, N, K, L, pool=P)
    x = _x(draft[0])
    lse = [logsumexp(x[d][_top(x[d], P)].astype(np.float64)) for d in range(L)]
    top = [_top(x[d], K) for d in range(L)]
    paths = [p for d in range(1, L + 1) for p in itertools.product(range(K), repeat=d)]

    def key(p):
        return sum(float(x[j][top[j][r]]) - lse[j] for j, r in enumerate(p))

    def cmp(a, b):  # distinct continuous logits: no exact ties
        ka, kb = key(a), key(b)
        if ka != kb:
            return -1 if ka > kb else 1
        return -1 if len(a) < len(b) else 1

    paths.sort(key=functools.cmp_to_key(cmp))
    assert _tree_paths(tree) == paths[:N]
    np.testing.assert_allclose(tree["score"][0, 1:], [key(p) for p in paths[:N]], rtol=1e-12, atol=1e-12)


def test_pool_of_the_whole_vocabulary_is_the_full_planner(orc):
    rng = np.random.default_rng(3003)
    V, K, L, N = 200, 8, 6, 60
    draft = (3.0 * rng.standard_normal((4, L, V))).astype(np.float32)
    full = orc.plan(draft, 1.0, N, K, L)
    pooled = orc.plan(draft, 1.0, N, K, L, pool=V)
    for k in ("parent", "depth", "rank", "plan_token", "child_off", "child_ids"):
        assert np.array_equal(full[k], pooled[k]), k
    np.testing.assert_allclose(full["score"], pooled["score"], rtol=1e-12, atol=1e-12)


def test_pooled_replay_law(orc):
    """Ordered WoR pairs from the pooled law of a star tree's root (chi-square over 1e5 seeds)."""
    rng = np.random.default_rng(3004)
    V, P, m = 32, 8, 3
    row = (2.0 * rng.standard_normal(V)).astype(np.float32)
    q = np.broadcast_to(row[None, None, :], (TRIALS, 1, V))
    tree = helpers.star_tree(m, TRIALS)
    pool = np.broadcast_to(_top(_x(row), P).astype(np.int32)[None, None, :], (TRIALS, 1, P))
    tok, ex = orc.replay_pooled(q, 1.0, tree, 7, pool)
    assert ex.mean() < 1e-3
    draws = tok[:, 1:]
    assert np.isin(draws, pool[0, 0]).all()
    assert (draws[:, 0] != draws[:, 1]).all() and (draws[:, 1] != draws[:, 2]).all()
    pl = pool[0, 0]
    qp = _pooled_q(_x(row), pl)
    assert helpers.chi2_pvalue(np.bincount(draws[:, 0], minlength=V)[pl], qp[pl]) > P_MIN
    # ordered pairs inside the pool: q(a) q(b) / (1 - q(a)), a != b
    pair = qp[pl][:, None] * qp[pl][None, :] / (1.0 - qp[pl][:, None])
    cnt = np.bincount(draws[:, 0] * V + draws[:, 1], minlength=V * V).reshape(V, V)[np.ix_(pl, pl)]
    off = ~np.eye(P, dtype=bool)
    assert helpers.chi2_pvalue(cnt[off], pair[off]) > P_MIN


def test_pool_of_the_whole_vocabulary_is_the_flat_sampler(orc):
    rng = np.random.default_rng(3005)
    V, K, L, N, B = 50, 4, 4, 24, 6
    draft = (2.0 * rng.standard_normal((B, L, V))).astype(np.float32)
    tree = orc.plan(draft, 1.0, N, K, L)
    pool = orc.pools(draft, 1.0, V)
    tok, _ = orc.replay_pooled(draft, 1.0, tree, 9, pool)
    flat = orc.replay(draft, 1.0, tree, 9, flat=True)
    assert np.array_equal(tok, flat)


def _star_target(base_row, m, B):
    return np.ascontiguousarray(np.broadcast_to(base_row[None, None, :], (B, m + 1, base_row.shape[0])))


@pytest.mark.parametrize("V,P,m", [(32, 6, 3), (40, 10, 1)])
def test_pooled_rrs_is_lossless(orc, V, P, m):
    """Pooled draft law, WoR children from it, full-vocabulary target: the first emitted token
    follows the target law (Prop. 1 with any draft law)."""
    rng = np.random.default_rng(3006 + m)
    drow = (2.0 * rng.standard_normal(V)).astype(np.float32)
    trow = (drow + rng.standard_normal(V)).astype(np.float32)
    B = TRIALS
    q = np.broadcast_to(drow[None, None, :], (B, 1, V))
    tree = helpers.star_tree(m, B)
    pool = np.ascontiguousarray(np.broadcast_to(_top(_x(drow), P).astype(np.int32)[None, None, :], (B, 1, P)))
    tok, _ = orc.replay_pooled(q, 1.0, tree, 11, pool)
    out = orc.verify_rrs(_star_target(trow, m, B), q, 1.0, tree, tok, 13, 1, pool_ids=pool)
    p = helpers.softmax64(_x(trow))
    assert helpers.chi2_pvalue(np.bincount(out["tokens"][:, 0], minlength=V), p) > P_MIN
    if m == 1:  # single candidate: acceptance probability sum_v min(p, q_pool) (Eq. rs-overlap)
        qp = _pooled_q(_x(drow), pool[0, 0])
        alpha = np.minimum(p, qp).sum()
        acc = (out["len"] == 2).mean()
        assert abs(acc - alpha) < 5 * np.sqrt(alpha * (1 - alpha) / B)


def test_pool_of_the_whole_vocabulary_is_the_full_verifier(orc):
    rng = np.random.default_rng(3008)
    V, K, L, N, B = 64, 4, 4, 20, 8
    draft = (2.0 * rng.standard_normal((B, L, V))).astype(np.float32)
    tree = orc.plan(draft, 1.0, N, K, L)
    tok, _ = orc.replay(draft, 1.0, tree, 3)
    idx = np.minimum(tree["depth"], L - 1)
    target = np.ascontiguousarray(np.take_along_axis(draft, idx[:, :, None], axis=1) +
                                  rng.standard_normal((B, N + 1, V)).astype(np.float32))
    full = orc.verify_rrs(target, draft, 1.0, tree, tok, 5, L)
    pooled = orc.verify_rrs(target, draft, 1.0, tree, tok, 5, L, pool_ids=orc.pools(draft, 1.0, V))
    ok = ~(full["exempt"] | pooled["exempt"])
    assert ok.mean() > 0.8
    for k in ("tokens", "nodes", "len"):
        assert np.array_equal(full[k][ok], pooled[k][ok]), k
