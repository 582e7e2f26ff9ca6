"""The pooled verifier's representation of the residual (CPU, fp64). With a pooled draft law q
(zero outside a pool of P tokens), recursive rejection sampling (Sec. 2.3, App. A; q normalised
within the pool, Sec. 3.3) never changes the target law outside the pool except by the common
normalisation: after any number of rejections the current law is p(v) * out / mout for v
outside the pool, where mout is the target mass outside the pool and out the current one. The
GPU walk therefore keeps only the P pool entries and `out`; here that form is checked against
the recursion over the whole vocabulary: the same acceptance decisions for the same uniforms,
and the same final residual (children inside the pool, and children outside it, which have
draft probability 0 and are accepted)."""
import numpy as np
import pytest


def _full(p, q, ys, us):
    """The recursion over all V tokens: accept test, residual, renormalisation."""
    P, t, drawn = p.copy(), 1.0, np.zeros(len(p), bool)
    for i, (y, u) in enumerate(zip(ys, us)):
        qp = q[y] / t if (q[y] > 0 and t > 0) else 0.0
        if u * qp < P[y]:
            return "accept", i, None
        R = np.maximum(P - np.where(drawn, 0.0, q / t), 0.0)
        Z = R.sum()
        if not Z > 0:
            return "degenerate", i, None
        if i == len(ys) - 1:
            return "residual", i, R
        P, drawn[y], t = R / Z, True, t - q[y]
    raise AssertionError("unreachable")


def _pooled(p, pool, qp_pool, ys, us):
    """The GPU walk's form: pool entries explicitly, the rest as one mass `out`."""
    inpool = np.zeros(len(p), bool)
    inpool[pool] = True
    mout = p[~inpool].sum()
    cur, out, t, drawn = p[pool].copy(), mout, 1.0, np.zeros(len(pool), bool)
    for i, (y, u) in enumerate(zip(ys, us)):
        hit = np.nonzero(pool == y)[0]
        if len(hit):
            k = hit[0]
            qk, pk = qp_pool[k], cur[k]
        else:
            k, qk, pk = -1, 0.0, (out / mout) * p[y] if mout > 0 else 0.0
        qp = qk / t if (qk > 0 and t > 0) else 0.0
        if u * qp < pk:
            return "accept", i, None
        R = np.maximum(cur - np.where(drawn, 0.0, qp_pool / t), 0.0)
        Z = R.sum() + out
        if not Z > 0:
            return "degenerate", i, None
        if i == len(ys) - 1:
            w = p * (out / mout if mout > 0 else 0.0)
            w[pool] = R
            return "residual", i, w
        cur, out = R / Z, out / Z
        if k >= 0:
            drawn[k] = True
        t -= qk
    raise AssertionError("unreachable")


@pytest.mark.parametrize("seed", range(10))
def test_pooled_form_matches_full_recursion(seed):
    rng = np.random.default_rng(100 + seed)
    checked = {"accept": 0, "residual": 0}
    for _ in range(300):
        V = int(rng.integers(5, 60))
        P = int(rng.integers(1, min(V, 32) + 1))
        m = int(rng.integers(1, P + 1))
        xt = 2.0 * rng.standard_normal(V)
        xq = xt + rng.standard_normal(V)
        p = np.exp(xt - xt.max())
        p /= p.sum()
        pool = np.lexsort((np.arange(V), -xq))[:P]
        qp_pool = np.exp(xq[pool] - xq[pool].max())
        qp_pool /= qp_pool.sum()
        q = np.zeros(V)
        q[pool] = qp_pool
        ys = list(rng.choice(pool, size=m, replace=False))
        if P < V and rng.random() < 0.2:  # a child outside the pool (draft probability 0)
            ys[-1] = int(rng.choice(np.setdiff1d(np.arange(V), pool)))
        us = rng.random(m)
        a, b = _full(p, q, ys, us), _pooled(p, pool, qp_pool, ys, us)
        assert a[:2] == b[:2]
        if a[2] is not None:
            np.testing.assert_allclose(b[2], a[2], rtol=1e-10, atol=1e-16)
        if a[0] in checked:
            checked[a[0]] += 1
    assert checked["accept"] > 0 and checked["residual"] > 0


def test_child_outside_the_pool_is_accepted():
    """q(y) = 0 for a token outside the pool: U * 0 < p(y) holds whenever p(y) > 0."""
    rng = np.random.default_rng(7)
    V, P = 20, 4
    xt = rng.standard_normal(V)
    p = np.exp(xt - xt.max())
    p /= p.sum()
    pool = np.arange(P)
    qp_pool = np.full(P, 1.0 / P)
    q = np.zeros(V)
    q[pool] = qp_pool
    for u in (1e-9, 0.5, 1 - 1e-9):
        assert _full(p, q, [P + 3], [u])[0] == "accept"
        assert _pooled(p, pool, qp_pool, [P + 3], [u])[0] == "accept"
