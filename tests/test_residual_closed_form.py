"""The verifier's residual in closed form (CPU, fp64). Recursive rejection sampling with
candidates drawn without replacement updates, after rejecting candidate y_i,
    p_{i+1} = max(p_i - q_i, 0) / Z_{i+1},   q_{i+1} = q_i without y_i, renormalised
(Sec. 2.3, App. A). Because subtracting non-negative multiples of q and clamping at zero
compose, p_i = max(P0 - A_i q, 0) / D_i with A_0 = 0, D_0 = 1, A_{i+1} = A_i + D_i / t_i,
D_{i+1} = sum max(P0 - A_{i+1} q, 0) and t_i = 1 - (mass of the drawn candidates). The CUDA
walk uses that form; here it is checked against the recursion as the paper states it."""
import numpy as np
import pytest


def _recursion(p0, q, drawn):
    """p_i for i = 0..len(drawn) by the recursive definition (drawn tokens leave q)."""
    ps, p, qi = [p0], p0.copy(), q.copy()
    for y in drawn:
        r = np.maximum(p - qi, 0.0)
        p = r / r.sum()
        qi = qi.copy()
        qi[y] = 0.0
        qi = qi / qi.sum()
        ps.append(p)
    return ps


def _closed_form(p0, q, drawn):
    ps, A, D, t = [p0], 0.0, 1.0, 1.0
    for y in drawn:
        A = A + D / t
        r = np.maximum(p0 - A * q, 0.0)
        D = r.sum()
        t -= q[y]
        ps.append(r / D)
    return ps


@pytest.mark.parametrize("seed", range(20))
def test_closed_form_matches_recursion(seed):
    rng = np.random.default_rng(seed)
    V = int(rng.integers(8, 400))
    p0 = rng.dirichlet(np.full(V, rng.uniform(0.05, 2.0)))
    q = rng.dirichlet(np.full(V, rng.uniform(0.05, 2.0)))
    m = int(rng.integers(1, 9))
    # candidates a rejection can follow: drawn without replacement from q, each with p_i < q_i
    drawn, ps = [], [p0]
    qi = q.copy()
    for _ in range(m):
        cand = [v for v in range(V) if v not in drawn and ps[-1][v] < qi[v]]
        if not cand:
            break
        y = int(rng.choice(cand))
        drawn.append(y)
        ps = _recursion(p0, q, drawn)
        qi = q.copy()
        qi[drawn] = 0.0
        qi /= qi.sum()
    rec, cf = _recursion(p0, q, drawn), _closed_form(p0, q, drawn)
    for a, b in zip(rec, cf):
        np.testing.assert_allclose(b, a, rtol=1e-9, atol=1e-15)
    for i, y in enumerate(drawn):  # a rejected candidate keeps zero residual
        for p in cf[i + 1:]:
            assert p[y] == 0.0


def test_closed_form_needs_the_rejection_condition():
    """The composition uses that a rejected candidate had p_i(y) < q_i(y): the recursion then
    zeroes it. For an accepted-or-rejected-at-random token with p_i(y) >= q_i(y) the two forms
    differ (the recursion would exclude it from q only), so the walk applies the closed form
    only after a rejection, where the acceptance test guarantees the condition."""
    p0 = np.array([0.5, 0.3, 0.2])
    q = np.array([0.4, 0.1, 0.5])
    # token 0 has p0 >= q (never rejected in a real walk), then token 2 is a valid rejection
    rec, cf = _recursion(p0, q, [0, 2]), _closed_form(p0, q, [0, 2])
    np.testing.assert_allclose(rec[2], [0.4, 0.6, 0.0])
    np.testing.assert_allclose(cf[2], [0.0, 1.0, 0.0])
