"""Pins of the oracle's block verification of a sampled chain (Sun et al. 2025, cited in
Sec. 1, Table 2 and App. A), CPU only.

1. Exact enumeration over every chain X in V^g with prefix-dependent target and draft laws:
   the emitted sequence, extended by target sampling to length g+1, has the target law.
   (A stop-at-first-failure variant of the same weights fails this check, which shows the
   enumeration has the power to see a wrong acceptance rule.)
2. g = 1 is exactly token-wise rejection sampling (Eq. rs-overlap).
3. Optimality among chain verifiers: E[accepted] >= that of token-wise rejection sampling.
4. Sampled chain, 1e5 trials: chi-square of the first emitted token against the target.
"""
import itertools

import numpy as np
import pytest

import helpers
from paper_2609_33652_gb300 import synth

P_MIN = 1e-4


def _laws(rng, V, g):
    """Random prefix-dependent target Mb(.|prefix) for len <= g, draft Ms(.|prefix) for len < g."""
    Mb, Ms = {}, {}
    for n in range(g + 1):
        for pre in itertools.product(range(V), repeat=n):
            Mb[pre] = helpers.softmax64(1.5 * rng.standard_normal(V))
            if n < g:
                Ms[pre] = helpers.softmax64(1.5 * rng.standard_normal(V))
    return Mb, Ms


def _output_law(orc, Mb, Ms, V, g, rule="max"):
    """{emitted tuple: probability} by exact enumeration of X and of tau."""
    out = {}
    for X in itertools.product(range(V), repeat=g):
        px = 1.0
        for i in range(g):
            px *= Ms[X[:i]][X[i]]
        mb = np.array([Mb[X[:i]] for i in range(g + 1)])
        ms = np.array([Ms[X[:i]] for i in range(g)])
        w, h, resid = orc.blockv_law(mb, ms, X)
        ptau = np.zeros(g + 1)
        if rule == "max":  # tau = max{i >= 1 : eta_i <= h_i}, independent eta
            for t in range(g + 1):
                pt = h[t] if t >= 1 else 1.0
                for j in range(t + 1, g + 1):
                    pt *= 1.0 - h[j]
                ptau[t] = pt
        else:  # stop at the first failure
            run = 1.0
            for t in range(g + 1):
                nxt = h[t + 1] if t + 1 <= g else 0.0
                ptau[t] = run * (1.0 - nxt)
                run *= nxt
        for t in range(g + 1):
            if ptau[t] == 0.0:
                continue
            if t == g:
                ylaw = mb[g]
            else:
                s = resid[t].sum()
                ylaw = resid[t] / s if s > 0 else mb[t]
            for y in range(V):
                key = tuple(X[:t]) + (y,)
                out[key] = out.get(key, 0.0) + px * ptau[t] * ylaw[y]
    return out


def _extended_error(Mb, V, g, law):
    worst = 0.0
    for s in itertools.product(range(V), repeat=g + 1):
        target = 1.0
        for i in range(g + 1):
            target *= Mb[s[:i]][s[i]]
        got = 0.0
        for k in range(1, g + 2):
            pk = law.get(s[:k], 0.0)
            if pk == 0.0:
                continue
            ext = 1.0
            for i in range(k, g + 1):
                ext *= Mb[s[:i]][s[i]]
            got += pk * ext
        worst = max(worst, abs(got - target))
    return worst


@pytest.mark.parametrize("V,g,seed", [(3, 1, 1), (3, 2, 2), (4, 2, 3), (3, 3, 4), (5, 2, 5)])
def test_block_verification_is_lossless(orc, V, g, seed):
    rng = np.random.default_rng(seed)
    Mb, Ms = _laws(rng, V, g)
    assert _extended_error(Mb, V, g, _output_law(orc, Mb, Ms, V, g)) < 1e-12


def test_enumeration_detects_wrong_rule(orc):
    rng = np.random.default_rng(2)
    V, g = 3, 2
    Mb, Ms = _laws(rng, V, g)
    assert _extended_error(Mb, V, g, _output_law(orc, Mb, Ms, V, g, rule="first")) > 1e-3


def test_gamma1_is_rejection_sampling(orc):
    rng = np.random.default_rng(3)
    V = 9
    for _ in range(5):
        p = helpers.softmax64(rng.standard_normal(V))
        q = helpers.softmax64(rng.standard_normal(V))
        p1 = helpers.softmax64(rng.standard_normal(V))
        for x in range(V):
            w, h, resid = orc.blockv_law(np.array([p, p1]), np.array([q]), [x])
            assert h[1] == pytest.approx(min(1.0, p[x] / q[x]), rel=1e-15)
            r = np.maximum(p - q, 0.0)
            assert np.allclose(resid[0], r, atol=1e-16)
        # acceptance of a sampled token: sum_x q(x) min(1, p/q) = sum min(p, q)
        acc = sum(q[x] * orc.blockv_law(np.array([p, p1]), np.array([q]), [x])[1][1] for x in range(V))
        assert acc == pytest.approx(np.minimum(p, q).sum(), abs=1e-14)


def test_expected_length_not_below_tokenwise_rs(orc):
    rng = np.random.default_rng(4)
    V, g = 4, 3
    for _ in range(3):
        Mb, Ms = _laws(rng, V, g)
        law = _output_law(orc, Mb, Ms, V, g)
        e_bv = sum(p * (len(k) - 1) for k, p in law.items())
        e_rs = 0.0
        for X in itertools.product(range(V), repeat=g):
            px = 1.0
            for i in range(g):
                px *= Ms[X[:i]][X[i]]
            run = 1.0
            for i in range(g):
                run *= min(1.0, Mb[X[:i]][X[i]] / Ms[X[:i]][X[i]])
                e_rs += px * run
        assert e_bv >= e_rs - 1e-12


def test_sampled_chain_is_lossless(orc):
    B, V, g = 100_000, 16, 3
    rng = np.random.default_rng(6)
    draft = (1.5 * rng.standard_normal((1, g, V))).astype(np.float32)
    tree = helpers.chain_tree(g, B)
    qb = np.broadcast_to(draft, (B, g, V))
    tok, _ = orc.replay(qb, 1.0, tree, seed=11)
    base = np.concatenate([draft[0], draft[0, -1:]], axis=0)  # g+1 per-depth base rows
    target = synth.path_keyed_rows(base, tree["parent"], tree["depth"], tok, 1.0, seed=78)
    out = orc.verify_block(target, qb, 1.0, tree, tok, seed=11, L=g)
    p_root = helpers.softmax64(synth.path_keyed_row(base, [], 1.0, 78))
    first = out["tokens"][:, 0]
    assert helpers.chi2_pvalue(np.bincount(first, minlength=V), p_root) > P_MIN
    two = out["len"] >= 2
    vals, cnt = np.unique(first[two], return_counts=True)
    a = int(vals[np.argmax(cnt)])
    sel = two & (first == a)
    p_a = helpers.softmax64(synth.path_keyed_row(base, [a], 1.0, 78))
    assert helpers.chi2_pvalue(np.bincount(out["tokens"][sel, 1], minlength=V), p_a) > P_MIN
    assert np.all(out["tau"] == out["len"] - 1)
    assert out["exempt"].mean() < 1e-3
