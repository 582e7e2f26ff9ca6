"""Pins of the oracle's traversal verification (sequence-level recursive rejection sampling
with WoR candidates; Weng et al. 2025 as cited in Sec. 2.3, Table 2 and App. A), CPU only.

1. Exact enumeration over every WoR token assignment of small trees of several shapes, with
   prefix-dependent target and draft laws: the emitted sequence, extended by target sampling
   to the tree's depth + 1, has the target law (losslessness). Dropping the sequence-weight
   update (a plausible slip) fails this check.
2. On a chain the law equals block verification's (tau = the deepest accepted position), and
   on a star it equals token-wise recursive rejection sampling's: both are pinned on their own.
3. The sampler follows the exact law: chi-square of (accepted node, final token) over 1e5
   seeded trials, in one vocabulary chunk and across chunks.
4. Whole sampled paths (plan -> replay -> traversal) with path-keyed targets: chi-square of
   the first token and of the first two tokens (extended by target sampling).
5. Expected emitted length of traversal >= recursive rejection sampling's on the same trees
   (the sequence-level gain the paper reports in Table 2 / Sec. 4.2), by exact enumeration.
"""
import itertools

import numpy as np
import pytest

import helpers
from paper_2609_33652_gb300 import synth

P_MIN = 1e-4


def _tree_from_parents(parents):
    """child_off / child_ids / depth of a tree whose nodes are numbered so parent[i] < i; the
    children of u in slot order are its children by increasing id."""
    NN = len(parents)
    kids = [[] for _ in range(NN)]
    for i in range(1, NN):
        kids[parents[i]].append(i)
    off = [0]
    ids = []
    for u in range(NN):
        ids.extend(kids[u])
        off.append(len(ids))
    depth = [0] * NN
    for i in range(1, NN):
        depth[i] = depth[parents[i]] + 1
    return np.array(off, dtype=np.int32), np.array(ids, dtype=np.int32), depth, kids


def _random_laws(rng, V, D, scale=1.5):
    """Target laws P[prefix] for prefixes of length <= D and draft laws Q[prefix] for < D."""
    P, Q = {}, {}
    for n in range(D + 1):
        for pre in itertools.product(range(V), repeat=n):
            P[pre] = helpers.softmax64(scale * rng.standard_normal(V))
            if n < D:
                Q[pre] = helpers.softmax64(scale * rng.standard_normal(V))
    return P, Q


def _assignments(kids, Q, V):
    """Every WoR token assignment of the tree (parents fill their children's slots in order)
    with its probability: yields (tokens, paths, prob)."""
    NN = len(kids)
    parents_with_kids = [u for u in range(NN) if kids[u]]

    def rec(k, tokens, paths, prob):
        if k == len(parents_with_kids):
            yield list(tokens), dict(paths), prob
            return
        u = parents_with_kids[k]
        q = Q[paths[u]]
        for ys in itertools.permutations(range(V), len(kids[u])):
            w = helpers.wor_tuple_prob(q, ys)
            if w == 0.0:
                continue
            for c, y in zip(kids[u], ys):
                tokens[c] = y
                paths[c] = paths[u] + (y,)
            yield from rec(k + 1, tokens, paths, prob * w)

    yield from rec(0, [-1] * NN, {0: ()}, 1.0)


def _emitted_law(orc, parents, V, P, Q, law_fn=None):
    """{emitted sequence: probability} of traversal verification over every assignment."""
    off, ids, depth, kids = _tree_from_parents(parents)
    NN = len(parents)
    out = {}
    for tokens, paths, prob in _assignments(kids, Q, V):
        Prow = np.array([P[paths[u]] for u in range(NN)])
        Qrow = np.array([Q[paths[u]] if kids[u] else np.full(V, 1.0 / V) for u in range(NN)])
        acc, law, deg = (law_fn or orc.traversal_law)(off, ids, np.array(tokens, dtype=np.int32), Prow, Qrow)
        assert not deg
        for u in range(NN):
            if acc[u] == 0.0:
                continue
            for f in range(V):
                key = paths[u] + (f,)
                out[key] = out.get(key, 0.0) + prob * acc[u] * law[u, f]
    return out, max(depth)


def _extended_error(out, P, V, D):
    """max over z in V^(D+1) of |extended emitted law - target law|."""
    err = 0.0
    for z in itertools.product(range(V), repeat=D + 1):
        want = 1.0
        for k in range(D + 1):
            want *= P[z[:k]][z[k]]
        got = 0.0
        for n in range(1, D + 2):
            e = z[:n]
            if e in out:
                ext = 1.0
                for k in range(n, D + 1):
                    ext *= P[z[:k]][z[k]]
                got += out[e] * ext
        err = max(err, abs(got - want))
    return err


TREES = {
    "chain3": [-1, 0, 1, 2],
    "star3": [-1, 0, 0, 0],
    "two_levels": [-1, 0, 0, 1, 1, 2],       # root {1, 2}, 1 {3, 4}, 2 {5}
    "deep_branch": [-1, 0, 1, 1, 2],         # root {1}, 1 {2, 3}, 2 {4}
    "wide_root": [-1, 0, 0, 0, 1, 3],        # root {1, 2, 3}, 1 {4}, 3 {5}
}


@pytest.mark.parametrize("name,V,seed", [("chain3", 3, 1), ("star3", 4, 2), ("two_levels", 4, 3),
                                         ("deep_branch", 4, 4), ("wide_root", 4, 5), ("two_levels", 3, 6)])
def test_traversal_is_lossless_by_enumeration(orc, name, V, seed):
    parents = TREES[name]
    _, _, depth, _ = _tree_from_parents(parents)
    rng = np.random.default_rng(seed)
    P, Q = _random_laws(rng, V, max(depth))
    out, D = _emitted_law(orc, parents, V, P, Q)
    assert abs(sum(out.values()) - 1.0) < 1e-12
    assert _extended_error(out, P, V, D) < 1e-12


def test_enumeration_sees_a_dropped_weight_update(orc):
    """The same enumeration applied to a variant that keeps p_a(u) after a rejected subtree
    (only the residual law is updated) is not lossless: the check has the power to see it."""

    def law_without_pa_update(off, ids, tokens, Prow, Qrow):
        NN, V = Prow.shape
        acc = np.zeros(NN)
        law = np.zeros((NN, V))

        def visit(u, pa, reach):
            Mb, Qu, t, drawn = Prow[u].copy(), Qrow[u], 1.0, np.zeros(V, dtype=bool)
            cont, rejected, R = reach, False, None
            for c in ids[off[u]:off[u + 1]]:
                y = tokens[c]
                qy = 0.0 if drawn[y] else Qu[y] / t
                w = min(pa * Mb[y] / qy, 1.0) if qy > 0 else 1.0
                cont = visit(c, w, cont)
                rejected = True
                qv = np.where(drawn, 0.0, Qu / t)
                R = np.maximum(pa * Mb - qv, 0.0)
                Mb = R / max(R.sum(), 1e-300)  # p_a(u) is not updated: the slip
                drawn[y] = True
                t -= Qu[y]
            pacc = 1.0 if u == 0 else pa
            acc[u] += cont * pacc
            law[u] = Prow[u] if not rejected else R / max(R.sum(), 1e-300)
            return cont * (1.0 - pacc)

        visit(0, 1.0, 1.0)
        return acc, law, False

    parents = TREES["deep_branch"]
    rng = np.random.default_rng(4)
    P, Q = _random_laws(rng, 4, 3)
    out, D = _emitted_law(orc, parents, 4, P, Q, law_fn=law_without_pa_update)
    assert _extended_error(out, P, 4, D) > 1e-3


@pytest.mark.parametrize("g,V,seed", [(1, 5, 11), (2, 4, 12), (4, 6, 13), (6, 8, 14)])
def test_chain_is_block_verification(orc, g, V, seed):
    rng = np.random.default_rng(seed)
    for _ in range(5):
        Mb = np.array([helpers.softmax64(1.5 * rng.standard_normal(V)) for _ in range(g + 1)])
        Ms = np.array([helpers.softmax64(1.5 * rng.standard_normal(V)) for _ in range(g)])
        X = rng.integers(0, V, g).astype(np.int32)
        w, h, resid = orc.blockv_law(Mb, Ms, X)
        off, ids, _, _ = _tree_from_parents([-1] + list(range(g)))
        tokens = np.array([-1] + list(X), dtype=np.int32)
        Qrow = np.vstack([Ms, np.full((1, V), 1.0 / V)])
        acc, law, deg = orc.traversal_law(off, ids, tokens, Mb, Qrow)
        assert not deg
        for t in range(g + 1):  # P(tau = t) = h_t prod_{j > t} (1 - h_j), h_0 = 1
            pt = (h[t] if t >= 1 else 1.0) * np.prod(1.0 - h[t + 1:])
            assert acc[t] == pytest.approx(pt, abs=1e-13)
            if pt > 1e-12:
                want = Mb[g] if t == g else resid[t] / resid[t].sum()
                np.testing.assert_allclose(law[t], want, atol=1e-12)


@pytest.mark.parametrize("m,V,seed", [(1, 6, 21), (2, 5, 22), (4, 8, 23)])
def test_star_is_recursive_rejection_sampling(orc, m, V, seed):
    rng = np.random.default_rng(seed)
    for _ in range(5):
        P = helpers.softmax64(2.0 * rng.standard_normal(V))
        Q = helpers.softmax64(2.0 * rng.standard_normal(V))
        ys = rng.choice(V, m, replace=False).astype(np.int32)
        a_rrs, fin, _ = orc.rrs_node_law(P, Q, ys)
        off, ids, _, _ = _tree_from_parents([-1] + [0] * m)
        Prow = np.vstack([P] + [helpers.softmax64(rng.standard_normal(V)) for _ in range(m)])
        Qrow = np.vstack([Q] + [np.full(V, 1.0 / V)] * m)
        acc, law, _ = orc.traversal_law(off, ids, np.array([-1] + list(ys), dtype=np.int32), Prow, Qrow)
        reach = 1.0
        for i in range(m):
            assert acc[1 + i] == pytest.approx(reach * a_rrs[i], abs=1e-14)
            if acc[1 + i] > 0:
                np.testing.assert_allclose(law[1 + i], Prow[1 + i], atol=1e-15)  # bonus rows
            reach *= 1.0 - a_rrs[i]
        assert acc[0] == pytest.approx(reach, abs=1e-14)
        if reach > 1e-12:
            np.testing.assert_allclose(law[0], fin, atol=1e-12)


@pytest.mark.parametrize("V", [6, 300])
def test_sampler_follows_the_exact_law(orc, V):
    """1e5 trees share one topology, token assignment and rows (batch stride 0); each tree
    draws its own uniforms. The joint law of (accepted node, final token) is acc * law."""
    B = 100_000
    parents = TREES["two_levels"]
    off, ids, depth, kids = _tree_from_parents(parents)
    NN = len(parents)
    rng = np.random.default_rng(31 + V)
    zt = (1.2 * rng.standard_normal((1, NN, V))).astype(np.float32)
    zq = (1.2 * rng.standard_normal((1, NN, V))).astype(np.float32)
    tokens = np.array([-1, 0, 1, 2, 3, 4], dtype=np.int32)  # distinct siblings
    tree = {"parent": np.array([parents], dtype=np.int32), "depth": np.array([depth], dtype=np.int32),
            "child_off": off[None], "child_ids": ids[None]}
    treeB = helpers.repeat_tree(tree, B)
    tokB = np.repeat(tokens[None], B, axis=0)
    qidx = np.repeat(np.arange(NN, dtype=np.int32)[None], B, axis=0)
    target = np.broadcast_to(zt, (B, NN, V))
    q = np.broadcast_to(zq, (B, NN, V))
    out = orc.verify_traversal(target, q, 1.0, treeB, tokB, 7, 2, qrow_of_node=qidx)
    Prow = np.array([helpers.softmax64(zt[0, u].astype(np.float64)) for u in range(NN)])
    Qrow = np.array([helpers.softmax64(zq[0, u].astype(np.float64)) for u in range(NN)])
    acc, law, _ = orc.traversal_law(off, ids, tokens, Prow, Qrow)
    n = out["len"] - 1
    node = np.where(n > 0, out["nodes"][np.arange(B), np.maximum(n - 1, 0)], 0)
    fin = out["tokens"][np.arange(B), n]
    counts = np.bincount(node * V + fin, minlength=NN * V)
    expect = (acc[:, None] * law).ravel()
    assert helpers.chi2_pvalue(counts, expect) > P_MIN
    # the emitted prefix is the accepted node's path with its replayed tokens
    for b in range(100):
        a, k = node[b], n[b] - 1
        while a != 0:
            assert out["nodes"][b, k] == a and out["tokens"][b, k] == tokens[a]
            a, k = parents[a], k - 1
        assert k == -1
    assert out["exempt"].mean() < 1e-3


def _rrs_expected_len(orc, u, kids, tokens, Prow, Qrow):
    if not kids[u]:
        return 1.0
    ys = [tokens[c] for c in kids[u]]
    a, _, _ = orc.rrs_node_law(Prow[u], Qrow[u], np.array(ys, dtype=np.int32))
    e, reach = 0.0, 1.0
    for i, c in enumerate(kids[u]):
        e += reach * a[i] * (1.0 + _rrs_expected_len(orc, c, kids, tokens, Prow, Qrow))
        reach *= 1.0 - a[i]
    return e + reach


@pytest.mark.parametrize("name,V,seed", [("two_levels", 4, 41), ("deep_branch", 4, 42), ("wide_root", 3, 43),
                                         ("chain3", 4, 44)])
def test_traversal_accepts_at_least_as_much_as_rrs(orc, name, V, seed):
    parents = TREES[name]
    off, ids, depth, kids = _tree_from_parents(parents)
    NN = len(parents)
    rng = np.random.default_rng(seed)
    P, Q = _random_laws(rng, V, max(depth), scale=1.0)
    e_trav = e_rrs = 0.0
    for tokens, paths, prob in _assignments(kids, Q, V):
        Prow = np.array([P[paths[u]] for u in range(NN)])
        Qrow = np.array([Q[paths[u]] if kids[u] else np.full(V, 1.0 / V) for u in range(NN)])
        acc, _, _ = orc.traversal_law(off, ids, np.array(tokens, dtype=np.int32), Prow, Qrow)
        e_trav += prob * float(np.dot(acc, np.array(depth) + 1))
        e_rrs += prob * _rrs_expected_len(orc, 0, kids, tokens, Prow, Qrow)
    assert e_trav >= e_rrs - 1e-12


# --------------------------------------------------------------------------------------
@pytest.mark.parametrize("T", [1.0, 0.6])
def test_sampled_path_is_lossless(orc, T):
    """Plan -> replay -> traversal on the tiny workload, 1e5 trials, targets keyed by the token
    path (a function of the prefix): the first token follows the root target law, and the first
    two tokens (the second drawn from the target when only one was emitted) follow the joint
    target law."""
    w = synth.WORKLOADS["tiny"]
    B, V, L = 100_000, w["V"], w["L"]
    draft = synth.to_host(synth.draft_logits(1, L, V, "normal2", "f32", 1000))
    tree = helpers.repeat_tree(orc.plan(draft, T, w["N"], w["K"], L), B)
    qb = np.broadcast_to(draft, (B,) + draft.shape[1:])
    tok, _ = orc.replay(qb, T, tree, 103)
    base = draft[0]
    target = synth.path_keyed_rows(base, tree["parent"], tree["depth"], tok, 1.0, seed=77)
    out = orc.verify_traversal(target, qb, T, tree, tok, 103, L)
    inv = np.float32(np.float32(1.0) / np.float32(T))

    def p_after(prefix):
        return helpers.softmax64(synth.path_keyed_row(base, list(prefix), 1.0, 77) * inv)

    first = out["tokens"][:, 0]
    p_root = p_after([])
    assert helpers.chi2_pvalue(np.bincount(first, minlength=V), p_root) > P_MIN
    second = out["tokens"][:, 1].copy()
    ext = np.random.default_rng(5)
    for b in np.nonzero(out["len"] == 1)[0]:
        second[b] = ext.choice(V, p=p_after([first[b]]))
    joint = np.bincount(first * V + second, minlength=V * V)
    want = np.concatenate([p_root[a] * p_after([a]) for a in range(V)])
    assert helpers.chi2_pvalue(joint, want) > P_MIN
    assert out["exempt"].mean() < 1e-3
