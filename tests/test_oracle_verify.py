"""Pins of the oracle's tree verifier (recursive rejection sampling, WoR variant; Sec. 2.3
Eq. rs-overlap, App. A, Prop. 1), CPU only.

1. Exact enumeration: for every ordered child tuple at a node, weight the per-tuple law of
   the emitted token by the closed-form WoR tuple probability; the sum must be the target
   law (losslessness) to rounding.
2. Closed form for one child: P(accept) = sum_v min(p(v), q(v)).
3. Whole sampled path (plan -> replay -> verify), 1e5 seeded trials with prefix-keyed
   target rows: chi-square of the first emitted token against the root target law and of
   the second token against the target law after the first.
"""
import itertools

import numpy as np
import pytest

import helpers
from paper_2609_33652_gb300 import synth

TRIALS = 100_000
P_MIN = 1e-4


def _emitted_law(orc, P, Q, m):
    V = len(P)
    total = np.zeros(V)
    for ys in itertools.permutations(range(V), m):
        w = helpers.wor_tuple_prob(Q, ys)
        if w == 0.0:
            continue
        acc, fin, deg = orc.rrs_node_law(P, Q, ys)
        assert not deg
        reach = 1.0
        for i, y in enumerate(ys):
            total[y] += w * reach * acc[i]
            reach *= 1.0 - acc[i]
        total += w * reach * fin
    return total


@pytest.mark.parametrize("V,m,seed", [(6, 1, 1), (6, 2, 2), (6, 3, 3), (8, 4, 4), (32, 2, 5), (5, 5, 6)])
def test_node_law_is_target_law(orc, V, m, seed):
    rng = np.random.default_rng(seed)
    P = helpers.softmax64(2.0 * rng.standard_normal(V))
    Q = helpers.softmax64(2.0 * rng.standard_normal(V))
    law = _emitted_law(orc, P, Q, m)
    assert np.max(np.abs(law - P)) < 1e-12


def test_node_law_peaked_draft(orc):
    """A draft far from the target (large rejection mass) still gives the target law."""
    V = 7
    P = helpers.softmax64(np.array([3.0, 0, 0, 1, 2, -1, 0.5]))
    Q = helpers.softmax64(np.array([-2.0, 4, 3, 0, -1, 2, 0]))
    for m in (1, 2, 3, 4):
        assert np.max(np.abs(_emitted_law(orc, P, Q, m) - P)) < 1e-12


def test_single_child_acceptance_closed_form(orc):
    rng = np.random.default_rng(8)
    for _ in range(5):
        V = 20
        P = helpers.softmax64(rng.standard_normal(V))
        Q = helpers.softmax64(rng.standard_normal(V))
        accept = sum(Q[y] * orc.rrs_node_law(P, Q, [y])[0][0] for y in range(V))
        assert accept == pytest.approx(np.minimum(P, Q).sum(), abs=1e-14)


def test_equal_laws_accept_first_slot(orc):
    rng = np.random.default_rng(9)
    P = helpers.softmax64(rng.standard_normal(10))
    acc, _, _ = orc.rrs_node_law(P, P, [3, 1, 4])
    assert acc[0] == 1.0


# --------------------------------------------------------------------------------------
def _tiny_setup(orc, seed_data=1000, T=1.0):
    w = synth.WORKLOADS["tiny"]
    draft = synth.to_host(synth.draft_logits(1, w["L"], w["V"], "normal2", "f32", seed_data))
    tree1 = orc.plan(draft, T, w["N"], w["K"], w["L"])
    return w, draft, tree1


def _sampled_path(orc, w, draft, tree1, seed, T=1.0, base_noise=1.0, B=TRIALS):
    tree = helpers.repeat_tree(tree1, B)
    qb = np.broadcast_to(draft, (B,) + draft.shape[1:])
    tok, ex_r = orc.replay(qb, T, tree, seed)
    base = draft[0]
    target = synth.path_keyed_rows(base, tree["parent"], tree["depth"], tok, base_noise, seed=77)
    out = orc.verify_rrs(target, qb, T, tree, tok, seed, w["L"])
    return tree, tok, out, base


@pytest.mark.parametrize("T", [1.0, 0.6])
def test_sampled_path_is_lossless(orc, T):
    w, draft, tree1 = _tiny_setup(orc, T=T)
    tree, tok, out, base = _sampled_path(orc, w, draft, tree1, seed=101, T=T)
    V = w["V"]
    inv = np.float32(np.float32(1.0) / np.float32(T))
    p_root = helpers.softmax64(synth.path_keyed_row(base, [], 1.0, 77) * inv)
    first = out["tokens"][:, 0]
    assert np.all((first >= 0) & (first < V))
    assert helpers.chi2_pvalue(np.bincount(first, minlength=V), p_root) > P_MIN
    # second token given the first (when the first was an accepted draft token)
    two = out["len"] >= 2
    vals, cnt = np.unique(first[two], return_counts=True)
    for a in vals[np.argsort(-cnt)][:3]:
        sel = two & (first == a)
        p_a = helpers.softmax64(synth.path_keyed_row(base, [int(a)], 1.0, 77) * inv)
        assert helpers.chi2_pvalue(np.bincount(out["tokens"][sel, 1], minlength=V), p_a) > P_MIN
    # structure: accepted nodes form a root path and carry their replayed tokens
    for b in range(200):
        n = out["len"][b] - 1
        prev = 0
        for k in range(n):
            node = out["nodes"][b, k]
            assert tree["parent"][b, node] == prev
            assert out["tokens"][b, k] == tok[b, node]
            prev = node
    assert out["exempt"].mean() < 1e-3


def test_target_equal_to_draft_accepts_first_child_chain(orc):
    """p_u = q_u at every node: slot 1 is always accepted, so the walk follows first
    children to a leaf and ends with the leaf's bonus token."""
    w, draft, tree1 = _tiny_setup(orc)
    B = 500
    tree = helpers.repeat_tree(tree1, B)
    qb = np.ascontiguousarray(np.broadcast_to(draft, (B,) + draft.shape[1:]))
    tok, _ = orc.replay(qb, 1.0, tree, seed=3)
    depth = tree["depth"]
    target = qb[np.arange(B)[:, None], np.minimum(depth, w["L"] - 1)]
    out = orc.verify_rrs(np.ascontiguousarray(target), qb, 1.0, tree, tok, seed=3, L=w["L"])
    off, ids = tree1["child_off"][0], tree1["child_ids"][0]
    chain = []
    u = 0
    while off[u + 1] > off[u]:
        u = ids[off[u]]
        chain.append(u)
    assert np.all(out["len"] == len(chain) + 1)
    assert np.all(out["nodes"][:, :len(chain)] == np.array(chain))


def test_verify_outputs_padding(orc):
    w, draft, tree1 = _tiny_setup(orc)
    tree, tok, out, base = _sampled_path(orc, w, draft, tree1, seed=5, B=64)
    L = w["L"]
    for b in range(64):
        n = out["len"][b]
        assert 1 <= n <= L + 1
        assert np.all(out["tokens"][b, n:] == -1)
        assert np.all(out["nodes"][b, n - 1:] == -1)


def test_final_token_law_across_chunks(orc):
    """V = 1000 spans four chunks (the last ragged), so the final token's two-level draw (chunk,
    then token inside it) is exercised both for the residual after rejections and for the
    bonus token at a leaf. Draft and target laws differ strongly, so every child is often
    rejected. First emitted token vs the root target law; second vs the child's target law."""
    B, V, m = 30_000, 1000, 3
    rng = np.random.default_rng(31)
    zq = rng.standard_normal((1, V)).astype(np.float32)
    zq[0, [5, 400, 990]] += np.float32(6.0)
    zt = rng.standard_normal((2, V)).astype(np.float32)
    zt[0, [7, 260, 600, 995]] += np.float32(4.0)
    zt[1, [12, 700]] += np.float32(5.0)
    tree = helpers.star_tree(m, B)
    qb = np.broadcast_to(zq[None], (B, 1, V))
    tok, ex_r = orc.replay(qb, 1.0, tree, seed=41)
    target = synth.path_keyed_rows(zt, tree["parent"], tree["depth"], tok, 0.5, seed=79)
    out = orc.verify_rrs(target, qb, 1.0, tree, tok, seed=41, L=1)
    first = out["tokens"][:, 0]
    p_root = helpers.softmax64(synth.path_keyed_row(zt, [], 0.5, 79))
    assert (out["len"] == 1).mean() > 0.2  # all children rejected reasonably often
    assert helpers.chi2_pvalue(np.bincount(first, minlength=V), p_root) > P_MIN
    two = out["len"] == 2
    vals, cnt = np.unique(first[two], return_counts=True)
    a = int(vals[np.argmax(cnt)])
    sel = two & (first == a)
    p_a = helpers.softmax64(synth.path_keyed_row(zt, [a], 0.5, 79))
    assert helpers.chi2_pvalue(np.bincount(out["tokens"][sel, 1], minlength=V), p_a) > P_MIN
