"""Pins of the oracle's mixed-sampling replay (Sec. 3.2, App. A) and target-sample-matching
verifier ("Naive", Table 2 / Sec. 2.3), CPU only.

Mixed sampling: the m-1 deterministic slots must be a stable sort of (-x, id), and the last
slot must follow q renormalised over the other tokens (chi-square over 1e5 seeded trials, in
one chunk and across chunks, where the excluded tokens sit in different chunks and may hold
their chunk's maximum). Naive verification: every emitted token must follow the target law
at its prefix (chi-square), a child carrying token v is accepted with probability p(v)
(closed form), and a target that puts all its mass on a child's token always accepts it.
"""
import numpy as np
import pytest

import helpers

TRIALS = 100_000
P_MIN = 1e-4


def _x(row, T=1.0):
    return row.astype(np.float32) * np.float32(np.float32(1.0) / np.float32(T))


def _topk(x, k):
    return np.lexsort((np.arange(len(x)), -x.astype(np.float64)))[:k]


def _mixed_star(orc, row, m, B=TRIALS, seed=1):
    q = np.broadcast_to(row.astype(np.float32)[None, None, :], (B, 1, row.shape[0]))
    tree = helpers.star_tree(m, B)
    tok, ex = orc.replay_mixed(q, 1.0, tree, seed)
    assert ex.mean() < 1e-3
    return tok[:, 1:]


@pytest.mark.parametrize("V,m,spread", [(32, 3, 2.0), (32, 1, 2.0), (1000, 4, 2.5), (700, 8, 1.0)])
def test_mixed_slots(orc, V, m, spread):
    rng = np.random.default_rng(40 + m + V)
    row = (spread * rng.standard_normal(V)).astype(np.float32)
    if V >= 700:
        # heavy tokens in several chunks, one of them the maximum of its chunk
        row[[3, 300, 301, 650]] += np.float32(4.0)
    draws = _mixed_star(orc, row, m)
    x = _x(row)
    top = _topk(x, m - 1)
    assert np.all(draws[:, : m - 1] == top[None, :])  # deterministic slots, most probable first
    last = draws[:, m - 1]
    assert not np.isin(last, top).any()
    keep = np.setdiff1d(np.arange(V), top)
    q = helpers.softmax64(x)[keep]
    q /= q.sum()
    assert helpers.chi2_pvalue(np.bincount(last, minlength=V)[keep], q) > P_MIN


def test_mixed_ties_are_stable(orc):
    """Equal logits: the deterministic slots take the lower token id first."""
    row = np.zeros(64, dtype=np.float32)
    row[[5, 9, 40, 41]] = 3.0
    draws = _mixed_star(orc, row, 4, B=200)
    assert np.all(draws[:, :3] == np.array([5, 9, 40]))
    assert np.all(draws[:, 3] != 5) and np.all(draws[:, 3] != 9) and np.all(draws[:, 3] != 40)


def test_mixed_single_child_is_the_wor_draw(orc):
    """With one child nothing is excluded: the draw is the replay sampler's own draw."""
    rng = np.random.default_rng(6)
    V, L, B = 900, 5, 8
    draft = (3.0 * rng.standard_normal((B, L, V))).astype(np.float32)
    tree = orc.plan(draft, 1.0, L, 1, L)  # a chain: every parent has one child
    t_mixed, _ = orc.replay_mixed(draft, 1.0, tree, 99)
    t_wor, _ = orc.replay(draft, 1.0, tree, 99)
    assert np.array_equal(t_mixed, t_wor)


def test_mixed_on_planned_tree(orc):
    """Every parent of a planned tree: its children's first slots are its row's top tokens in
    order, and siblings are distinct."""
    rng = np.random.default_rng(12)
    V, K, L, N, B = 600, 4, 5, 30, 4
    draft = (3.0 * rng.standard_normal((B, L, V))).astype(np.float32)
    tree = orc.plan(draft, 1.0, N, K, L)
    tok, _ = orc.replay_mixed(draft, 1.0, tree, 5)
    for b in range(B):
        off, ids = tree["child_off"][b], tree["child_ids"][b]
        for u in range(N + 1):
            ch = ids[off[u]:off[u + 1]]
            if len(ch) == 0:
                continue
            top = _topk(_x(draft[b, tree["depth"][b, u]]), len(ch) - 1)
            assert list(tok[b, ch[:-1]]) == list(top)
            assert len(set(tok[b, ch].tolist())) == len(ch)


# --------------------------------------------------------------------------------------
def _naive_star(orc, target_row, child_tokens, B=TRIALS, seed=3):
    m = len(child_tokens)
    V = target_row.shape[0]
    tgt = np.broadcast_to(target_row.astype(np.float32)[None, None, :], (B, m + 1, V))
    tree = helpers.star_tree(m, B)
    tok = np.zeros((B, m + 1), dtype=np.int32)
    tok[:, 0] = -1
    tok[:, 1:] = np.asarray(child_tokens, dtype=np.int32)[None, :]
    return orc.verify_naive(tgt, 1.0, tree, tok, seed, L=1)


@pytest.mark.parametrize("V,children", [(32, [3, 7, 11]), (1000, [0, 299, 300, 999]), (32, [])])
def test_naive_emits_target_law(orc, V, children):
    rng = np.random.default_rng(50 + V + len(children))
    row = (2.0 * rng.standard_normal(V)).astype(np.float32)
    if children:
        row[children[0]] += np.float32(2.0)
    out = _naive_star(orc, row, children)
    p = helpers.softmax64(_x(row))
    first = out["tokens"][:, 0]
    assert helpers.chi2_pvalue(np.bincount(first, minlength=V), p) > P_MIN
    acc = out["len"] == 2
    # an emitted token equal to a child's token is that child's acceptance, and vice versa
    assert np.array_equal(acc, np.isin(first, children))
    if children:
        pa = p[children].sum()
        z = (acc.mean() - pa) / np.sqrt(pa * (1 - pa) / TRIALS)
        assert abs(z) < 5.0
        assert np.all(out["nodes"][acc, 0] == 1 + np.array([children.index(t) for t in first[acc]]))
    assert np.all(out["tokens"][~acc, 1] == -1)


def test_naive_forced_acceptance_down_a_chain(orc):
    """Target rows that put (numerically) all mass on the chain's tokens accept every node;
    the bonus token then comes from the leaf's row."""
    V, g, B = 64, 4, 50
    tree = helpers.chain_tree(g, B)
    chain = np.array([7, 21, 33, 60], dtype=np.int32)
    tgt = np.zeros((B, g + 1, V), dtype=np.float32)
    for i in range(g):
        tgt[:, i, chain[i]] = 200.0
    tgt[:, g, 5] = 200.0
    tok = np.zeros((B, g + 1), dtype=np.int32)
    tok[:, 0] = -1
    tok[:, 1:] = chain
    out = orc.verify_naive(tgt, 1.0, tree, tok, 11, L=g)
    assert np.all(out["len"] == g + 1)
    assert np.all(out["tokens"] == np.append(chain, 5)[None, :])
    assert np.all(out["nodes"] == np.arange(1, g + 1)[None, :])


def test_naive_second_token_follows_child_target(orc):
    """Two levels with different target rows: given that child c was accepted, the next
    emitted token follows child c's target row (the prefix-conditional law)."""
    rng = np.random.default_rng(77)
    V, B = 32, TRIALS
    # root -> children 1, 2 (tokens 4, 9); node 1 -> child 3 (token 0)
    tree = {
        "parent": np.array([[-1, 0, 0, 1]] * B, dtype=np.int32),
        "depth": np.array([[0, 1, 1, 2]] * B, dtype=np.int32),
        "rank": np.array([[-1, 0, 1, 0]] * B, dtype=np.int32),
        "child_off": np.array([[0, 2, 3, 3, 3]] * B, dtype=np.int32),
        "child_ids": np.array([[1, 2, 3]] * B, dtype=np.int32),
    }
    rows = (1.5 * rng.standard_normal((4, V))).astype(np.float32)
    rows[0, [4, 9]] += 2.0
    tgt = np.broadcast_to(rows[None], (B, 4, V))
    tok = np.array([[-1, 4, 9, 0]] * B, dtype=np.int32)
    out = orc.verify_naive(tgt, 1.0, tree, tok, 21, L=2)
    p = [helpers.softmax64(_x(r)) for r in rows]
    after1 = out["nodes"][:, 0] == 1
    after2 = out["nodes"][:, 0] == 2
    assert helpers.chi2_pvalue(np.bincount(out["tokens"][after1, 1], minlength=V), p[1]) > P_MIN
    # node 2 is a leaf: its bonus token follows its own row
    assert helpers.chi2_pvalue(np.bincount(out["tokens"][after2, 1], minlength=V), p[2]) > P_MIN
    # node 3 accepted only through node 1 and token 0
    deep = out["nodes"][:, 1] == 3
    assert np.all(out["tokens"][deep, 1] == 0)
    assert np.all(out["len"][deep] == 3)
