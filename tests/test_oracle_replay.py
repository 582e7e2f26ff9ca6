"""Pins of the oracle's replay sampler (Sec. 3.2; WoR as in App. A), CPU only.

Ordered draws of the hierarchical (chunked) Gumbel-top-k sampler and of the flat one are
both checked by chi-square against the closed-form law of sampling without replacement,
prod_j q(y_j) / (1 - sum_{l<j} q(y_l)), over 1e5 seeded trials.
"""
import numpy as np
import pytest

import helpers

TRIALS = 100_000
P_MIN = 1e-4


def _q(x, T=1.0):
    x32 = x.astype(np.float32) * np.float32(np.float32(1.0) / np.float32(T))
    return helpers.softmax64(x32)


def _star_draws(orc, row, m, seed, flat, T=1.0, B=TRIALS):
    q = np.broadcast_to(row.astype(np.float32)[None, None, :], (B, 1, row.shape[0]))
    tree = helpers.star_tree(m, B)
    if flat:
        tok = orc.replay(q, T, tree, seed, flat=True)
    else:
        tok, ex = orc.replay(q, T, tree, seed)
        assert ex.mean() < 1e-3
    return tok[:, 1:]


def _marginals_exact(q, m):
    """P(slot j = v) for j < m by explicit summation over prefixes (small m)."""
    V = len(q)
    marg = np.zeros((m, V))
    marg[0] = q
    if m >= 2:
        # P(y1=a, y2=b) = q(a) q(b) / (1 - q(a))
        pair = q[:, None] * q[None, :] / (1.0 - q[:, None])
        np.fill_diagonal(pair, 0.0)
        marg[1] = pair.sum(axis=0)
    if m >= 3:
        for c in range(V):
            qa = q[:, None]
            qb = q[None, :]
            t = qa * qb / (1.0 - qa) * q[c] / (1.0 - qa - qb)
            mask = np.ones((V, V), bool)
            np.fill_diagonal(mask, False)
            mask[c, :] = False
            mask[:, c] = False
            marg[2, c] = t[mask].sum()
    return marg


@pytest.mark.parametrize("flat", [False, True])
def test_wor_single_chunk(orc, flat):
    rng = np.random.default_rng(21)
    V, m = 32, 3
    row = (2.0 * rng.standard_normal(V)).astype(np.float32)
    draws = _star_draws(orc, row, m, seed=1, flat=flat)
    q = _q(row)
    # without replacement: siblings are distinct
    assert np.all(draws[:, 0] != draws[:, 1]) and np.all(draws[:, 1] != draws[:, 2])
    assert np.all(draws[:, 0] != draws[:, 2])
    marg = _marginals_exact(q, m)
    for j in range(m):
        counts = np.bincount(draws[:, j], minlength=V)
        assert helpers.chi2_pvalue(counts, marg[j]) > P_MIN, f"slot {j}"
    pair = q[:, None] * q[None, :] / (1.0 - q[:, None])
    np.fill_diagonal(pair, 0.0)
    counts = np.bincount(draws[:, 0] * V + draws[:, 1], minlength=V * V)
    assert helpers.chi2_pvalue(counts, pair.ravel()) > P_MIN


@pytest.mark.parametrize("flat", [False, True])
def test_wor_across_chunks(orc, flat):
    """V = 1000 spans four chunks (the last one ragged); heavy tokens sit in the same and in
    different chunks, so chunk selection and the conditional shift both matter."""
    rng = np.random.default_rng(22)
    V, m = 1000, 3
    row = rng.standard_normal(V).astype(np.float32)
    heavy = [3, 10, 300, 700, 999]
    row[heavy] += np.float32(5.0)
    draws = _star_draws(orc, row, m, seed=2, flat=flat)
    q = _q(row)
    marg = _marginals_exact(q, 2)
    for j in range(2):
        counts = np.bincount(draws[:, j], minlength=V)
        assert helpers.chi2_pvalue(counts, marg[j]) > P_MIN, f"slot {j}"
    pair = q[:, None] * q[None, :] / (1.0 - q[:, None])
    np.fill_diagonal(pair, 0.0)
    idx = draws[:, 0].astype(np.int64) * V + draws[:, 1]
    counts = np.bincount(idx, minlength=V * V)
    assert helpers.chi2_pvalue(counts, pair.ravel()) > P_MIN
    # third slot: only the heavy tokens carry enough mass to test individually
    qa = q[:, None]
    qb = q[None, :]
    base = qa * qb / (1.0 - qa)
    np.fill_diagonal(base, 0.0)
    probs = []
    for c in heavy:
        t = base * q[c] / (1.0 - qa - qb)
        t[c, :] = 0.0
        t[:, c] = 0.0
        probs.append(t.sum())
    counts = [np.sum(draws[:, 2] == c) for c in heavy]
    probs.append(1.0 - sum(probs))
    counts.append(TRIALS - sum(counts))
    assert helpers.chi2_pvalue(np.array(counts), np.array(probs)) > P_MIN


def test_single_draw_is_categorical(orc):
    rng = np.random.default_rng(23)
    V = 600
    row = (3.0 * rng.standard_normal(V)).astype(np.float32)
    draws = _star_draws(orc, row, 1, seed=3, flat=False, T=0.6)
    q = _q(row, 0.6)
    assert helpers.chi2_pvalue(np.bincount(draws[:, 0], minlength=V), q) > P_MIN


def test_replay_fills_slots_in_key_order_and_keeps_topology(orc):
    """Replay on a planned tree: every parent's children are distinct tokens; parents at the
    same depth share a row but use independent streams (node in the counter)."""
    rng = np.random.default_rng(24)
    V, K, L, N = 700, 4, 4, 30
    draft = (2.0 * rng.standard_normal((3, L, V))).astype(np.float32)
    tree = orc.plan(draft, 1.0, N, K, L)
    tok, ex = orc.replay(draft, 1.0, tree, seed=5)
    assert np.all(tok[:, 0] == -1)
    for b in range(3):
        off, ids = tree["child_off"][b], tree["child_ids"][b]
        for u in range(N + 1):
            ch = ids[off[u]:off[u + 1]]
            t = tok[b, ch]
            assert len(set(t.tolist())) == len(t)
            assert np.all((t >= 0) & (t < V))
    # reproducible, and a different seed changes the draws
    tok2, _ = orc.replay(draft, 1.0, tree, seed=5)
    tok3, _ = orc.replay(draft, 1.0, tree, seed=6)
    assert np.array_equal(tok, tok2) and not np.array_equal(tok, tok3)
    # per-node rows: qrow_of_node selects the row of each parent
    qrows = (2.0 * rng.standard_normal((3, N + 1, V))).astype(np.float32)
    qidx = np.tile(np.arange(N + 1, dtype=np.int32), (3, 1))
    tok4, _ = orc.replay(qrows, 1.0, tree, seed=5, qrow_of_node=qidx)
    assert not np.array_equal(tok, tok4)
