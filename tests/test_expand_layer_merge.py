"""The GPU expand-then-prune planner's algorithm restated on the CPU (integer keys, as its 64-bit
fixed-point path sums): each layer ranked by counting the candidates before each (index order
f*K + r for equal keys), the frontier the layer's first W, then the first N of a merge of the
sorted layers by (key desc, depth asc). Checked against the oracle's definition of the
expand-then-prune tree (Sec. 3.1, App. B.3), which sorts all generated candidates at once."""
import numpy as np
import pytest


def _fixed(x):
    return np.rint(x.astype(np.float64) * 2.0**30).astype(np.int64)


def _layer_merge_plan(topk_x, lse, K, L, N, W):
    """topk_x [L, K] (sorted desc), lse [L]; returns node list of (depth, parent position, rank)
    in node order, and the layers."""
    fx = _fixed(topk_x)
    CL = np.concatenate([[0], _fixed(np.cumsum(lse.astype(np.float64)))])  # each prefix rounded once
    layers = []  # per depth: list of (key, f, r) sorted
    cur = [(int(fx[0, r] - CL[1]), 0, r) for r in range(K)]
    layers.append(cur)
    for d in range(1, L):
        prev = layers[-1]
        nf = min(W, len(prev))
        cand = []
        for f in range(nf):
            sx = prev[f][0] + int(CL[d])
            for r in range(K):
                cand.append((sx + int(fx[d, r]) - int(CL[d + 1]), f, r))
        n = len(cand)
        pos = [sum(1 for i2 in range(n) if cand[i2][0] > cand[j][0] or (cand[i2][0] == cand[j][0] and i2 < j))
               for j in range(n)]
        srt = [None] * n
        for j in range(n):
            srt[pos[j]] = cand[j]
        layers.append(srt)
    heads = [0] * L
    nodes = []
    for _ in range(N):
        best = None
        for d in range(L):
            if heads[d] < len(layers[d]):
                k = layers[d][heads[d]][0]
                if best is None or k > best[0]:  # equal keys: the shallower layer first
                    best = (k, d)
        k, d = best
        _, f, r = layers[d][heads[d]]
        nodes.append((d + 1, f, r, heads[d]))
        heads[d] += 1
    return nodes


@pytest.mark.parametrize("seed,V,K,L,N,W", [(4000, 64, 4, 5, 30, 3), (4001, 300, 8, 8, 64, 10),
                                            (4002, 40, 3, 6, 30, 2), (4003, 128, 8, 16, 64, 10)])
def test_layer_merge_matches_oracle_definition(orc, seed, V, K, L, N, W):
    rng = np.random.default_rng(seed)
    draft = (3.0 * rng.standard_normal((1, L, V))).astype(np.float32)
    st = orc.row_stats(draft, 1.0, K)
    nodes = _layer_merge_plan(st["topk_x"][0], st["lse"][0], K, L, N, W)
    tree = orc.plan_expand(draft, 1.0, N, K, L, W)
    assert not tree["exempt"][0], "near tie: choose another seed"
    # node i: depth and rank agree; its parent is the node holding position f of the layer above
    num = {}
    for i, (d, f, r, p) in enumerate(nodes, start=1):
        num[(d, p)] = i
        assert tree["depth"][0, i] == d and tree["rank"][0, i] == r
        assert tree["parent"][0, i] == (0 if d == 1 else num[(d - 1, f)])
