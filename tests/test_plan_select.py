"""The GPU first pass's selection algorithm restated on the CPU, with its integer keys (64-bit
fixed-point path sums), and checked against the oracle's best-first expansion (Sec. 3.1,
App. B.3).

Keys never increase along a path's links (a first child's key is its parent's plus a
log-probability <= 0, a sibling's key is at most its left neighbour's), so the max-heap's N
pops are the N first paths of the global order (key desc, depth asc, parent's position asc,
rank asc). The algorithm finds them without popping one at a time:

1. a lower bound tau0 on the N-th key: every path of the family F0 (the top-1 chain of each
   length, and every path that leaves it once, at depth i with rank r >= 1, then follows rank 0
   to depth d) is a real path, so the N-th largest key of F0 is at most the N-th largest key
   overall. Two histogram rounds over F0's keys (64 power-of-two bins, then 64 sub-bins of the
   bin holding the N-th) give a bin edge tau0 with at least N keys of F0 at or above it;
2. every path with key >= tau0, enumerated as chains: the top-1 chain from the root as far as
   it stays >= tau0, then level by level, every rank >= 1 child of a node found in the level
   before (the root and the top-1 chain first) that reaches tau0, each followed by its rank-0
   continuation as far as it reaches tau0;
3. each path's position in the global order by counting the paths before it; parents' positions
   decide only between equal keys at equal depths, so those positions are settled depth by
   depth when such ties occur. The paths at positions 0..N-1 are nodes 1..N.
"""
import numpy as np
import pytest


def _fixed(x):
    return np.rint(x.astype(np.float64) * 2.0**30).astype(np.int64)


def nth_bound(keys, N, hi, lo=None):
    """A bin edge t <= the N-th largest of keys (all in [lo, hi]) with at least N keys >= t: 64
    power-of-two bins of hi - key, then 64 sub-bins of the bin holding the N-th."""
    lo = min(keys) if lo is None else lo
    s1 = 0
    while ((hi - lo) >> s1) >= 64:
        s1 += 1
    h1 = [0] * 64
    for e in keys:
        h1[(hi - e) >> s1] += 1
    cum, j = 0, 0
    while cum + h1[j] < N:
        cum += h1[j]
        j += 1
    s2 = max(s1 - 6, 0)
    h2 = [0] * 64
    for e in keys:
        if (hi - e) >> s1 == j:
            h2[((hi - e) >> s2) - (j << (s1 - s2))] += 1
    k = 0
    while cum + h2[k] < N:
        cum += h2[k]
        k += 1
    return hi - (((j << (s1 - s2)) + k + 1) << s2) + 1


def enumerate_paths(delta, B, K, L, tau, cap):
    """Every path with key >= tau as entries (key, depth, rank, parent entry); stops once more
    than cap entries exist."""
    ent = []
    e_prev = -1
    for d in range(1, L + 1):
        if B[d] < tau:
            break
        ent.append((B[d], d, 0, e_prev))
        e_prev = len(ent) - 1
    anchors = [(-1, 0, 0)] + [(e, ent[e][1], ent[e][0]) for e in range(len(ent))]  # (entry, depth, key)
    while anchors:
        start = len(ent)
        for a, da, ka in anchors:
            d = da + 1
            if d > L:
                continue
            for r in range(1, K):
                key = ka + delta[d][r]
                if key < tau:
                    break
                ent.append((key, d, r, a))
                p = len(ent) - 1
                for dd in range(d + 1, L + 1):
                    kk = key + B[dd] - B[d]
                    if kk < tau:
                        break
                    ent.append((kk, dd, 0, p))
                    p = len(ent) - 1
                if len(ent) > cap:
                    return ent
        anchors = [(e, ent[e][1], ent[e][0]) for e in range(start, len(ent))]
    return ent


def select_plan(topk_x, lse, K, L, N, cap=None):
    """topk_x [L, K] (sorted desc), lse [L]. Returns a list of (depth, parent node, rank) for
    nodes 1..N, or None where the GPU kernel falls back to the serial heap."""
    fx = [[int(v) for v in row] for row in _fixed(topk_x)]
    CL = [0] + [int(v) for v in _fixed(np.cumsum(lse.astype(np.float64)))]
    delta = [[0] * K] + [[fx[d - 1][r] - (CL[d] - CL[d - 1]) for r in range(K)] for d in range(1, L + 1)]
    if any(delta[d][0] > 0 for d in range(1, L + 1)):
        return None  # a first child above its parent: not monotone
    B = [0] * (L + 1)
    for d in range(1, L + 1):
        B[d] = B[d - 1] + delta[d][0]
    # 1. tau0 from F0
    F0 = [B[d] for d in range(1, L + 1)]
    for i in range(1, L + 1):
        for r in range(1, K):
            c = delta[i][0] - delta[i][r]
            F0 += [B[d] - c for d in range(i, L + 1)]
    tau = nth_bound(F0, N, B[1]) if len(F0) >= N else -(1 << 62)
    cap = cap or 4 * N + 64
    for _attempt in range(4):
        ent = enumerate_paths(delta, B, K, L, tau, cap)
        if len(ent) <= cap:
            break
        # more than cap paths reach tau: the N-th largest key among cap of them bounds it better
        t2 = nth_bound([e[0] for e in ent[:cap]], N, B[1])
        if t2 <= tau:
            return None
        tau = t2
    else:
        return None
    M = len(ent)
    if M < N:
        return None
    # 3. positions by counting; between equal keys at equal depths with different parents, the
    #    ancestors' keys compared upwards, then the ranks of the common ancestor's two children
    def before(y, x):
        ky, dy, ry, py = ent[y]
        kx, dx, rx, px = ent[x]
        if ky != kx:
            return ky > kx
        if dy != dx:
            return dy < dx
        if py == px:
            return ry < rx
        cx, cy, ax, ay = x, y, px, py
        while ax != ay:
            if ent[ax][0] != ent[ay][0]:
                return ent[ay][0] > ent[ax][0]
            cx, cy, ax, ay = ax, ay, ent[ax][3], ent[ay][3]
        return ent[cy][2] < ent[cx][2]
    # with many more paths than N, only those reaching a second bound get positions (their
    # predecessors and parents all reach it)
    kept = list(range(M))
    if M > N + N // 8:
        t = nth_bound([e[0] for e in ent], N, B[1], tau)
        kept = [x for x in range(M) if ent[x][0] >= t]
    pos = {x: sum(1 for y in kept if before(y, x)) for x in kept}
    nodes = [None] * N
    for x in kept:
        if pos[x] < N:
            kx, dx, rx, px = ent[x]
            nodes[pos[x]] = (dx, 0 if px < 0 else pos[px] + 1, rx)
    return nodes


def heap_plan(topk_x, lse, K, L, N):
    """The serial best-first expansion on the same integer keys (the kernel's fallback)."""
    import heapq
    fx = [[int(v) for v in row] for row in _fixed(topk_x)]
    CL = [0] + [int(v) for v in _fixed(np.cumsum(lse.astype(np.float64)))]
    heap = [(-(fx[0][0] - CL[1]), 1, 0, 0, fx[0][0])]  # (-key, depth, parent, rank, path sum)
    nodes = []
    while len(nodes) < N:
        nk, d, p, r, sx = heapq.heappop(heap)
        nodes.append((d, p, r))
        i = len(nodes)
        if r + 1 < K:
            s2 = sx - fx[d - 1][r] + fx[d - 1][r + 1]
            heapq.heappush(heap, (-(s2 - CL[d]), d, p, r + 1, s2))
        if d < L:
            s3 = sx + fx[d][0]
            heapq.heappush(heap, (-(s3 - CL[d + 1]), d + 1, i, 0, s3))
    return nodes


def _check(orc, draft, K, L, N, fast=True):
    st = orc.row_stats(draft, 1.0, K)
    tree = orc.plan(draft, 1.0, N, K, L)
    nodes = select_plan(st["topk_x"][0], st["lse"][0], K, L, N)
    assert (nodes is not None) == fast
    heap = heap_plan(st["topk_x"][0], st["lse"][0], K, L, N)
    if nodes is not None:
        assert nodes == heap  # the selection reproduces the heap on the same keys, ties included
    else:
        nodes = heap
    if tree["exempt"][0]:
        return False
    for i, (d, p, r) in enumerate(nodes, start=1):
        assert (tree["depth"][0, i], tree["parent"][0, i], tree["rank"][0, i]) == (d, p, r), i
    return True


@pytest.mark.parametrize("seed,V,K,L,N,fast", [(5000, 64, 4, 5, 30, True), (5001, 300, 8, 8, 64, True),
                                               (5002, 40, 3, 6, 60, True), (5003, 512, 8, 16, 64, True),
                                               (5004, 200, 8, 16, 256, True), (5005, 64, 2, 10, 200, True),
                                               (5006, 100, 1, 12, 12, True), (5007, 1000, 32, 4, 300, True),
                                               (5009, 2000, 8, 64, 1024, True)])
def test_selection_matches_heap(orc, seed, V, K, L, N, fast):
    """Flat rows (3 N(0, 1) logits): F0's bound is loose and the first enumeration overflows;
    the bound from the paths it found ends the second or third."""
    rng = np.random.default_rng(seed)
    draft = (3.0 * rng.standard_normal((1, L, V))).astype(np.float32)
    assert _check(orc, draft, K, L, N, fast), "near tie: choose another seed"


@pytest.mark.parametrize("seed", range(6))
def test_selection_with_exact_ties(orc, seed):
    """Integer logits, identical rows: many paths with exactly equal keys at equal depths."""
    rng = np.random.default_rng(6000 + seed)
    L, V, K, N = 6, 24, 4, 80
    row = rng.integers(-3, 3, V).astype(np.float32)
    draft = np.broadcast_to(row, (1, L, V)).copy()
    assert _check(orc, draft, K, L, N)


def test_selection_planted_rows(orc):
    """Rows shaped like the serving workload: one planted token per row."""
    rng = np.random.default_rng(7000)
    L, V, K, N = 16, 4096, 8, 64
    draft = (3.0 * rng.standard_normal((1, L, V))).astype(np.float32)
    for d in range(L):
        draft[0, d, rng.integers(V)] = 12.0 + rng.uniform(-1, 1)
    assert _check(orc, draft, K, L, N)
