"""Small helpers shared by the tests (no method arithmetic here)."""
from __future__ import annotations

import itertools

import numpy as np
from scipy import stats


def star_tree(m: int, B: int = 1):
    """Root with m leaf children (slots 0..m-1 = nodes 1..m)."""
    NN = m + 1
    tree = {
        "parent": np.array([[-1] + [0] * m] * B, dtype=np.int32),
        "depth": np.array([[0] + [1] * m] * B, dtype=np.int32),
        "rank": np.array([[-1] + list(range(m))] * B, dtype=np.int32),
        "child_off": np.array([[0] + [m] * NN] * B, dtype=np.int32),
        "child_ids": np.array([list(range(1, m + 1))] * B, dtype=np.int32),
    }
    return tree


def chain_tree(g: int, B: int = 1):
    """Chain 0 -> 1 -> ... -> g."""
    NN = g + 1
    tree = {
        "parent": np.array([[-1] + list(range(g))] * B, dtype=np.int32),
        "depth": np.array([list(range(NN))] * B, dtype=np.int32),
        "rank": np.array([[-1] + [0] * g] * B, dtype=np.int32),
        "child_off": np.array([list(range(g + 1)) + [g]] * B, dtype=np.int32),
        "child_ids": np.array([list(range(1, g + 1))] * B, dtype=np.int32),
    }
    return tree


def repeat_tree(tree, B: int):
    """Broadcast a single tree (B=1) to B identical trees."""
    out = {}
    for k, v in tree.items():
        if isinstance(v, np.ndarray) and v.ndim == 2 and v.shape[0] == 1:
            out[k] = np.ascontiguousarray(np.repeat(v, B, axis=0))
        else:
            out[k] = v
    return out


def wor_tuple_prob(q: np.ndarray, ys) -> float:
    """Closed-form probability of the ordered draw sequence ys under sampling without
    replacement from q: prod_j q(y_j) / (1 - sum_{l<j} q(y_l))."""
    p, used = 1.0, 0.0
    for y in ys:
        p *= q[y] / (1.0 - used)
        used += q[y]
    return p


def all_wor_tuples(V: int, m: int):
    return itertools.permutations(range(V), m)


def chi2_pvalue(counts: np.ndarray, probs: np.ndarray, min_expected: float = 20.0) -> float:
    """Chi-square goodness of fit; categories with small expectation are pooled."""
    counts = np.asarray(counts, dtype=np.float64)
    probs = np.asarray(probs, dtype=np.float64)
    if (counts[probs <= 0.0] > 0).any():  # an outcome the law gives probability 0
        return 0.0
    keep = probs > 0.0
    counts, probs = counts[keep], probs[keep]
    n = counts.sum()
    exp = probs * n
    big = exp >= min_expected
    obs = list(counts[big])
    ex = list(exp[big])
    if (~big).any():
        obs.append(counts[~big].sum())
        ex.append(exp[~big].sum())
    obs = np.array(obs)
    ex = np.array(ex)
    ex *= obs.sum() / ex.sum()
    if len(obs) < 2:
        return 1.0
    return float(stats.chisquare(obs, ex).pvalue)


def softmax64(x):
    x = np.asarray(x, dtype=np.float64)
    m = x.max()
    e = np.exp(x - m)
    return e / e.sum()
