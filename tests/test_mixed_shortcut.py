"""The mixed-sampling kernel's shortcut (CPU, fp64). The sampled slot is the largest Gumbel key
among the tokens outside the m-1 deterministic ones, with the keys of the top-down construction:
chunk keys K_c, element keys shifted to their chunk's maximum (Sec. 3.2, App. A; Kool et al.
2019). The kernel expands only the chunks holding an excluded token and the best clean chunk,
and in each shifts only its largest non-excluded raw key (the shift is increasing in the raw
key, and a clean chunk's largest key is its chunk key). Here that shortcut is checked against
the definition: every chunk expanded, every key shifted."""
import numpy as np
import pytest


def _shift(T, Z, g):
    with np.errstate(divide="ignore"):  # g = Z (the chunk's maximum) is replaced by T by the caller
        u = T - g + np.log1p(-np.exp(g - Z))
    return T - (np.maximum(u, 0.0) + np.log1p(np.exp(-np.abs(u))))


def _keys_all(x, C, cs, chunk_keys, raw):
    """Every element's shifted key (the definition)."""
    k = np.empty_like(x)
    for c in range(C):
        lo, hi = c * cs, min(len(x), (c + 1) * cs)
        g = raw[lo:hi]
        j = int(np.argmax(g))
        kk = _shift(chunk_keys[c], g[j], g)
        kk[j] = chunk_keys[c]
        k[lo:hi] = kk
    return k


def _shortcut(x, C, cs, chunk_keys, raw, excluded):
    dirty = sorted({int(v) // cs for v in excluded})
    clean = [c for c in range(C) if c not in dirty]
    cands = []
    if clean:  # the best clean chunk: its largest key is its chunk key, held by its largest raw key
        c = max(clean, key=lambda c: (chunk_keys[c], -c))
        lo, hi = c * cs, min(len(x), (c + 1) * cs)
        cands.append((chunk_keys[c], lo + int(np.argmax(raw[lo:hi]))))
    for c in dirty:
        lo, hi = c * cs, min(len(x), (c + 1) * cs)
        g = raw[lo:hi]
        z = int(np.argmax(g))
        keep = [i for i in range(hi - lo) if (lo + i) not in excluded]
        if not keep:
            continue
        b = max(keep, key=lambda i: (g[i], -i))
        key = chunk_keys[c] if b == z else _shift(chunk_keys[c], g[z], g[b])
        cands.append((key, lo + b))
    return max(cands, key=lambda t: (t[0], -t[1]))[1]


@pytest.mark.parametrize("seed", range(8))
def test_shortcut_matches_definition(seed):
    rng = np.random.default_rng(500 + seed)
    for _ in range(200):
        cs = int(rng.choice([4, 8, 16]))
        V = int(rng.integers(cs, 8 * cs + 3))
        C = (V + cs - 1) // cs
        x = 2.5 * rng.standard_normal(V)
        m = int(rng.integers(1, min(V, 9) + 1))
        excluded = set(np.lexsort((np.arange(V), -x))[: m - 1].tolist())
        A = np.array([np.logaddexp.reduce(x[c * cs:(c + 1) * cs]) for c in range(C)])
        chunk_keys = A + rng.gumbel(size=C)
        raw = x + rng.gumbel(size=V)
        keys = _keys_all(x, C, cs, chunk_keys, raw)
        allowed = [v for v in range(V) if v not in excluded]
        want = max(allowed, key=lambda v: (keys[v], -v))
        assert _shortcut(x, C, cs, chunk_keys, raw, excluded) == want
