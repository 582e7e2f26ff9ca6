"""Pins of the oracle's row statistics (step a1 of the first pass, Sec. 3.1), CPU only.

``orc_row_stats`` returns, per row of x = fp32(z) * fp32(1/T): the maximum, the row's
log-normaliser log sum_v exp(x_v), the log-mass of every 256-token chunk, and the top-K by
(x desc, id asc). Each output is checked against a computation that shares nothing with the
oracle's C code: numpy's max, scipy's logsumexp on numpy slices, and numpy's lexsort (a
stable sort). The cases cover a row shorter than one chunk, a ragged last chunk, bf16 input,
a temperature other than 1, heavy ties and a row whose mass sits on one token.
"""
import numpy as np
import pytest
from scipy.special import logsumexp

CHUNK = 256


def _x(rows, T):
    """x = fp32(z) * fp32(1/T) with one fp32 rounding (bf16 rows widened exactly first)."""
    if rows.dtype == np.uint16:
        z = (rows.astype(np.uint32) << 16).view(np.float32)
    else:
        z = rows.astype(np.float32)
    return z * np.float32(np.float32(1.0) / np.float32(T))


def _bf16_bits(a):
    """Round-to-nearest-even fp32 -> bf16 bit patterns."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def _rows(B, R, V, dtype, seed, scale=3.0):
    rng = np.random.default_rng(seed)
    z = (scale * rng.standard_normal((B, R, V))).astype(np.float32)
    return _bf16_bits(z) if dtype == "bf16" else z


def _check(orc, rows, T, K):
    B, R, V = rows.shape
    C = (V + CHUNK - 1) // CHUNK
    got = orc.row_stats(rows, T, K)
    x = _x(rows, T).astype(np.float64)
    for b in range(B):
        for r in range(R):
            xr = x[b, r]
            assert got["max"][b, r] == xr.max()
            np.testing.assert_allclose(got["lse"][b, r], logsumexp(xr), rtol=1e-13, atol=1e-13)
            want_c = [logsumexp(xr[c * CHUNK:min(V, (c + 1) * CHUNK)]) for c in range(C)]
            np.testing.assert_allclose(got["chunk_lse"][b, r], want_c, rtol=1e-13, atol=1e-13)
            order = np.lexsort((np.arange(V), -xr))[:K]
            assert np.array_equal(got["topk_id"][b, r], order)
            assert np.array_equal(got["topk_x"][b, r], xr[order].astype(np.float32))
    return got


@pytest.mark.parametrize("V", [1, 5, 32, 255, 256, 257, 1000, 5003])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_row_stats_against_numpy_and_scipy(orc, V, dtype):
    rows = _rows(2, 3, V, dtype, seed=V)
    _check(orc, rows, 1.0, min(V, 8))


@pytest.mark.parametrize("T", [0.6, 1.0, 1.7])
def test_row_stats_temperature(orc, T):
    rows = _rows(2, 2, 1001, "bf16", seed=7)
    got = _check(orc, rows, T, 5)
    # a temperature only rescales x: the top-K ids are those at T = 1
    base = orc.row_stats(rows, 1.0, 5)
    assert np.array_equal(got["topk_id"], base["topk_id"])


def test_row_stats_ragged_last_chunk_is_its_own(orc):
    """A large logit in the ragged tail (V = 600: chunks of 256, 256, 88) belongs to chunk 2
    only: moving it by one position across the 512 boundary moves the mass with it."""
    V = 600
    rows = np.zeros((1, 2, V), dtype=np.float32)
    rows[0, 0, 512] = 20.0  # first element of the tail chunk
    rows[0, 1, 511] = 20.0  # last element of chunk 1
    got = _check(orc, rows, 1.0, 3)
    cl = got["chunk_lse"][0]
    assert cl[0, 2] > 19.0 and cl[0, 1] < 6.0
    assert cl[1, 1] > 19.0 and cl[1, 2] < 5.0
    # the tail holds 88 tokens: an all-zero tail chunk has log-mass log(88)
    np.testing.assert_allclose(cl[1, 2], np.log(88.0), rtol=1e-14)


def test_row_stats_ties_and_one_hot(orc):
    """A flat row (every id ties: top-K = ids 0..K-1), a repeated maximum (the lowest ids win),
    and a row with one token at +1000 (log-normaliser = that logit)."""
    V = 700
    rows = np.zeros((1, 3, V), dtype=np.float32)
    rows[0, 1, [600, 5, 300, 42]] = 4.0
    rows[0, 2, 77] = 1000.0
    got = _check(orc, rows, 1.0, 6)
    assert list(got["topk_id"][0, 0]) == [0, 1, 2, 3, 4, 5]
    assert list(got["topk_id"][0, 1][:4]) == [5, 42, 300, 600]
    np.testing.assert_allclose(got["lse"][0, 2], 1000.0, rtol=0, atol=1e-12)
    np.testing.assert_allclose(got["lse"][0, 0], np.log(V), rtol=1e-14)


def test_row_stats_broadcast_rows(orc):
    """A zero batch stride gives every tree the same statistics."""
    base = _rows(1, 2, 300, "f32", seed=3)
    rows = np.broadcast_to(base, (4, 2, 300))
    got = orc.row_stats(rows, 1.0, 4)
    for b in range(4):
        assert np.array_equal(got["lse"][b], got["lse"][0])
        assert np.array_equal(got["topk_id"][b], got["topk_id"][0])
