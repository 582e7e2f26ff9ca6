"""CPU oracle of the Tsubame per-step logit path (plan / replay / verify).

TEST INFRASTRUCTURE ONLY. Only the test suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline / reference legs may import this package. It is a plain, slow,
single-threaded fp64 reference written from the paper; it shares no code with the CUDA
library and never imports it. The arithmetic lives in ``tsb_oracle.c`` (plain C, built with
``-ffp-contract=off``); this module only marshals numpy arrays through ctypes.

Logit arrays are numpy arrays of shape [B, R, V], either ``float32`` or ``uint16`` holding
raw bf16 bit patterns. A zero batch stride (``np.broadcast_to``) shares one set of rows
across every tree.

Parity status of each function (what pins it, see tests/test_oracle_*.py):
  philox / uniform : published Philox4x32-10 known-answer vectors.
  row_stats        : numpy max, scipy logsumexp on numpy slices (row and every chunk),
                     numpy lexsort for the top-K (tests/test_oracle_row_stats.py).
  plan             : brute-force enumeration of every path + exact same-depth order;
                     exhaustive search for the maximum-probability prefix-closed set.
  replay           : chi-square against the closed-form ordered WoR law (flat and
                     hierarchical samplers separately).
  verify_rrs       : exact enumeration of the emitted-token law over all ordered child
                     tuples (= target law, Prop. 1); closed-form single-child acceptance
                     (Eq. rs-overlap); chi-square of the sampled path against the target.
  verify_traversal : exact enumeration of the extended output law on several topologies
                     (= target law); a chain gives block verification's law and a star
                     gives recursive rejection sampling's; the sampler against the exact
                     law (chi-square); sampled paths with path-keyed targets.
  verify_block     : exact enumeration of the extended output law (= target law);
                     gamma = 1 reduces to rejection sampling; E[tau] >= token-wise RS.
  plan_expand      : equals the heap planner once the frontier holds N; brute-force
                     path enumeration of the layer-wise frontiers; prefix closure; its
                     i-th path probability never above the heap's.
  replay_mixed     : deterministic slots vs a stable sort; chi-square of the sampled slot
                     against q renormalised over the remaining tokens; m = 1 is the WoR draw.
  verify_naive     : chi-square of the emitted tokens against the target law; acceptance
                     frequency vs the closed form p(y) (Sec. 2.3); forced acceptances.
  plan (pool=P)    : brute-force path enumeration with pooled normalisers; P = V is the
                     full-vocabulary planner.
  replay_pooled    : chi-square of ordered draws vs the WoR law of the pooled q; tokens stay
                     in the pool; P = V is the flat sampler token for token.
  verify_rrs(pool) : chi-square losslessness with pooled q; single-child acceptance
                     sum min(p, q_pool); P = V is the full-vocabulary verifier.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sys

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tsb_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None

CHUNK = 256

# Bound on another implementation's error in one draft row's log-normaliser (absolute, nats).
# The planner's near-tie flag for a pop between candidates at depths da and db is
# PLAN_LSE_ERR * |da - db| + 2^-30 * (da + db + 2) (see plan_band in tsb_oracle.c). An fp32
# implementation whose per-logit terms carry a relative error of a few 2^-24 (an exp2
# approximation, fp32 partial sums of 32 terms) and whose row sums and logarithm are carried in
# float-float stays well inside 1e-6; tests/test_gpu_accuracy.py holds the CUDA path's
# log-normalisers to this bound on every row of the workloads' draft rows.
PLAN_LSE_ERR = 1e-6
(PURPOSE_REPLAY_CHUNK, PURPOSE_REPLAY_ELEM, PURPOSE_ACCEPT, PURPOSE_FINAL, PURPOSE_BLOCK_ETA,
 PURPOSE_FINAL_CHUNK) = 0, 1, 2, 3, 4, 5


def build_command(out=_LIB_PATH):
    return ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
            "-o", out, _SRC, "-lm"]


def build(force: bool = False) -> str:
    """Compile the oracle into oracle/liboracle.so (skipped when up to date)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.run(build_command(tmp), check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Logits(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("dtype", ctypes.c_int32), ("B", ctypes.c_int32),
                ("R", ctypes.c_int32), ("V", ctypes.c_int32), ("batch_stride", ctypes.c_int64),
                ("row_stride", ctypes.c_int64)]


_P = ctypes.c_void_p
_I = ctypes.c_int32


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = ctypes.CDLL(_LIB_PATH)
    sig = {
        "orc_philox4x32_10": (None, [_P, _P, _P]),
        "orc_uniform": (ctypes.c_double, [ctypes.c_uint64, _I, _I, _I, _I]),
        "orc_row_stats": (_I, [_P, ctypes.c_float, _I, _P, _P, _P, _P, _P]),
        "orc_plan": (_I, [_P, ctypes.c_float, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, ctypes.c_double, _P, _P]),
        "orc_replay": (_I, [_P, ctypes.c_float, _P, _I, _P, _P, _P, ctypes.c_uint64, _P, _P, _P]),
        "orc_replay_flat": (_I, [_P, ctypes.c_float, _P, _I, _P, _P, _P, ctypes.c_uint64, _P, _P]),
        "orc_rrs_node_law": (_I, [_I, _P, _P, _I, _P, _P, _P]),
        "orc_verify_rrs": (_I, [_P, _P, ctypes.c_float, _P, _I, _I, _P, _P, _P, _P, ctypes.c_uint64, _P, _P, _P, _P,
                                _P]),
        "orc_blockv_law": (_I, [_I, _I, _P, _P, _P, _P, _P, _P]),
        "orc_plan_expand": (_I, [_P, ctypes.c_float, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, ctypes.c_double,
                                 _P]),
        "orc_replay_mixed": (_I, [_P, ctypes.c_float, _P, _I, _P, _P, _P, ctypes.c_uint64, _P, _P, _P]),
        "orc_verify_naive": (_I, [_P, ctypes.c_float, _I, _I, _P, _P, _P, ctypes.c_uint64, _P, _P, _P, _P, _P]),
        "orc_plan_pooled": (_I, [_P, ctypes.c_float, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, ctypes.c_double, _P,
                                 _P]),
        "orc_replay_pooled": (_I, [_P, ctypes.c_float, _P, _I, _P, _P, _P, _P, _I, _I, ctypes.c_uint64, _P, _P, _P]),
        "orc_verify_rrs_pooled": (_I, [_P, _P, ctypes.c_float, _P, _I, _I, _P, _P, _P, _P, ctypes.c_uint64, _P, _P, _I,
                                       _I, _P, _P, _P, _P]),
        "orc_verify_block": (_I, [_P, _P, ctypes.c_float, _P, _I, _I, _P, _P, _P, _P, ctypes.c_uint64, _P, _P, _P,
                                  _P, _P, _P]),
        "orc_verify_traversal": (_I, [_P, _P, ctypes.c_float, _P, _I, _I, _P, _P, _P, _P, _P, ctypes.c_uint64, _P,
                                      _P, _P, _P, _P]),
        "orc_traversal_law": (_I, [_I, _I, _P, _P, _P, _P, _P, _P, _P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _logits(arr: np.ndarray):
    """Describe a [B, R, V] float32 / bf16-bits array (last axis contiguous)."""
    if arr.ndim != 3:
        raise ValueError("logits must be [B, R, V]")
    if arr.dtype == np.float32:
        dt = 0
    elif arr.dtype == np.uint16:
        dt = 1
    else:
        raise TypeError("logits must be float32 or uint16 (bf16 bits)")
    it = arr.itemsize
    if arr.strides[2] != it:
        raise ValueError("vocabulary axis must be contiguous")
    d = _Logits(arr.ctypes.data, dt, arr.shape[0], arr.shape[1], arr.shape[2],
                arr.strides[0] // it, arr.strides[1] // it)
    return d, arr  # keep the array alive with the descriptor


def _i32(a):
    return None if a is None else np.ascontiguousarray(a, dtype=np.int32)


def _check(rc, what):
    if rc != 0:
        raise RuntimeError(f"oracle {what} failed with code {rc}")


# ---------------------------------------------------------------------------------------
def philox(ctr, key):
    lib = _load()
    c = np.asarray(ctr, dtype=np.uint32)
    k = np.asarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib.orc_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return out


def uniform(seed, purpose, batch, node, draw):
    return _load().orc_uniform(int(seed) & (2**64 - 1), purpose, batch, node, draw)


def row_stats(rows: np.ndarray, temperature: float, K: int = 1):
    lib = _load()
    B, R, V = rows.shape
    C = (V + CHUNK - 1) // CHUNK
    d, keep = _logits(rows)
    mx = np.zeros(B * R)
    lse = np.zeros(B * R)
    tid = np.zeros(B * R * K, dtype=np.int32)
    tx = np.zeros(B * R * K, dtype=np.float32)
    clse = np.zeros(B * R * C)
    _check(lib.orc_row_stats(ctypes.byref(d), temperature, K, _ptr(mx), _ptr(lse), _ptr(tid), _ptr(tx), _ptr(clse)),
           "row_stats")
    return {"max": mx.reshape(B, R), "lse": lse.reshape(B, R), "topk_id": tid.reshape(B, R, K),
            "topk_x": tx.reshape(B, R, K), "chunk_lse": clse.reshape(B, R, C)}


def plan(draft: np.ndarray, temperature: float, N: int, K: int, L: int, lse_err: float = PLAN_LSE_ERR,
         pool: int = 0):
    """First pass; ``pool`` = P > 0 normalises each depth's law over its P most probable tokens."""
    lib = _load()
    B = draft.shape[0]
    NN = N + 1
    d, keep = _logits(draft)
    out = {k: np.zeros(B * NN, dtype=np.int32) for k in ("parent", "depth", "rank", "plan_token")}
    score = np.zeros(B * NN)
    child_off = np.zeros(B * (NN + 1), dtype=np.int32)
    child_ids = np.zeros(B * N, dtype=np.int32)
    exempt = np.zeros(B, dtype=np.uint8)
    margin = np.zeros(B)
    if pool:
        rc = lib.orc_plan_pooled(ctypes.byref(d), temperature, N, K, L, int(pool), _ptr(out["parent"]),
                                 _ptr(out["depth"]), _ptr(out["rank"]), _ptr(out["plan_token"]), _ptr(score),
                                 _ptr(child_off), _ptr(child_ids), lse_err, _ptr(exempt), _ptr(margin))
    else:
        rc = lib.orc_plan(ctypes.byref(d), temperature, N, K, L, _ptr(out["parent"]), _ptr(out["depth"]),
                          _ptr(out["rank"]), _ptr(out["plan_token"]), _ptr(score), _ptr(child_off), _ptr(child_ids),
                          lse_err, _ptr(exempt), _ptr(margin))
    _check(rc, "plan")
    tree = {k: v.reshape(B, NN) for k, v in out.items()}
    tree["score"] = score.reshape(B, NN)
    tree["child_off"] = child_off.reshape(B, NN + 1)
    tree["child_ids"] = child_ids.reshape(B, N)
    tree["exempt"] = exempt.astype(bool)
    tree["min_margin"] = margin
    return tree


def plan_expand(draft: np.ndarray, temperature: float, N: int, K: int, L: int, W: int,
                lse_err: float = PLAN_LSE_ERR):
    """Expand-then-prune first pass with frontier width W; same outputs as ``plan``."""
    lib = _load()
    B = draft.shape[0]
    NN = N + 1
    d, keep = _logits(draft)
    out = {k: np.zeros(B * NN, dtype=np.int32) for k in ("parent", "depth", "rank", "plan_token")}
    score = np.zeros(B * NN)
    child_off = np.zeros(B * (NN + 1), dtype=np.int32)
    child_ids = np.zeros(B * N, dtype=np.int32)
    exempt = np.zeros(B, dtype=np.uint8)
    _check(lib.orc_plan_expand(ctypes.byref(d), temperature, N, K, L, W, _ptr(out["parent"]), _ptr(out["depth"]),
                               _ptr(out["rank"]), _ptr(out["plan_token"]), _ptr(score), _ptr(child_off),
                               _ptr(child_ids), lse_err, _ptr(exempt)), "plan_expand")
    tree = {k: v.reshape(B, NN) for k, v in out.items()}
    tree["score"] = score.reshape(B, NN)
    tree["child_off"] = child_off.reshape(B, NN + 1)
    tree["child_ids"] = child_ids.reshape(B, N)
    tree["exempt"] = exempt.astype(bool)
    return tree


def _tree_ptrs(tree):
    return (_i32(tree["depth"]), _i32(tree["child_off"]), _i32(tree["child_ids"]))


def replay(q: np.ndarray, temperature: float, tree, seed: int, qrow_of_node=None, flat: bool = False,
           batch_ids=None):
    """Tokens [B, N+1] (root -1) and, for the hierarchical sampler, a per-parent near-tie flag.
    ``batch_ids`` gives the Philox batch index of each tree (default 0..B-1)."""
    lib = _load()
    bids = _i32(batch_ids)
    B = q.shape[0]
    NN = tree["depth"].shape[1]
    d, keep = _logits(q)
    depth, off, ids = _tree_ptrs(tree)
    qr = _i32(qrow_of_node)
    token = np.zeros(B * NN, dtype=np.int32)
    if flat:
        _check(lib.orc_replay_flat(ctypes.byref(d), temperature, _ptr(qr), NN - 1, _ptr(depth), _ptr(off), _ptr(ids),
                                   int(seed), _ptr(bids), _ptr(token)), "replay_flat")
        return token.reshape(B, NN)
    exempt = np.zeros(B * NN, dtype=np.uint8)
    _check(lib.orc_replay(ctypes.byref(d), temperature, _ptr(qr), NN - 1, _ptr(depth), _ptr(off), _ptr(ids),
                          int(seed), _ptr(bids), _ptr(token), _ptr(exempt)), "replay")
    return token.reshape(B, NN), exempt.reshape(B, NN).astype(bool)


def replay_mixed(q: np.ndarray, temperature: float, tree, seed: int, qrow_of_node=None, batch_ids=None):
    """Mixed sampling: tokens [B, N+1] (root -1) and a per-parent near-tie flag."""
    lib = _load()
    bids = _i32(batch_ids)
    B = q.shape[0]
    NN = tree["depth"].shape[1]
    d, keep = _logits(q)
    depth, off, ids = _tree_ptrs(tree)
    qr = _i32(qrow_of_node)
    token = np.zeros(B * NN, dtype=np.int32)
    exempt = np.zeros(B * NN, dtype=np.uint8)
    _check(lib.orc_replay_mixed(ctypes.byref(d), temperature, _ptr(qr), NN - 1, _ptr(depth), _ptr(off), _ptr(ids),
                                int(seed), _ptr(bids), _ptr(token), _ptr(exempt)), "replay_mixed")
    return token.reshape(B, NN), exempt.reshape(B, NN).astype(bool)


def verify_naive(target: np.ndarray, temperature: float, tree, token, seed: int, L: int, batch_ids=None):
    """Target-sample matching down the tree; outputs as ``verify_rrs``."""
    lib = _load()
    bids = _i32(batch_ids)
    B = target.shape[0]
    NN = tree["child_off"].shape[1] - 1
    dt, keep_t = _logits(target)
    off, ids = _i32(tree["child_off"]), _i32(tree["child_ids"])
    tok = _i32(token)
    otok = np.zeros(B * (L + 1), dtype=np.int32)
    onode = np.zeros(B * L, dtype=np.int32)
    olen = np.zeros(B, dtype=np.int32)
    ex = np.zeros(B, dtype=np.uint8)
    _check(lib.orc_verify_naive(ctypes.byref(dt), temperature, NN - 1, L, _ptr(off), _ptr(ids), _ptr(tok), int(seed),
                                _ptr(bids), _ptr(otok), _ptr(onode), _ptr(olen), _ptr(ex)), "verify_naive")
    return {"tokens": otok.reshape(B, L + 1), "nodes": onode.reshape(B, L), "len": olen, "exempt": ex.astype(bool)}


def pools(draft: np.ndarray, temperature: float, P: int):
    """Per (tree, depth row) the P most probable tokens by (x desc, id asc): [B, R, P] int32."""
    return np.ascontiguousarray(row_stats(draft, temperature, P)["topk_id"])


def replay_pooled(q: np.ndarray, temperature: float, tree, seed: int, pool_ids: np.ndarray, qrow_of_node=None,
                  batch_ids=None):
    """WoR draws from the pooled draft laws; pool_ids [B, Lp, P]. Tokens [B, N+1] and near-tie flags."""
    lib = _load()
    bids = _i32(batch_ids)
    B = q.shape[0]
    NN = tree["depth"].shape[1]
    d, keep = _logits(q)
    depth, off, ids = _tree_ptrs(tree)
    qr = _i32(qrow_of_node)
    pl = _i32(pool_ids)
    token = np.zeros(B * NN, dtype=np.int32)
    exempt = np.zeros(B * NN, dtype=np.uint8)
    _check(lib.orc_replay_pooled(ctypes.byref(d), temperature, _ptr(qr), NN - 1, _ptr(depth), _ptr(off), _ptr(ids),
                                 _ptr(pl), pl.shape[2], pl.shape[1], int(seed), _ptr(bids), _ptr(token),
                                 _ptr(exempt)), "replay_pooled")
    return token.reshape(B, NN), exempt.reshape(B, NN).astype(bool)


def verify_rrs(target: np.ndarray, q: np.ndarray, temperature: float, tree, token, seed: int, L: int,
               qrow_of_node=None, batch_ids=None, pool_ids=None):
    """Recursive rejection sampling; with ``pool_ids`` [B, Lp, P] the draft laws are pooled."""
    lib = _load()
    bids = _i32(batch_ids)
    B = target.shape[0]
    NN = tree["depth"].shape[1]
    dt, keep_t = _logits(target)
    dq, keep_q = _logits(q)
    depth, off, ids = _tree_ptrs(tree)
    tok = _i32(token)
    qr = _i32(qrow_of_node)
    otok = np.zeros(B * (L + 1), dtype=np.int32)
    onode = np.zeros(B * L, dtype=np.int32)
    olen = np.zeros(B, dtype=np.int32)
    ex = np.zeros(B, dtype=np.uint8)
    if pool_ids is not None:
        pl = _i32(pool_ids)
        rc = lib.orc_verify_rrs_pooled(ctypes.byref(dt), ctypes.byref(dq), temperature, _ptr(qr), NN - 1, L,
                                       _ptr(depth), _ptr(off), _ptr(ids), _ptr(tok), int(seed), _ptr(bids), _ptr(pl),
                                       pl.shape[2], pl.shape[1], _ptr(otok), _ptr(onode), _ptr(olen), _ptr(ex))
    else:
        rc = lib.orc_verify_rrs(ctypes.byref(dt), ctypes.byref(dq), temperature, _ptr(qr), NN - 1, L, _ptr(depth),
                                _ptr(off), _ptr(ids), _ptr(tok), int(seed), _ptr(bids), _ptr(otok), _ptr(onode),
                                _ptr(olen), _ptr(ex))
    _check(rc, "verify_rrs")
    return {"tokens": otok.reshape(B, L + 1), "nodes": onode.reshape(B, L), "len": olen, "exempt": ex.astype(bool)}


def verify_block(target: np.ndarray, q: np.ndarray, temperature: float, tree, token, seed: int, L: int,
                 qrow_of_node=None, batch_ids=None):
    lib = _load()
    bids = _i32(batch_ids)
    B = target.shape[0]
    NN = tree["depth"].shape[1]
    dt, keep_t = _logits(target)
    dq, keep_q = _logits(q)
    depth, off, ids = _tree_ptrs(tree)
    tok = _i32(token)
    qr = _i32(qrow_of_node)
    otok = np.zeros(B * (L + 1), dtype=np.int32)
    onode = np.zeros(B * L, dtype=np.int32)
    olen = np.zeros(B, dtype=np.int32)
    ex = np.zeros(B, dtype=np.uint8)
    tau = np.zeros(B, dtype=np.int32)
    _check(lib.orc_verify_block(ctypes.byref(dt), ctypes.byref(dq), temperature, _ptr(qr), NN - 1, L, _ptr(depth),
                                _ptr(off), _ptr(ids), _ptr(tok), int(seed), _ptr(bids), _ptr(otok), _ptr(onode),
                                _ptr(olen), _ptr(ex), _ptr(tau)), "verify_block")
    return {"tokens": otok.reshape(B, L + 1), "nodes": onode.reshape(B, L), "len": olen, "exempt": ex.astype(bool),
            "tau": tau}


def verify_traversal(target: np.ndarray, q: np.ndarray, temperature: float, tree, token, seed: int, L: int,
                     qrow_of_node=None, batch_ids=None):
    """Traversal verification (sequence-level recursive rejection sampling); outputs as
    ``verify_rrs``."""
    lib = _load()
    bids = _i32(batch_ids)
    B = target.shape[0]
    NN = tree["depth"].shape[1]
    dt, keep_t = _logits(target)
    dq, keep_q = _logits(q)
    depth, off, ids = _tree_ptrs(tree)
    parent = _i32(tree["parent"])
    tok = _i32(token)
    qr = _i32(qrow_of_node)
    otok = np.zeros(B * (L + 1), dtype=np.int32)
    onode = np.zeros(B * L, dtype=np.int32)
    olen = np.zeros(B, dtype=np.int32)
    ex = np.zeros(B, dtype=np.uint8)
    _check(lib.orc_verify_traversal(ctypes.byref(dt), ctypes.byref(dq), temperature, _ptr(qr), NN - 1, L,
                                    _ptr(parent), _ptr(depth), _ptr(off), _ptr(ids), _ptr(tok), int(seed), _ptr(bids),
                                    _ptr(otok), _ptr(onode), _ptr(olen), _ptr(ex)), "verify_traversal")
    return {"tokens": otok.reshape(B, L + 1), "nodes": onode.reshape(B, L), "len": olen, "exempt": ex.astype(bool)}


def traversal_law(child_off, child_ids, token, P_rows, Q_rows):
    """Exact law of traversal verification on one tree: (acc[NN], final_law[NN, V], degenerate)."""
    lib = _load()
    P_rows = np.ascontiguousarray(P_rows, dtype=np.float64)
    Q_rows = np.ascontiguousarray(Q_rows, dtype=np.float64)
    NN, V = P_rows.shape
    off, ids, tok = _i32(child_off), _i32(child_ids), _i32(token)
    acc = np.zeros(NN)
    law = np.zeros(NN * V)
    deg = lib.orc_traversal_law(NN, V, _ptr(off), _ptr(ids), _ptr(tok), _ptr(P_rows), _ptr(Q_rows), _ptr(acc),
                                _ptr(law))
    if deg < 0:
        raise RuntimeError(f"oracle traversal_law failed with code {deg}")
    return acc, law.reshape(NN, V), bool(deg)


def rrs_node_law(P, Q, y):
    """Per-slot acceptance probabilities and final-token law of one node, fixed tuple y."""
    lib = _load()
    P = np.ascontiguousarray(P, dtype=np.float64)
    Q = np.ascontiguousarray(Q, dtype=np.float64)
    yy = _i32(y)
    acc = np.zeros(len(yy))
    fin = np.zeros(len(P))
    deg = lib.orc_rrs_node_law(len(P), _ptr(P), _ptr(Q), len(yy), _ptr(yy), _ptr(acc), _ptr(fin))
    return acc, fin, bool(deg)


def blockv_law(Mb, Ms, X):
    """(w, h, unnormalised residuals) of block verification for one chain X."""
    lib = _load()
    Mb = np.ascontiguousarray(Mb, dtype=np.float64)
    Ms = np.ascontiguousarray(Ms, dtype=np.float64)
    XX = _i32(X)
    g = len(XX)
    V = Mb.shape[1]
    w = np.zeros(g + 1)
    h = np.zeros(g + 1)
    resid = np.zeros(g * V)
    lib.orc_blockv_law(g, V, _ptr(Mb), _ptr(Ms), _ptr(XX), _ptr(w), _ptr(h), _ptr(resid))
    return w, h, resid.reshape(g, V)


if __name__ == "__main__":  # pragma: no cover
    build(force="--force" in sys.argv)
    print(_LIB_PATH)
