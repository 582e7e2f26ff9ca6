"""ctypes binding of libtsb (include/tsb.h). Argument marshalling only: every step of the
path runs in the library's CUDA kernels. Tensors are torch CUDA tensors (torch provides the
device memory and the current stream); nothing here computes on their contents.

The functions carry the C names: tsb_row_stats, tsb_plan, tsb_replay, tsb_verify, ...
They raise TsbError on any status other than TSB_OK. ``TsbBuffers`` allocates (with torch)
every output and scratch buffer one configuration needs.
"""
from __future__ import annotations

import contextlib
import ctypes
import os
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libtsb.so")
LIB_CHECKED_PATH = os.path.join(_HERE, "libtsb_checked.so")

TSB_OK = 0
STATUS_NAMES = {0: "TSB_OK", 1: "TSB_ERR_ARG", 2: "TSB_ERR_SHAPE", 3: "TSB_ERR_DTYPE", 4: "TSB_ERR_ALIGN",
                5: "TSB_ERR_WORKSPACE", 6: "TSB_ERR_CUDA", 7: "TSB_ERR_DEVICE"}
TSB_F32, TSB_BF16 = 0, 1
TSB_VERIFY_RRS, TSB_VERIFY_BLOCK, TSB_VERIFY_NAIVE, TSB_VERIFY_TRAVERSAL = 0, 1, 2, 3
TSB_DEV_NONFINITE, TSB_DEV_BAD_INDEX, TSB_DEV_BAD_TREE, TSB_DEV_CHECK = 0x1, 0x2, 0x4, 0x8
TSB_CHUNK = 256

EXPORTS = ("tsb_version", "tsb_status_str", "tsb_stats_bytes", "tsb_workspace_bytes", "tsb_workspace_init",
           "tsb_device_status", "tsb_row_stats", "tsb_plan", "tsb_replay", "tsb_verify", "tsb_plan_noalloc",
           "tsb_plan_rows", "tsb_plan_expand", "tsb_plan_rows_expand", "tsb_replay_mixed", "tsb_plan_pooled",
           "tsb_replay_pooled", "tsb_verify_pooled", "tsb_replay_verify")
TSB_NOALLOC_SCRATCH_BYTES = 1 << 20
TSB_MAX_WIDTH = 1024
TSB_MAX_EXPAND_CANDIDATES = 8192
TSB_MAX_POOL = 64


class TsbError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {STATUS_NAMES.get(status, status)}")


class Logits(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("dtype", ctypes.c_int32), ("B", ctypes.c_int32), ("R", ctypes.c_int32),
                ("V", ctypes.c_int32), ("batch_stride", ctypes.c_int64), ("row_stride", ctypes.c_int64)]


class Cfg(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("L", ctypes.c_int32), ("N", ctypes.c_int32), ("K", ctypes.c_int32),
                ("V", ctypes.c_int32), ("temperature", ctypes.c_float)]


class Tree(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("parent", "depth", "rank", "plan_token", "score", "child_off",
                                               "child_ids")]


_lib = None
_P = ctypes.c_void_p
_SZ = ctypes.c_size_t
_I32 = ctypes.c_int32


def library_path() -> str:
    return LIB_PATH


def load():
    """Load libtsb.so; fails loudly if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    _lib = _open(LIB_PATH)
    return _lib


@contextlib.contextmanager
def checked_library():
    """Within the block every call goes to libtsb_checked.so (the TSB_CHECKED build)."""
    global _lib
    saved = load()
    _lib = _open(LIB_CHECKED_PATH)
    try:
        yield _lib
    finally:
        _lib = saved


def _open(path):
    if not os.path.exists(path):
        raise RuntimeError(f"{os.path.basename(path)} not found at {path}; build it with "
                           "`python -m paper_2609_33652_gb300.build` (or __graft_entry__.build())")
    lib = ctypes.CDLL(path)
    sig = {
        "tsb_version": (_I32, []),
        "tsb_status_str": (ctypes.c_char_p, [_I32]),
        "tsb_stats_bytes": (_SZ, [_I32, _I32, _I32]),
        "tsb_workspace_bytes": (_SZ, [_P]),
        "tsb_workspace_init": (_I32, [_P, _SZ, _P]),
        "tsb_device_status": (_I32, [_P, _P, _P]),
        "tsb_row_stats": (_I32, [_P, ctypes.c_float, _P, _SZ, _P, _SZ, _P]),
        "tsb_plan": (_I32, [_P, _P, _P, _SZ, _P, _P, _SZ, _P]),
        "tsb_plan_noalloc": (_I32, [_P, _P, _P, _SZ, _P, _P, _P]),
        "tsb_plan_rows": (_I32, [_P, _P, _P, _SZ, _P, _P, _SZ, _P]),
        "tsb_replay": (_I32, [_P, _P, _P, _SZ, _P, _P, ctypes.c_uint64, _P, _P, _SZ, _P]),
        "tsb_replay_mixed": (_I32, [_P, _P, _P, _SZ, _P, _P, ctypes.c_uint64, _P, _P, _SZ, _P]),
        "tsb_plan_expand": (_I32, [_P, _I32, _P, _P, _SZ, _P, _P, _SZ, _P]),
        "tsb_plan_rows_expand": (_I32, [_P, _I32, _P, _P, _SZ, _P, _P, _SZ, _P]),
        "tsb_plan_pooled": (_I32, [_P, _I32, _P, _P, _SZ, _P, _P, _P, _SZ, _P]),
        "tsb_replay_pooled": (_I32, [_P, _I32, _P, _P, _P, _P, ctypes.c_uint64, _P, _P, _SZ, _P]),
        "tsb_verify_pooled": (_I32, [_P, _I32, _P, _P, _P, _P, _P, _P, ctypes.c_uint64, _P, _P, _P, _P, _SZ, _P]),
        "tsb_verify": (_I32, [_P, _I32, _P, _P, _P, _SZ, _P, _P, _P, ctypes.c_uint64, _P, _P, _P, _P, _SZ, _P]),
        "tsb_replay_verify": (_I32, [_P, _P, _P, _P, _SZ, _P, _P, ctypes.c_uint64, _P, _P, _P, _P, _P, _SZ, _P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


def _check(rc: int, what: str):
    if rc != TSB_OK:
        raise TsbError(rc, what)


def _stream(stream=None):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def logits_desc(t: torch.Tensor) -> Logits:
    """Descriptor of a [B, R, V] float32 / bfloat16 CUDA tensor (vocabulary axis contiguous;
    a broadcast batch axis, stride 0, is allowed)."""
    if t.dim() != 3:
        raise ValueError("logits must be [B, R, V]")
    if t.dtype == torch.float32:
        dt = TSB_F32
    elif t.dtype == torch.bfloat16:
        dt = TSB_BF16
    else:
        raise TypeError(f"logits dtype {t.dtype} not supported (float32 or bfloat16)")
    if t.stride(2) != 1:
        raise ValueError("the vocabulary axis must be contiguous")
    B, R, V = t.shape
    return Logits(t.data_ptr(), dt, B, R, V, t.stride(0), t.stride(1))


def make_cfg(B, L, N, K, V, temperature) -> Cfg:
    return Cfg(B, L, N, K, V, float(temperature))


def tsb_version() -> int:
    return load().tsb_version()


def tsb_status_str(status: int) -> str:
    return load().tsb_status_str(status).decode()


def tsb_stats_bytes(B: int, R: int, V: int) -> int:
    return load().tsb_stats_bytes(B, R, V)


def tsb_workspace_bytes(cfg: Cfg) -> int:
    return load().tsb_workspace_bytes(ctypes.byref(cfg))


def tsb_workspace_init(ws: torch.Tensor, stream=None):
    _check(load().tsb_workspace_init(_ptr(ws), ws.numel() * ws.element_size(), _stream(stream)),
           "tsb_workspace_init")


def tsb_device_status(ws: torch.Tensor, stream=None) -> int:
    """Device status bits since the last call (0 = clean); waits for the stream."""
    bits = ctypes.c_uint32(0)
    rc = load().tsb_device_status(_ptr(ws), _stream(stream), ctypes.byref(bits))
    if rc not in (TSB_OK, 7):
        raise TsbError(rc, "tsb_device_status")
    return bits.value


def tsb_row_stats(rows: torch.Tensor, temperature: float, stats: torch.Tensor, ws: torch.Tensor, stream=None):
    d = logits_desc(rows)
    _check(load().tsb_row_stats(ctypes.byref(d), float(temperature), _ptr(stats), stats.numel() * stats.element_size(),
                                _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)), "tsb_row_stats")


def tree_struct(tree: dict) -> Tree:
    return Tree(*[(tree[k].data_ptr() if tree.get(k) is not None else None)
                  for k in ("parent", "depth", "rank", "plan_token", "score", "child_off", "child_ids")])


def tsb_plan(cfg: Cfg, draft: torch.Tensor, stats: torch.Tensor, tree: dict, ws: torch.Tensor, stream=None):
    d = logits_desc(draft)
    t = tree_struct(tree)
    _check(load().tsb_plan(ctypes.byref(cfg), ctypes.byref(d), _ptr(stats), stats.numel() * stats.element_size(),
                           ctypes.byref(t), _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)), "tsb_plan")


def tsb_plan_rows(cfg: Cfg, draft: torch.Tensor, stats: torch.Tensor, tree: dict, ws: torch.Tensor, stream=None):
    """tsb_row_stats of draft rows 0..L-1 (written into ``stats``) and tsb_plan in one pass."""
    d = logits_desc(draft)
    t = tree_struct(tree)
    _check(load().tsb_plan_rows(ctypes.byref(cfg), ctypes.byref(d), _ptr(stats), stats.numel() * stats.element_size(),
                                ctypes.byref(t), _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)),
           "tsb_plan_rows")


def tsb_plan_expand(cfg: Cfg, width: int, draft: torch.Tensor, stats: torch.Tensor, tree: dict, ws: torch.Tensor,
                    stream=None):
    """Expand-then-prune first pass with frontier width ``width`` (stats from tsb_row_stats)."""
    d = logits_desc(draft)
    t = tree_struct(tree)
    _check(load().tsb_plan_expand(ctypes.byref(cfg), int(width), ctypes.byref(d), _ptr(stats),
                                  stats.numel() * stats.element_size(), ctypes.byref(t), _ptr(ws),
                                  ws.numel() * ws.element_size(), _stream(stream)), "tsb_plan_expand")


def tsb_plan_rows_expand(cfg: Cfg, width: int, draft: torch.Tensor, stats: torch.Tensor, tree: dict,
                         ws: torch.Tensor, stream=None):
    """Statistics of draft rows 0..L-1 (written into ``stats``) and the expand-then-prune pass."""
    d = logits_desc(draft)
    t = tree_struct(tree)
    _check(load().tsb_plan_rows_expand(ctypes.byref(cfg), int(width), ctypes.byref(d), _ptr(stats),
                                       stats.numel() * stats.element_size(), ctypes.byref(t), _ptr(ws),
                                       ws.numel() * ws.element_size(), _stream(stream)), "tsb_plan_rows_expand")


def tsb_plan_pooled(cfg: Cfg, P: int, draft: torch.Tensor, stats: torch.Tensor, pool_ids: torch.Tensor, tree: dict,
                    ws: torch.Tensor, stream=None):
    """First pass with pooled draft laws; writes the pools [B, L, P] int32 into ``pool_ids``."""
    d = logits_desc(draft)
    t = tree_struct(tree)
    _check(load().tsb_plan_pooled(ctypes.byref(cfg), int(P), ctypes.byref(d), _ptr(stats),
                                  stats.numel() * stats.element_size(), _ptr(pool_ids), ctypes.byref(t), _ptr(ws),
                                  ws.numel() * ws.element_size(), _stream(stream)), "tsb_plan_pooled")


def tsb_replay_pooled(cfg: Cfg, P: int, qrows: torch.Tensor, qrow_of_node, pool_ids: torch.Tensor, tree: dict,
                      seed: int, token: torch.Tensor, ws: torch.Tensor, stream=None):
    d = logits_desc(qrows)
    t = tree_struct(tree)
    _check(load().tsb_replay_pooled(ctypes.byref(cfg), int(P), ctypes.byref(d), _ptr(qrow_of_node), _ptr(pool_ids),
                                    ctypes.byref(t), int(seed) & (2**64 - 1), _ptr(token), _ptr(ws),
                                    ws.numel() * ws.element_size(), _stream(stream)), "tsb_replay_pooled")


def tsb_verify_pooled(cfg: Cfg, P: int, target: torch.Tensor, qrows: torch.Tensor, qrow_of_node, pool_ids, tree: dict,
                      token: torch.Tensor, seed: int, out_tokens: torch.Tensor, out_nodes: torch.Tensor,
                      out_len: torch.Tensor, ws: torch.Tensor, stream=None):
    dt = logits_desc(target)
    dq = logits_desc(qrows)
    t = tree_struct(tree)
    _check(load().tsb_verify_pooled(ctypes.byref(cfg), int(P), ctypes.byref(dt), ctypes.byref(dq), _ptr(qrow_of_node),
                                    _ptr(pool_ids), ctypes.byref(t), _ptr(token), int(seed) & (2**64 - 1),
                                    _ptr(out_tokens), _ptr(out_nodes), _ptr(out_len), _ptr(ws),
                                    ws.numel() * ws.element_size(), _stream(stream)), "tsb_verify_pooled")


def tsb_plan_noalloc(cfg: Cfg, draft: torch.Tensor, stats: torch.Tensor, tree: dict, dev_status=None, stream=None):
    """tsb_plan with the library's static device scratch instead of a workspace; the C call
    allocates nothing. ``dev_status``: optional int32 CUDA tensor whose first word receives
    the device status bits."""
    d = logits_desc(draft)
    t = tree_struct(tree)
    _check(load().tsb_plan_noalloc(ctypes.byref(cfg), ctypes.byref(d), _ptr(stats),
                                   stats.numel() * stats.element_size(), ctypes.byref(t), _ptr(dev_status),
                                   _stream(stream)), "tsb_plan_noalloc")


def tsb_replay(cfg: Cfg, qrows: torch.Tensor, qstats: torch.Tensor, qrow_of_node, tree: dict, seed: int,
               token: torch.Tensor, ws: torch.Tensor, stream=None):
    d = logits_desc(qrows)
    t = tree_struct(tree)
    _check(load().tsb_replay(ctypes.byref(cfg), ctypes.byref(d), _ptr(qstats), qstats.numel() * qstats.element_size(),
                             _ptr(qrow_of_node), ctypes.byref(t), int(seed) & (2**64 - 1), _ptr(token), _ptr(ws),
                             ws.numel() * ws.element_size(), _stream(stream)), "tsb_replay")


def tsb_replay_mixed(cfg: Cfg, qrows: torch.Tensor, qstats: torch.Tensor, qrow_of_node, tree: dict, seed: int,
                     token: torch.Tensor, ws: torch.Tensor, stream=None):
    """Mixed sampling: the m-1 most probable tokens, then one draw from the rest."""
    d = logits_desc(qrows)
    t = tree_struct(tree)
    _check(load().tsb_replay_mixed(ctypes.byref(cfg), ctypes.byref(d), _ptr(qstats),
                                   qstats.numel() * qstats.element_size(), _ptr(qrow_of_node), ctypes.byref(t),
                                   int(seed) & (2**64 - 1), _ptr(token), _ptr(ws), ws.numel() * ws.element_size(),
                                   _stream(stream)), "tsb_replay_mixed")


def tsb_verify(cfg: Cfg, mode: int, target: torch.Tensor, qrows, qstats, qrow_of_node,
               tree: dict, token: torch.Tensor, seed: int, out_tokens: torch.Tensor, out_nodes: torch.Tensor,
               out_len: torch.Tensor, ws: torch.Tensor, stream=None):
    """``qrows`` / ``qstats`` may be None for TSB_VERIFY_NAIVE."""
    dt = logits_desc(target)
    dq = logits_desc(qrows) if qrows is not None else None
    t = tree_struct(tree)
    qsb = qstats.numel() * qstats.element_size() if qstats is not None else 0
    _check(load().tsb_verify(ctypes.byref(cfg), int(mode), ctypes.byref(dt), ctypes.byref(dq) if dq is not None else None,
                             _ptr(qstats), qsb, _ptr(qrow_of_node), ctypes.byref(t), _ptr(token),
                             int(seed) & (2**64 - 1), _ptr(out_tokens), _ptr(out_nodes), _ptr(out_len), _ptr(ws),
                             ws.numel() * ws.element_size(), _stream(stream)), "tsb_verify")


def tsb_replay_verify(cfg: Cfg, target: torch.Tensor, qrows: torch.Tensor, qstats: torch.Tensor, qrow_of_node,
                      tree: dict, seed: int, token: torch.Tensor, out_tokens: torch.Tensor, out_nodes: torch.Tensor,
                      out_len: torch.Tensor, ws: torch.Tensor, stream=None):
    """tsb_replay then tsb_verify (recursive rejection sampling) in one call."""
    dt = logits_desc(target)
    dq = logits_desc(qrows)
    t = tree_struct(tree)
    _check(load().tsb_replay_verify(ctypes.byref(cfg), ctypes.byref(dt), ctypes.byref(dq), _ptr(qstats),
                                    qstats.numel() * qstats.element_size(), _ptr(qrow_of_node), ctypes.byref(t),
                                    int(seed) & (2**64 - 1), _ptr(token), _ptr(out_tokens), _ptr(out_nodes),
                                    _ptr(out_len), _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)),
           "tsb_replay_verify")


# ---------------------------------------------------------------------------------------
@dataclass
class TsbBuffers:
    """Device buffers for one configuration (allocated with torch, owned by this object)."""
    cfg: Cfg
    ws: torch.Tensor
    stats: torch.Tensor
    tree: dict
    token: torch.Tensor
    out_tokens: torch.Tensor
    out_nodes: torch.Tensor
    out_len: torch.Tensor

    @staticmethod
    def allocate(B, L, N, K, V, temperature, draft_rows=None, device="cuda"):
        cfg = make_cfg(B, L, N, K, V, temperature)
        wsb = tsb_workspace_bytes(cfg)
        if wsb == 0:
            raise TsbError(2, "invalid configuration")
        R = draft_rows if draft_rows is not None else L
        ws = torch.zeros((wsb + 255) // 256 * 256, dtype=torch.uint8, device=device)
        stats = torch.empty(tsb_stats_bytes(B, R, V) // 4, dtype=torch.float32, device=device)
        NN = N + 1
        i32 = dict(dtype=torch.int32, device=device)
        tree = {"parent": torch.empty(B, NN, **i32), "depth": torch.empty(B, NN, **i32),
                "rank": torch.empty(B, NN, **i32), "plan_token": torch.empty(B, NN, **i32),
                "score": torch.empty(B, NN, dtype=torch.float32, device=device),
                "child_off": torch.empty(B, NN + 1, **i32), "child_ids": torch.empty(B, max(N, 1), **i32)}
        return TsbBuffers(cfg, ws, stats, tree, torch.empty(B, NN, **i32), torch.empty(B, L + 1, **i32),
                          torch.empty(B, L, **i32), torch.empty(B, **i32))


class PreparedStep:
    """One plan -> replay -> verify step with every ctypes argument built in advance, so a
    timing loop pays only the C calls. ``calls`` holds (name, function, args) in launch order:
    tsb_plan_rows (or, with ``width``, tsb_plan_rows_expand), tsb_replay (``replay="wor"``),
    tsb_replay_mixed (``"mixed"``) or nothing (``"plan"``: the first pass's tokens are
    verified), then tsb_verify in ``mode``. With ``fused=False`` the first pass is
    tsb_row_stats + tsb_plan instead; with ``plan_only`` only the first pass runs. With
    ``qrows`` (per-node draft rows [B, Rq, V]), ``qstats`` (their statistics buffer) and
    ``qrow_of_node`` ([B, N+1]), the step also runs tsb_row_stats on the q rows, and replay and
    verification draw from them (the corrected-drafter workload). With ``together`` (the default;
    WoR replay and recursive rejection sampling only) the two are one tsb_replay_verify call."""

    def __init__(self, buf: TsbBuffers, draft: torch.Tensor, target: torch.Tensor, seed: int, mode=TSB_VERIFY_RRS,
                 out_tokens=None, out_nodes=None, out_len=None, stream=None, fused=True, width=None, replay="wor",
                 plan_only=False, qrows=None, qstats=None, qrow_of_node=None, together=True):
        lib = load()
        self._keep = []
        s = _stream(stream)
        dd = logits_desc(draft)
        dt = logits_desc(target)
        tr = tree_struct(buf.tree)
        cfg = buf.cfg
        self._keep += [dd, dt, tr, cfg, draft, target, buf]
        sb = buf.stats.numel() * buf.stats.element_size()
        wb = buf.ws.numel() * buf.ws.element_size()
        ot = buf.out_tokens if out_tokens is None else out_tokens
        on = buf.out_nodes if out_nodes is None else out_nodes
        ol = buf.out_len if out_len is None else out_len
        self._keep += [ot, on, ol]
        seed = int(seed) & (2**64 - 1)
        if width is not None:
            plan = [("tsb_plan_rows_expand", lib.tsb_plan_rows_expand,
                     (ctypes.byref(cfg), int(width), ctypes.byref(dd), _ptr(buf.stats), sb, ctypes.byref(tr),
                      _ptr(buf.ws), wb, s))]
        elif fused:
            plan = [("tsb_plan_rows", lib.tsb_plan_rows, (ctypes.byref(cfg), ctypes.byref(dd), _ptr(buf.stats), sb,
                                                          ctypes.byref(tr), _ptr(buf.ws), wb, s))]
        else:
            plan = [("tsb_row_stats", lib.tsb_row_stats,
                     (ctypes.byref(dd), ctypes.c_float(cfg.temperature), _ptr(buf.stats), sb, _ptr(buf.ws), wb, s)),
                    ("tsb_plan", lib.tsb_plan, (ctypes.byref(cfg), ctypes.byref(dd), _ptr(buf.stats), sb,
                                                ctypes.byref(tr), _ptr(buf.ws), wb, s))]
        tok = buf.tree["plan_token"] if replay == "plan" else buf.token
        qcalls = []
        if qrows is not None:  # per-node draft rows: their statistics first
            dq = logits_desc(qrows)
            self._keep += [dq, qrows, qstats, qrow_of_node]
            qsb_ = qstats.numel() * qstats.element_size()
            qcalls = [("tsb_row_stats_q", lib.tsb_row_stats,
                       (ctypes.byref(dq), ctypes.c_float(cfg.temperature), _ptr(qstats), qsb_, _ptr(buf.ws), wb, s))]
            qref, qst, qstb, qidx = ctypes.byref(dq), _ptr(qstats), qsb_, _ptr(qrow_of_node)
        else:
            qref, qst, qstb, qidx = ctypes.byref(dd), _ptr(buf.stats), sb, None
        if replay == "plan":
            rep = []
        else:
            fn, name = (lib.tsb_replay_mixed, "tsb_replay_mixed") if replay == "mixed" else (lib.tsb_replay,
                                                                                              "tsb_replay")
            rep = [(name, fn, (ctypes.byref(cfg), qref, qst, qstb, qidx, ctypes.byref(tr), seed, _ptr(tok),
                               _ptr(buf.ws), wb, s))]
        if mode == TSB_VERIFY_NAIVE:
            qd, qs, qsb, qi = None, None, 0, None
        else:
            qd, qs, qsb, qi = qref, qst, qstb, qidx
        self.calls = plan + qcalls + rep + [
            ("tsb_verify", lib.tsb_verify, (ctypes.byref(cfg), int(mode), ctypes.byref(dt), qd, qs, qsb, qi,
                                            ctypes.byref(tr), _ptr(tok), seed, _ptr(ot), _ptr(on), _ptr(ol),
                                            _ptr(buf.ws), wb, s)),
        ]
        if together and replay == "wor" and mode == TSB_VERIFY_RRS:  # replay and verification in one call
            self.calls = plan + qcalls + [
                ("tsb_replay_verify", lib.tsb_replay_verify,
                 (ctypes.byref(cfg), ctypes.byref(dt), qref, qst, qstb, qidx, ctypes.byref(tr), seed, _ptr(tok),
                  _ptr(ot), _ptr(on), _ptr(ol), _ptr(buf.ws), wb, s)),
            ]
        if plan_only:  # the first pass alone
            self.calls = plan

    def run(self, events=None):
        """Launch the calls; with ``events`` (len(calls) + 1 torch.cuda.Event), record one
        before the first call and one after each."""
        if events is not None:
            events[0].record()
        for i, (name, fn, args) in enumerate(self.calls):
            rc = fn(*args)
            if rc != TSB_OK:
                raise TsbError(rc, name)
            if events is not None:
                events[i + 1].record()
