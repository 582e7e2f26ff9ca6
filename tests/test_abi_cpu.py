"""The C ABI library builds, loads and exports every function include/tsb.h declares; host
validation rejects bad arguments before any CUDA call (no GPU needed: the pointers below are
fake device addresses that validation never dereferences)."""
import ctypes
import math
import os
import re

import pytest

from paper_2609_33652_gb300 import build as libbuild
from paper_2609_33652_gb300 import tsb

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "tsb.h")

OK, ARG, SHAPE, DTYPE, ALIGN, WS = 0, 1, 2, 3, 4, 5
FAKE = 0x7F00_0000_0000  # 256-aligned fake device address


@pytest.fixture(scope="module")
def lib():
    libbuild.build()
    return tsb.load()


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(tsb_\w+)\s*\(", text)))


def test_exports_every_declared_function(lib):
    names = _declared()
    assert set(names) == set(tsb.EXPORTS)
    for n in names:
        assert hasattr(lib, n), n


def test_checked_build_exports_the_same_functions(lib):
    """libtsb_checked.so (the TSB_CHECKED build) loads and exports every declared function;
    the binding switches to it inside tsb.checked_library() and back afterwards."""
    with tsb.checked_library() as checked:
        for n in _declared():
            assert hasattr(checked, n), n
        assert tsb.load() is checked
        assert tsb.tsb_version() >= 100
    assert tsb.load() is lib


def test_header_is_plain_c(tmp_path):
    """include/tsb.h is a C header: it compiles as strict C99 (and as C++) on its own."""
    import shutil
    import subprocess

    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no gcc")
    src = tmp_path / "use_tsb.c"
    src.write_text('#include "tsb.h"\nint main(void) { return (int)tsb_version(); }\n')
    inc = os.path.join(ROOT, "include")
    for cmd in ([gcc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-fsyntax-only", "-I", inc, str(src)],
                [gcc, "-x", "c++", "-std=c++17", "-Wall", "-Werror", "-fsyntax-only", "-I", inc, str(src)]):
        r = subprocess.run(cmd, capture_output=True, text=True)
        assert r.returncode == 0, r.stderr


def test_c_program_links_and_validates(tmp_path, lib):
    """A plain C program linked against libtsb.so (no Python, no torch) queries sizes and gets
    host-validation errors back; nothing reaches a GPU."""
    import shutil
    import subprocess

    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no gcc")
    libdir = os.path.dirname(tsb.library_path())
    src = tmp_path / "abi.c"
    src.write_text(r"""
#include <stdio.h>
#include "tsb.h"
int main(void) {
    tsb_cfg cfg = {16, 16, 64, 8, 151936, 1.0f};
    size_t ws = tsb_workspace_bytes(&cfg);
    if (ws != 256 + 16 * 65 * 32 + 16 * 1024 + 16 * 16 * (8 + 8 * 8)) return 1;
    if (tsb_stats_bytes(16, 16, 151936) != (size_t)16 * 16 * 594 * 8) return 2;
    tsb_cfg bad = cfg;
    bad.temperature = 0.0f;
    if (tsb_workspace_bytes(&bad) != 0) return 3;
    if (tsb_plan(&bad, 0, 0, 0, 0, 0, 0, 0) != TSB_ERR_ARG) return 4;
    if (tsb_replay_mixed(0, 0, 0, 0, 0, 0, 1, 0, 0, 0, 0) != TSB_ERR_ARG) return 5;
    printf("%s\n", tsb_status_str(TSB_ERR_SHAPE));
    return 0;
}
""")
    exe = tmp_path / "abi"
    r = subprocess.run([gcc, "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-L", libdir, "-ltsb",
                        f"-Wl,-rpath,{libdir}", "-o", str(exe)], capture_output=True, text=True)
    if r.returncode != 0 and "cannot find -ltsb" in r.stderr:
        pytest.skip("libtsb.so not linkable here")
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True)
    assert r.returncode == 0, (r.returncode, r.stderr)
    assert r.stdout.strip() == "shape out of range or inconsistent"


def test_host_queries(lib):
    assert tsb.tsb_version() >= 100
    for s in range(8):
        assert tsb.tsb_status_str(s)
    assert tsb.tsb_status_str(99) == "unknown status"
    assert tsb.tsb_stats_bytes(2, 3, 151936) == 2 * 3 * 594 * 8
    assert tsb.tsb_stats_bytes(1, 1, 257) == 2 * 8
    assert tsb.tsb_stats_bytes(0, 1, 10) == 0
    cfg = tsb.make_cfg(16, 16, 64, 8, 151936, 1.0)
    assert tsb.tsb_workspace_bytes(cfg) == 256 + 16 * 65 * 32 + 16 * 1024 + 16 * 16 * (8 + 8 * 8)
    assert tsb.tsb_workspace_bytes(tsb.make_cfg(1, 2, 7, 2, 8, 1.0)) == 0  # N above K + K^2


def _logits(B, R, V, dtype=0, data=FAKE, bstride=None, rstride=None):
    rs = V if rstride is None else rstride
    return tsb.Logits(data, dtype, B, R, V, R * rs if bstride is None else bstride, rs)


def _tree():
    return tsb.Tree(*([FAKE] * 7))


def _plan(lib, cfg, draft, stats_bytes=1 << 30, ws_bytes=1 << 30, ws=FAKE, tree=None):
    t = tree if tree is not None else _tree()
    return lib.tsb_plan(ctypes.byref(cfg) if cfg is not None else None, ctypes.byref(draft), FAKE, stats_bytes,
                        ctypes.byref(t), ws, ws_bytes, None)


def test_plan_validation(lib):
    good = tsb.make_cfg(4, 16, 64, 8, 1024, 1.0)
    d = _logits(4, 16, 1024)
    assert _plan(lib, None, d) == ARG
    for T in (0.0, -1.0, math.nan, math.inf):
        assert _plan(lib, tsb.make_cfg(4, 16, 64, 8, 1024, T), d) == ARG
    assert _plan(lib, tsb.make_cfg(4, 16, 64, 33, 1024, 1.0), d) == SHAPE  # K > 32
    assert _plan(lib, tsb.make_cfg(4, 16, 64, 8, 4, 1.0), _logits(4, 16, 4)) == SHAPE  # K > V
    assert _plan(lib, tsb.make_cfg(4, 2, 7, 2, 1024, 1.0), _logits(4, 2, 1024)) == SHAPE  # N > K + K^2
    assert _plan(lib, tsb.make_cfg(4, 65, 64, 8, 1024, 1.0), _logits(4, 65, 1024)) == SHAPE  # L > 64
    assert _plan(lib, tsb.make_cfg(4, 16, 1025, 8, 1024, 1.0), d) == SHAPE  # N > 1024
    assert _plan(lib, tsb.make_cfg(0, 16, 64, 8, 1024, 1.0), _logits(0, 16, 1024)) == SHAPE
    assert _plan(lib, good, _logits(4, 15, 1024)) == SHAPE  # fewer draft rows than L
    assert _plan(lib, good, _logits(5, 16, 1024)) == SHAPE  # batch mismatch
    assert _plan(lib, good, _logits(4, 16, 1024, dtype=2)) == DTYPE
    assert _plan(lib, good, _logits(4, 16, 1024, data=FAKE + 4)) == ALIGN
    assert _plan(lib, good, _logits(4, 16, 1024, rstride=1026)) == ALIGN  # 1026 * 4 bytes
    assert _plan(lib, good, _logits(4, 16, 1024, dtype=1, rstride=1028)) == ALIGN  # 1028 * 2 bytes
    assert _plan(lib, good, _logits(4, 16, 1024, rstride=1000)) == SHAPE  # row stride < V
    assert _plan(lib, good, d, stats_bytes=4 * 16 * 4 * 8 - 8) == WS
    assert _plan(lib, good, d, ws_bytes=255) == WS
    assert _plan(lib, good, d, ws=FAKE + 8) == WS
    assert _plan(lib, good, d, ws=None) == ARG
    t = _tree()
    t.child_ids = None
    assert _plan(lib, good, d, tree=t) == ARG
    # broadcast rows (batch stride 0) are accepted by validation
    cfg1 = tsb.make_cfg(4, 2, 6, 2, 8, 1.0)
    assert lib.tsb_workspace_bytes(ctypes.byref(cfg1)) == 256 + 4 * 7 * 32 + 4 * 1024 + 4 * 2 * (8 + 8 * 2)


def test_plan_rows_validation(lib):
    good = tsb.make_cfg(4, 16, 64, 8, 1024, 1.0)
    d = _logits(4, 16, 1024)

    def call(cfg=good, draft=d, stats=FAKE, stats_bytes=1 << 30, ws=FAKE, ws_bytes=1 << 30, tree=None):
        t = tree if tree is not None else _tree()
        return lib.tsb_plan_rows(ctypes.byref(cfg) if cfg is not None else None, ctypes.byref(draft), stats,
                                 stats_bytes, ctypes.byref(t), ws, ws_bytes, None)

    assert call(cfg=None) == ARG
    assert call(stats=None) == ARG
    assert call(stats=FAKE + 4) == WS
    assert call(stats_bytes=4 * 16 * 4 * 8 - 8) == WS
    assert call(draft=_logits(4, 15, 1024)) == SHAPE
    assert call(draft=_logits(4, 16, 1024, dtype=2)) == DTYPE
    assert call(ws_bytes=255) == WS
    t = _tree()
    t.score = None
    assert call(tree=t) == ARG


def test_replay_verify_validation(lib):
    cfg = tsb.make_cfg(2, 4, 8, 4, 64, 1.0)
    q = _logits(2, 4, 64)
    t = _tree()

    def replay(cfg=cfg, q=q, qrow=None, token=FAKE):
        return lib.tsb_replay(ctypes.byref(cfg), ctypes.byref(q), FAKE, 1 << 30, qrow, ctypes.byref(t), 1, token,
                              FAKE, 1 << 30, None)

    assert replay(token=None) == ARG
    assert replay(q=_logits(2, 3, 64)) == SHAPE  # per-depth rows need L rows
    assert replay(q=_logits(2, 3, 64), qrow=FAKE) != SHAPE  # per-node rows: any row count (validated on device)

    def verify(mode=0, target=None, q=q, cfg=cfg, out=FAKE):
        tg = target if target is not None else _logits(2, 9, 64)
        return lib.tsb_verify(ctypes.byref(cfg), mode, ctypes.byref(tg), ctypes.byref(q), FAKE, 1 << 30, None,
                              ctypes.byref(t), FAKE, 1, out, FAKE, FAKE, FAKE, 1 << 30, None)

    assert verify(mode=4) == ARG
    assert verify(target=_logits(2, 8, 64)) == SHAPE  # needs N+1 target rows
    assert verify(target=_logits(2, 9, 64, dtype=1)) == DTYPE  # target / q dtypes differ
    assert verify(out=None) == ARG
    assert verify(mode=1, cfg=tsb.make_cfg(2, 4, 5, 4, 64, 1.0)) == SHAPE  # block: chain longer than L


def test_naive_and_mixed_validation(lib):
    cfg = tsb.make_cfg(2, 4, 8, 4, 64, 1.0)
    t = _tree()
    tg = _logits(2, 9, 64)

    def naive(target=tg, token=FAKE, out=FAKE, ws_bytes=1 << 30):
        # target-sample matching takes no draft rows: qrows / qstats may be NULL
        return lib.tsb_verify(ctypes.byref(cfg), tsb.TSB_VERIFY_NAIVE, ctypes.byref(target), None, None, 0, None,
                              ctypes.byref(t), token, 1, out, FAKE, FAKE, FAKE, ws_bytes, None)

    assert naive(target=_logits(2, 8, 64)) == SHAPE  # needs N+1 target rows
    assert naive(target=_logits(2, 9, 64, dtype=2)) == DTYPE
    assert naive(token=None) == ARG
    assert naive(out=None) == ARG
    assert naive(ws_bytes=255) == WS
    q = _logits(2, 4, 64)

    def mixed(q=q, token=FAKE, ws_bytes=1 << 30):
        return lib.tsb_replay_mixed(ctypes.byref(cfg), ctypes.byref(q), FAKE, 1 << 30, None, ctypes.byref(t), 1,
                                    token, FAKE, ws_bytes, None)

    assert mixed(token=None) == ARG
    assert mixed(q=_logits(2, 3, 64)) == SHAPE  # per-depth rows need L rows
    assert mixed(ws_bytes=255) == WS


def test_plan_expand_validation(lib):
    good = tsb.make_cfg(4, 16, 64, 8, 1024, 1.0)
    d = _logits(4, 16, 1024)

    def call(width, cfg=good, draft=d, stats=FAKE, fused=False):
        fn = lib.tsb_plan_rows_expand if fused else lib.tsb_plan_expand
        return fn(ctypes.byref(cfg), width, ctypes.byref(draft), stats, 1 << 30, ctypes.byref(_tree()), FAKE,
                  1 << 30, None)

    for fused in (False, True):
        assert call(0, fused=fused) == SHAPE
        assert call(tsb.TSB_MAX_WIDTH + 1, fused=fused) == SHAPE
        assert call(10, stats=None, fused=fused) == ARG
        assert call(10, draft=_logits(4, 15, 1024), fused=fused) == SHAPE
        # W = 1, K = 2, L = 3: 2 + 2 + 2 = 6 candidates cannot hold N = 7
        assert call(1, cfg=tsb.make_cfg(4, 3, 7, 2, 1024, 1.0), draft=_logits(4, 3, 1024), fused=fused) == SHAPE
        # K = 32, W = 64, L = 16: far more than TSB_MAX_EXPAND_CANDIDATES candidates
        assert call(64, cfg=tsb.make_cfg(4, 16, 64, 32, 1024, 1.0), fused=fused) == SHAPE


def test_pooled_validation(lib):
    cfg = tsb.make_cfg(2, 4, 8, 4, 64, 1.0)
    t = _tree()
    d = _logits(2, 4, 64)

    def plan(P, draft=d, pools=FAKE):
        return lib.tsb_plan_pooled(ctypes.byref(cfg), P, ctypes.byref(draft), FAKE, 1 << 30, pools,
                                   ctypes.byref(t), FAKE, 1 << 30, None)

    assert plan(3) == SHAPE  # P < K
    assert plan(tsb.TSB_MAX_POOL + 1) == SHAPE
    assert plan(8, pools=None) == ARG
    assert plan(8, draft=_logits(2, 3, 64)) == SHAPE

    def replay(P, pools=FAKE, token=FAKE):
        return lib.tsb_replay_pooled(ctypes.byref(cfg), P, ctypes.byref(d), None, pools, ctypes.byref(t), 1, token,
                                     FAKE, 1 << 30, None)

    assert replay(2) == SHAPE
    assert replay(8, pools=None) == ARG
    assert replay(8, token=None) == ARG

    def verify(P, target=None, pools=FAKE):
        tg = target if target is not None else _logits(2, 9, 64)
        return lib.tsb_verify_pooled(ctypes.byref(cfg), P, ctypes.byref(tg), ctypes.byref(d), None, pools,
                                     ctypes.byref(t), FAKE, 1, FAKE, FAKE, FAKE, FAKE, 1 << 30, None)

    assert verify(65) == SHAPE  # P > V
    assert verify(8, target=_logits(2, 8, 64)) == SHAPE
    assert verify(8, target=_logits(2, 9, 64, dtype=1)) == DTYPE
    assert verify(8, pools=None) == ARG


def test_workspace_and_status_validation(lib):
    assert lib.tsb_workspace_init(None, 256, None) == ARG
    assert lib.tsb_workspace_init(FAKE, 100, None) == WS
    bits = ctypes.c_uint32(0)
    assert lib.tsb_device_status(None, None, ctypes.byref(bits)) == ARG
    assert lib.tsb_row_stats(None, 1.0, FAKE, 1 << 20, FAKE, 256, None) == ARG
    rows = _logits(1, 2, 300)
    assert lib.tsb_row_stats(ctypes.byref(rows), 0.0, FAKE, 1 << 20, FAKE, 256, None) == ARG
    assert lib.tsb_row_stats(ctypes.byref(rows), 1.0, FAKE, 2 * 2 * 8 - 1, FAKE, 256, None) == WS
    assert lib.tsb_row_stats(ctypes.byref(_logits(1, 2, 409601)), 1.0, FAKE, 1 << 30, FAKE, 256, None) == SHAPE
