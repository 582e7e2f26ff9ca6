"""Accuracy of the GPU's row log-normalisers against the oracle's fp64 values.

The first pass ranks candidates of different depths by path log-probabilities that contain
the prefix sums of the draft rows' log-normalisers (Sec. 3.1), so the oracle's near-tie flag
for a planner pop is derived from a bound on the GPU's error in one row's log-normaliser:
LSE_ERR_BOUND in ``oracle.PLAN_LSE_ERR``. This test measures that error on every row of the
workloads' draft rows (bf16 and fp32, T = 1 and 0.6, ragged V) and holds it to the bound.
"""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2609_33652_gb300 import synth, tsb

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_33652_gb300 import build

    build.build()
    oracle.build()
    tsb.load()


def _gpu_row_lse(buf, B, L, N):
    """The first pass's per-draft-row log-normaliser (float-float) from the workspace: after
    the 256-byte header, B*(N+1) 32-byte slots and B 1024-byte pre-pass partials come B*L
    float2 values."""
    off = 256 + B * (N + 1) * 32 + B * 1024
    v = buf.ws[off:off + B * L * 8].view(torch.float32).view(B, L, 2).cpu().numpy().astype(np.float64)
    return v[..., 0] + v[..., 1]


@pytest.mark.parametrize("B,V,kind,dtype,T", [
    (16, 151936, "planted", "bf16", 1.0),
    (16, 151936, "planted", "bf16", 0.6),
    (8, 151936, "planted", "f32", 1.0),
    (16, 128256, "normal3", "bf16", 1.0),
    (64, 5003, "normal3", "f32", 0.6),
    (64, 32, "normal2", "f32", 1.0),
])
@pytest.mark.parametrize("fused", [False, True])
def test_row_lse_error_within_the_planner_bound(B, V, kind, dtype, T, fused):
    L, N, K = 16, 64, 8
    draft = synth.draft_logits(B, L, V, kind, dtype, 4242 + V, device=DEV)
    buf = tsb.TsbBuffers.allocate(B, L, N, K, V, T, device=DEV)
    if fused:
        tsb.tsb_plan_rows(buf.cfg, draft, buf.stats, buf.tree, buf.ws)
    else:
        tsb.tsb_row_stats(draft, T, buf.stats, buf.ws)
        tsb.tsb_plan(buf.cfg, draft, buf.stats, buf.tree, buf.ws)
    assert tsb.tsb_device_status(buf.ws) == 0
    got = _gpu_row_lse(buf, B, L, N)
    want = oracle.row_stats(synth.to_host(draft), T)["lse"]
    err = np.abs(got - want)
    log = os.environ.get("TSB_PARITY_LOG")
    if log:
        with open(log, "a") as f:
            f.write(json.dumps({"test": os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0],
                                "row_lse_err_max": float(err.max()), "row_lse_err_rms": float(np.sqrt((err ** 2).mean())),
                                "rows": int(err.size)}) + "\n")
    assert err.max() <= oracle.PLAN_LSE_ERR, (err.max(), oracle.PLAN_LSE_ERR)
