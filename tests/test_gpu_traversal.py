"""GPU parity of traversal verification (tsb_verify mode TSB_VERIFY_TRAVERSAL) against the
oracle's orc_verify_traversal, through the C ABI, on every workload shape and the edge cases
of the walk (chains, stars, full trees, a per-node draft row per node, ragged V, K = 32, the
depth cap, a budget of one node). The comparison rule and difference budget are those of the
other parity tests (tests/gpu_harness.py)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_harness import gpu_plan, run_step
from paper_2609_33652_gb300 import synth, tsb

pytestmark = pytest.mark.gpu
DEV = "cuda"
TRAV = tsb.TSB_VERIFY_TRAVERSAL


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_33652_gb300 import build

    build.build()
    oracle.build()
    tsb.load()


def _draft(B, L, V, kind, dtype, seed):
    return synth.draft_logits(B, L, V, kind, dtype, seed, device=DEV)


@pytest.mark.parametrize("V", [151936, 128256])
def test_traversal_batched(V):
    w = synth.WORKLOADS["batched"]
    draft = _draft(w["B"], w["L"], V, "planted", "bf16", 1503)
    _, _, gout = run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=5, target_noise=w["target_noise"], mode=TRAV)
    assert (gout["len"] >= 1).all() and (gout["len"] <= w["L"] + 1).all()


@pytest.mark.parametrize("seed", [1, 2])
def test_traversal_tiny(seed):
    w = synth.WORKLOADS["tiny"]
    draft = _draft(256, w["L"], w["V"], "normal2", "f32", 1500 + seed)
    run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=seed, target_noise=1.0, mode=TRAV)


def test_traversal_single_stream():
    w = synth.WORKLOADS["single"]
    draft = _draft(4, w["L"], w["V"], "planted", "bf16", 1501)
    run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=11, target_noise=w["target_noise"], mode=TRAV)


@pytest.mark.parametrize("T", [0.6, 1.0])
def test_traversal_per_node_rows(T):
    w = synth.WORKLOADS["corrected"]
    B = 4
    draft = _draft(B, w["L"], w["V"], "planted", "bf16", 1502)
    buf = gpu_plan(draft, w["L"], w["N"], w["K"], T)
    qrows = synth.rows_from_depth(draft, buf.tree["depth"], w["per_node_noise"], seed=3000)
    qidx = torch.arange(w["N"] + 1, dtype=torch.int32, device=DEV).repeat(B, 1).contiguous()
    run_step(draft, w["L"], w["N"], w["K"], T, seed=9, target_noise=w["target_noise"], qrows=qrows, qrow_of_node=qidx,
             mode=TRAV)


def test_traversal_sweep_sampled():
    """B = 64 at the largest budget; the oracle checks a sample of trees."""
    w = synth.WORKLOADS["sweep"]
    draft = _draft(64, w["L"], w["V"], "planted", "f32", 1504)
    run_step(draft, w["L"], 256, w["K"], w["T"], seed=3, target_noise=w["target_noise"], trees=[0, 21, 42, 63],
             mode=TRAV)


def test_traversal_edges():
    run_step(_draft(8, 6, 1000, "normal3", "f32", 7), 6, 6, 1, 1.0, seed=1, target_noise=0.7, mode=TRAV)  # chain
    run_step(_draft(8, 3, 640, "normal3", "bf16", 8), 3, 14, 2, 1.0, seed=2, target_noise=0.7, mode=TRAV)  # full
    run_step(_draft(8, 4, 1001, "normal3", "f32", 9), 4, 20, 4, 0.8, seed=3, target_noise=0.7, mode=TRAV)  # ragged
    run_step(_draft(8, 3, 5, "normal2", "f32", 10), 3, 12, 5, 1.0, seed=4, target_noise=1.0, mode=TRAV)  # K = V
    run_step(_draft(8, 1, 300, "normal3", "bf16", 11), 1, 1, 1, 1.0, seed=5, target_noise=0.7, mode=TRAV)  # N = 1
    run_step(_draft(4, 4, 4096, "normal3", "bf16", 12), 4, 200, 32, 1.0, seed=6, target_noise=0.7, mode=TRAV)  # K=32
    run_step(_draft(8, 4, 1000, "normal2", "f32", 31), 4, 40, 8, 1.0, seed=13, target_noise=0.7, mode=TRAV)
    # a star (depth cap 1): traversal is recursive rejection sampling at the root
    draft = _draft(16, 1, 2048, "normal3", "f32", 14)
    _, _, g_trav = run_step(draft, 1, 8, 8, 1.0, seed=7, target_noise=0.7, mode=TRAV)
    _, _, g_rrs = run_step(draft, 1, 8, 8, 1.0, seed=7, target_noise=0.7, mode=tsb.TSB_VERIFY_RRS)
    for k in g_trav:
        assert np.array_equal(g_trav[k], g_rrs[k]), k


def test_traversal_sampled_chains():
    """Sampled chains (K = 1, the block-verification input) verified by traversal, against the
    oracle on the batched workload's draft rows."""
    w = synth.WORKLOADS["batched"]
    draft = _draft(w["B"], w["L"], 151936, "planted", "bf16", 1003)
    _, _, g_trav = run_step(draft, w["L"], 16, 1, 1.0, seed=21, target_noise=0.7, mode=TRAV)
    assert (g_trav["len"] >= 1).all() and (g_trav["len"] <= 17).all()


def test_traversal_flags_bad_tree():
    """A child list pointing outside the tree sets TSB_DEV_BAD_TREE (nothing is read out of range)."""
    w = synth.WORKLOADS["tiny"]
    draft = _draft(4, w["L"], 512, "normal3", "f32", 15)
    buf = gpu_plan(draft, w["L"], w["N"], w["K"], 1.0)
    tsb.tsb_replay(buf.cfg, draft, buf.stats, None, buf.tree, 1, buf.token, buf.ws)
    target = synth.rows_from_depth(draft, buf.tree["depth"], 0.7, 2000)
    buf.tree["child_off"][1, 1] = 1000  # inconsistent offsets
    tsb.tsb_verify(buf.cfg, TRAV, target, draft, buf.stats, None, buf.tree, buf.token, 1, buf.out_tokens,
                   buf.out_nodes, buf.out_len, buf.ws)
    assert tsb.tsb_device_status(buf.ws) & tsb.TSB_DEV_BAD_TREE
