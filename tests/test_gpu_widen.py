"""GPU parity of the widened path against the CPU oracle: the expand-then-prune first pass
(Sec. 3.1 / App. B.3), mixed-sampling replay (Sec. 3.2 / App. A) and target-sample-matching
verification ("Naive", Table 2), through the C ABI, on the workload shapes and edge cases."""
import numpy as np
import pytest
import torch

import helpers
import oracle
from gpu_harness import Report, check_status, compare_plan, compare_trials, gpu_plan, run_step
from paper_2609_33652_gb300 import synth, tsb

pytestmark = pytest.mark.gpu
DEV = "cuda"
TREE_KEYS = ("parent", "depth", "rank", "plan_token", "score", "child_off", "child_ids")


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




# --------------------------------------------------------------------------------------
# expand-then-prune first pass
@pytest.mark.parametrize("wl,V,B,width,dtype", [("batched", 151936, 16, 10, "bf16"), ("batched", 128256, 16, 4, "bf16"),
                                                ("tiny", 32, 256, 2, "f32"), ("single", 151936, 4, 1, "bf16")])
def test_expand_step_matches_oracle(wl, V, B, width, dtype):
    """Expand-then-prune tree, WoR replay and recursive rejection sampling on it."""
    w = synth.WORKLOADS[wl]
    draft = _draft(B, w["L"], V, "planted" if V > 100 else "normal2", dtype, 1203)
    rep, _, gout = run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=7, target_noise=w["target_noise"],
                            width=width)
    assert (gout["len"] >= 1).all()


def test_expand_sweep_budget_256_sampled():
    w = synth.WORKLOADS["sweep"]
    draft = _draft(64, w["L"], w["V"], "planted", "bf16", 1204)
    rep, _, _ = run_step(draft, w["L"], 256, w["K"], w["T"], seed=3, target_noise=w["target_noise"], width=10,
                         trees=[0, 31, 63])


@pytest.mark.parametrize("B,L,N,K,V,kind,dtype", [
    (16, 16, 64, 8, 151936, "planted", "bf16"),
    (4, 6, 100, 4, 3001, "normal3", "f32"),
    (2, 24, 150, 2, 1000, "planted", "bf16"),  # 510 + 16 * 300 = 5310 candidates at W = N
])
def test_expand_wide_frontier_is_the_heap_tree(B, L, N, K, V, kind, dtype):
    """A frontier of N candidates gives the max-heap tree, bit for bit, on the GPU too."""
    draft = _draft(B, L, V, kind, dtype, 1205)
    heap = gpu_plan(draft, L, N, K, 1.0)
    ept = gpu_plan(draft, L, N, K, 1.0, width=N)
    torch.cuda.synchronize()
    check_status(heap)
    check_status(ept)
    for k in TREE_KEYS:
        assert torch.equal(heap.tree[k], ept.tree[k]), k


def test_expand_fused_rows_match_separate_calls():
    w = synth.WORKLOADS["batched"]
    draft = _draft(w["B"], w["L"], 151936, "planted", "bf16", 1206)
    ref = gpu_plan(draft, w["L"], w["N"], w["K"], 1.0, width=10)
    got = tsb.TsbBuffers.allocate(w["B"], w["L"], w["N"], w["K"], 151936, 1.0, device=DEV)
    tsb.tsb_plan_rows_expand(got.cfg, 10, draft, got.stats, got.tree, got.ws)
    torch.cuda.synchronize()
    check_status(ref)
    check_status(got)
    assert torch.equal(got.stats, ref.stats)
    for k in TREE_KEYS:
        assert torch.equal(got.tree[k], ref.tree[k]), k


def test_expand_large_layers_and_edges():
    """Wide frontiers (W*K = 1024 per layer), K = 32, and a budget equal to the candidates."""
    for (B, L, N, K, V, W) in [(2, 8, 500, 32, 5003, 32), (3, 5, 20, 2, 700, 3), (2, 4, 2 + 3 * 2, 2, 300, 1)]:
        draft = _draft(B, L, V, "normal3", "f32", 1207 + N)
        buf = gpu_plan(draft, L, N, K, 1.0, width=W)
        check_status(buf)
        ref = oracle.plan_expand(synth.to_host(draft), 1.0, N, K, L, W)
        rep = Report()
        compare_plan(buf, ref, rep, list(range(B)))
        rep.check()


def test_expand_rejects_bad_width():
    buf = tsb.TsbBuffers.allocate(2, 3, 10, 2, 300, 1.0, device=DEV)
    draft = _draft(2, 3, 300, "normal3", "f32", 1)
    tsb.tsb_row_stats(draft, 1.0, buf.stats, buf.ws)
    for width in (0, tsb.TSB_MAX_WIDTH + 1):
        with pytest.raises(tsb.TsbError) as e:
            tsb.tsb_plan_expand(buf.cfg, width, draft, buf.stats, buf.tree, buf.ws)
        assert e.value.status == 2
    with pytest.raises(tsb.TsbError):  # W = 1, K = 2, L = 3: 6 candidates < N = 10
        tsb.tsb_plan_expand(buf.cfg, 1, draft, buf.stats, buf.tree, buf.ws)


# --------------------------------------------------------------------------------------
# mixed sampling and target-sample matching
@pytest.mark.parametrize("wl,V,B", [("batched", 151936, 16), ("tiny", 32, 256), ("single", 151936, 4)])
def test_mixed_replay_naive_verify(wl, V, B):
    w = synth.WORKLOADS[wl]
    draft = _draft(B, w["L"], V, "planted" if V > 100 else "normal2", "bf16" if V > 100 else "f32", 1301)
    rep, _, gout = run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=17, target_noise=w["target_noise"],
                            replay="mixed", mode=tsb.TSB_VERIFY_NAIVE)
    assert (gout["len"] >= 1).all()


def test_mixed_replay_per_node_rows_k32():
    """Per-node q rows (the corrected-drafter layout) and K = 32 candidates per row."""
    B, L, N, K, V = 4, 4, 120, 32, 5003
    draft = _draft(B, L, V, "normal3", "bf16", 1302)
    buf = gpu_plan(draft, L, N, K, 0.6)
    qrows = synth.rows_from_depth(draft, buf.tree["depth"], 0.3, seed=3001)
    qidx = torch.arange(N + 1, dtype=torch.int32, device=DEV).repeat(B, 1).contiguous()
    rep, _, _ = run_step(draft, L, N, K, 0.6, seed=19, target_noise=0.7, qrows=qrows, qrow_of_node=qidx,
                         replay="mixed", mode=tsb.TSB_VERIFY_NAIVE)


@pytest.mark.parametrize("wl,V,B,K", [("batched", 151936, 16, 8), ("tiny", 32, 256, 4), ("batched", 151936, 16, 1)])
def test_first_pass_tokens_naive_verify(wl, V, B, K):
    """The deterministic tree (First / TopK with Naive) and, with K = 1, the Top1 chain."""
    w = synth.WORKLOADS[wl]
    N = w["N"] if K > 1 else w["L"]
    draft = _draft(B, w["L"], V, "planted" if V > 100 else "normal2", "bf16" if V > 100 else "f32", 1303)
    rep, _, _ = run_step(draft, w["L"], N, K, w["T"], seed=23, target_noise=w["target_noise"], replay="plan",
                         mode=tsb.TSB_VERIFY_NAIVE)


def test_mixed_single_child_equals_wor():
    """With one child per parent nothing is excluded: mixed and WoR replays agree bit for bit."""
    draft = _draft(16, 16, 151936, "planted", "bf16", 1304)
    buf = gpu_plan(draft, 16, 16, 1, 1.0)
    tok_mixed = torch.empty_like(buf.token)
    tsb.tsb_replay(buf.cfg, draft, buf.stats, None, buf.tree, 5, buf.token, buf.ws)
    tsb.tsb_replay_mixed(buf.cfg, draft, buf.stats, None, buf.tree, 5, tok_mixed, buf.ws)
    check_status(buf)
    assert torch.equal(tok_mixed, buf.token)


def test_naive_losslessness_on_gpu():
    """1e5 trees share the tiny workload's rows; target rows are functions of the token path.
    The first emitted token must follow the root's target law (chi-square), and every tree
    must match the oracle wherever it flags no near tie."""
    w = synth.WORKLOADS["tiny"]
    B, L, N, K, V, T = 100_000, w["L"], w["N"], w["K"], w["V"], w["T"]
    base1 = _draft(1, L, V, "normal2", "f32", 1000)
    draft = base1.expand(B, -1, -1)
    buf = gpu_plan(draft, L, N, K, T)
    seed = 41
    tsb.tsb_replay_mixed(buf.cfg, draft, buf.stats, None, buf.tree, seed, buf.token, buf.ws)
    check_status(buf)
    tree = {k: v.cpu().numpy() for k, v in buf.tree.items()}
    tok = buf.token.cpu().numpy()
    base = synth.to_host(base1)[0]
    target_h = synth.path_keyed_rows(base, tree["parent"], tree["depth"], tok, 1.0, seed=78)
    target = torch.from_numpy(target_h).to(DEV)
    tsb.tsb_verify(buf.cfg, tsb.TSB_VERIFY_NAIVE, target, None, None, None, buf.tree, buf.token, seed,
                   buf.out_tokens, buf.out_nodes, buf.out_len, buf.ws)
    check_status(buf)
    first = buf.out_tokens[:, 0].cpu().numpy()
    p_root = helpers.softmax64(synth.path_keyed_row(base, [], 1.0, 78))
    assert helpers.chi2_pvalue(np.bincount(first, minlength=V), p_root) > 1e-4
    h_draft = np.ascontiguousarray(np.broadcast_to(base[None], (B, L, V)))
    ref = oracle.plan(h_draft, T, N, K, L)
    rtok, rex = oracle.replay_mixed(h_draft, T, ref, seed)
    rt = synth.path_keyed_rows(base, ref["parent"], ref["depth"], rtok, 1.0, seed=78)
    rout = oracle.verify_naive(rt, T, ref, rtok, seed, L)
    compare_trials(buf, tok, rtok, rex, rout)


def test_naive_flags_nonfinite_target():
    w = synth.WORKLOADS["tiny"]
    draft = _draft(4, w["L"], 600, "normal3", "f32", 1305)
    buf = gpu_plan(draft, w["L"], w["N"], w["K"], 1.0)
    target = synth.rows_from_depth(draft, buf.tree["depth"], 0.7, 2000).clone()
    target[2, 0, 17] = float("nan")
    buf.token.copy_(buf.tree["plan_token"])
    tsb.tsb_verify(buf.cfg, tsb.TSB_VERIFY_NAIVE, target, None, None, None, buf.tree, buf.token, 1, buf.out_tokens,
                   buf.out_nodes, buf.out_len, buf.ws)
    assert tsb.tsb_device_status(buf.ws) & tsb.TSB_DEV_NONFINITE
