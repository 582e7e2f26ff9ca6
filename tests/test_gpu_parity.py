"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on identical seeded
inputs, for every workload shape, plus edge cases, losslessness and device status bits."""
import numpy as np
import pytest
import torch

import helpers
import oracle
from gpu_harness import Report, check_status, compare_plan, compare_trials, gpu_plan, run_step
from paper_2609_33652_gb300 import synth, tsb

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_33652_gb300 import build

    build.build()
    oracle.build()
    tsb.load()


DEV = "cuda"


def _draft(B, L, V, kind, dtype, seed):
    return synth.draft_logits(B, L, V, kind, dtype, seed, device=DEV)




# --------------------------------------------------------------------------------------
@pytest.mark.parametrize("B,R,V,dtype,T", [(3, 4, 32, "f32", 1.0), (2, 3, 1000, "bf16", 1.0),
                                           (2, 2, 1001, "f32", 0.6), (2, 3, 151936, "bf16", 1.0),
                                           (1, 2, 128256, "f32", 0.6)])
def test_row_stats(B, R, V, dtype, T):
    rows = _draft(B, R, V, "planted" if V > 100 else "normal2", dtype, 1)
    stats = torch.empty(tsb.tsb_stats_bytes(B, R, V) // 4, dtype=torch.float32, device=DEV)
    ws = torch.zeros(256, dtype=torch.uint8, device=DEV)
    tsb.tsb_row_stats(rows, T, stats, ws)
    assert tsb.tsb_device_status(ws) == 0
    C = (V + 255) // 256
    st = stats.view(B, R, C, 2).cpu().numpy().astype(np.float64)
    h = synth.to_host(rows.contiguous())
    ref = oracle.row_stats(h, T)
    x = (h.astype(np.float32) if h.dtype == np.float32 else (h.astype(np.uint32) << 16).view(np.float32))
    x = x * np.float32(np.float32(1.0) / np.float32(T))
    for c in range(C):
        np.testing.assert_array_equal(st[:, :, c, 0], x[:, :, c * 256:(c + 1) * 256].max(axis=2))
    np.testing.assert_allclose(st[..., 0] + np.log(st[..., 1]), ref["chunk_lse"], rtol=1e-6, atol=2e-6)


@pytest.mark.parametrize("seed", [1, 2])
def test_step_tiny(seed):
    w = synth.WORKLOADS["tiny"]
    draft = _draft(256, w["L"], w["V"], "normal2", "f32", 1000 + seed)
    rep, buf, _ = run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=seed, target_noise=1.0)


def test_step_single_stream():
    w = synth.WORKLOADS["single"]
    draft = _draft(4, w["L"], w["V"], "planted", "bf16", 1001)
    rep, _, _ = run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=11, target_noise=w["target_noise"])


@pytest.mark.parametrize("V", [151936, 128256])
def test_step_batched(V):
    w = synth.WORKLOADS["batched"]
    draft = _draft(w["B"], w["L"], V, "planted", "bf16", 1003)
    rep, _, gout = run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=5, target_noise=w["target_noise"])
    assert (gout["len"] >= 1).all()


@pytest.mark.parametrize("T", [0.6, 1.0])
def test_step_corrected_per_node_rows(T):
    w = synth.WORKLOADS["corrected"]
    B = 4
    draft = _draft(B, w["L"], w["V"], "planted", "bf16", 1002)
    buf = gpu_plan(draft, w["L"], w["N"], w["K"], T)
    qrows = synth.rows_from_depth(draft, buf.tree["depth"], w["per_node_noise"], seed=3000)
    qidx = torch.arange(w["N"] + 1, dtype=torch.int32, device=DEV).repeat(B, 1).contiguous()
    rep, _, _ = run_step(draft, w["L"], w["N"], w["K"], T, seed=9, target_noise=w["target_noise"], qrows=qrows,
                         qrow_of_node=qidx)


@pytest.mark.parametrize("N,dtype", [(16, "bf16"), (256, "f32")])
def test_step_sweep_sampled(N, dtype):
    """Full-size batch (B=64); the oracle checks a sample of trees one by one."""
    w = synth.WORKLOADS["sweep"]
    draft = _draft(64, w["L"], w["V"], "planted", dtype, 1004)
    rep, _, _ = run_step(draft, w["L"], N, w["K"], w["T"], seed=3, target_noise=w["target_noise"],
                         trees=[0, 21, 42, 63])


def test_step_small_vocab_many_children():
    """Parents with more children than vocabulary chunks (V=1000: 4 chunks, up to 8 children):
    every element of the kept chunks is a replay candidate, more than the key buffer holds."""
    draft = _draft(8, 4, 1000, "normal2", "f32", 31)
    rep, _, _ = run_step(draft, 4, 40, 8, 1.0, seed=13, target_noise=0.7)


def test_block_verification_chain():
    """Sampled chain (plan with K=1, replay = one draw per node) verified by block
    verification, on the batched workload's draft rows."""
    w = synth.WORKLOADS["batched"]
    g = 16
    draft = _draft(w["B"], w["L"], 151936, "planted", "bf16", 1003)
    rep, buf, gout = run_step(draft, w["L"], g, 1, w["T"], seed=21, target_noise=w["target_noise"],
                              mode=tsb.TSB_VERIFY_BLOCK)
    assert (gout["len"] >= 1).all() and (gout["len"] <= g + 1).all()


def test_block_verification_tiny_many():
    w = synth.WORKLOADS["tiny"]
    draft = _draft(300, w["L"], w["V"], "normal2", "f32", 1010)
    rep, _, _ = run_step(draft, w["L"], w["L"], 1, 1.0, seed=4, target_noise=1.0, mode=tsb.TSB_VERIFY_BLOCK)


# --------------------------------------------------------------------------------------
# edge cases
def test_edges_chain_full_tree_ragged():
    # K = 1 (chain of length min(N, L))
    draft = _draft(8, 6, 1000, "normal3", "f32", 7)
    run_step(draft, 6, 6, 1, 1.0, seed=1, target_noise=0.7)
    # N = full capacity of a K=2, L=3 tree
    draft = _draft(8, 3, 640, "normal3", "bf16", 8)
    run_step(draft, 3, 14, 2, 1.0, seed=2, target_noise=0.7)
    # V not a multiple of 8 (scalar tail), V below one chunk, K = V
    run_step(_draft(8, 4, 1001, "normal3", "f32", 9), 4, 20, 4, 0.8, seed=3, target_noise=0.7)
    run_step(_draft(8, 4, 1001, "normal3", "bf16", 9), 4, 20, 4, 0.8, seed=3, target_noise=0.7)
    run_step(_draft(8, 3, 5, "normal2", "f32", 10), 3, 12, 5, 1.0, seed=4, target_noise=1.0)
    # N = 1, L = 1
    run_step(_draft(8, 1, 300, "normal3", "bf16", 11), 1, 1, 1, 1.0, seed=5, target_noise=0.7)
    # K = 32 (largest candidate list)
    run_step(_draft(4, 4, 4096, "normal3", "bf16", 12), 4, 200, 32, 1.0, seed=6, target_noise=0.7)


def test_edges_broadcast_rows():
    """Every tree shares the same draft rows (batch stride 0): identical topology, different
    draws per tree."""
    w = synth.WORKLOADS["tiny"]
    base = _draft(1, w["L"], 512, "normal3", "f32", 13)
    draft = base.expand(64, -1, -1)
    rep, buf, _ = run_step(draft, w["L"], w["N"], w["K"], 1.0, seed=8, target_noise=0.7)
    p = buf.tree["parent"].cpu().numpy()
    assert (p == p[0]).all()
    tok = buf.token.cpu().numpy()
    assert len({tuple(t) for t in tok}) > 1


@pytest.mark.parametrize("B,R,L,N,K,V,kind,dtype", [
    (16, 16, 16, 64, 8, 151936, "planted", "bf16"),  # the batched workload
    (3, 6, 4, 40, 12, 5003, "normal3", "f32"),       # ragged V, K > 8, rows beyond L
    (64, 4, 4, 8, 4, 32, "normal2", "f32"),          # tiny rows, one chunk
])
def test_plan_rows_matches_separate_calls(B, R, L, N, K, V, kind, dtype):
    """tsb_plan_rows = tsb_row_stats (rows < L, same bits) + tsb_plan (same tree)."""
    draft = _draft(B, R, V, kind, dtype, 71)
    ref = tsb.TsbBuffers.allocate(B, L, N, K, V, 1.0, draft_rows=R, device=DEV)
    tsb.tsb_row_stats(draft, 1.0, ref.stats, ref.ws)
    tsb.tsb_plan(ref.cfg, draft, ref.stats, ref.tree, ref.ws)
    got = tsb.TsbBuffers.allocate(B, L, N, K, V, 1.0, draft_rows=R, device=DEV)
    got.stats.fill_(-7.0)
    tsb.tsb_plan_rows(got.cfg, draft, got.stats, got.tree, got.ws)
    torch.cuda.synchronize()
    check_status(ref)
    check_status(got)
    C = (V + 255) // 256
    rs = ref.stats.view(B, R, C, 2)
    gs = got.stats.view(B, R, C, 2)
    assert torch.equal(gs[:, :L], rs[:, :L])
    assert bool((gs[:, L:] == -7.0).all())  # rows the plan does not read are not written
    for k in ("parent", "depth", "rank", "plan_token", "score", "child_off", "child_ids"):
        assert torch.equal(got.tree[k], ref.tree[k]), k


@pytest.mark.parametrize("B,L,N,K,V,kind,dtype", [
    (2, 4, 1024, 32, 5003, "normal3", "f32"),   # the largest budget, 33 frontier slots per lane
    (2, 64, 1024, 2, 1000, "planted", "bf16"),  # the deepest tree (64 levels)
    (3, 16, 500, 8, 5003, "planted", "bf16"),   # 16 slots per lane
    (3, 16, 200, 4, 2048, "normal2", "f32"),    # 8 slots per lane
])
def test_plan_large_budgets(B, L, N, K, V, kind, dtype):
    """Topology of large and deep budgets against the oracle's best-first expansion."""
    draft = _draft(B, L, V, kind, dtype, 1010 + N)
    buf = gpu_plan(draft, L, N, K, 1.0)
    check_status(buf)
    ref = oracle.plan(synth.to_host(draft), 1.0, N, K, L)
    rep = Report()
    same = compare_plan(buf, ref, rep, list(range(B)))
    g = {k: v.cpu().numpy() for k, v in buf.tree.items()}
    for b in range(B):
        if same[b]:
            continue
        # a tree with flagged near ties that differs: still a best-first expansion, i.e. a
        # valid tree whose path scores are the oracle's top-N scores up to the near ties
        par, dep, rk = g["parent"][b], g["depth"][b], g["rank"][b]
        assert (par[1:] < np.arange(1, N + 1)).all() and (dep[1:] == dep[par[1:]] + 1).all()
        for u in range(N + 1):
            kids = g["child_ids"][b][g["child_off"][b][u]:g["child_off"][b][u + 1]]
            assert (par[kids] == u).all() and (rk[kids] == np.arange(len(kids))).all()
        np.testing.assert_allclose(np.sort(g["score"][b]), np.sort(ref["score"][b]), rtol=1e-5, atol=1e-5)
    rep.check()


def _topk_scratch(buf, B, L, N, K):
    """The first pass's per-row top-K (x, id) from the workspace: after the 256-byte header,
    B*(N+1) 32-byte slots and B 1024-byte pre-pass partials come B*L float2 log-normalisers,
    B*L*K x, B*L*K ids."""
    off = 256 + B * (N + 1) * 32 + B * 1024 + B * L * 8
    x = buf.ws[off:off + B * L * K * 4].view(torch.float32).view(B * L, K).cpu().numpy()
    ids = buf.ws[off + B * L * K * 4:off + B * L * K * 8].view(torch.int32).view(B * L, K).cpu().numpy()
    return x, ids


@pytest.mark.parametrize("dtype,K", [("f32", 8), ("bf16", 12), ("f32", 32)])
@pytest.mark.parametrize("fused", [False, True])
def test_topk_rows_exact(dtype, K, fused):
    """Per-row top-K by (x desc, id asc) against a host sort, on rows with heavy ties: a flat
    row (every logit reaches tau), a row whose maximum repeats 100 times, a planted row, and
    random rows (ragged V)."""
    B, L, N, V = 2, 4, 16, 5003
    g = torch.Generator().manual_seed(77)
    z = torch.randn(B, L, V, generator=g) * 3
    z[0, 1] = 0.5
    pos = torch.randperm(V, generator=g)[:100]
    z[0, 2, pos] = z[0, 2].max() + 1.0
    z[0, 3, 1234] = 12.0
    rows = z.to(torch.bfloat16 if dtype == "bf16" else torch.float32)
    stride = (V + 7) // 8 * 8
    store = torch.zeros(B, L, stride, dtype=rows.dtype)
    store[..., :V] = rows
    draft = store.to(DEV)[..., :V]
    buf = tsb.TsbBuffers.allocate(B, L, N, K, V, 1.0, device=DEV)
    if fused:
        tsb.tsb_plan_rows(buf.cfg, draft, buf.stats, buf.tree, buf.ws)
    else:
        tsb.tsb_row_stats(draft, 1.0, buf.stats, buf.ws)
        tsb.tsb_plan(buf.cfg, draft, buf.stats, buf.tree, buf.ws)
    check_status(buf)
    gx, gid = _topk_scratch(buf, B, L, N, K)
    x = rows.float().numpy().reshape(B * L, V)
    for r in range(B * L):
        order = np.lexsort((np.arange(V), -x[r]))[:K]
        assert np.array_equal(gid[r], order), r
        assert np.array_equal(gx[r], x[r][order]), r


def test_plan_rows_flags_nonfinite():
    draft = _draft(2, 3, 512, "normal3", "f32", 15).clone()
    draft[1, 2, 100] = float("inf")
    buf = tsb.TsbBuffers.allocate(2, 3, 10, 3, 512, 1.0, device=DEV)
    tsb.tsb_plan_rows(buf.cfg, draft, buf.stats, buf.tree, buf.ws)
    assert tsb.tsb_device_status(buf.ws) & tsb.TSB_DEV_NONFINITE


def test_determinism_and_launch_independence():
    w = synth.WORKLOADS["tiny"]
    draft = _draft(32, w["L"], 2000, "normal3", "bf16", 14)
    _, _, g1 = run_step(draft, w["L"], 30, 4, 1.0, seed=9, target_noise=0.7)
    _, _, g2 = run_step(draft, w["L"], 30, 4, 1.0, seed=9, target_noise=0.7)
    for k in g1:
        assert np.array_equal(g1[k], g2[k])


# --------------------------------------------------------------------------------------
def test_losslessness_on_gpu():
    """1e5 trees share the tiny workload's draft rows; targets are functions of the token
    path. The first emitted token must follow the root target law (chi-square), and the GPU
    outputs must equal the oracle's on every non-exempt tree."""
    w = synth.WORKLOADS["tiny"]
    B, L, N, K, V, T = 100_000, w["L"], w["N"], w["K"], w["V"], w["T"]
    base1 = _draft(1, L, V, "normal2", "f32", 1000)
    draft = base1.expand(B, -1, -1)
    buf = gpu_plan(draft, L, N, K, T)
    seed = 31
    tsb.tsb_replay(buf.cfg, draft, buf.stats, None, buf.tree, seed, buf.token, buf.ws)
    check_status(buf)
    tree = {k: v.cpu().numpy() for k, v in buf.tree.items()}
    tok = buf.token.cpu().numpy()
    base = synth.to_host(base1)[0]
    target_h = synth.path_keyed_rows(base, tree["parent"], tree["depth"], tok, 1.0, seed=77)
    target = torch.from_numpy(target_h).to(DEV)
    tsb.tsb_verify(buf.cfg, tsb.TSB_VERIFY_RRS, target, draft, buf.stats, None, buf.tree, buf.token, seed,
                   buf.out_tokens, buf.out_nodes, buf.out_len, buf.ws)
    check_status(buf)
    first = buf.out_tokens[:, 0].cpu().numpy()
    p_root = helpers.softmax64(synth.path_keyed_row(base, [], 1.0, 77))
    assert helpers.chi2_pvalue(np.bincount(first, minlength=V), p_root) > 1e-4
    # oracle on the same inputs (its own plan, replay and path-keyed targets)
    h_draft = np.ascontiguousarray(np.broadcast_to(base[None], (B, L, V)))
    ref = oracle.plan(h_draft, T, N, K, L)
    for k in ("parent", "child_ids"):
        assert np.array_equal(ref[k], tree[k])
    rtok, rex = oracle.replay(h_draft, T, ref, seed)
    rt = synth.path_keyed_rows(base, ref["parent"], ref["depth"], rtok, 1.0, seed=77)
    rout = oracle.verify_rrs(rt, h_draft, T, ref, rtok, seed, L)
    compare_trials(buf, tok, rtok, rex, rout)


def test_device_status_bits():
    draft = _draft(2, 3, 512, "normal3", "f32", 15).clone()
    draft[1, 2, 100] = float("nan")
    buf = gpu_plan(draft, 3, 10, 3, 1.0)
    assert tsb.tsb_device_status(buf.ws) & tsb.TSB_DEV_NONFINITE
    assert tsb.tsb_device_status(buf.ws) == 0  # cleared by the read
    draft = _draft(2, 3, 512, "normal3", "f32", 16)
    buf = gpu_plan(draft, 3, 10, 3, 1.0)
    check_status(buf)
    bad = torch.full((2, 11), 7, dtype=torch.int32, device=DEV)  # row 7 of a 3-row tensor
    tsb.tsb_replay(buf.cfg, draft, buf.stats, bad, buf.tree, 1, buf.token, buf.ws)
    assert tsb.tsb_device_status(buf.ws) & tsb.TSB_DEV_BAD_INDEX
