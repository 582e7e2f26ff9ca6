"""GPU parity of the pooled draft laws (Sec. 3.1-3.3: each position's draft law restricted to
its P most probable tokens) against the CPU oracle, through the C ABI: pooled first pass
(pools bit-exact, topology), pooled WoR replay, recursive rejection sampling with pooled q and
a full-vocabulary target, on the workload shapes; losslessness on the GPU."""
import numpy as np
import pytest
import torch

import helpers
import oracle
from gpu_harness import Report, check_status, compare_plan, compare_tokens, compare_trials, compare_verify, host_tree
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


def _draft(B, L, V, kind, dtype, seed):
    return synth.draft_logits(B, L, V, kind, dtype, seed, device=DEV)


def pooled_step(draft, L, N, K, P, T, seed, target_noise, qrows=None, qrow_of_node=None, trees=None):
    """Pooled plan -> replay -> verify on both sides, compared stage by stage."""
    rep = Report()
    B, R, V = draft.shape
    buf = tsb.TsbBuffers.allocate(B, L, N, K, V, T, draft_rows=R, device=DEV)
    pools = torch.empty(B, L, P, dtype=torch.int32, device=DEV)
    tsb.tsb_row_stats(draft, T, buf.stats, buf.ws)
    tsb.tsb_plan_pooled(buf.cfg, P, draft, buf.stats, pools, buf.tree, buf.ws)
    check_status(buf)
    sel = list(range(B)) if trees is None else list(trees)
    bids = np.array(sel, dtype=np.int32)
    h_draft = synth.to_host(draft[sel])
    ref_pools = np.ascontiguousarray(oracle.pools(h_draft, T, P)[:, :L])
    assert np.array_equal(pools.cpu().numpy()[sel], ref_pools)  # (x desc, id asc): exact
    ref = oracle.plan(h_draft, T, N, K, L, pool=P)
    same = compare_plan(buf, ref, rep, sel)
    if qrows is None:
        q, qidx, h_q, h_qidx = draft, None, h_draft, None
    else:
        q, qidx = qrows, qrow_of_node
        h_q, h_qidx = synth.to_host(qrows[sel]), qrow_of_node[sel].cpu().numpy()
    tsb.tsb_replay_pooled(buf.cfg, P, q, qidx, pools, buf.tree, seed, buf.token, buf.ws)
    check_status(buf)
    rtok, rex = oracle.replay_pooled(h_q, T, ref, seed, ref_pools, qrow_of_node=h_qidx, batch_ids=bids)
    gtok = buf.token.cpu().numpy()
    same = compare_tokens(gtok, rtok, rex, host_tree(buf), same, rep, sel)
    target = synth.rows_from_depth(draft, buf.tree["depth"], target_noise, 2000)
    rd = buf.tree["depth"].clone()
    rd[sel] = torch.from_numpy(ref["depth"]).to(DEV)
    h_target = synth.to_host(synth.rows_from_depth(draft, rd, target_noise, 2000)[sel])
    tsb.tsb_verify_pooled(buf.cfg, P, target, q, qidx, pools, buf.tree, buf.token, seed, buf.out_tokens,
                          buf.out_nodes, buf.out_len, buf.ws)
    check_status(buf)
    rout = oracle.verify_rrs(h_target, h_q, T, ref, rtok, seed, L, qrow_of_node=h_qidx, batch_ids=bids,
                             pool_ids=ref_pools)
    gout = {"len": buf.out_len.cpu().numpy(), "tokens": buf.out_tokens.cpu().numpy(),
            "nodes": buf.out_nodes.cpu().numpy()}
    compare_verify(gout, rout, same, rep, sel)
    rep.check()
    return rep, buf, gout


@pytest.mark.parametrize("wl,V,B,P,dtype", [("batched", 151936, 16, 16, "bf16"), ("batched", 128256, 16, 8, "bf16"),
                                            ("tiny", 32, 256, 6, "f32"), ("single", 151936, 4, 32, "bf16"),
                                            ("batched", 151936, 16, 64, "bf16"), ("single", 151936, 4, 33, "bf16")])
def test_pooled_step(wl, V, B, P, dtype):
    w = synth.WORKLOADS[wl]
    draft = _draft(B, w["L"], V, "planted" if V > 100 else "normal2", dtype, 1401)
    rep, _, gout = pooled_step(draft, w["L"], w["N"], w["K"], P, w["T"], seed=29, target_noise=w["target_noise"])
    assert (gout["len"] >= 1).all()


@pytest.mark.parametrize("T", [0.6, 1.0])
def test_pooled_per_node_rows(T):
    """Per-node (corrected) q rows normalised over the pools of the first pass."""
    w = synth.WORKLOADS["corrected"]
    B = 4
    draft = _draft(B, w["L"], w["V"], "planted", "bf16", 1402)
    buf = tsb.TsbBuffers.allocate(B, w["L"], w["N"], w["K"], w["V"], T, device=DEV)
    pools = torch.empty(B, w["L"], 16, dtype=torch.int32, device=DEV)
    tsb.tsb_row_stats(draft, T, buf.stats, buf.ws)
    tsb.tsb_plan_pooled(buf.cfg, 16, draft, buf.stats, pools, buf.tree, buf.ws)  # the pooled tree's depths
    qrows = synth.rows_from_depth(draft, buf.tree["depth"], w["per_node_noise"], seed=3000)
    qidx = torch.arange(w["N"] + 1, dtype=torch.int32, device=DEV).repeat(B, 1).contiguous()
    rep, _, _ = pooled_step(draft, w["L"], w["N"], w["K"], 16, T, seed=31, target_noise=w["target_noise"], qrows=qrows,
                            qrow_of_node=qidx)


def test_pooled_edges():
    # P = K (the pool is the candidate list), ragged V, fp32
    rep, _, _ = pooled_step(_draft(8, 4, 1001, "normal3", "f32", 1403), 4, 20, 4, 4, 0.8, seed=3, target_noise=0.7)
    # P = V for a one-chunk vocabulary
    rep, _, _ = pooled_step(_draft(16, 3, 24, "normal2", "f32", 1404), 3, 12, 3, 24, 1.0, seed=4, target_noise=1.0)


@pytest.mark.parametrize("V,P", [(5003, 64), (700, 40), (151936, 48)])
def test_pool_selection_degenerate_rows(V, P):
    """Pools above 32 tokens on rows that defeat the chunk bound: a flat row (every logit ties,
    so every chunk reaches tau), a maximum repeated 300 times, a vocabulary with fewer chunks
    than P (every logit is a candidate), and random rows; bit-exact against the host's stable
    sort by (x desc, id asc)."""
    B, L, K, N = 2, 4, 4, 12
    g = torch.Generator().manual_seed(V + P)
    z = torch.randn(B, L, V, generator=g) * 3
    z[0, 0] = 0.25  # flat
    pos = torch.randperm(V, generator=g)[:min(300, V)]
    z[0, 1, pos] = z[0, 1].max() + 1.0  # repeated maximum
    z[1, 2, :V // 2] = 1.5  # half the row tied
    stride = (V + 7) // 8 * 8
    store = torch.zeros(B, L, stride, dtype=torch.float32)
    store[..., :V] = z
    draft = store.to(DEV)[..., :V]
    buf = tsb.TsbBuffers.allocate(B, L, N, K, V, 1.0, device=DEV)
    pools = torch.empty(B, L, P, dtype=torch.int32, device=DEV)
    tsb.tsb_row_stats(draft, 1.0, buf.stats, buf.ws)
    tsb.tsb_plan_pooled(buf.cfg, P, draft, buf.stats, pools, buf.tree, buf.ws)
    check_status(buf)
    got = pools.cpu().numpy()
    x = z.numpy().astype(np.float32)
    for b in range(B):
        for d in range(L):
            want = np.lexsort((np.arange(V), -x[b, d]))[:P]
            assert np.array_equal(got[b, d], want), (b, d)


@pytest.mark.parametrize("V,P", [(32, 8), (1000, 64)])
def test_pooled_losslessness_on_gpu(V, P):
    """1e5 trees share one set of draft rows, target rows keyed by the token path: the first
    emitted token follows the root's target law (and the second token, extended by a target
    draw, the law after the first), and a sample of the trees matches the oracle. At V = 1000
    the pools hold 64 tokens (two per lane) across four chunks."""
    w = synth.WORKLOADS["tiny"]
    B, L, N, K, T = 100_000, w["L"], w["N"], w["K"], w["T"]
    base1 = _draft(1, L, V, "normal2", "f32", 1000 + V)
    draft = base1.expand(B, -1, -1)
    buf = tsb.TsbBuffers.allocate(B, L, N, K, V, T, device=DEV)
    pools = torch.empty(B, L, P, dtype=torch.int32, device=DEV)
    tsb.tsb_row_stats(draft, T, buf.stats, buf.ws)
    tsb.tsb_plan_pooled(buf.cfg, P, draft, buf.stats, pools, buf.tree, buf.ws)
    seed = 43
    tsb.tsb_replay_pooled(buf.cfg, P, draft, None, pools, buf.tree, seed, buf.token, buf.ws)
    check_status(buf)
    tree = {k: v.cpu().numpy() for k, v in buf.tree.items()}
    tok = buf.token.cpu().numpy()
    base = synth.to_host(base1)[0]
    target = synth.path_keyed_rows_device(base1[0].contiguous(), tree["parent"], tree["depth"], tok, 1.0, seed=79)
    tsb.tsb_verify_pooled(buf.cfg, P, target, draft, None, pools, buf.tree, buf.token, seed, buf.out_tokens,
                          buf.out_nodes, buf.out_len, buf.ws)
    check_status(buf)
    out = {"len": buf.out_len.cpu().numpy(), "tokens": buf.out_tokens.cpu().numpy(),
           "nodes": buf.out_nodes.cpu().numpy()}
    first = out["tokens"][:, 0]
    p_root = helpers.softmax64(synth.path_keyed_row(base, [], 1.0, 79))
    assert helpers.chi2_pvalue(np.bincount(first, minlength=V), p_root) > 1e-4
    second = out["tokens"][:, 1].copy()
    ext = np.random.default_rng(P)
    vals, cnt = np.unique(first, return_counts=True)
    for a in vals[np.argsort(-cnt)][:2]:
        sel = first == a
        pa = helpers.softmax64(synth.path_keyed_row(base, [int(a)], 1.0, 79))
        short = sel & (out["len"] == 1)
        second[short] = ext.choice(V, size=int(short.sum()), p=pa)
        assert helpers.chi2_pvalue(np.bincount(second[sel], minlength=V), pa) > 1e-4
    # the oracle on a sample of the trees, with their own batch indices
    sel = list(range(0, B, B // 1500))[:1500]
    bids = np.array(sel, dtype=np.int32)
    h1 = synth.to_host(base1)
    ref1 = oracle.plan(h1, T, N, K, L, pool=P)
    for k in ("parent", "child_off", "child_ids"):
        assert np.array_equal(ref1[k][0], tree[k][0]), k
    ref = helpers.repeat_tree({k: v for k, v in ref1.items() if k not in ("exempt", "min_margin")}, len(sel))
    hq = np.ascontiguousarray(np.broadcast_to(h1, (len(sel),) + h1.shape[1:]))
    ref_pools = np.ascontiguousarray(oracle.pools(h1, T, P)[:, :L].repeat(len(sel), axis=0))
    assert np.array_equal(pools.cpu().numpy()[0], ref_pools[0])
    rtok, rex = oracle.replay_pooled(hq, T, ref, seed, ref_pools, batch_ids=bids)
    rep = Report()
    same = compare_tokens(tok, rtok, rex, tree, dict.fromkeys(sel, True), rep, sel)
    rout = oracle.verify_rrs(synth.to_host(target[sel].contiguous()), hq, T, ref, rtok, seed, L, batch_ids=bids,
                             pool_ids=ref_pools)
    compare_verify(out, rout, same, rep, sel)
    rep.check()
