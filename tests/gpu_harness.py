"""Runs the CUDA path (through the C ABI) and the CPU oracle on the same seeded inputs and
compares them stage by stage.

Comparison rule (the parity contract):
  * topology (parent, depth, rank, planning token, child lists) bit-exact, unless the oracle
    flags a near-tie pop in that tree (cross-depth keys within 1e-6 relative);
  * replayed tokens bit-exact, unless the oracle flags a near-tie Gumbel decision at that
    parent (a uniform within 1e-6 of the value that would swap the decision);
  * verification outputs bit-exact, unless the oracle flags a near-tie decision in that
    tree's walk (acceptance uniform within 1e-6 of p'/q', or a near-tie Gumbel-max);
  * a stage is compared only where every earlier stage of the same tree matched;
  * path scores within 1e-5 relative.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2609_33652_gb300 import synth, tsb


def gpu_plan(draft, L, N, K, T, stats_rows=None):
    B, R, V = draft.shape
    buf = tsb.TsbBuffers.allocate(B, L, N, K, V, T, draft_rows=R, device=draft.device)
    tsb.tsb_row_stats(draft, T, buf.stats, buf.ws)
    tsb.tsb_plan(buf.cfg, draft, buf.stats, buf.tree, buf.ws)
    return buf


def check_status(buf):
    bits = tsb.tsb_device_status(buf.ws)
    assert bits == 0, f"device status bits {bits:#x}"


def host_tree(buf):
    return {k: v.cpu().numpy() for k, v in buf.tree.items()}


class Report:
    def __init__(self):
        self.trees = 0
        self.skipped = {"plan": 0, "replay": 0, "verify": 0}
        self.compared = {"plan": 0, "replay": 0, "verify": 0}

    def __repr__(self):
        return f"Report(trees={self.trees}, compared={self.compared}, skipped={self.skipped})"


def compare_plan(buf, ref, rep: Report, trees=None):
    g = host_tree(buf)
    B = g["parent"].shape[0]
    idx = range(B) if trees is None else trees
    ok = np.ones(B, dtype=bool)
    for j, b in enumerate(idx):
        rb = j
        rep.trees += 1
        if ref["exempt"][rb]:
            rep.skipped["plan"] += 1
            ok[b] = False
            continue
        rep.compared["plan"] += 1
        for k in ("parent", "depth", "rank", "plan_token", "child_off", "child_ids"):
            assert np.array_equal(g[k][b], ref[k][rb]), f"tree {b}: plan {k} differs"
        np.testing.assert_allclose(g["score"][b], ref["score"][rb], rtol=1e-5, atol=1e-5)
    return ok


def compare_tokens(gtok, rtok, rex, ok, rep: Report, trees=None):
    B = gtok.shape[0]
    idx = range(B) if trees is None else trees
    ok2 = ok.copy()
    for j, b in enumerate(idx):
        if not ok[b]:
            continue
        if rex[j].any():
            rep.skipped["replay"] += 1
            ok2[b] = False
            continue
        rep.compared["replay"] += 1
        assert np.array_equal(gtok[b], rtok[j]), f"tree {b}: replayed tokens differ"
    return ok2


def compare_verify(gout, rout, ok, rep: Report, trees=None):
    B = gout["len"].shape[0]
    idx = range(B) if trees is None else trees
    for j, b in enumerate(idx):
        if not ok[b]:
            continue
        if rout["exempt"][j]:
            rep.skipped["verify"] += 1
            continue
        rep.compared["verify"] += 1
        assert gout["len"][b] == rout["len"][j], f"tree {b}: length {gout['len'][b]} vs {rout['len'][j]}"
        assert np.array_equal(gout["tokens"][b], rout["tokens"][j]), f"tree {b}: emitted tokens differ"
        assert np.array_equal(gout["nodes"][b], rout["nodes"][j]), f"tree {b}: accepted nodes differ"


def run_step(draft, L, N, K, T, seed, target_noise=0.7, target_seed=2000, qrows=None, qrow_of_node=None,
             trees=None, mode=tsb.TSB_VERIFY_RRS, target=None):
    """Full plan -> replay -> verify on both sides; returns the report and the GPU outputs.

    ``trees`` restricts the oracle to a sample of trees (large batches)."""
    rep = Report()
    buf = gpu_plan(draft, L, N, K, T)
    check_status(buf)
    B = draft.shape[0]
    sel = list(range(B)) if trees is None else list(trees)
    h_draft = synth.to_host(draft[sel])
    ref = oracle.plan(h_draft, T, N, K, L)
    ok = compare_plan(buf, ref, rep, sel)

    if qrows is None:
        q, qstats, qidx = draft, buf.stats, None
        h_q, h_qidx = h_draft, None
    else:
        q = qrows
        qstats = torch.empty(tsb.tsb_stats_bytes(B, qrows.shape[1], qrows.shape[2]) // 4, dtype=torch.float32,
                             device=draft.device)
        tsb.tsb_row_stats(qrows, T, qstats, buf.ws)
        qidx = qrow_of_node
        h_q = synth.to_host(qrows[sel])
        h_qidx = qrow_of_node[sel].cpu().numpy()
    tsb.tsb_replay(buf.cfg, q, qstats, qidx, buf.tree, seed, buf.token, buf.ws)
    check_status(buf)
    rtok, rex = oracle.replay(h_q, T, ref, seed, qrow_of_node=h_qidx)
    gtok = buf.token.cpu().numpy()
    ok = compare_tokens(gtok, rtok, rex, ok, rep, sel)

    if target is None:
        target = synth.rows_from_depth(draft, buf.tree["depth"], target_noise, target_seed)
        ref_depth = torch.from_numpy(ref["depth"]).to(draft.device)
        h_target = synth.to_host(synth.rows_from_depth(draft, _scatter_depth(buf.tree["depth"], ref_depth, sel),
                                                       target_noise, target_seed)[sel])
    else:
        h_target = synth.to_host(target[sel])
    tsb.tsb_verify(buf.cfg, mode, target, q, qstats, qidx, buf.tree, buf.token, seed, buf.out_tokens,
                   buf.out_nodes, buf.out_len, buf.ws)
    check_status(buf)
    if mode == tsb.TSB_VERIFY_RRS:
        rout = oracle.verify_rrs(h_target, h_q, T, ref, rtok, seed, L, qrow_of_node=h_qidx)
    else:
        rout = oracle.verify_block(h_target, h_q, T, ref, rtok, seed, L, qrow_of_node=h_qidx)
    gout = {"len": buf.out_len.cpu().numpy(), "tokens": buf.out_tokens.cpu().numpy(),
            "nodes": buf.out_nodes.cpu().numpy()}
    compare_verify(gout, rout, ok, rep, sel)
    return rep, buf, gout


def _scatter_depth(gdepth, rdepth, sel):
    """GPU depth array with the oracle's depths written into the sampled trees (so the
    oracle's target rows follow the oracle's own plan)."""
    d = gdepth.clone()
    d[sel] = rdepth
    return d
