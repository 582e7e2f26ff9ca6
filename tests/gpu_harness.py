"""Runs the CUDA path (through the C ABI) and the CPU oracle on the same seeded inputs and
compares them stage by stage.

Comparison rule (the parity contract): every output must be bit-exact, and a difference is
accepted only where the oracle flags the decision that produced it as a near tie:
  * topology (parent, depth, rank, planning token, child lists): a tree may differ only if
    the oracle flags a near-tie pop in it (cross-depth keys closer than the GPU's bound on
    the error of its log-normaliser prefixes);
  * replayed tokens: a parent's children may differ only if the oracle flags a near-tie
    Gumbel decision at that parent (a deciding uniform within 1e-6 of its flip value);
  * verification outputs: may differ only if the oracle flags a near-tie decision in that
    tree's walk (acceptance uniform within 1e-6 of p'/q', or a near-tie Gumbel decision);
  * a stage of a tree is compared only when every earlier stage of that tree matched
    exactly (otherwise its inputs differ);
  * path scores within 1e-5 relative.
Budget: the differences actually seen (not the flags) are counted per stage and may not
exceed BUDGET_RATE = 1e-4 of that stage's decisions: planner pops (N per tree), replayed
tokens (m_u per parent), emitted tokens (one decision each, the oracle's length per walk).
For the sizes of the parity tests that allows no difference at all; a report of every
test's counts is appended to the file named by TSB_PARITY_LOG when that variable is set.
"""
from __future__ import annotations

import json
import os

import numpy as np
import torch

import oracle
from paper_2609_33652_gb300 import synth, tsb


def gpu_plan(draft, L, N, K, T, width=None):
    """tsb_row_stats + tsb_plan (max-heap), or tsb_plan_expand with frontier ``width``."""
    B, R, V = draft.shape
    buf = tsb.TsbBuffers.allocate(B, L, N, K, V, T, draft_rows=R, device=draft.device)
    tsb.tsb_row_stats(draft, T, buf.stats, buf.ws)
    if width is None:
        tsb.tsb_plan(buf.cfg, draft, buf.stats, buf.tree, buf.ws)
    else:
        tsb.tsb_plan_expand(buf.cfg, width, draft, buf.stats, buf.tree, buf.ws)
    return buf


def check_status(buf):
    bits = tsb.tsb_device_status(buf.ws)
    assert bits == 0, f"device status bits {bits:#x}"


def host_tree(buf):
    return {k: v.cpu().numpy() for k, v in buf.tree.items()}


BUDGET_RATE = 1e-4
STAGES = ("plan", "replay", "verify")


class Report:
    """Per stage: items compared (trees / parents / walks), decisions they hold (pops /
    replayed tokens / emitted tokens), items the oracle flagged as near ties, and items that
    actually differ (each of which must be flagged)."""

    def __init__(self):
        self.trees = 0
        self.compared = dict.fromkeys(STAGES, 0)
        self.units = dict.fromkeys(STAGES, 0)
        self.flagged = dict.fromkeys(STAGES, 0)
        self.differ = dict.fromkeys(STAGES, 0)

    def __repr__(self):
        return (f"Report(trees={self.trees}, compared={self.compared}, decisions={self.units}, "
                f"flagged={self.flagged}, differ={self.differ})")

    def merge(self, other):
        self.trees += other.trees
        for st in STAGES:
            self.compared[st] += other.compared[st]
            self.units[st] += other.units[st]
            self.flagged[st] += other.flagged[st]
            self.differ[st] += other.differ[st]
        return self

    def check(self, rate=BUDGET_RATE):
        """Log the counts, then hold every stage to the budget of actual differences."""
        log = os.environ.get("TSB_PARITY_LOG")
        if log:
            rec = {"test": os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0], "trees": self.trees,
                   "compared": self.compared, "decisions": self.units, "flagged": self.flagged,
                   "differ": self.differ}
            with open(log, "a") as f:
                f.write(json.dumps(rec) + "\n")
        for st in STAGES:
            allowed = int(rate * self.units[st])
            assert self.differ[st] <= allowed, f"{st}: {self.differ[st]} differences > budget {allowed}: {self}"
        return self


PLAN_KEYS = ("parent", "depth", "rank", "plan_token", "child_off", "child_ids")


def compare_plan(buf, ref, rep: Report, trees):
    """Returns the trees whose topology matched exactly."""
    g = host_tree(buf)
    same = {}
    for j, b in enumerate(trees):
        rep.trees += 1
        rep.compared["plan"] += 1
        rep.units["plan"] += int(ref["parent"].shape[1]) - 1
        rep.flagged["plan"] += int(bool(ref["exempt"][j]))
        eq = all(np.array_equal(g[k][b], ref[k][j]) for k in PLAN_KEYS)
        if not eq:
            assert ref["exempt"][j], f"tree {b}: topology differs without a flagged near tie"
            rep.differ["plan"] += 1
            same[b] = False
            continue
        np.testing.assert_allclose(g["score"][b], ref["score"][j], rtol=1e-5, atol=1e-5)
        same[b] = True
    return same


def compare_tokens(gtok, rtok, rex, tree, same, rep: Report, trees):
    """Per parent: children's tokens equal, or the parent is flagged. Returns the trees whose
    tokens all matched."""
    out = {}
    for j, b in enumerate(trees):
        if not same[b]:
            out[b] = False
            continue
        off, ids = tree["child_off"][b], tree["child_ids"][b]
        all_eq = True
        for u in range(len(off) - 1):
            kids = ids[off[u]:off[u + 1]]
            if len(kids) == 0:
                continue
            rep.compared["replay"] += 1
            rep.units["replay"] += len(kids)
            rep.flagged["replay"] += int(bool(rex[j, u]))
            if not np.array_equal(gtok[b, kids], rtok[j, kids]):
                assert rex[j, u], f"tree {b} parent {u}: replayed tokens differ without a flagged near tie"
                rep.differ["replay"] += 1
                all_eq = False
        if all_eq:
            assert gtok[b, 0] == rtok[j, 0] == -1
        out[b] = all_eq
    return out


def compare_verify(gout, rout, same, rep: Report, trees):
    for j, b in enumerate(trees):
        if not same[b]:
            continue
        rep.compared["verify"] += 1
        rep.units["verify"] += int(rout["len"][j])
        rep.flagged["verify"] += int(bool(rout["exempt"][j]))
        eq = (gout["len"][b] == rout["len"][j] and np.array_equal(gout["tokens"][b], rout["tokens"][j])
              and np.array_equal(gout["nodes"][b], rout["nodes"][j]))
        if not eq:
            assert rout["exempt"][j], (f"tree {b}: verification differs without a flagged near tie "
                                       f"(gpu len {gout['len'][b]} tokens {gout['tokens'][b]}, "
                                       f"oracle len {rout['len'][j]} tokens {rout['tokens'][j]})")
            rep.differ["verify"] += 1


def compare_trials(buf, tok, rtok, rex, rout):
    """Many trees on one topology (the losslessness trials): replayed tokens and verification
    outputs against the oracle, held to the difference budget."""
    tree = host_tree(buf)
    gout = {"len": buf.out_len.cpu().numpy(), "tokens": buf.out_tokens.cpu().numpy(),
            "nodes": buf.out_nodes.cpu().numpy()}
    rep = Report()
    trees = list(range(tok.shape[0]))
    same = compare_tokens(tok, rtok, rex, tree, dict.fromkeys(trees, True), rep, trees)
    compare_verify(gout, rout, same, rep, trees)
    return rep.check()


def run_step(draft, L, N, K, T, seed, target_noise=0.7, target_seed=2000, qrows=None, qrow_of_node=None,
             trees=None, mode=tsb.TSB_VERIFY_RRS, target=None, width=None, replay="wor", check=True):
    """Full plan -> replay -> verify on both sides; returns the report, the GPU buffers and
    the GPU outputs. ``trees`` restricts the oracle to a sample of trees (large batches); the
    oracle then draws with the sampled trees' own batch indices. ``width``: expand-then-prune
    first pass with that frontier (default: max-heap). ``replay``: "wor" (tsb_replay), "mixed"
    (tsb_replay_mixed) or "plan" (no replay: the first pass's tokens are verified). With
    ``check`` the report is held to the difference budget before returning."""
    rep = Report()
    buf = gpu_plan(draft, L, N, K, T, width)
    check_status(buf)
    B = draft.shape[0]
    sel = list(range(B)) if trees is None else list(trees)
    bids = np.array(sel, dtype=np.int32)
    h_draft = synth.to_host(draft[sel])
    ref = oracle.plan(h_draft, T, N, K, L) if width is None else oracle.plan_expand(h_draft, T, N, K, L, width)
    same = compare_plan(buf, ref, rep, sel)

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
    if replay == "plan":
        buf.token.copy_(buf.tree["plan_token"])
        rtok, rex = ref["plan_token"], np.zeros(ref["plan_token"].shape, dtype=bool)
    elif replay == "mixed":
        tsb.tsb_replay_mixed(buf.cfg, q, qstats, qidx, buf.tree, seed, buf.token, buf.ws)
        rtok, rex = oracle.replay_mixed(h_q, T, ref, seed, qrow_of_node=h_qidx, batch_ids=bids)
    else:
        tsb.tsb_replay(buf.cfg, q, qstats, qidx, buf.tree, seed, buf.token, buf.ws)
        rtok, rex = oracle.replay(h_q, T, ref, seed, qrow_of_node=h_qidx, batch_ids=bids)
    check_status(buf)
    gtok = buf.token.cpu().numpy()
    same = compare_tokens(gtok, rtok, rex, host_tree(buf), same, rep, sel)

    if target is None:
        target = synth.rows_from_depth(draft, buf.tree["depth"], target_noise, target_seed)
        ref_depth = torch.from_numpy(ref["depth"]).to(draft.device)
        h_target = synth.to_host(synth.rows_from_depth(draft, _scatter_depth(buf.tree["depth"], ref_depth, sel),
                                                       target_noise, target_seed)[sel])
    else:
        h_target = synth.to_host(target[sel])
    if mode == tsb.TSB_VERIFY_NAIVE:  # no draft rows needed
        tsb.tsb_verify(buf.cfg, mode, target, None, None, None, buf.tree, buf.token, seed, buf.out_tokens,
                       buf.out_nodes, buf.out_len, buf.ws)
    else:
        tsb.tsb_verify(buf.cfg, mode, target, q, qstats, qidx, buf.tree, buf.token, seed, buf.out_tokens,
                       buf.out_nodes, buf.out_len, buf.ws)
    check_status(buf)
    if mode == tsb.TSB_VERIFY_RRS:
        rout = oracle.verify_rrs(h_target, h_q, T, ref, rtok, seed, L, qrow_of_node=h_qidx, batch_ids=bids)
    elif mode == tsb.TSB_VERIFY_TRAVERSAL:
        rout = oracle.verify_traversal(h_target, h_q, T, ref, rtok, seed, L, qrow_of_node=h_qidx, batch_ids=bids)
    elif mode == tsb.TSB_VERIFY_NAIVE:
        rout = oracle.verify_naive(h_target, T, ref, rtok, seed, L, batch_ids=bids)
    else:
        rout = oracle.verify_block(h_target, h_q, T, ref, rtok, seed, L, qrow_of_node=h_qidx, batch_ids=bids)
    gout = {"len": buf.out_len.cpu().numpy(), "tokens": buf.out_tokens.cpu().numpy(),
            "nodes": buf.out_nodes.cpu().numpy()}
    compare_verify(gout, rout, same, rep, sel)
    if check:
        rep.check()
    return rep, buf, gout


def _scatter_depth(gdepth, rdepth, sel):
    """GPU depth array with the oracle's depths written into the sampled trees (so the
    oracle's target rows follow the oracle's own plan)."""
    d = gdepth.clone()
    d[sel] = rdepth
    return d
