"""tsb_replay_verify (replay and recursive rejection sampling in one call, the verifier's
pre-pass in the replay's grid) against tsb_replay followed by tsb_verify: the same tokens and
outputs bit for bit, on the batched serving shape, small vocabularies, K > 8 (the 32-slot
replay lists) and per-node q rows; and against the oracle through the parity harness."""
import pytest
import torch

from gpu_harness import check_status, gpu_plan
from paper_2609_33652_gb300 import synth, tsb

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0")


def _two_ways(buf, target, q, qstats, qidx, seed):
    """Outputs of the two calls and of the one call, each from fresh output buffers."""
    res = []
    for together in (False, True):
        tok = torch.full_like(buf.token, -7)
        ot = torch.full_like(buf.out_tokens, -7)
        on = torch.full_like(buf.out_nodes, -7)
        ol = torch.full_like(buf.out_len, -7)
        if together:
            tsb.tsb_replay_verify(buf.cfg, target, q, qstats, qidx, buf.tree, seed, tok, ot, on, ol, buf.ws)
        else:
            tsb.tsb_replay(buf.cfg, q, qstats, qidx, buf.tree, seed, tok, buf.ws)
            tsb.tsb_verify(buf.cfg, tsb.TSB_VERIFY_RRS, target, q, qstats, qidx, buf.tree, tok, seed, ot, on, ol,
                           buf.ws)
        check_status(buf)
        res.append({k: v.cpu() for k, v in (("token", tok), ("tokens", ot), ("nodes", on), ("len", ol))})
    return res


@pytest.mark.parametrize("B,V,L,N,K,T,dtype,kind,seed", [
    (16, 151936, 16, 64, 8, 1.0, "bf16", "planted", 11),  # the batched serving shape
    (16, 151936, 16, 64, 8, 0.6, "bf16", "planted", 12),
    (5, 1000, 6, 30, 4, 1.0, "f32", "normal2", 13),        # four chunks, a ragged tail
    (3, 700, 5, 40, 12, 0.8, "bf16", "planted", 14),       # K > 8
    (2, 37, 4, 9, 3, 1.0, "f32", "normal2", 15),           # one chunk, a short chain
])
def test_one_call_equals_two(B, V, L, N, K, T, dtype, kind, seed):
    draft = synth.draft_logits(B, L, V, kind, dtype, 900 + seed, device=DEV)
    buf = gpu_plan(draft, L, N, K, T)
    check_status(buf)
    target = synth.rows_from_depth(draft, buf.tree["depth"], 0.7, 2000 + seed)
    for step_seed in (seed, seed + 1000):
        a, b = _two_ways(buf, target, draft, buf.stats, None, step_seed)
        for k in a:
            assert torch.equal(a[k], b[k]), k
        assert (b["len"] >= 1).all()


def test_one_call_equals_two_per_node_rows():
    w = synth.WORKLOADS["corrected"]
    B, T = 4, 0.6
    draft = synth.draft_logits(B, w["L"], w["V"], "planted", "bf16", 1002, device=DEV)
    buf = gpu_plan(draft, w["L"], w["N"], w["K"], T)
    qrows = synth.rows_from_depth(draft, buf.tree["depth"], w["per_node_noise"], seed=3000)
    qstats = torch.empty(tsb.tsb_stats_bytes(B, qrows.shape[1], qrows.shape[2]) // 4, dtype=torch.float32,
                         device=DEV)
    tsb.tsb_row_stats(qrows, T, qstats, buf.ws)
    qidx = torch.arange(w["N"] + 1, dtype=torch.int32, device=DEV).repeat(B, 1).contiguous()
    target = synth.rows_from_depth(draft, buf.tree["depth"], w["target_noise"], 2000)
    a, b = _two_ways(buf, target, qrows, qstats, qidx, 9)
    for k in a:
        assert torch.equal(a[k], b[k]), k


def test_prepared_step_together():
    """The bench's step with the one call gives the outputs of the three-call step."""
    w = synth.WORKLOADS["batched"]
    draft = synth.draft_logits(w["B"], w["L"], w["V"], "planted", "bf16", 1003, device=DEV)
    outs = []
    for together in (False, True):
        buf = tsb.TsbBuffers.allocate(w["B"], w["L"], w["N"], w["K"], w["V"], w["T"], device=DEV)
        tsb.tsb_workspace_init(buf.ws)
        plan = tsb.PreparedStep(buf, draft, draft, 5, plan_only=True)
        plan.run()
        target = synth.rows_from_depth(draft, buf.tree["depth"], w["target_noise"], 2000)
        step = tsb.PreparedStep(buf, draft, target, 5, together=together)
        assert [c[0] for c in step.calls][-1] == ("tsb_replay_verify" if together else "tsb_verify")
        step.run()
        check_status(buf)
        outs.append((buf.token.cpu(), buf.out_tokens.cpu(), buf.out_len.cpu()))
    for x, y in zip(*outs):
        assert torch.equal(x, y)
