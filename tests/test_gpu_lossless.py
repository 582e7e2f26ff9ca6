"""Losslessness of the GPU path (Prop. 1 for recursive rejection sampling; the cited works for
traversal and block verification), 1e5 seeded trials each, through the C ABI.

Every trial is a tree over the same draft rows (batch stride 0) with its own replayed tokens
and uniforms; target rows are a function of the token path (a real target model's
p(. | prefix)), generated on the device. Checked per verifier, at V = 32 (one 256-token chunk)
and V = 1000 (four chunks, so the chunk level of the replay sampler and of the two-level final
draw is exercised):
  * the first emitted token follows the root's target law (chi-square);
  * the second token, extended by a target draw when only one token was emitted, follows the
    target law after the first (chi-square for the most frequent first tokens);
  * a sample of the trials matches the oracle (plan, replay and verification), held to the
    difference budget of the parity tests.
"""
import numpy as np
import pytest
import torch

import helpers
import oracle
from gpu_harness import Report, compare_tokens, compare_verify, gpu_plan
from paper_2609_33652_gb300 import synth, tsb

pytestmark = pytest.mark.gpu
DEV = "cuda"
P_MIN = 1e-4
TRIALS = 100_000
SAMPLE = 1500  # trials also run through the oracle


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_33652_gb300 import build

    build.build()
    oracle.build()
    tsb.load()


def _trials(mode, V, seed, L=4, N=8, K=4, T=1.0):
    if mode == tsb.TSB_VERIFY_BLOCK:
        N, K = L, 1  # the sampled chain of length L
    base1 = synth.draft_logits(1, L, V, "normal2", "f32", 1000 + V, device=DEV)
    draft = base1.expand(TRIALS, -1, -1)
    buf = gpu_plan(draft, L, N, K, T)
    tsb.tsb_replay(buf.cfg, draft, buf.stats, None, buf.tree, seed, buf.token, buf.ws)
    assert tsb.tsb_device_status(buf.ws) == 0
    tree = {k: v.cpu().numpy() for k, v in buf.tree.items()}
    tok = buf.token.cpu().numpy()
    target = synth.path_keyed_rows_device(base1[0].contiguous(), tree["parent"], tree["depth"], tok, 1.0, seed=77)
    tsb.tsb_verify(buf.cfg, mode, target, draft, buf.stats, None, buf.tree, buf.token, seed, buf.out_tokens,
                   buf.out_nodes, buf.out_len, buf.ws)
    assert tsb.tsb_device_status(buf.ws) == 0
    out = {"len": buf.out_len.cpu().numpy(), "tokens": buf.out_tokens.cpu().numpy(),
           "nodes": buf.out_nodes.cpu().numpy()}
    return dict(buf=buf, draft=draft, base=synth.to_host(base1)[0], tree=tree, tok=tok, target=target, out=out,
                L=L, N=N, K=K, T=T, V=V, seed=seed)


def _check_laws(r):
    V, base, out = r["V"], r["base"], r["out"]
    inv = np.float32(np.float32(1.0) / np.float32(r["T"]))

    def p_after(prefix):
        return helpers.softmax64(synth.path_keyed_row(base, list(prefix), 1.0, 77) * inv)

    first = out["tokens"][:, 0]
    assert ((first >= 0) & (first < V)).all() and (out["len"] >= 1).all()
    assert helpers.chi2_pvalue(np.bincount(first, minlength=V), p_after([])) > P_MIN
    second = out["tokens"][:, 1].copy()
    ext = np.random.default_rng(r["seed"])
    vals, cnt = np.unique(first, return_counts=True)
    for a in vals[np.argsort(-cnt)][:3]:
        sel = first == a
        pa = p_after([int(a)])
        short = sel & (out["len"] == 1)
        second[short] = ext.choice(V, size=int(short.sum()), p=pa)
        assert helpers.chi2_pvalue(np.bincount(second[sel], minlength=V), pa) > P_MIN, (a, int(sel.sum()))


def _check_oracle(r, mode):
    """The oracle on SAMPLE trials (their own batch indices), same inputs."""
    sel = list(range(0, TRIALS, TRIALS // SAMPLE))[:SAMPLE]
    bids = np.array(sel, dtype=np.int32)
    L, N, K, T, seed = r["L"], r["N"], r["K"], r["T"], r["seed"]
    h1 = synth.to_host(r["draft"][:1].contiguous())
    ref1 = oracle.plan(h1, T, N, K, L)
    for k in ("parent", "depth", "rank", "plan_token", "child_off", "child_ids"):
        assert np.array_equal(ref1[k][0], r["tree"][k][0]), k
    ref = helpers.repeat_tree({k: v for k, v in ref1.items() if k not in ("exempt", "min_margin")}, len(sel))
    hq = np.ascontiguousarray(np.broadcast_to(h1, (len(sel),) + h1.shape[1:]))
    rtok, rex = oracle.replay(hq, T, ref, seed, batch_ids=bids)
    rep = Report()
    same = compare_tokens(r["tok"], rtok, rex, r["tree"], dict.fromkeys(sel, True), rep, sel)
    ht = synth.to_host(r["target"][sel].contiguous())
    fn = {tsb.TSB_VERIFY_RRS: oracle.verify_rrs, tsb.TSB_VERIFY_TRAVERSAL: oracle.verify_traversal,
          tsb.TSB_VERIFY_BLOCK: oracle.verify_block}[mode]
    rout = fn(ht, hq, T, ref, rtok, seed, L, batch_ids=bids)
    compare_verify(r["out"], rout, same, rep, sel)
    rep.check()


MODES = {"rrs": tsb.TSB_VERIFY_RRS, "traversal": tsb.TSB_VERIFY_TRAVERSAL, "block": tsb.TSB_VERIFY_BLOCK}


@pytest.mark.parametrize("V", [32, 1000])
@pytest.mark.parametrize("name", ["rrs", "traversal", "block"])
def test_lossless_on_gpu(name, V):
    r = _trials(MODES[name], V, seed={"rrs": 51, "traversal": 52, "block": 53}[name])
    _check_laws(r)
    _check_oracle(r, MODES[name])
