"""tsb_plan_noalloc (the first pass on the library's static device scratch) against tsb_plan
(the same pass on a caller workspace): identical trees on two calls in a row that reuse the
scratch with different shapes. Collected last so that it runs after every other test in a
full session, and self-contained so that it also runs alone in a fresh process."""
import ctypes

import pytest
import torch

from paper_2609_33652_gb300 import build as libbuild
from paper_2609_33652_gb300 import synth, tsb

FAKE = 0x7F00_0000_0000  # 256-aligned fake device address, never dereferenced by validation
SHAPE = 2


@pytest.fixture(scope="module")
def lib():
    libbuild.build()
    return tsb.load()


def test_noalloc_rejects_configs_beyond_its_scratch(lib):
    """256 + B*L*(8 + 8K) bytes must fit in TSB_NOALLOC_SCRATCH_BYTES; checked on the host
    before any CUDA call."""
    L, K, V = 16, 8, 1024
    per_tree = L * (8 + 8 * K)
    fits = (tsb.TSB_NOALLOC_SCRATCH_BYTES - 256) // per_tree
    assert fits == 910
    tree = tsb.Tree(*([FAKE] * 7))
    for B, ok in ((fits + 1, False), (4096, False)):
        cfg = tsb.make_cfg(B, L, 64, K, V, 1.0)
        d = tsb.Logits(FAKE, 0, B, L, V, L * V, V)
        rc = lib.tsb_plan_noalloc(ctypes.byref(cfg), ctypes.byref(d), FAKE, 1 << 40, ctypes.byref(tree), None, None)
        assert rc == SHAPE


def _case(B, L, N, K, V, dtype, seed, device):
    draft = synth.draft_logits(B, L, V, "planted", dtype, seed, device=device)
    ref = tsb.TsbBuffers.allocate(B, L, N, K, V, 1.0, device=device)
    tsb.tsb_row_stats(draft, 1.0, ref.stats, ref.ws)
    tsb.tsb_plan(ref.cfg, draft, ref.stats, ref.tree, ref.ws)
    out = {k: torch.full_like(v, -7) for k, v in ref.tree.items()}
    return draft, ref, out


def _assert_same_tree(ref_tree, tree):
    for k in ("parent", "depth", "rank", "plan_token", "child_off", "child_ids"):
        assert torch.equal(ref_tree[k], tree[k]), k
    torch.testing.assert_close(tree["score"], ref_tree["score"], rtol=1e-5, atol=1e-6)


@pytest.mark.gpu
def test_noalloc_plan_matches_workspace_plan_twice(lib):
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    # call 1: 16 trees over a 151,936-token bf16 vocabulary (the batched serving shape);
    # call 2: a different shape (f32, ragged V, K > 8) that reuses the same scratch
    d1, r1, o1 = _case(16, 16, 64, 8, 151936, "bf16", seed=11, device=dev)
    d2, r2, o2 = _case(6, 5, 150, 12, 5003, "f32", seed=12, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    torch.cuda.synchronize()
    before = torch.cuda.memory_allocated(dev)

    tsb.tsb_plan_noalloc(r1.cfg, d1, r1.stats, o1, dev_status=status)
    tsb.tsb_plan_noalloc(r2.cfg, d2, r2.stats, o2, dev_status=None)
    torch.cuda.synchronize()

    assert torch.cuda.memory_allocated(dev) == before
    assert int(status.item()) == 0
    assert tsb.tsb_device_status(r1.ws) == 0 and tsb.tsb_device_status(r2.ws) == 0
    _assert_same_tree(r1.tree, o1)
    _assert_same_tree(r2.tree, o2)

    # the same two calls again, with the device's free memory (cudaMemGetInfo, which also
    # sees allocations made outside torch's caching allocator) read on both sides: the
    # module and its static array are loaded by now, so nothing may change it
    for o in (o1, o2):
        for v in o.values():
            v.fill_(-7)
    torch.cuda.synchronize()
    free_before, _ = torch.cuda.mem_get_info(dev)
    tsb.tsb_plan_noalloc(r1.cfg, d1, r1.stats, o1, dev_status=status)
    tsb.tsb_plan_noalloc(r2.cfg, d2, r2.stats, o2, dev_status=None)
    torch.cuda.synchronize()
    free_after, _ = torch.cuda.mem_get_info(dev)
    assert free_after == free_before
    assert int(status.item()) == 0
    _assert_same_tree(r1.tree, o1)
    _assert_same_tree(r2.tree, o2)


@pytest.mark.gpu
def test_noalloc_plan_at_the_exact_scratch_limit(lib):
    """The largest batch whose scratch fits (910 trees at L = 16, K = 8: 256 + 910*16*72 bytes
    of the 1 MiB) runs, fills every tree like tsb_plan, and sets no status bit."""
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    B, L, N, K, V = 910, 16, 12, 8, 256
    assert 256 + B * L * (8 + 8 * K) <= tsb.TSB_NOALLOC_SCRATCH_BYTES < 256 + (B + 1) * L * (8 + 8 * K)
    d, r, o = _case(B, L, N, K, V, "bf16", seed=13, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    tsb.tsb_plan_noalloc(r.cfg, d, r.stats, o, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert tsb.tsb_device_status(r.ws) == 0
    _assert_same_tree(r.tree, o)
