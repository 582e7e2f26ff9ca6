"""The parity suite's tiny cases through libtsb_checked.so, the TSB_CHECKED build: every
data-dependent shared-memory fill position (atomic counters) and index is bounds-checked there,
and a failed check sets TSB_DEV_CHECK in the status word (the access is skipped). The outputs
must still equal the oracle's, and no check may fail."""
import numpy as np
import pytest
import torch

import oracle
from gpu_harness import gpu_plan, run_step
from paper_2609_33652_gb300 import build, synth, tsb

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()
    oracle.build()
    tsb.load()


DEV = "cuda"


def _draft(B, L, V, kind, dtype, seed):
    return synth.draft_logits(B, L, V, kind, dtype, seed, device=DEV)


@pytest.mark.parametrize("seed", [0, 1])
def test_checked_step_tiny(seed):
    w = synth.WORKLOADS["tiny"]
    draft = _draft(64, w["L"], w["V"], "normal2", "f32", 1000 + seed)
    with tsb.checked_library():
        run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=seed, target_noise=1.0)


def test_checked_small_vocab_many_children():
    draft = _draft(8, 4, 1000, "normal2", "f32", 31)
    with tsb.checked_library():
        run_step(draft, 4, 40, 8, 1.0, seed=13, target_noise=0.7)


@pytest.mark.parametrize("mode", [tsb.TSB_VERIFY_NAIVE, tsb.TSB_VERIFY_TRAVERSAL])
def test_checked_other_verifiers(mode):
    w = synth.WORKLOADS["tiny"]
    draft = _draft(32, w["L"], w["V"], "normal2", "f32", 1100)
    with tsb.checked_library():
        run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=3, target_noise=1.0, mode=mode)


def test_checked_mixed_and_expand():
    w = synth.WORKLOADS["tiny"]
    draft = _draft(32, w["L"], w["V"], "normal2", "f32", 1200)
    with tsb.checked_library():
        run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=4, target_noise=1.0, replay="mixed",
                 mode=tsb.TSB_VERIFY_NAIVE)
        run_step(draft, w["L"], w["N"], w["K"], w["T"], seed=4, target_noise=1.0, width=2)


def test_checked_status_bit_is_distinct():
    """The checked build sets its own bit; a clean run leaves the word at zero."""
    assert tsb.TSB_DEV_CHECK not in (tsb.TSB_DEV_NONFINITE, tsb.TSB_DEV_BAD_INDEX, tsb.TSB_DEV_BAD_TREE)
    w = synth.WORKLOADS["tiny"]
    draft = _draft(4, w["L"], w["V"], "normal2", "f32", 1300)
    with tsb.checked_library():
        buf = gpu_plan(draft, w["L"], w["N"], w["K"], 1.0)
        assert tsb.tsb_device_status(buf.ws) == 0
