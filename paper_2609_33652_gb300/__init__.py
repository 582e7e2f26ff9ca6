"""GB300-native (sm_103a) library for the per-step logit path of Tsubame's two-pass tree
speculative decoding: plan (row top-k + best-first expansion), replay (Gumbel-top-k
sampling without replacement of every node's token) and verify (recursive rejection
sampling down the tree, and block verification of a sampled chain).

The compute lives in ``libtsb.so`` (hand-written CUDA behind a C ABI, ``include/tsb.h``);
``paper_2609_33652_gb300.tsb`` is the thin ctypes binding. Importing this package does not
load the library; the first call does, and fails loudly if it is missing.
"""
__all__ = ["tsb", "synth"]
