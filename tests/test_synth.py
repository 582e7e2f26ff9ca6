"""The seeded input generators (no method arithmetic): the device-side path-keyed target rows
are the host generator's rows bit for bit (run here on torch's CPU device)."""
import numpy as np
import torch

from paper_2609_33652_gb300 import synth


def test_path_keyed_rows_device_matches_host():
    rng = np.random.default_rng(1)
    base = rng.standard_normal((4, 300)).astype(np.float32)
    B = 50
    parent = np.tile(np.array([-1, 0, 0, 1, 1, 2, 3, 3, 4]), (B, 1)).astype(np.int32)
    depth = np.tile(np.array([0, 1, 1, 2, 2, 2, 3, 3, 3]), (B, 1)).astype(np.int32)
    tok = rng.integers(0, 300, parent.shape).astype(np.int32)
    host = synth.path_keyed_rows(base, parent, depth, tok, 1.0, 77)
    dev = synth.path_keyed_rows_device(torch.from_numpy(base), parent, depth, tok, 1.0, 77, trees_per_batch=7)
    assert np.array_equal(host, dev.numpy())
    # the row at the end of an explicit path is the same row
    b, u = 3, 7
    path = [int(tok[b, 1]), int(tok[b, 3]), int(tok[b, 7])]
    assert np.array_equal(synth.path_keyed_row(base, path, 1.0, 77), host[b, u])
