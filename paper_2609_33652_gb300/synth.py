"""Seeded synthetic inputs shaped like the paper's workloads.

This module holds none of the method's arithmetic: it only draws random logits with the
shapes and value distributions of the workloads, and builds target rows from a tree's
depths or token paths. It is the one module that both the CUDA path's callers and the CPU
oracle's callers use, so both sides always see identical inputs.

Workloads (all synthetic; the paper's datasets, drafters and target models are not used):

* ``tiny``      B=1, V=32, L=4, fp32 draft logits z ~ N(0, 2^2), N=8, K=4, T=1.
* ``single``    B=1, V=151,936, L=16, bf16 draft logits 3*N(0,1) with one planted token per
                row whose probability is drawn from U(0.3, 0.9); N=32, K=8, T=1; target
                row of node u = draft row of depth(u) + N(0, 0.7^2).
* ``corrected`` as ``single`` with N=64 plus per-node draft rows (depth row + N(0, 0.3^2)),
                T in {0.6, 1.0}.
* ``batched``   B=16, V=128,256 (and 151,936), L=16, N=64, K=8, T=1, target [16, 65, V];
                plus a sampled chain of length 16 for block verification.
* ``sweep``     B=64, V=151,936, L=16, N in {16, 32, 64, 128, 256}, fp32 and bf16.

The planted-token recipe: the literal "+10" of the workload description gives a top-1
probability far below 0.3 at V=151,936, so the stated probability range wins: the planted
logit is LSE(background without that token) + log(p/(1-p)), p ~ U(0.3, 0.9), computed in
fp64 before the cast.
"""
from __future__ import annotations

import numpy as np
import torch

WORKLOADS = {
    "tiny": dict(B=1, V=32, L=4, N=8, K=4, T=1.0, dtype="f32", draft="normal2", target_noise=1.0),
    "single": dict(B=1, V=151936, L=16, N=32, K=8, T=1.0, dtype="bf16", draft="planted", target_noise=0.7),
    "corrected": dict(B=1, V=151936, L=16, N=64, K=8, T=1.0, dtype="bf16", draft="planted", target_noise=0.7,
                      per_node_noise=0.3),
    "batched": dict(B=16, V=151936, L=16, N=64, K=8, T=1.0, dtype="bf16", draft="planted", target_noise=0.7),
    "batched128k": dict(B=16, V=128256, L=16, N=64, K=8, T=1.0, dtype="bf16", draft="planted", target_noise=0.7),
    "sweep": dict(B=64, V=151936, L=16, N=64, K=8, T=1.0, dtype="bf16", draft="planted", target_noise=0.7),
}

_TORCH_DTYPES = {"f32": torch.float32, "bf16": torch.bfloat16}


def torch_dtype(name: str) -> torch.dtype:
    return _TORCH_DTYPES[name]


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _padded(V: int) -> int:
    """Row length rounded up to 8 elements, so every row starts on a 16-byte boundary."""
    return (V + 7) // 8 * 8


def draft_logits(B: int, L: int, V: int, kind: str, dtype: str, seed: int, device="cpu") -> torch.Tensor:
    """Per-depth draft logits [B, L, V] in ``dtype`` ("f32" or "bf16"); rows are padded to a
    multiple of 8 elements (the returned tensor is a view when V is not)."""
    Vp = _padded(V)
    if Vp != V:
        return draft_logits(B, L, Vp, kind, dtype, seed, device)[..., :V]
    g = _gen(seed, device)
    if kind == "normal2":
        z = 2.0 * torch.randn(B, L, V, generator=g, device=device, dtype=torch.float32)
    elif kind == "planted":
        z = 3.0 * torch.randn(B, L, V, generator=g, device=device, dtype=torch.float32)
        p = 0.3 + 0.6 * torch.rand(B, L, generator=g, device=device, dtype=torch.float64)
        tok = torch.randint(0, V, (B, L), generator=g, device=device)
        zz = z.to(torch.float64)
        zz.scatter_(2, tok.unsqueeze(-1), float("-inf"))
        lse_bg = torch.logsumexp(zz, dim=2)
        planted = lse_bg + torch.log(p / (1.0 - p))
        z.scatter_(2, tok.unsqueeze(-1), planted.to(torch.float32).unsqueeze(-1))
    elif kind == "normal3":
        z = 3.0 * torch.randn(B, L, V, generator=g, device=device, dtype=torch.float32)
    else:
        raise ValueError(kind)
    return z.to(_TORCH_DTYPES[dtype]).contiguous()


def rows_from_depth(draft: torch.Tensor, depth: torch.Tensor, noise_std: float, seed: int) -> torch.Tensor:
    """Row u of tree b = draft[b, min(depth[b, u], L-1)] + N(0, noise_std^2), cast back to the
    draft's dtype. Used for target rows (noise 0.7) and per-node draft rows (noise 0.3)."""
    B, L, V = draft.shape
    NN = depth.shape[1]
    idx = depth.to(device=draft.device, dtype=torch.long).clamp(max=L - 1)
    base = torch.gather(draft.to(torch.float32), 1, idx.unsqueeze(-1).expand(B, NN, V))
    g = _gen(seed, draft.device)
    noise = torch.randn(B, NN, V, generator=g, device=draft.device, dtype=torch.float32)
    rows = (base + noise_std * noise).to(draft.dtype)
    out = torch.empty(B, NN, _padded(V), dtype=draft.dtype, device=draft.device)[..., :V]
    out.copy_(rows)
    return out


def to_host(t: torch.Tensor) -> np.ndarray:
    """Host copy for the oracle: float32, or raw bf16 bit patterns as uint16."""
    t = t.detach().to("cpu").contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    if t.dtype == torch.float32:
        return t.numpy()
    raise TypeError(t.dtype)


# --------------------------------------------------------------------------------------
# Prefix-keyed target rows (for the losslessness tests): the target law at a node must be a
# function of the token path that reaches it, as for a real target model p(. | prefix).

_M64 = np.uint64(0xFFFFFFFFFFFFFFFF)


def _mix64(x: np.ndarray) -> np.ndarray:
    """splitmix64 finaliser (Steele, Lea & Flood 2014), vectorised over uint64 arrays."""
    with np.errstate(over="ignore"):
        z = x + np.uint64(0x9E3779B97F4A7C15)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return z ^ (z >> np.uint64(31))


def path_hashes(parent: np.ndarray, token: np.ndarray, seed: int) -> np.ndarray:
    """Hash of the token path root -> u for every node (nodes are in pop order, parent < u)."""
    B, NN = parent.shape
    h = np.zeros((B, NN), dtype=np.uint64)
    h[:, 0] = _mix64(np.full(B, seed, dtype=np.uint64))
    for u in range(1, NN):
        p = parent[:, u].astype(np.int64)
        hp = h[np.arange(B), p]
        h[:, u] = _mix64(hp ^ _mix64(token[:, u].astype(np.uint64) + np.uint64(1)))
    return h


def prefix_noise(h: np.ndarray, V: int) -> np.ndarray:
    """Standard normal noise [*, V] keyed by path hash (Box-Muller on hashed uniforms)."""
    v = np.arange(V, dtype=np.uint64)
    a = _mix64(h[..., None] ^ (np.uint64(2) * v + np.uint64(1)))
    b = _mix64(h[..., None] ^ (np.uint64(2) * v + np.uint64(2)) ^ np.uint64(0x5851F42D4C957F2D))
    u1 = ((a >> np.uint64(11)).astype(np.float64) + 0.5) * 2.0**-53
    u2 = ((b >> np.uint64(11)).astype(np.float64) + 0.5) * 2.0**-53
    return np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * np.pi * u2)


def path_keyed_rows(base: np.ndarray, parent: np.ndarray, depth: np.ndarray, token: np.ndarray, noise_std: float,
                    seed: int) -> np.ndarray:
    """Target rows [B, N+1, V] float32: base[min(depth, L-1)] + noise_std * noise(path hash).

    ``base`` is one set of per-depth rows [L, V] (float32) shared by every tree."""
    L, V = base.shape
    h = path_hashes(parent, token, seed)
    rows = base[np.minimum(depth, L - 1)] + noise_std * prefix_noise(h, V)
    return rows.astype(np.float32)


def path_keyed_row(base: np.ndarray, path_tokens, noise_std: float, seed: int) -> np.ndarray:
    """The target row [V] at the end of one explicit token path (for expected laws)."""
    L, V = base.shape
    h = _mix64(np.array([seed], dtype=np.uint64))
    for t in path_tokens:
        h = _mix64(h ^ _mix64(np.array([t], dtype=np.uint64) + np.uint64(1)))
    d = min(len(path_tokens), L - 1)
    return (base[d] + noise_std * prefix_noise(h, V)[0]).astype(np.float32)


def _signed64(c: int) -> int:
    return c - (1 << 64) if c >= 1 << 63 else c


def _lsr_t(x: torch.Tensor, k: int) -> torch.Tensor:
    """Logical right shift of int64 tensors holding uint64 bit patterns."""
    return (x >> k) & ((1 << (64 - k)) - 1)


def _mix64_t(x: torch.Tensor) -> torch.Tensor:
    """_mix64 on int64 tensors (two's-complement wraparound gives the uint64 arithmetic)."""
    z = x + _signed64(0x9E3779B97F4A7C15)
    z = (z ^ _lsr_t(z, 30)) * _signed64(0xBF58476D1CE4E5B9)
    z = (z ^ _lsr_t(z, 27)) * _signed64(0x94D049BB133111EB)
    return z ^ _lsr_t(z, 31)


def path_keyed_rows_device(base: torch.Tensor, parent: np.ndarray, depth: np.ndarray, token: np.ndarray,
                           noise_std: float, seed: int, trees_per_batch: int = 8192) -> torch.Tensor:
    """``path_keyed_rows`` generated on base's device (the same path hashes and noise formula),
    for trial counts whose rows do not fit the host comfortably. base: [L, V] float32."""
    L, V = base.shape
    dev = base.device
    h = torch.from_numpy(path_hashes(parent, token, seed).view(np.int64)).to(dev)
    d = torch.from_numpy(np.minimum(depth, L - 1).astype(np.int64)).to(dev)
    B, NN = h.shape
    out = torch.empty(B, NN, V, dtype=torch.float32, device=dev)
    v = torch.arange(V, dtype=torch.int64, device=dev)
    for b0 in range(0, B, trees_per_batch):
        hb = h[b0:b0 + trees_per_batch].unsqueeze(-1)
        a = _mix64_t(hb ^ (2 * v + 1))
        c = _mix64_t(hb ^ (2 * v + 2) ^ _signed64(0x5851F42D4C957F2D))
        u1 = (_lsr_t(a, 11).to(torch.float64) + 0.5) * 2.0**-53
        u2 = (_lsr_t(c, 11).to(torch.float64) + 0.5) * 2.0**-53
        noise = torch.sqrt(-2.0 * torch.log(u1)) * torch.cos(2.0 * np.pi * u2)
        rows = base.to(torch.float64)[d[b0:b0 + trees_per_batch]] + noise_std * noise
        out[b0:b0 + trees_per_batch] = rows.to(torch.float32)
    return out
