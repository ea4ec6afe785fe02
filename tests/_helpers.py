"""Shared helpers for the GPU parity tests: building segment tensors in several
layouts, converting them to the oracle's bf16 bit arrays, and the tolerances."""
import math

import numpy as np
import torch

import oracle

ROLES = ("text", "ref", "tgt")

# Parity tolerances of the hot path against the fp64 oracle: O max relative
# error 1e-2 (bf16 P and O round at 2^-9 relative), M 1e-3 absolute, D 1e-4
# relative; gate modes exact except where |gbar - theta| < 1e-4, where the
# GPU's fp32 score and the oracle's fp64 score may fall on either side.
O_REL = 1e-2
M_ABS = 1e-3
D_REL = 1e-4
TIE_BAND = 1e-4


def bits(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor (any device) -> uint16 numpy array of its bit patterns."""
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def f64(t: torch.Tensor) -> np.ndarray:
    return oracle.bf16_to_f64(bits(t))


def make_segments(B, H, d, n, layout="separate", scale=None, gen=None, device="cuda", std=None):
    """Random q, k, v segments per role.

    layout: 'separate' (one contiguous [B,H,n,d] tensor per role and kind),
            'joint' (one [B,H,N,d] tensor per kind, roles are slices along N),
            'token' (one [B,N,H,d] tensor per kind viewed as [B,H,N,d], roles sliced).
    std: element standard deviation (default 1/sqrt(d)).
    Returns dict role -> [q, k, v] CUDA bf16 views.
    """
    g = gen or torch.Generator().manual_seed(0)
    sd = (1.0 / math.sqrt(d)) if std is None else std
    N = sum(n[r] for r in ROLES)
    out = {r: [None, None, None] for r in ROLES}
    for z in range(3):
        if layout == "separate":
            for r in ROLES:
                x = (torch.randn((B, H, n[r], d), generator=g) * sd).to(torch.bfloat16)
                out[r][z] = x.to(device)
        else:
            if layout == "joint":
                full = (torch.randn((B, H, N, d), generator=g) * sd).to(torch.bfloat16).to(device)
            elif layout == "token":
                full = (torch.randn((B, N, H, d), generator=g) * sd).to(torch.bfloat16).to(device)
                full = full.permute(0, 2, 1, 3)
            else:
                raise ValueError(layout)
            o = 0
            for r in ROLES:
                out[r][z] = full[:, :, o:o + n[r], :]
                o += n[r]
    return out


def empty_outputs(B, H, d, n, device="cuda", fill=float("nan")):
    return {r: torch.full((B, H, n[r], d), fill, dtype=torch.bfloat16, device=device) for r in ROLES}


def oracle_block(segs, s, mode, scale, bias=None, mass_rows=0):
    """Oracle block attention for sample s of GPU segment tensors."""
    q = {r: f64(segs[r][0][s]) for r in ROLES}
    k = {r: f64(segs[r][1][s]) for r in ROLES}
    v = {r: f64(segs[r][2][s]) for r in ROLES}
    return oracle.block_attention(q, k, v, mode, scale, bias, mass_rows)


def o_close(got, ref, rel=O_REL):
    """|o - r| <= rel * (|r| + rms(r)) elementwise, per (head) slab. Returns
    (ok, worst ratio, normwise relative error)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    if ref.size == 0:
        return True, 0.0, 0.0
    rms = np.sqrt(np.mean(ref ** 2, axis=tuple(range(1, ref.ndim)), keepdims=True)) + 1e-30
    ratio = np.abs(got - ref) / (rel * (np.abs(ref) + rms))
    worst = float(np.nanmax(ratio)) if np.all(np.isfinite(got)) else float("inf")
    normwise = float(np.linalg.norm(got - ref) / (np.linalg.norm(ref) + 1e-30))
    return worst <= 1.0, worst, normwise


def mass_from_partials(partial, n_rows):
    """[B, H, L] tile partials -> [B, H] mean mass."""
    return partial.double().sum(-1).cpu().numpy() / float(n_rows)
