"""Oracle for the DiT block around the hot path: fp64, plain numpy.

TEST INFRASTRUCTURE (see the package header): only tests/, smoke() and
bench.py's CPU legs may use it; it shares nothing with the CUDA library.

What the paper fixes and what it leaves open. The paper runs distilled
multi-reference DiTs whose blocks attend jointly over [text; reference;
target] rows (Sec. 3, "Setting"); under reuse, reference-side QKV projections
and the other reference-stream operations are skipped because the layer-wise
reference K/V are cached (App. A.4); at the boundary block the cached
reference hidden state is restored, the reference query runs against the
current target and the reference output is stored as the next block's cached
hidden state (Algorithm 1, App. A.3). D is measured on the post-RoPE target
query (Sec. 4). The block's layers themselves are not given; this module takes
a dual-stream MMDiT block (one weight set for text rows, one for image rows =
reference + target), with

* AdaLN modulation per block, stream and sample: shift, scale, gate for the
  attention branch and for the MLP branch (six vectors of width C = H d,
  inputs of the block);
* x = LN(h) (1 + scale) + shift, LN without affine, eps 1e-6;
* q, k, v = split(x W_qkv^T + b_qkv) per head; q and k RMS-normalised over d
  with a per-stream weight, eps 1e-6, then rotated by RoPE on interleaved
  pairs (2i, 2i+1) by angle pos * base^(-2i/d), base 1e4, pos = the row's
  index in the joint sequence;
* h <- h + gate_a * (O W_o^T + b_o) after the joint attention;
* h <- h + gate_m * (GELU_tanh(x' W_1^T + b_1) W_2^T + b_2), x' the MLP
  branch's modulated LN, MLP width 4C.

Every tensor the block stores between operations is bf16 (x, q, k, v, O, h,
the MLP hidden); each operation is computed here in fp64 from the stored
values and its result rounded to bf16 (nearest, ties to even) at the same
points, so the CUDA path's fp32 arithmetic differs only below bf16 rounding.
"""
import math

import numpy as np

from .core import (BOUNDARY, COMPUTE, FULL, REUSE, ROLES, Gate, block_attention, bf16_to_f64,
                   q_change)

STREAM_OF = {"text": "text", "ref": "image", "tgt": "image"}


def round_bf16(x) -> np.ndarray:
    """Round float64 values to the nearest bf16 value (8 significant bits,
    ties to even), returned as float64. Finite values in bf16's normal range."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                  # x = m 2^e, 0.5 <= |m| < 1
    return np.ldexp(np.rint(m * 256.0) / 256.0, e)


def linear(x, W, b=None) -> np.ndarray:
    """x W^T + b for x [n, K], W [N, K], b [N] (a library matmul as one step)."""
    y = np.asarray(x, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T
    return y if b is None else y + np.asarray(b, dtype=np.float64)


def layer_norm_modulate(h, shift, scale, eps=1e-6) -> np.ndarray:
    """LN(h) (1 + scale) + shift over the last axis (LN without affine)."""
    h = np.asarray(h, dtype=np.float64)
    mu = h.mean(axis=-1, keepdims=True)
    var = ((h - mu) ** 2).mean(axis=-1, keepdims=True)
    return (h - mu) / np.sqrt(var + eps) * (1.0 + np.asarray(scale, np.float64)) + np.asarray(shift, np.float64)


def rms_norm(x, w, eps=1e-6) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * w over the last axis."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt((x * x).mean(axis=-1, keepdims=True) + eps) * np.asarray(w, np.float64)


def rope_angles(pos, d, base=10000.0) -> np.ndarray:
    """Angles [n, d/2]: pos * base^(-2i/d)."""
    i = np.arange(d // 2, dtype=np.float64)
    return np.asarray(pos, dtype=np.float64)[:, None] * base ** (-2.0 * i / d)[None, :]


def apply_rope(x, pos, base=10000.0) -> np.ndarray:
    """Rotate each interleaved pair (x_{2i}, x_{2i+1}) of the last axis by
    pos * base^(-2i/d). x [..., n, d], pos [n]."""
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    ang = rope_angles(pos, d, base)
    c, s = np.cos(ang), np.sin(ang)
    x0, x1 = x[..., 0::2], x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = x0 * c - x1 * s
    out[..., 1::2] = x0 * s + x1 * c
    return out


def gelu_tanh(x) -> np.ndarray:
    """GELU, tanh form: 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))."""
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def qkv_project(h, mod, W, pos, H, d, eps=1e-6, base=10000.0):
    """Attention-branch input of a block for rows h [n, C] of one stream:
    modulated LN (stored bf16), the QKV linear, per-head RMS norm of q and k,
    RoPE of q and k; returns q, k, v as bf16-valued float64 [H, n, d].
    mod: dict shift_a, scale_a (C); W: dict w_qkv [3C, C], b_qkv [3C],
    q_norm [d], k_norm [d]."""
    n = h.shape[0]
    C = H * d
    x = round_bf16(layer_norm_modulate(h, mod["shift_a"], mod["scale_a"], eps))
    y = linear(x, W["w_qkv"], W["b_qkv"])
    q = y[:, 0:C].reshape(n, H, d).transpose(1, 0, 2)
    k = y[:, C:2 * C].reshape(n, H, d).transpose(1, 0, 2)
    v = y[:, 2 * C:3 * C].reshape(n, H, d).transpose(1, 0, 2)
    q = apply_rope(rms_norm(q, W["q_norm"], eps), pos, base)
    k = apply_rope(rms_norm(k, W["k_norm"], eps), pos, base)
    return round_bf16(q), round_bf16(k), round_bf16(v)


def post_attention(h, o, mod, W, eps=1e-6):
    """Rest of the block for rows h [n, C] (bf16 values) given their attention
    output o [H, n, d] (bf16 values): output projection with gated residual,
    modulated LN, GELU MLP with gated residual. Returns bf16-valued [n, C]."""
    H, n, d = o.shape
    of = o.transpose(1, 0, 2).reshape(n, H * d)
    h1 = round_bf16(h + np.asarray(mod["gate_a"], np.float64) * linear(of, W["w_o"], W["b_o"]))
    x2 = round_bf16(layer_norm_modulate(h1, mod["shift_m"], mod["scale_m"], eps))
    u = round_bf16(gelu_tanh(linear(x2, W["w_1"], W["b_1"])))
    return round_bf16(h1 + np.asarray(mod["gate_m"], np.float64) * linear(u, W["w_2"], W["b_2"]))


def dit_closed_loop(h_in, mods, weights, n_steps, n_blocks, B, H, d, *, theta, delta_max, eps=1e-6,
                    ln_eps=1e-6, rope_base=10000.0, mass_rows=0, forced_boundary=-1, tie=None,
                    tie_band=1e-4, cue="product", nthreads=None):
    """Algorithm 1 over a stack of DiT blocks (the block of this module).

    h_in(t) -> dict role -> uint16 bf16 bits [B, n_role, C]: the stack's input
    rows at step t (text and reference rows are the same at every step in the
    workloads used here; target rows follow the sampler).
    mods(t, b) -> dict stream -> dict of six fp32 arrays [B, C] (shift_a,
    scale_a, gate_a, shift_m, scale_m, gate_m); stream in {text, image}.
    weights(b) -> dict stream -> dict w_qkv, w_o, w_1, w_2 (uint16 bf16 bits)
    and b_qkv, b_o, b_1, b_2, q_norm, k_norm (fp32).

    Reference stream (Algorithm 1, App. A.3): Hbar[b] is the cached input
    hidden state of block b's reference rows; Hbar[0] is the reference input.
    REUSE: reference rows do nothing; text and target rows attend to the
    cached reference K/V. BOUNDARY: the reference rows restore Hbar[b], form
    their query (their K/V stay the cached ones), attend, finish the block and
    store Hbar[b+1]. COMPUTE / FULL: the reference rows form Q, K, V from
    Hbar[b], the cache takes K, V (a_b = t), all rows attend, the reference
    output is stored as Hbar[b+1]. D is Eq. 1 on the post-RoPE target query,
    M the executed attention's exposure, both recorded for the next step.

    ``tie(t, b, s)`` and ``tie_band``: as in ``Gate.decide`` (a score within
    the band of theta adopts the given decision).

    Returns records[t][b] = dict(mode, gbar, D, M, a_b) and per step
    outputs[t] = dict(text, tgt [B, n, C], hbar [n_blocks + 1][B] arrays or
    None) with the stack's output rows and the reference hidden states.
    """
    gate = Gate(B, theta, delta_max, forced_boundary, cue)
    C = H * d
    sc = 1.0 / math.sqrt(d)
    cache = [[None] * B for _ in range(n_blocks)]
    a_b = [[-1] * B for _ in range(n_blocks)]
    hbar = [[None] * B for _ in range(n_blocks + 1)]
    prev_q = [None] * n_blocks
    prev_M = [None] * n_blocks
    records, outputs = [], []
    for t in range(n_steps):
        gate.begin_step(t)
        x0 = {r: bf16_to_f64(a) for r, a in h_in(t).items()}
        n = {r: x0[r].shape[1] for r in ROLES}
        pos = {"text": np.arange(n["text"]), "ref": n["text"] + np.arange(n["ref"]),
               "tgt": n["text"] + n["ref"] + np.arange(n["tgt"])}
        hcur = {"text": x0["text"].copy(), "tgt": x0["tgt"].copy()}
        for s in range(B):
            hbar[0][s] = x0["ref"][s]
        step_rec = []
        for b in range(n_blocks):
            mb = mods(t, b)
            Wb = weights(b)
            Wf = {st: {k: (bf16_to_f64(v) if k.startswith("w_") else np.asarray(v, np.float64))
                       for k, v in Wb[st].items()} for st in ("text", "image")}
            md = {st: {k: np.asarray(v, np.float64) for k, v in mb[st].items()} for st in ("text", "image")}
            qkv = {}
            for r in ("text", "tgt"):
                st = STREAM_OF[r]
                qkv[r] = [qkv_project(hcur[r][s], {k: v[s] for k, v in md[st].items()}, Wf[st], pos[r], H, d,
                                      ln_eps, rope_base) for s in range(B)]
            q_tgt = np.stack([qkv["tgt"][s][0] for s in range(B)])
            D = q_change(q_tgt, prev_q[b], eps) if (t >= 1 and prev_q[b] is not None) else None
            modes, gbars = gate.decide(t, b, D, prev_M[b], tie=tie, tie_band=tie_band)
            M = np.zeros((B, H))
            for s in range(B):
                mode = modes[s]
                mi = {k: v[s] for k, v in md["image"].items()}
                q_ref = None
                if mode != REUSE:
                    q_ref, k_ref, v_ref = qkv_project(hbar[b][s], mi, Wf["image"], pos["ref"], H, d, ln_eps,
                                                      rope_base)
                    if mode in (COMPUTE, FULL):
                        cache[b][s] = (k_ref, v_ref)
                        a_b[b][s] = t
                kc, vc = cache[b][s]
                qd = {"text": qkv["text"][s][0], "ref": q_ref, "tgt": qkv["tgt"][s][0]}
                kd = {"text": qkv["text"][s][1], "ref": kc, "tgt": qkv["tgt"][s][1]}
                vd = {"text": qkv["text"][s][2], "ref": vc, "tgt": qkv["tgt"][s][2]}
                res = block_attention(qd, kd, vd, mode, sc, None, mass_rows, None, True, nthreads)
                M[s] = res["M"]
                for r in ("text", "tgt"):
                    st = STREAM_OF[r]
                    hcur[r][s] = post_attention(hcur[r][s], round_bf16(res["O"][r]),
                                                {k: v[s] for k, v in md[st].items()}, Wf[st], ln_eps)
                if mode != REUSE:
                    hbar[b + 1][s] = post_attention(hbar[b][s], round_bf16(res["O"]["ref"]), mi, Wf["image"],
                                                    ln_eps)
            step_rec.append({"mode": modes, "gbar": gbars, "D": None if D is None else np.asarray(D),
                             "M": M, "a_b": list(a_b[b])})
            prev_q[b] = q_tgt
            prev_M[b] = M
        records.append(step_rec)
        outputs.append({"text": hcur["text"].copy(), "tgt": hcur["tgt"].copy(),
                        "hbar": [[None if x is None else np.array(x) for x in row] for row in hbar]})
    return records, outputs


def dit_block_flops(n_rows, C, mlp_ratio=4):
    """GEMM FLOPs of one block's linear layers over n_rows rows: QKV (3C),
    output projection (C), MLP (mlp_ratio C, twice)."""
    return 2 * n_rows * C * (3 * C + C + 2 * mlp_ratio * C)
