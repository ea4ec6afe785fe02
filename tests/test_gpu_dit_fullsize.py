"""Parity of one DiT block at the image-edit size (C = 3072, text 256 +
reference 8192 + target 4096 rows, the launch configuration bench.py --dit
times) on outputs the oracle can compute row by row: step 0 (FULL) and step 1
(REUSE), sampled output rows of every role, sampled rows of the K/V cache
slot, D of every head, and the exposure of two target tiles.

The oracle forms K and V of every row in fp64 with the same layer functions
(its per-row cost is what makes the full-size check sampled), then runs the
sampled rows through attention and the rest of the block. Tolerances are those
of the DiT closed-loop test (one block is within the stack bound)."""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import FULL, REUSE
from oracle import dit
from _helpers import M_ABS, bits, f64, o_close

pytestmark = pytest.mark.gpu

D_REL_DIT = 1e-3
ROWS_REL_DIT = 3e-2
ROWS_NORMWISE_DIT = 1e-2


def _np(t):
    return t.double().cpu().numpy()


def _qkv_all(x, md, W, pos, H, d):
    """q, k, v [H, n, d] of rows x with the oracle's layers (dit.qkv_project)."""
    return dit.qkv_project(x, md, W, pos, H, d)


def test_dit_block_image_edit_size(cuda_ok):
    from paper_2609_32415_gb300 import DiTExecutor, synth
    wl = synth.make_workload("c2")
    wl.n_blocks, wl.n_steps = 1, 2
    H, d, C = wl.H, wl.d, wl.H * wl.d
    di = synth.DiTInputs(wl, device="cuda")
    ex = DiTExecutor(1, wl.B, H, d, wl.n_text, wl.n_ref, wl.n_tgt, float("inf"), 10, log_steps=2)
    snaps = {}
    for t in range(2):
        hin = {r: x.clone() for r, x in di.h_in(t).items()}
        ex.step(t, hin, di.mods, di.weights)
        torch.cuda.synchronize()
        snaps[t] = {"in": {r: f64(x[0]) for r, x in hin.items()},
                    "text": f64(ex.h["text"][0]), "tgt": f64(ex.h["tgt"][0]),
                    "hbar1": f64(ex.hbar[1][0]), "k": f64(ex.cache_k[0, 0]), "v": f64(ex.cache_v[0, 0]),
                    "mass": _np(ex.mass[0, 0]), "D": _np(ex.D[0, 0]), "mode": int(ex.modes[t, 0, 0])}
    ex.check()
    assert snaps[0]["mode"] == FULL and snaps[1]["mode"] == REUSE

    Wd = {st: {k: (f64(v) if k.startswith("w_") else _np(v)) for k, v in w.items()}
          for st, w in di.weights(0).items()}
    n = {"text": wl.n_text, "ref": wl.n_ref, "tgt": wl.n_tgt}
    pos = {"text": np.arange(n["text"]), "ref": n["text"] + np.arange(n["ref"]),
           "tgt": n["text"] + n["ref"] + np.arange(n["tgt"])}
    stream = {"text": "text", "ref": "image", "tgt": "image"}
    rng = np.random.default_rng(0)
    sample = {r: np.unique(np.concatenate([np.arange(4), np.arange(n[r] - 4, n[r]),
                                           rng.choice(n[r], size=24, replace=False)])) for r in n}
    sc = 1.0 / math.sqrt(d)
    r0, r1 = n["text"], n["text"] + n["ref"]
    cache = None
    q_tgt_prev = None
    for t in range(2):
        md = {st: {k: _np(v[0]) for k, v in m.items()} for st, m in di.mods(t, 0).items()}
        x = snaps[t]["in"]
        q, k, v = {}, {}, {}
        for r in ("text", "tgt") if t == 1 else ("text", "ref", "tgt"):
            q[r], k[r], v[r] = _qkv_all(x[r], md[stream[r]], Wd[stream[r]], pos[r], H, d)
        if t == 0:
            cache = (k["ref"], v["ref"])
            # the cache slot holds this step's reference K/V (written by the QKV epilogue)
            for z, want in ((snaps[0]["k"], k["ref"]), (snaps[0]["v"], v["ref"])):
                rows = sample["ref"]
                ok, worst, nw = o_close(z[:, rows], want[:, rows], ROWS_REL_DIT)
                assert ok, ("cache", worst, nw)
        else:
            Dw = oracle.q_change(q["tgt"][None], q_tgt_prev[None], 1e-6)[0]
            assert (np.abs(snaps[1]["D"] - Dw) / Dw).max() <= D_REL_DIT
        q_tgt_prev = q["tgt"]
        keys = np.concatenate([k["text"], cache[0], k["tgt"]], axis=1)
        vals = np.concatenate([v["text"], cache[1], v["tgt"]], axis=1)
        roles = ("text", "ref", "tgt") if t == 0 else ("text", "tgt")
        for r in roles:
            rows = sample[r]
            o, _ = oracle.joint_attention(q[r][:, rows], keys, vals, sc, ref_range=(r0, r1))
            h_in = x[r][rows] if r != "ref" else x["ref"][rows]
            want = dit.post_attention(h_in, dit.round_bf16(o), md[stream[r]], Wd[stream[r]])
            got = (snaps[t]["hbar1"] if r == "ref" else snaps[t][r])[rows]
            ok, worst, nw = o_close(got[None], want[None], ROWS_REL_DIT)
            assert ok and nw <= ROWS_NORMWISE_DIT, (t, r, worst, nw)
        # exposure of the first and last target tiles (mass partials of the executed attention)
        base = (n["text"] + 127) // 128
        nt = (n["tgt"] + 127) // 128
        for tile in (0, nt - 1):
            rows = np.arange(tile * 128, min(n["tgt"], tile * 128 + 128))
            _, m = oracle.joint_attention(q["tgt"][:, rows], keys, vals, sc, ref_range=(r0, r1), want_o=False)
            got = snaps[t]["mass"][:, base + tile] / len(rows)
            assert np.abs(got - m.mean(axis=1)).max() <= M_ABS, (t, tile)
