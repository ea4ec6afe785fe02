"""Pins for the DiT-block oracle (oracle/dit.py): closed forms, library special
cases, invariants and the cache semantics of Algorithm 1 (no GPU)."""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import BOUNDARY, COMPUTE, FULL, REUSE
from oracle import dit


def _bits(t):
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


# --------------------------------------------------------------------------- bf16 rounding
def test_round_bf16_ties_and_known_values():
    one = 1.0
    cases = [(one + 2.0 ** -8, one),                      # tie, even neighbour 1.0
             (one + 3 * 2.0 ** -8, one + 2.0 ** -6),      # tie, even neighbour 1 + 2^-6
             (one + 2.0 ** -8 + 2.0 ** -30, one + 2.0 ** -7),
             (-(one + 2.0 ** -8), -one),
             (3.14159265, 3.140625), (0.0, 0.0), (2.0 ** -100, 2.0 ** -100)]
    for x, want in cases:
        assert dit.round_bf16(np.array([x]))[0] == want, (x, want)


def test_round_bf16_matches_torch_on_fp32_values():
    # For inputs exactly representable in fp32, torch's fp32 -> bf16 rounding
    # (nearest, ties to even) is the same operation.
    x = (torch.randn(1 << 16, dtype=torch.float32) * 10.0)
    x = torch.cat([x, torch.tensor([1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5 - 2 ** -7], dtype=torch.float32)])
    want = x.to(torch.bfloat16).to(torch.float64).numpy()
    got = dit.round_bf16(x.to(torch.float64).numpy())
    np.testing.assert_array_equal(got, want)


# --------------------------------------------------------------------------- layers
def test_linear_matches_loops():
    rng = np.random.default_rng(1)
    x, W, b = rng.standard_normal((3, 5)), rng.standard_normal((4, 5)), rng.standard_normal(4)
    y = dit.linear(x, W, b)
    for i in range(3):
        for j in range(4):
            assert abs(y[i, j] - (sum(x[i, k] * W[j, k] for k in range(5)) + b[j])) < 1e-12


def test_layer_norm_modulate_closed_forms():
    rng = np.random.default_rng(2)
    h = rng.standard_normal((7, 64)) * 3.0 + 1.5
    z = dit.layer_norm_modulate(h, np.zeros(64), np.zeros(64), eps=0.0)
    np.testing.assert_allclose(z.mean(-1), 0.0, atol=1e-12)
    np.testing.assert_allclose((z ** 2).mean(-1), 1.0, rtol=1e-12)
    # two elements [a, b]: (+-)(b - a)/2 / sqrt(((b - a)/2)^2 + eps)
    a, bb, eps = 0.3, 1.7, 0.01
    half = (bb - a) / 2
    z2 = dit.layer_norm_modulate(np.array([[a, bb]]), np.array([0.5, -0.5]), np.array([1.0, 0.0]), eps)
    r = half / math.sqrt(half * half + eps)
    np.testing.assert_allclose(z2[0], [-r * 2.0 + 0.5, r - 0.5], rtol=1e-14)


def test_rms_norm_constant_vector():
    w = np.linspace(0.5, 1.5, 8)
    x = np.full((1, 8), -2.0)
    np.testing.assert_allclose(dit.rms_norm(x, w, eps=0.0)[0], -w, rtol=1e-15)
    np.testing.assert_allclose(dit.rms_norm(x, w, eps=1.0)[0], -2.0 / math.sqrt(5.0) * w, rtol=1e-15)


def test_rope_rotation_properties():
    rng = np.random.default_rng(3)
    d = 16
    x = rng.standard_normal((5, d))
    # position 0 is the identity
    np.testing.assert_array_equal(dit.apply_rope(x, np.zeros(5)), x)
    # each pair keeps its norm
    pos = rng.integers(0, 10000, size=5)
    y = dit.apply_rope(x, pos)
    np.testing.assert_allclose(y[:, 0::2] ** 2 + y[:, 1::2] ** 2, x[:, 0::2] ** 2 + x[:, 1::2] ** 2, rtol=1e-12)
    # the first pair turns by exactly pos radians, counter-clockwise
    e = np.zeros((1, d))
    e[0, 0] = 1.0
    r = dit.apply_rope(e, np.array([0.7]))
    assert abs(r[0, 0] - math.cos(0.7)) < 1e-15 and abs(r[0, 1] - math.sin(0.7)) < 1e-15
    # the last pair turns by pos * base^(-(d-2)/d)
    e = np.zeros((1, d))
    e[0, d - 2] = 1.0
    r = dit.apply_rope(e, np.array([3.0]))
    ang = 3.0 * 10000.0 ** (-(d - 2) / d)
    assert abs(r[0, d - 2] - math.cos(ang)) < 1e-14 and abs(r[0, d - 1] - math.sin(ang)) < 1e-14


def test_rope_scores_depend_on_relative_position_only():
    rng = np.random.default_rng(4)
    d = 32
    q, k = rng.standard_normal((1, d)), rng.standard_normal((1, d))
    s = []
    for shift in (0, 17, 1234):
        rq = dit.apply_rope(q, np.array([40 + shift]))
        rk = dit.apply_rope(k, np.array([11 + shift]))
        s.append(float((rq @ rk.T)[0, 0]))
    np.testing.assert_allclose(s, s[0], rtol=1e-9)
    rk2 = dit.apply_rope(k, np.array([12]))
    assert abs(float((dit.apply_rope(q, np.array([40])) @ rk2.T)[0, 0]) - s[0]) > 1e-6


def test_gelu_tanh_against_exact_gelu():
    from scipy.special import ndtr
    x = np.linspace(-6, 6, 2001)
    g = dit.gelu_tanh(x)
    assert np.max(np.abs(g - x * ndtr(x))) < 1e-3      # the tanh form's approximation error
    np.testing.assert_allclose(g - dit.gelu_tanh(-x), x, atol=1e-12)   # odd part is x / 2 each side
    assert dit.gelu_tanh(np.array([0.0]))[0] == 0.0


# --------------------------------------------------------------------------- block and stack
def _tiny(B=1, H=2, d=16, n_text=5, n_ref=12, n_tgt=9, n_blocks=3, n_steps=3, tgt_drift=0.2, mod_drift=0.05,
          seed=0):
    from paper_2609_32415_gb300 import synth
    wl = synth.custom_workload(B, H, d, n_text, n_ref, n_tgt, n_blocks=n_blocks, n_steps=n_steps, seed=seed)
    di = synth.DiTInputs(wl, tgt_drift=tgt_drift, mod_drift=mod_drift)

    def h_in(t):
        return {r: _bits(x) for r, x in di.h_in(t).items()}

    def mods(t, b):
        return {st: {k: v.numpy() for k, v in m.items()} for st, m in di.mods(t, b).items()}

    def weights(b):
        return {st: {k: (_bits(v) if k.startswith("w_") else v.numpy()) for k, v in w.items()}
                for st, w in di.weights(b).items()}

    return wl, h_in, mods, weights


def test_zero_gates_leave_the_rows_unchanged():
    wl, h_in, mods, weights = _tiny(n_blocks=2, n_steps=1)

    def zmods(t, b):
        m = mods(t, b)
        for st in m:
            m[st]["gate_a"] = np.zeros_like(m[st]["gate_a"])
            m[st]["gate_m"] = np.zeros_like(m[st]["gate_m"])
        return m

    rec, out = dit.dit_closed_loop(h_in, zmods, weights, 1, 2, wl.B, wl.H, wl.d, theta=0.1, delta_max=4)
    x0 = {r: oracle.bf16_to_f64(a) for r, a in h_in(0).items()}
    np.testing.assert_array_equal(out[0]["tgt"], x0["tgt"])
    np.testing.assert_array_equal(out[0]["text"], x0["text"])
    np.testing.assert_array_equal(out[0]["hbar"][2][0], x0["ref"][0])


def test_stack_without_drift_repeats_itself_under_any_schedule():
    """No target or timestep drift: D = 0, every later block reuses, and the
    cached K/V are what would be recomputed, so every step's outputs equal
    step 0's exactly (Eqs. 8-9 with a = t); a forced boundary at block 1 (the
    cached hidden state restored) gives the same outputs again."""
    wl, h_in, mods, weights = _tiny(n_steps=3, tgt_drift=0.0, mod_drift=0.0)
    rec, out = dit.dit_closed_loop(h_in, mods, weights, 3, 3, wl.B, wl.H, wl.d, theta=1e-9, delta_max=10)
    for t in (1, 2):
        assert [r["mode"][0] for r in rec[t]] == [REUSE] * 3
        assert np.all(rec[t][0]["D"] == 0.0)
        np.testing.assert_array_equal(out[t]["tgt"], out[0]["tgt"])
        np.testing.assert_array_equal(out[t]["text"], out[0]["text"])
    rec2, out2 = dit.dit_closed_loop(h_in, mods, weights, 3, 3, wl.B, wl.H, wl.d, theta=float("inf"),
                                     delta_max=10, forced_boundary=1)
    assert [r["mode"][0] for r in rec2[1]] == [REUSE, BOUNDARY, COMPUTE]
    for t in (1, 2):
        np.testing.assert_array_equal(out2[t]["tgt"], out[0]["tgt"])
        for b in range(4):
            np.testing.assert_array_equal(out2[t]["hbar"][b][0], out[0]["hbar"][b][0])


def test_reuse_changes_target_rows_only_through_stale_reference():
    """With target drift, a REUSE step differs from the always-refresh run;
    with delta_max = 1 (always refresh) every step is FULL and the reference
    hidden states are recomputed each step."""
    wl, h_in, mods, weights = _tiny(n_steps=2)
    rec_f, out_f = dit.dit_closed_loop(h_in, mods, weights, 2, 3, wl.B, wl.H, wl.d, theta=0.1, delta_max=1)
    assert all(r["mode"][0] == FULL for step in rec_f for r in step)
    rec_r, out_r = dit.dit_closed_loop(h_in, mods, weights, 2, 3, wl.B, wl.H, wl.d, theta=1e9, delta_max=10)
    assert [r["mode"][0] for r in rec_r[1]] == [REUSE] * 3
    # step 0 identical; step 1 target outputs differ (stale reference), but stay close
    np.testing.assert_array_equal(out_r[0]["tgt"], out_f[0]["tgt"])
    diff = np.abs(out_r[1]["tgt"] - out_f[1]["tgt"])
    assert diff.max() > 0.0
    assert np.linalg.norm(out_r[1]["tgt"] - out_f[1]["tgt"]) < 0.2 * np.linalg.norm(out_f[1]["tgt"])
    # REUSE leaves the cached reference hidden states of step 0 in place
    for b in range(1, 4):
        np.testing.assert_array_equal(out_r[1]["hbar"][b][0], out_r[0]["hbar"][b][0])


def test_block_matches_a_row_by_row_restatement():
    """One FULL block for one sample, checked against a restatement that
    forms every row separately with explicit per-head loops (only the
    attention and the library matmul are shared)."""
    wl, h_in, mods, weights = _tiny(n_blocks=1, n_steps=1, H=2, d=8, n_text=3, n_ref=4, n_tgt=5)
    rec, out = dit.dit_closed_loop(h_in, mods, weights, 1, 1, wl.B, wl.H, wl.d, theta=0.1, delta_max=4)
    H, d = wl.H, wl.d
    C = H * d
    x = {r: oracle.bf16_to_f64(a)[0] for r, a in h_in(0).items()}
    m = mods(0, 0)
    w = weights(0)
    rows = [("text", i) for i in range(3)] + [("ref", i) for i in range(4)] + [("tgt", i) for i in range(5)]
    Q, K, V = [], [], []
    for p, (r, i) in enumerate(rows):
        st = "text" if r == "text" else "image"
        W = {k: (oracle.bf16_to_f64(v) if k.startswith("w_") else v.astype(np.float64)) for k, v in w[st].items()}
        h = x[r][i]
        mu = sum(h) / C
        var = sum((hh - mu) ** 2 for hh in h) / C
        xn = dit.round_bf16(np.array([(hh - mu) / math.sqrt(var + 1e-6) * (1 + m[st]["scale_a"][0][c])
                                      + m[st]["shift_a"][0][c] for c, hh in enumerate(h)]))
        y = W["w_qkv"] @ xn + W["b_qkv"]
        qh, kh, vh = [], [], []
        for hd in range(H):
            for part, dst, nw in ((0, qh, W["q_norm"]), (1, kh, W["k_norm"]), (2, vh, None)):
                seg = y[part * C + hd * d: part * C + (hd + 1) * d]
                if nw is not None:
                    seg = seg / math.sqrt(sum(s * s for s in seg) / d + 1e-6) * nw
                    rot = np.empty(d)
                    for i2 in range(d // 2):
                        a = p * 10000.0 ** (-2.0 * i2 / d)
                        rot[2 * i2] = seg[2 * i2] * math.cos(a) - seg[2 * i2 + 1] * math.sin(a)
                        rot[2 * i2 + 1] = seg[2 * i2] * math.sin(a) + seg[2 * i2 + 1] * math.cos(a)
                    seg = rot
                dst.append(dit.round_bf16(seg))
        Q.append(qh), K.append(kh), V.append(vh)
    Qa = np.array(Q).transpose(1, 0, 2)
    Ka = np.array(K).transpose(1, 0, 2)
    Va = np.array(V).transpose(1, 0, 2)
    o, _ = oracle.joint_attention(Qa, Ka, Va, 1.0 / math.sqrt(d), ref_range=(3, 7))
    o = dit.round_bf16(o)
    for p, (r, i) in enumerate(rows):
        st = "text" if r == "text" else "image"
        W = {k: (oracle.bf16_to_f64(v) if k.startswith("w_") else v.astype(np.float64)) for k, v in w[st].items()}
        of = o[:, p, :].reshape(C)
        h1 = dit.round_bf16(x[r][i] + m[st]["gate_a"][0] * (W["w_o"] @ of + W["b_o"]))
        mu = h1.mean()
        var = ((h1 - mu) ** 2).mean()
        x2 = dit.round_bf16((h1 - mu) / math.sqrt(var + 1e-6) * (1 + m[st]["scale_m"][0]) + m[st]["shift_m"][0])
        z = W["w_1"] @ x2 + W["b_1"]
        u = dit.round_bf16(np.array([0.5 * zz * (1 + math.tanh(math.sqrt(2 / math.pi) * (zz + 0.044715 * zz ** 3)))
                                     for zz in z]))
        h2 = dit.round_bf16(h1 + m[st]["gate_m"][0] * (W["w_2"] @ u + W["b_2"]))
        want = out[0]["text"][0][i] if r == "text" else (out[0]["tgt"][0][i] if r == "tgt" else
                                                          out[0]["hbar"][1][0][i])
        # the two differ only in rounding order: a bf16 step at most, rarely
        assert np.all(np.abs(h2 - want) <= 1e-12 + 2.0 ** -7 * np.abs(want)), (r, i)
        assert np.mean(h2 == want) > 0.98, (r, i)


def test_dit_block_flops():
    assert dit.dit_block_flops(1, 1) == 2 * 12
    assert dit.dit_block_flops(12544, 3072) == 2 * 12544 * 3072 * 3072 * 12


def test_boundary_block_keeps_cached_reference_kv():
    """Algorithm 1 at the boundary: the target still attends to the block's
    cached reference K/V (materialised at step 0), and the reference query is
    formed from the restored hidden state with this step's modulation. The
    recorded exposure M of the boundary block equals one assembled by hand
    that way, and differs from the one with freshly formed reference K/V."""
    wl, h_in, mods, weights = _tiny(n_steps=2, n_blocks=3)
    H, d = wl.H, wl.d
    rec, out = dit.dit_closed_loop(h_in, mods, weights, 2, 3, wl.B, wl.H, wl.d, theta=float("inf"),
                                   delta_max=10, forced_boundary=1)
    assert [r["mode"][0] for r in rec[1]] == [REUSE, BOUNDARY, COMPUTE]
    # block 0's outputs at step 1 (it reused): the same stack cut after block 0
    _, out0 = dit.dit_closed_loop(h_in, mods, weights, 2, 1, wl.B, wl.H, wl.d, theta=float("inf"),
                                  delta_max=10, forced_boundary=1)
    n = {"text": wl.n_text, "ref": wl.n_ref, "tgt": wl.n_tgt}
    pos = {"text": np.arange(n["text"]), "ref": n["text"] + np.arange(n["ref"]),
           "tgt": n["text"] + n["ref"] + np.arange(n["tgt"])}
    W = {st: {k: (oracle.bf16_to_f64(v) if k.startswith("w_") else v.astype(np.float64))
              for k, v in w.items()} for st, w in weights(1).items()}
    m0 = {st: {k: v[0] for k, v in mm.items()} for st, mm in mods(0, 1).items()}
    m1 = {st: {k: v[0] for k, v in mm.items()} for st, mm in mods(1, 1).items()}
    hbar1 = out[0]["hbar"][1][0]
    np.testing.assert_array_equal(out[1]["hbar"][1][0], hbar1)          # block 0 reused: not rewritten
    _, k_c, v_c = dit.qkv_project(hbar1, m0["image"], W["image"], pos["ref"], H, d)
    q_r, k_f, v_f = dit.qkv_project(hbar1, m1["image"], W["image"], pos["ref"], H, d)
    qt, kt, vt = dit.qkv_project(out0[1]["text"][0], m1["text"], W["text"], pos["text"], H, d)
    qy, ky, vy = dit.qkv_project(out0[1]["tgt"][0], m1["image"], W["image"], pos["tgt"], H, d)
    sc = 1.0 / math.sqrt(d)
    cached = oracle.block_attention({"text": qt, "ref": q_r, "tgt": qy}, {"text": kt, "ref": k_c, "tgt": ky},
                                    {"text": vt, "ref": v_c, "tgt": vy}, BOUNDARY, sc)
    fresh = oracle.block_attention({"text": qt, "ref": q_r, "tgt": qy}, {"text": kt, "ref": k_f, "tgt": ky},
                                   {"text": vt, "ref": v_f, "tgt": vy}, BOUNDARY, sc)
    np.testing.assert_array_equal(rec[1][1]["M"][0], cached["M"])
    assert np.abs(fresh["M"] - cached["M"]).max() > 1e-6
