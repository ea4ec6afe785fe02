"""Pins for the CPU oracle: brute force, closed forms, library special cases and
invariants fixed by the paper and by the mathematics (no GPU)."""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import BOUNDARY, COMPUTE, FULL, REUSE

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _rand(rng, *shape, scale=1.0):
    return rng.standard_normal(shape) * scale


# --------------------------------------------------------------------------- bf16
def test_bf16_widening_known_patterns():
    bits = np.array([0x0000, 0x3F80, 0xC000, 0x3F81, 0x7F80, 0xFF80, 0x0001, 0x4049],
                    dtype=np.uint16)
    got = oracle.bf16_to_f64(bits)
    exp = [0.0, 1.0, -2.0, 1.0 + 2.0 ** -7, math.inf, -math.inf, 2.0 ** -133, 3.140625]
    for g, e in zip(got.tolist(), exp):
        assert g == e


def test_bf16_widening_matches_torch():
    x = torch.randn(4096, dtype=torch.float32).mul_(7.0).to(torch.bfloat16)
    bits = x.view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(oracle.bf16_to_f64(bits), x.to(torch.float64).numpy())


# --------------------------------------------------------------------------- attention
def _brute_attention(q, k, v, scale, bias, row_biased, r0, r1):
    """Explicit score matrix, then row softmax, by Python loops."""
    H, nq, d = len(q), len(q[0]), len(q[0][0])
    nk = len(k[0])
    o = [[[0.0] * d for _ in range(nq)] for _ in range(H)]
    mass = [[0.0] * nq for _ in range(H)]
    for h in range(H):
        for i in range(nq):
            s = []
            for j in range(nk):
                x = scale * sum(q[h][i][c] * k[h][j][c] for c in range(d))
                if bias is not None and row_biased[i] and r0 <= j < r1:
                    x += bias[h]
                s.append(x)
            mx = max(s)
            e = [math.exp(x - mx) for x in s]
            z = sum(e)
            p = [x / z for x in e]
            for j in range(nk):
                for c in range(d):
                    o[h][i][c] += p[j] * v[h][j][c]
            mass[h][i] = sum(p[r0:r1])
    return np.array(o), np.array(mass)


@pytest.mark.parametrize("with_bias", [False, True])
def test_attention_brute_force_tiny(with_bias):
    rng = np.random.default_rng(1)
    H, nq, nk, d = 2, 5, 7, 4
    q, k, v = _rand(rng, H, nq, d), _rand(rng, H, nk, d), _rand(rng, H, nk, d)
    bias = np.array([0.7, -1.3]) if with_bias else None
    rb = np.array([0, 1, 1, 0, 1], dtype=np.uint8)
    o, m = oracle.joint_attention(q, k, v, 0.37, bias, rb, (2, 5))
    ob, mb = _brute_attention(q.tolist(), k.tolist(), v.tolist(), 0.37,
                              None if bias is None else bias.tolist(), rb.tolist(), 2, 5)
    np.testing.assert_allclose(o, ob, rtol=0, atol=1e-13)
    np.testing.assert_allclose(m, mb, rtol=0, atol=1e-13)


def test_attention_matches_library_softmax():
    """Special case: torch's fp64 softmax(QK^T * scale) V on the CPU."""
    rng = np.random.default_rng(2)
    H, nq, nk, d = 3, 40, 57, 16
    q, k, v = _rand(rng, H, nq, d), _rand(rng, H, nk, d), _rand(rng, H, nk, d)
    scale = 1.0 / math.sqrt(d)
    o, m = oracle.joint_attention(q, k, v, scale, ref_range=(10, 30), nthreads=3)
    tq, tk, tv = (torch.from_numpy(x) for x in (q, k, v))
    p = torch.softmax(tq @ tk.transpose(1, 2) * scale, dim=-1)
    np.testing.assert_allclose(o, (p @ tv).numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(m, p[:, :, 10:30].sum(-1).numpy(), rtol=0, atol=1e-12)


def test_attention_thread_count_invariant():
    rng = np.random.default_rng(3)
    q, k, v = _rand(rng, 2, 33, 8), _rand(rng, 2, 50, 8), _rand(rng, 2, 50, 8)
    o1, m1 = oracle.joint_attention(q, k, v, 0.3, ref_range=(5, 20), nthreads=1)
    o7, m7 = oracle.joint_attention(q, k, v, 0.3, ref_range=(5, 20), nthreads=7)
    np.testing.assert_array_equal(o1, o7)
    np.testing.assert_array_equal(m1, m7)


def test_rows_sum_to_one():
    """With V = 1 every output element equals the row sum of the probabilities."""
    rng = np.random.default_rng(4)
    q, k = _rand(rng, 2, 20, 8, scale=3.0), _rand(rng, 2, 31, 8, scale=3.0)
    o, m = oracle.joint_attention(q, k, np.ones((2, 31, 8)), 1.0, ref_range=(0, 31))
    np.testing.assert_allclose(o, 1.0, rtol=0, atol=1e-13)
    np.testing.assert_allclose(m, 1.0, rtol=0, atol=1e-13)


def test_equal_logits_give_mean_value_and_share_mass():
    rng = np.random.default_rng(5)
    nk, r0, r1 = 37, 4, 19
    v = _rand(rng, 2, nk, 6)
    o, m = oracle.joint_attention(np.zeros((2, 9, 6)), _rand(rng, 2, nk, 6), v, 0.5,
                                  ref_range=(r0, r1))
    np.testing.assert_allclose(o, np.broadcast_to(v.mean(axis=1, keepdims=True), o.shape),
                               rtol=0, atol=1e-13)
    np.testing.assert_allclose(m, (r1 - r0) / nk, rtol=0, atol=1e-14)


def test_single_key_returns_its_value():
    rng = np.random.default_rng(6)
    v = _rand(rng, 2, 1, 5)
    o, m = oracle.joint_attention(_rand(rng, 2, 4, 5), _rand(rng, 2, 1, 5), v, 1.0,
                                  ref_range=(0, 1))
    np.testing.assert_allclose(o, np.broadcast_to(v, o.shape), rtol=0, atol=1e-15)
    np.testing.assert_allclose(m, 1.0, rtol=0, atol=1e-15)


def test_bias_closed_form_mass():
    """Equal logits plus bias beta on n_ref keys: M = n_ref e^b / (n_ref e^b + n_other)."""
    n_other, n_ref = 50, 30
    beta = np.array([-3.0, -0.5, 0.0, 1.25])
    H = len(beta)
    rng = np.random.default_rng(7)
    k = _rand(rng, H, n_other + n_ref, 4)
    q = np.zeros((H, 3, 4))
    rb = np.array([1, 0, 1], dtype=np.uint8)
    _, m = oracle.joint_attention(q, k, _rand(rng, H, n_other + n_ref, 4), 1.0, beta, rb,
                                  (10, 10 + n_ref))
    want = n_ref * np.exp(beta) / (n_ref * np.exp(beta) + n_other)
    np.testing.assert_allclose(m[:, 0], want, rtol=0, atol=1e-14)
    np.testing.assert_allclose(m[:, 2], want, rtol=0, atol=1e-14)
    np.testing.assert_allclose(m[:, 1], n_ref / (n_ref + n_other), rtol=0, atol=1e-14)


def test_no_reference_keys_gives_zero_mass():
    rng = np.random.default_rng(8)
    _, m = oracle.joint_attention(_rand(rng, 1, 6, 4), _rand(rng, 1, 9, 4),
                                  _rand(rng, 1, 9, 4), 1.0, ref_range=(3, 3))
    assert np.all(m == 0.0)


def test_reference_and_complement_mass_partition():
    """Ref mass + mass on every other key = 1 per row (the partition behind Tab. 1)."""
    rng = np.random.default_rng(9)
    q, k, v = _rand(rng, 2, 11, 8, scale=2), _rand(rng, 2, 40, 8, scale=2), _rand(rng, 2, 40, 8)
    _, m_ref = oracle.joint_attention(q, k, v, 1.0, ref_range=(12, 30))
    _, m_a = oracle.joint_attention(q, k, v, 1.0, ref_range=(0, 12))
    _, m_b = oracle.joint_attention(q, k, v, 1.0, ref_range=(30, 40))
    np.testing.assert_allclose(m_ref + m_a + m_b, 1.0, rtol=0, atol=1e-13)


def test_paper_table1_partition_fixture():
    """Tab. 1 prints Ref mass, Tgt mass and their ratio; the partition must close."""
    with open(os.path.join(GOLDEN, "paper_table1.json")) as f:
        rows = json.load(f)["rows"]
    for r in rows:
        assert abs(r["ref_mass_pct"] + r["tgt_mass_pct"] - 100.0) < 0.011
        assert abs(r["tgt_mass_pct"] / r["ref_mass_pct"] - r["tgt_over_ref"]) < 0.006
        ex = oracle.exposure(np.array([[r["ref_mass_pct"] / 100.0]]))
        assert abs(ex[0] * 100.0 - r["ref_mass_pct"]) < 1e-12


# --------------------------------------------------------------------------- drift D
def test_q_change_closed_forms():
    rng = np.random.default_rng(10)
    q = _rand(rng, 2, 3, 17, 8)
    assert np.all(oracle.q_change(q, q) == 0.0)
    for c in (-0.7, 0.05, 0.3, 2.0):
        eps = 1e-6
        nrm = np.sqrt((q ** 2).sum(axis=(-2, -1)))
        got = oracle.q_change((1.0 + c) * q, q, eps)
        np.testing.assert_allclose(got, abs(c) * nrm / (nrm + eps), rtol=1e-13, atol=0)


def test_q_change_brute_force():
    rng = np.random.default_rng(11)
    a, b = _rand(rng, 3, 4), _rand(rng, 3, 4)
    num = math.sqrt(sum((a[i, j] - b[i, j]) ** 2 for i in range(3) for j in range(4)))
    den = math.sqrt(sum(b[i, j] ** 2 for i in range(3) for j in range(4))) + 0.125
    assert abs(oracle.q_change(a, b, 0.125) - num / den) < 1e-14


def test_exposure_mean_over_rows():
    m_tgt = np.array([[0.1, 0.3, 0.2], [0.5, 0.5, 0.5]])
    m_text = np.array([[0.9], [0.0]])
    np.testing.assert_allclose(oracle.exposure(m_tgt), [0.2, 0.5], atol=1e-15)
    np.testing.assert_allclose(oracle.exposure(m_tgt, m_text), [1.5 / 4, 1.5 / 4], atol=1e-15)


# --------------------------------------------------------------------------- accounting
def test_compute_accounting():
    """App. A.4: 2 n_q n_k d MACs for scores and values per head, and the cached-step
    score fraction N_Y (N_R + N_Y) / (N_R + N_Y)^2, checked against entry counts."""
    assert oracle.attention_flops(3, 5, 2, 4) == 4 * 4 * 2 * 3 * 5
    for n_ref, n_y in ((8192, 4352), (16380, 16892), (16384, 4352), (0, 10)):
        n = n_ref + n_y
        full_entries = n * n
        cached_entries = n_y * n
        assert oracle.reuse_score_fraction(n_ref, n_y) == pytest.approx(
            cached_entries / full_entries, rel=1e-15)


# --------------------------------------------------------------------------- gate
def _run_gate(gbar_rows, theta, delta_max, forced=-1):
    """gbar_rows[t][b] -> modes[t][b] with D = gbar (one head), M = 1."""
    g = oracle.Gate(1, theta, delta_max, forced)
    out = []
    for t, row in enumerate(gbar_rows):
        g.begin_step(t)
        modes = []
        for b, x in enumerate(row):
            m, _ = g.decide(t, b, [[x]], [[1.0]])
            modes.append(m[0])
        out.append(modes)
    return out


def test_gate_first_crossing_table():
    rows = [[0.0] * 5, [0.01, 0.02, 0.06, 0.01, 0.09], [0.05, 0.0, 0.0, 0.0, 0.0],
            [0.01, 0.01, 0.01, 0.01, 0.01]]
    got = _run_gate(rows, 0.05, 100)
    R, Bd, C, F = REUSE, BOUNDARY, COMPUTE, FULL
    assert got == [[F] * 5, [R, R, Bd, C, C], [Bd, C, C, C, C], [R] * 5]


def test_gate_head_mean_of_products():
    """Eq. 12 forms D*M per head before the mean: mean(D)*mean(M) would differ."""
    g = oracle.Gate(1, 0.25, 100)
    g.begin_step(1)
    D = [[1.0, 0.0]]
    M = [[0.5, 1.0]]
    modes, gbar = g.decide(1, 0, D, M)
    assert gbar[0] == pytest.approx(0.25)     # (1*0.5 + 0*1)/2
    assert modes[0] == BOUNDARY
    g.begin_step(2)
    modes, gbar = g.decide(2, 0, [[0.0, 1.0]], [[1.0, 0.49]])
    assert gbar[0] == pytest.approx(0.245) and modes[0] == REUSE


def test_gate_bounded_age_refresh():
    rows = [[0.0] * 3] * 8
    got = _run_gate(rows, 1.0, 3)
    for t in range(8):
        if t in (0, 3, 6):
            assert got[t] == [FULL] * 3
        else:
            assert got[t] == [REUSE] * 3


def test_gate_always_refresh_and_degenerate_thresholds():
    rng = np.random.default_rng(12)
    rows = rng.uniform(0, 1, size=(6, 7)).tolist()
    assert all(m == [FULL] * 7 for m in _run_gate(rows, 0.5, 1))
    inf = _run_gate(rows, math.inf, 10 ** 6)
    assert inf[0] == [FULL] * 7 and all(m == [REUSE] * 7 for m in inf[1:])
    zero = _run_gate(rows, 0.0, 10 ** 6)
    assert all(m == [BOUNDARY] + [COMPUTE] * 6 for m in zero[1:])


def test_gate_monotone_suffix_invariant():
    rng = np.random.default_rng(13)
    for _ in range(50):
        rows = rng.uniform(0, 0.2, size=(5, 9)).tolist()
        for modes in _run_gate(rows, 0.15, 10 ** 6)[1:]:
            nb = modes.count(BOUNDARY)
            assert nb <= 1
            if nb == 0:
                assert modes == [REUSE] * 9
            else:
                k = modes.index(BOUNDARY)
                assert modes[:k] == [REUSE] * k and modes[k + 1:] == [COMPUTE] * (8 - k)


def test_gate_forced_boundary():
    rows = [[0.0] * 6] * 3
    got = _run_gate(rows, math.inf, 100, forced=2)
    assert got[1] == [REUSE, REUSE, BOUNDARY, COMPUTE, COMPUTE, COMPUTE]
    assert _run_gate(rows, math.inf, 100, forced=6)[2] == [REUSE] * 6


def test_gate_tie_adopts_given_decision():
    g = oracle.Gate(1, 0.1, 100)
    g.begin_step(1)
    modes, _ = g.decide(1, 0, [[0.10004]], [[1.0]], tie=lambda t, b, s: False)
    assert modes == [REUSE]


# --------------------------------------------------------------------------- closed loop
def _tiny_inputs(B=2, H=2, d=8, n=(3, 10, 7), steps=4, blocks=3, ref_drift=0.0,
                 tgt_drift=0.3, seed=0):
    rng = np.random.default_rng(seed)
    base = {r: [rng.standard_normal((3, B, H, nn, d)) / math.sqrt(d) for _ in range(blocks)]
            for r, nn in zip(oracle.ROLES, n)}
    traj = {}
    for b in range(blocks):
        cur = {r: base[r][b] for r in oracle.ROLES}
        for t in range(steps):
            if t > 0:
                for r in oracle.ROLES:
                    dl = ref_drift if r == "ref" else tgt_drift
                    cur[r] = cur[r] + dl * rng.standard_normal(cur[r].shape) / math.sqrt(d)
            traj[(t, b)] = {r: tuple(torch.from_numpy(cur[r][z]).to(torch.bfloat16)
                                     .view(torch.int16).numpy().view(np.uint16)
                                     for z in range(3)) for r in oracle.ROLES}
    return traj


def _plain_block(raw, s, scale, bias=None):
    f = {r: [oracle.bf16_to_f64(x)[s] for x in raw[r]] for r in oracle.ROLES}
    keys = np.concatenate([f["text"][1], f["ref"][1], f["tgt"][1]], axis=1)
    vals = np.concatenate([f["text"][2], f["ref"][2], f["tgt"][2]], axis=1)
    qs = np.concatenate([f["text"][0], f["ref"][0], f["tgt"][0]], axis=1)
    return oracle.joint_attention(qs, keys, vals, scale, ref_range=(f["text"][0].shape[1],
                                  f["text"][0].shape[1] + f["ref"][0].shape[1]))


def test_always_refresh_is_plain_joint_attention():
    traj = _tiny_inputs(ref_drift=0.05)
    rec = oracle.closed_loop(lambda t, b: traj[(t, b)], 4, 3, 2, theta=0.0, delta_max=1)
    for t in range(4):
        for b in range(3):
            assert rec[t][b]["mode"] == [FULL, FULL]
            for s in range(2):
                o, _ = _plain_block(traj[(t, b)], s, 1 / math.sqrt(8))
                got = np.concatenate([rec[t][b]["O"][s][r] for r in oracle.ROLES], axis=1)
                np.testing.assert_allclose(got, o, rtol=0, atol=1e-14)


def test_reuse_with_zero_reference_drift_equals_fresh():
    """Eqs. 8-9 with K_R^a = K_R^t: stale-KV output equals the fresh output."""
    traj = _tiny_inputs(ref_drift=0.0)
    fresh = oracle.closed_loop(lambda t, b: traj[(t, b)], 4, 3, 2, theta=0.0, delta_max=1)
    reuse = oracle.closed_loop(lambda t, b: traj[(t, b)], 4, 3, 2, theta=math.inf,
                               delta_max=10 ** 6)
    for t in range(1, 4):
        for b in range(3):
            assert reuse[t][b]["mode"] == [REUSE, REUSE]
            for s in range(2):
                assert reuse[t][b]["O"][s]["ref"] is None
                for r in ("text", "tgt"):
                    np.testing.assert_allclose(reuse[t][b]["O"][s][r], fresh[t][b]["O"][s][r],
                                               rtol=0, atol=1e-14)
                np.testing.assert_allclose(reuse[t][b]["M"], fresh[t][b]["M"], atol=1e-14)


def test_reuse_reads_keys_from_last_materialisation():
    """Eq. 9: a reusing block's target output is Attn with reference K/V of step a_b."""
    traj = _tiny_inputs(ref_drift=0.2, seed=3)
    rec = oracle.closed_loop(lambda t, b: traj[(t, b)], 4, 3, 2, theta=math.inf,
                             delta_max=10 ** 6)
    for t in range(1, 4):
        for b in range(3):
            assert rec[t][b]["a_b"] == [0, 0]
            for s in range(2):
                mixed = {"text": traj[(t, b)]["text"], "tgt": traj[(t, b)]["tgt"],
                         "ref": traj[(0, b)]["ref"]}
                o, m = _plain_block(mixed, s, 1 / math.sqrt(8))
                n_text = 3
                np.testing.assert_allclose(rec[t][b]["O"][s]["tgt"], o[:, n_text + 10:],
                                           rtol=0, atol=1e-14)
                np.testing.assert_allclose(rec[t][b]["M"][s], m[:, n_text + 10:].mean(axis=1),
                                           atol=1e-14)


def test_zero_threshold_puts_boundary_at_block_zero():
    traj = _tiny_inputs(ref_drift=0.1, seed=4)
    rec = oracle.closed_loop(lambda t, b: traj[(t, b)], 4, 3, 2, theta=0.0, delta_max=10 ** 6)
    for t in range(1, 4):
        assert [rec[t][b]["mode"][0] for b in range(3)] == [BOUNDARY, COMPUTE, COMPUTE]
        assert [rec[t][b]["a_b"][0] for b in range(3)] == [0, t, t]


def test_boundary_uses_cached_reference_kv():
    """At the boundary the target still reads block-b cached K/V (Sec. 4)."""
    traj = _tiny_inputs(ref_drift=0.3, seed=5)
    rec = oracle.closed_loop(lambda t, b: traj[(t, b)], 2, 1, 1, theta=0.0, delta_max=100)
    assert rec[1][0]["mode"] == [BOUNDARY]
    mixed = {"text": traj[(1, 0)]["text"], "tgt": traj[(1, 0)]["tgt"], "ref": traj[(0, 0)]["ref"]}
    o, _ = _plain_block(mixed, 0, 1 / math.sqrt(8))
    got = np.concatenate([rec[1][0]["O"][0][r] for r in oracle.ROLES], axis=1)
    np.testing.assert_allclose(got, o, rtol=0, atol=1e-14)


# --------------------------------------------------------------------------- controller ablation cues
def test_gate_cues_change_and_exposure():
    """Sec. 5.3 / Tab. 4: only the trigger changes; D alone or M alone per head."""
    D = [[0.3, 0.1]]
    M = [[0.5, 0.9]]
    for cue, want in (("product", (0.15 + 0.09) / 2), ("change", 0.2), ("exposure", 0.7)):
        g = oracle.Gate(1, 0.19, 100, cue=cue)
        g.begin_step(1)
        modes, gbar = g.decide(1, 0, D, M)
        assert gbar[0] == pytest.approx(want, abs=1e-15)
        assert modes[0] == (BOUNDARY if want >= 0.19 else REUSE)
    with pytest.raises(ValueError):
        oracle.Gate(1, 0.1, 4, cue="bogus")


def test_anchor_cue_measures_change_to_last_materialisation():
    """App. A.2: c^anchor = ||Q_t - Q_{a_b}|| / (||Q_{a_b}|| + eps). With theta = inf
    no block rematerialises after step 0, so the anchor stays at step 0."""
    traj = _tiny_inputs(ref_drift=0.1, tgt_drift=0.2, seed=8)
    rec = oracle.closed_loop(lambda t, b: traj[(t, b)], 4, 3, 2, theta=math.inf, delta_max=10 ** 6,
                             cue="anchor_product")
    for t in range(1, 4):
        for b in range(3):
            q0 = oracle.bf16_to_f64(traj[(0, b)]["tgt"][0])
            qt = oracle.bf16_to_f64(traj[(t, b)]["tgt"][0])
            np.testing.assert_allclose(rec[t][b]["D"], oracle.q_change(qt, q0), rtol=0, atol=1e-15)
    # consecutive-change cue for comparison: D_t is against step t-1
    rec2 = oracle.closed_loop(lambda t, b: traj[(t, b)], 4, 3, 2, theta=math.inf, delta_max=10 ** 6,
                              cue="change")
    q1 = oracle.bf16_to_f64(traj[(1, 0)]["tgt"][0])
    q2 = oracle.bf16_to_f64(traj[(2, 0)]["tgt"][0])
    np.testing.assert_allclose(rec2[2][0]["D"], oracle.q_change(q2, q1), rtol=0, atol=1e-15)


def test_anchor_moves_with_materialisation():
    """theta = 0: block 0 is the boundary every step (its anchor stays at step 0),
    blocks 1, 2 compute every step (their anchor is the previous step)."""
    traj = _tiny_inputs(ref_drift=0.1, tgt_drift=0.2, seed=9)
    rec = oracle.closed_loop(lambda t, b: traj[(t, b)], 4, 3, 2, theta=0.0, delta_max=10 ** 6,
                             cue="anchor_product")
    for t in range(2, 4):
        q = {k: oracle.bf16_to_f64(traj[(k, b)]["tgt"][0]) for k in range(4) for b in [0]}
        np.testing.assert_allclose(rec[t][0]["D"], oracle.q_change(q[t], q[0]), atol=1e-15)
        for b in (1, 2):
            qt = oracle.bf16_to_f64(traj[(t, b)]["tgt"][0])
            qp = oracle.bf16_to_f64(traj[(t - 1, b)]["tgt"][0])
            np.testing.assert_allclose(rec[t][b]["D"], oracle.q_change(qt, qp), atol=1e-15)


# --------------------------------------------------------------------------- staleness diagnostics
def test_diagnostics_vanish_without_reference_drift():
    """Eqs. 7-10: with no reference drift the cache equals the fresh K/V, so the
    endpoint drift and the local impact are zero and both exposures agree."""
    traj = _tiny_inputs(ref_drift=0.0, seed=10)
    rec = oracle.closed_loop(lambda t, b: traj[(t, b)], 3, 2, 2, theta=math.inf, delta_max=100,
                             diagnostics=True)
    for t in range(1, 3):
        for b in range(2):
            r = rec[t][b]
            assert np.all(r["E_K"] == 0) and np.all(r["E_V"] == 0) and np.all(r["E_KV"] == 0)
            np.testing.assert_allclose(r["I_KV"], 0.0, atol=1e-15)
            np.testing.assert_allclose(r["M_fresh"], r["M_cached"], atol=1e-15)


def test_diagnostics_match_their_definitions():
    """Eq. 7 on K and V against the step-0 cache; Eqs. 8-10 written out with
    fresh and anchor keys for every second target row."""
    traj = _tiny_inputs(ref_drift=0.3, seed=11)
    rec = oracle.closed_loop(lambda t, b: traj[(t, b)], 3, 1, 2, theta=math.inf, delta_max=100,
                             diagnostics=True, diag_row_stride=2)
    r = rec[2][0]
    for s in range(2):
        k0 = oracle.bf16_to_f64(traj[(0, 0)]["ref"][1])[s]
        k2 = oracle.bf16_to_f64(traj[(2, 0)]["ref"][1])[s]
        num = np.sqrt(((k2 - k0) ** 2).sum(axis=(1, 2)))
        den = np.sqrt((k0 ** 2).sum(axis=(1, 2))) + 1e-6
        np.testing.assert_allclose(r["E_K"][s], num / den, rtol=1e-13)
        fresh = {"text": traj[(2, 0)]["text"], "tgt": traj[(2, 0)]["tgt"], "ref": traj[(2, 0)]["ref"]}
        stale = {"text": traj[(2, 0)]["text"], "tgt": traj[(2, 0)]["tgt"], "ref": traj[(0, 0)]["ref"]}
        of, _ = _plain_block(fresh, s, 1 / math.sqrt(8))
        os_, _ = _plain_block(stale, s, 1 / math.sqrt(8))
        rows = np.arange(3 + 10, 3 + 10 + 7)[::2]
        a, b_ = os_[:, rows], of[:, rows]
        want = np.sqrt(((a - b_) ** 2).sum(axis=(1, 2))) / (np.sqrt((b_ ** 2).sum(axis=(1, 2))) + 1e-6)
        np.testing.assert_allclose(r["I_KV"][s], want, rtol=1e-12)
        assert np.all(r["I_KV"][s] > 0)


# --------------------------------------------------------------------------- sampled target rows
def test_sampled_rows_mass_is_the_brute_force_mean_over_the_sample():
    """Eq. 4 over the sampled target rows 0, k, 2k, ...: the mean of the
    brute-force row masses of exactly those rows (text rows too when counted)."""
    rng = np.random.default_rng(21)
    H, d = 2, 4
    n = {"text": 4, "ref": 5, "tgt": 7}
    q = {r: _rand(rng, H, n[r], d) for r in oracle.ROLES}
    k = {r: _rand(rng, H, n[r], d) for r in oracle.ROLES}
    v = {r: _rand(rng, H, n[r], d) for r in oracle.ROLES}
    keys = np.concatenate([k["text"], k["ref"], k["tgt"]], axis=1)
    vals = np.concatenate([v["text"], v["ref"], v["tgt"]], axis=1)
    r0, r1 = n["text"], n["text"] + n["ref"]
    for mass_rows in (0, 1):
        for ks in (1, 2, 3):
            res = oracle.block_attention(q, k, v, FULL, 0.5, mass_rows=mass_rows, sample_stride=ks)
            rows = []
            for r in (("tgt", "text") if mass_rows else ("tgt",)):
                _, m = _brute_attention(q[r].tolist(), keys.tolist(), vals.tolist(), 0.5, None, None, r0, r1)
                rows.append(m[:, ::ks])
            want = np.concatenate(rows, axis=1).mean(axis=1)
            np.testing.assert_allclose(res["M"], want, rtol=1e-12)


def test_sampled_rows_change_ignores_unsampled_rows():
    """Eq. 1 over the sampled target rows: doubling exactly the sampled rows
    gives D = 1/(1 + eps/||q_prev||) whatever the other rows do, while the
    every-row D differs."""
    rng = np.random.default_rng(22)
    B, H, d, ks = 1, 2, 8, 3
    n = (3, 6, 10)
    prev = rng.standard_normal((B, H, n[2], d))
    cur = rng.standard_normal((B, H, n[2], d))
    cur[:, :, ::ks] = 2.0 * prev[:, :, ::ks]
    bits = {}
    for t, tq in ((0, prev), (1, cur)):
        raw = {}
        for r, nn in zip(oracle.ROLES, n):
            z = [rng.standard_normal((B, H, nn, d)) for _ in range(3)]
            if r == "tgt":
                z[0] = tq
            raw[r] = tuple(torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
                           for x in z)
        bits[t] = raw
    rec = oracle.closed_loop(lambda t, b: bits[t], 2, 1, B, theta=1e9, delta_max=10, sample_stride=ks)
    qp = oracle.bf16_to_f64(bits[0]["tgt"][0])[:, :, ::ks]
    want = 1.0 / (1.0 + 1e-6 / np.sqrt((qp ** 2).sum(axis=(2, 3))))
    np.testing.assert_allclose(rec[1][0]["D"], want, rtol=1e-12)
    full = oracle.closed_loop(lambda t, b: bits[t], 2, 1, B, theta=1e9, delta_max=10)
    assert np.abs(full[1][0]["D"] - want).max() > 1e-2


def test_head_mean_exposure_eq5():
    """Eq. 5 is the plain mean over the head axis (the last one)."""
    M = np.array([[[0.1, 0.3, 0.2, 0.0]], [[0.5, 0.5, 0.5, 0.5]]])  # [T=2, B=1, H=4]
    got = oracle.head_mean_exposure(M)
    assert got.shape == (2, 1)
    assert got[0, 0] == pytest.approx(0.15) and got[1, 0] == pytest.approx(0.5)
    # one head: the mean is that head's exposure
    assert oracle.head_mean_exposure([[0.37]])[0] == pytest.approx(0.37)


def test_adjacent_ref_mass_change_eq6():
    """Eq. 6 in percentage points: 100/(T-1) times the summed absolute step-to-step
    change. Closed forms: a constant series gives 0, a linear ramp of slope c
    gives 100|c| whatever T, and a zig-zag counts every change with its size."""
    assert oracle.adjacent_ref_mass_change([0.2, 0.2, 0.2, 0.2]) == pytest.approx(0.0)
    for T in (2, 5, 9):
        up = [0.10 + 0.003 * t for t in range(T)]
        assert oracle.adjacent_ref_mass_change(up) == pytest.approx(0.3)
        assert oracle.adjacent_ref_mass_change(up[::-1]) == pytest.approx(0.3)
    # 0.10 -> 0.12 -> 0.11: (0.02 + 0.01) / 2 steps = 1.5 points (dividing by T would give 1.0)
    assert oracle.adjacent_ref_mass_change([0.10, 0.12, 0.11]) == pytest.approx(1.5)
    # per block and sample: the first axis is the step axis
    got = oracle.adjacent_ref_mass_change(np.array([[0.1, 0.4], [0.2, 0.4], [0.1, 0.1]]))
    assert got == pytest.approx([10.0, 15.0])
    with pytest.raises(ValueError):
        oracle.adjacent_ref_mass_change([0.1])
