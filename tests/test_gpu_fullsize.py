"""Parity at the workloads' full sizes, through the Executor (the launch
configuration bench.py times), on outputs the oracle can compute one by one:
sampled O rows, sampled mass-partial tiles, every D, and the gate's decisions
recomputed by the oracle's controller from the oracle's D."""
import math

import numpy as np
import pytest
import torch

import oracle
from _helpers import D_REL, M_ABS, TIE_BAND, bits, o_close

pytestmark = pytest.mark.gpu

ROLES = ("text", "ref", "tgt")
HEADS = (0, 7, 23)


def _wide(x):
    return oracle.bf16_to_f64(bits(x))


def _role(X, wl, r, z):
    o = wl.offsets()[r]
    return X[z, :, :, o:o + wl.n[r], :]


def _run_stack(wl, blocks, sample_stride=1):
    """Run the executor over `blocks` (indices into the workload's block
    stack, as a depth-reduced stack) for all steps; returns per (t, b) the
    inputs, outputs, D, modes, gbar and mass partials as seen after the block.
    sample_stride k > 1: D and M over the target rows 0, k, 2k, ..."""
    from paper_2609_32415_gb300 import Executor, roles_from_joint, synth
    sub = synth.Workload(**{**wl.__dict__})
    sub.n_blocks = len(blocks)
    sub.ref_drift = [wl.ref_drift[b] for b in blocks]
    sub.tgt_drift = [wl.tgt_drift[b] for b in blocks]
    traj = synth.Trajectory(sub, device="cuda")
    ex = Executor(sub.n_blocks, sub.B, sub.H, sub.d, sub.n_text, sub.n_ref, sub.n_tgt, sub.theta,
                  sub.delta_max, sub.eps, mass_rows=sub.mass_rows, forced_boundary=sub.forced_boundary,
                  bias=sub.bias, log_steps=sub.n_steps, sample_stride=sample_stride)
    rec = {}
    prev = {}
    last = {}  # (block, sample) -> (inputs, step) of the last materialisation
    for t in range(sub.n_steps):
        for b in range(sub.n_blocks):
            X = traj.get(t, b)
            out = {r: torch.full((sub.B, sub.H, sub.n[r], sub.d), float("nan"), dtype=torch.bfloat16,
                                 device="cuda") for r in ROLES}
            ex.block(t, b, roles_from_joint(X, sub.offsets(), sub.n), out)
            torch.cuda.synchronize()
            # Eq. 11: the cache slot holds the reference Q/K/V of the block's
            # last materialisation, bit for bit, and a_b its step
            for s, m in enumerate(ex.modes[t, b].tolist()):
                if m in (2, 3):
                    last[(b, s)] = (X, t)
                src, ts = last[(b, s)]
                for z, cache in enumerate((ex.cache_x, ex.cache_k, ex.cache_v)):
                    assert torch.equal(cache[b][s], _role(src, sub, "ref", z)[s]), (t, b, s, z)
                assert int(ex.a_b[b][s]) == ts, (t, b, s)
            rec[(t, b)] = {"X": X, "O": out, "D": ex.D[b].clone(), "mode": ex.modes[t, b].clone(),
                           "gbar": ex.gbar[t, b].clone(), "mass": ex.mass[b].clone(),
                           "M": ex.M[t, b].clone(), "Xprev": prev.get(b)}
            prev[b] = X
        # keep only what later checks need
    ex.check()
    return sub, rec


FULLSIZE = [("c2", {}), ("c3", {}), ("c4", {}),
            # sweep points: 64k tokens, 90 % reference, boundary forced at block 4
            # (block 0 reuses at step 1); 8k tokens, 50 % reference, boundary at block 7
            ("c5", dict(total=65536, ref_frac=0.9, reuse_frac=0.5)),
            ("c5", dict(total=8192, ref_frac=0.5, reuse_frac=0.9)),
            # two samples: per-sample strides and the grid's sample dimension at scale
            ("c5", dict(total=16384, ref_frac=0.7, reuse_frac=0.5, B=2))]


@pytest.mark.parametrize("name,over", FULLSIZE,
                         ids=["c2", "c3", "c4", "sweep-64k-90ref-50reuse", "sweep-8k-50ref-90reuse",
                              "sweep-16k-70ref-50reuse-B2"])
def test_fullsize_block_parity(cuda_ok, name, over):
    """First block of the stack, steps 0 and 1, every sample: sampled O rows
    of every executed role, two mass tiles per sampled head, D of every head,
    and the step-1 decisions from the oracle controller with the oracle's D."""
    from paper_2609_32415_gb300 import synth
    wl = synth.make_workload(name, **over)
    wl.n_steps = 2
    sub, rec = _run_stack(wl, [0])
    sc = 1.0 / math.sqrt(sub.d)
    bias = None if sub.bias is None else np.asarray(sub.bias)
    rng = np.random.default_rng(0)
    a_b = 0                                    # the cache holds step 0 after step 0's FULL
    hs = list(HEADS)
    r0, r1 = sub.n_text, sub.n_text + sub.n_ref
    for t in range(2):
        r = rec[(t, 0)]
        X = r["X"]
        for z in range(sub.B):
            mode = int(r["mode"][z])
            if t == 0:
                assert mode == 3
            fresh_ref = mode in (2, 3)
            Xk = X if fresh_ref else rec[(a_b, 0)]["X"]
            q = {ro: _wide(_role(X if ro != "ref" else Xk, sub, ro, 0)[z, hs]) for ro in ROLES}
            k = {ro: _wide(_role(X if ro != "ref" else Xk, sub, ro, 1)[z, hs]) for ro in ROLES}
            v = {ro: _wide(_role(X if ro != "ref" else Xk, sub, ro, 2)[z, hs]) for ro in ROLES}
            keys = np.concatenate([k["text"], k["ref"], k["tgt"]], axis=1)
            vals = np.concatenate([v["text"], v["ref"], v["tgt"]], axis=1)
            roles = ("text", "tgt") if mode == 0 else ROLES
            for ro in roles:
                n = sub.n[ro]
                idx = np.unique(np.concatenate([np.arange(min(8, n)), np.arange(max(0, n - 8), n),
                                                rng.choice(n, size=min(48, n), replace=False)]))
                rb = np.full(len(idx), 1 if ro == "tgt" else 0, dtype=np.uint8)
                o, _ = oracle.joint_attention(q[ro][:, idx], keys, vals, sc,
                                              None if bias is None else bias[hs],
                                              rb if bias is not None else None, (r0, r1))
                got = r["O"][ro][z, hs][:, idx].double().cpu().numpy()
                ok, worst, nw = o_close(got, o)
                assert ok, (name, t, z, ro, worst, nw)
            if mode == 0:
                assert torch.isnan(r["O"]["ref"][z].float()).all()
            # mass partials: first and last target tile of the sampled heads
            nt = (sub.n_tgt + 127) // 128
            base = (sub.n_text + 127) // 128
            for tile in (0, nt - 1):
                rows = np.arange(tile * 128, min(sub.n_tgt, tile * 128 + 128))
                rb = np.ones(len(rows), dtype=np.uint8)
                _, m = oracle.joint_attention(q["tgt"][:, rows], keys, vals, sc,
                                              None if bias is None else bias[hs],
                                              rb if bias is not None else None, (r0, r1), want_o=False)
                got = r["mass"][z, hs, base + tile].double().cpu().numpy() / len(rows)
                err = np.abs(got - m.mean(axis=1)).max()
                assert err <= M_ABS, (name, t, z, tile, err)
                assert err <= 2e-5, (name, t, z, tile, err)   # far below the gate's 1e-4 band
        if t == 1:
            qc = _wide(_role(X, sub, "tgt", 0))
            qp = _wide(_role(r["Xprev"], sub, "tgt", 0))
            D = oracle.q_change(qc, qp, sub.eps)                       # [B, H]
            got = r["D"].double().cpu().numpy()
            assert (np.abs(got - D) / D).max() <= D_REL
            # the controller's decisions from the oracle D and the mass of step 0
            # (the GPU's M, whose sampled tiles were checked above at step 0)
            M_prev = rec[(0, 0)]["mass"].double().sum(-1).cpu().numpy() / sub.n_tgt
            gate = oracle.Gate(sub.B, sub.theta, sub.delta_max, sub.forced_boundary)
            gate.begin_step(0)
            gate.decide(0, 0)
            gate.begin_step(1)
            gpu_modes = [int(x) for x in r["mode"]]
            modes, gbar = gate.decide(1, 0, D, M_prev,
                                      tie=lambda tt, bb, s: gpu_modes[s] == 1, tie_band=TIE_BAND)
            assert modes == gpu_modes, (name, modes, gpu_modes, gbar, sub.theta)
            for z in range(sub.B):
                assert abs(gbar[z] - float(r["gbar"][z])) < 1e-5 * max(1.0, abs(gbar[z]))


def test_fullsize_depth_reduced_trajectory(cuda_ok):
    """Image-edit workload on the depth-reduced stack {0, 1, 44, 45, 59}, all 8
    steps: every D against the oracle, every decision against the oracle's
    controller fed with the oracle's D (and the GPU's M), and the schedule's
    shape (full steps, monotone suffix)."""
    from paper_2609_32415_gb300 import synth
    wl = synth.make_workload("c2")
    blocks = [0, 1, 44, 45, 59]
    sub, rec = _run_stack(wl, blocks)
    gate = oracle.Gate(1, sub.theta, sub.delta_max, sub.forced_boundary)
    for t in range(sub.n_steps):
        gate.begin_step(t)
        gm = [int(rec[(t, b)]["mode"][0]) for b in range(len(blocks))]
        for b in range(len(blocks)):
            r = rec[(t, b)]
            if t >= 1:
                qc = _wide(_role(r["X"], sub, "tgt", 0)[0])
                qp = _wide(_role(r["Xprev"], sub, "tgt", 0)[0])
                D = oracle.q_change(qc, qp, sub.eps)
                got = r["D"][0].double().cpu().numpy()
                assert (np.abs(got - D) / D).max() <= D_REL, (t, b)
                M_prev = rec[(t - 1, b)]["mass"][0].double().sum(-1).cpu().numpy() / sub.n_tgt
                m, _ = gate.decide(t, b, D[None], M_prev[None],
                                   tie=lambda tt, bb, s: gm[bb] == 1, tie_band=TIE_BAND)
            else:
                m, _ = gate.decide(t, b)
            assert m[0] == gm[b], (t, b, m, gm)
        if t in (0, 4):
            assert gm == [3] * len(blocks)
        elif 1 in gm:
            k = gm.index(1)
            assert gm[:k] == [0] * k and gm[k + 1:] == [2] * (len(gm) - k - 1)
        else:
            assert gm == [0] * len(blocks)


@pytest.mark.parametrize("name,blocks,k", [("c2", [0, 1, 44, 45, 59], 16), ("c3", [0, 1, 20, 39], 64)],
                         ids=["image-edit", "video"])
def test_fullsize_trajectory_on_oracle_mass(cuda_ok, name, blocks, k):
    """Depth-reduced stacks of the image-edit (all 8 steps) and video (all 4
    steps, per-head target-to-reference bias) workloads, D and M over the
    sampled target rows 0, k, 2k, ... (256 rows): at every (t, b) the oracle
    computes M (Eq. 4) for all 24 heads from the keys the block executed (the
    reference keys of its last materialisation, kept by the oracle's own
    bookkeeping of Eq. 11) and D (Eq. 1) on the same rows; the GPU's M must
    agree within 2e-5 and its D within the Q-change tolerance, and the
    oracle's controller, fed with the oracle's own D and M only, must
    reproduce every decision."""
    from paper_2609_32415_gb300 import synth
    wl = synth.make_workload(name)
    sub, rec = _run_stack(wl, blocks, sample_stride=k)
    sc = 1.0 / math.sqrt(sub.d)
    bias = None if sub.bias is None else np.asarray(sub.bias)
    r0, r1 = sub.n_text, sub.n_text + sub.n_ref
    nb = len(blocks)
    gate = oracle.Gate(1, sub.theta, sub.delta_max, sub.forced_boundary)
    a_b = [-1] * nb                      # the oracle's own materialisation step per block
    m_prev = [None] * nb                 # the oracle's M of the previous step per block
    m_prev_gate = [None] * nb
    for t in range(sub.n_steps):
        gate.begin_step(t)
        gm = [int(rec[(t, b)]["mode"][0]) for b in range(nb)]
        for b in range(nb):
            r = rec[(t, b)]
            qt = _wide(_role(r["X"], sub, "tgt", 0)[0, :, ::k])            # [H, n_tgt / k, d]
            if t >= 1:
                qp = _wide(_role(r["Xprev"], sub, "tgt", 0)[0, :, ::k])
                D = oracle.q_change(qt, qp, sub.eps)                       # [H]
                got = r["D"][0].double().cpu().numpy()
                assert (np.abs(got - D) / D).max() <= D_REL, (t, b)
                m, _ = gate.decide(t, b, D[None], m_prev[b][None],
                                   tie=lambda tt, bb, s: gm[bb] == 1, tie_band=TIE_BAND)
            else:
                m, _ = gate.decide(t, b)
            assert m[0] == gm[b], (t, b, m, gm)
            if m[0] in (2, 3):
                a_b[b] = t
            Xk = r["X"] if m[0] in (2, 3) else rec[(a_b[b], b)]["X"]
            keys = np.concatenate([_wide(_role(r["X"], sub, "text", 1)[0]), _wide(_role(Xk, sub, "ref", 1)[0]),
                                   _wide(_role(r["X"], sub, "tgt", 1)[0])], axis=1)
            vals = np.concatenate([_wide(_role(r["X"], sub, "text", 2)[0]), _wide(_role(Xk, sub, "ref", 2)[0]),
                                   _wide(_role(r["X"], sub, "tgt", 2)[0])], axis=1)
            rb = np.ones(qt.shape[1], dtype=np.uint8) if bias is not None else None
            _, rm = oracle.joint_attention(qt, keys, vals, sc, bias, rb, (r0, r1), want_o=False)
            M = oracle.exposure(rm)                                         # [H]
            # the GPU's M of this step's attention: its mass partials over the
            # sampled rows (text tiles hold zero), as the next step's gate sums them
            got = r["mass"][0].double().sum(-1).cpu().numpy() / qt.shape[1]
            err = np.abs(got - M).max()
            assert err <= 2e-5, (t, b, err)
            m_prev[b] = M
            if t >= 1:   # the gate of step t read M of step t - 1 (its m_out)
                assert np.abs(r["M"][0].double().cpu().numpy() - m_prev_gate[b]).max() <= 2e-5, (t, b)
            m_prev_gate[b] = M
    gm_all = [[int(rec[(t, b)]["mode"][0]) for b in range(nb)] for t in range(sub.n_steps)]
    assert any(0 in row for row in gm_all[1:]) and any(1 in row for row in gm_all[1:]), gm_all
