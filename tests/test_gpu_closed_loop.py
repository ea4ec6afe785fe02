"""Closed-loop parity: Algorithm 1 run by the Executor over the C ABI against the
oracle's closed loop on the same seeded bf16 inputs (modes, D, M, O)."""
import numpy as np
import pytest
import torch

import oracle
from _helpers import D_REL, M_ABS, TIE_BAND, bits, o_close

pytestmark = pytest.mark.gpu

ROLES = ("text", "ref", "tgt")


def _run_both(wl, o_sample=None, cue="product", diagnostics=False, diag_row_stride=1):
    from paper_2609_32415_gb300 import Executor, roles_from_joint, synth
    traj = synth.Trajectory(wl, device="cuda")
    ex = Executor(wl.n_blocks, wl.B, wl.H, wl.d, wl.n_text, wl.n_ref, wl.n_tgt, wl.theta, wl.delta_max,
                  wl.eps, mass_rows=wl.mass_rows, forced_boundary=wl.forced_boundary, bias=wl.bias,
                  log_steps=wl.n_steps, cue=cue, diagnostics=diagnostics, diag_row_stride=diag_row_stride)
    keep, outs, D = {}, {}, np.zeros((wl.n_steps, wl.n_blocks, wl.B, wl.H))
    for t in range(wl.n_steps):
        xs, os_ = [], []
        for b in range(wl.n_blocks):
            X = traj.get(t, b)
            keep[(t, b)] = X
            xs.append(roles_from_joint(X, wl.offsets(), wl.n))
            os_.append({r: torch.full((wl.B, wl.H, wl.n[r], wl.d), float("nan"), dtype=torch.bfloat16,
                                      device="cuda") for r in ROLES})

        def grab(tt, bb):
            D[tt, bb] = ex.D[bb].double().cpu().numpy()

        ex.step(t, xs, os_, after_block=grab)
        outs[t] = os_
    torch.cuda.synchronize()
    ex.check()
    modes = ex.modes.cpu().numpy()
    gbar = ex.gbar.double().cpu().numpy()
    Mlog = ex.M.double().cpu().numpy()

    def raw(t, b):
        X = keep[(t, b)]
        off = wl.offsets()
        return {r: tuple(bits(X[z, :, :, off[r]:off[r] + wl.n[r], :]) for z in range(3)) for r in ROLES}

    def tie(t, b, s):
        return modes[t, b, s] == 1

    rec = oracle.closed_loop(raw, wl.n_steps, wl.n_blocks, wl.B, theta=wl.theta, delta_max=wl.delta_max,
                             eps=wl.eps, bias=wl.bias, mass_rows=wl.mass_rows,
                             forced_boundary=wl.forced_boundary, tie=tie, o_rows=o_sample, cue=cue,
                             diagnostics=diagnostics, diag_row_stride=diag_row_stride)
    if diagnostics:
        rows_s = ex.n_tgt_sampled
        diag = {"E_K": ex.E_K.double().cpu().numpy(), "E_V": ex.E_V.double().cpu().numpy(),
                "I_KV": ex.I_KV.double().cpu().numpy(),
                "M_fresh": ex.M_fresh_part.double().sum(-1).cpu().numpy() / rows_s,
                "summary": ex.exposure_summary(wl.n_steps),
                "summary_fresh": ex.exposure_summary(wl.n_steps, fresh=True)}
        return modes, gbar, Mlog, D, outs, rec, diag
    return modes, gbar, Mlog, D, outs, rec


def _compare(wl, modes, gbar, Mlog, D, outs, rec, o_sample=None):
    ties = 0
    for t in range(wl.n_steps):
        for b in range(wl.n_blocks):
            r = rec[t][b]
            assert list(modes[t, b]) == r["mode"], (t, b, modes[t, b], r["mode"])
            for s in range(wl.B):
                if np.isfinite(r["gbar"][s]) and abs(r["gbar"][s] - wl.theta) < TIE_BAND:
                    ties += 1
            if t >= 1:
                rel = np.abs(D[t, b] - r["D"]) / np.abs(r["D"])
                assert rel.max() <= D_REL, (t, b, rel.max())
                np.testing.assert_allclose(gbar[t, b], r["gbar"], rtol=1e-4, atol=1e-6)
            if t + 1 < wl.n_steps:
                dm = np.abs(Mlog[t + 1, b] - r["M"]).max()
                assert dm <= M_ABS, (t, b, dm)
            for s in range(wl.B):
                for role in ROLES:
                    ref = r["O"][s][role]
                    got = outs[t][b][role][s]
                    if ref is None:
                        assert torch.isnan(got.float()).all()
                        continue
                    g = got.double().cpu().numpy()
                    if o_sample is not None:
                        g = g[:, o_sample(t, b, s)[role], :]
                    ok, worst, nw = o_close(g, ref)
                    assert ok, (t, b, s, role, worst, nw)
    return ties


@pytest.mark.parametrize("theta", [0.05, 0.1, 0.2])
def test_closed_loop_single_block_workload(cuda_ok, theta):
    from paper_2609_32415_gb300 import synth
    wl = synth.make_workload("c1", theta=theta)
    res = _run_both(wl)
    _compare(wl, *res)


def test_closed_loop_multi_block_depth_profile(cuda_ok):
    """Five blocks, B=2, ragged segments, increasing target drift with depth so
    the boundary moves; delta_max=3 forces a full refresh mid-trajectory."""
    from paper_2609_32415_gb300 import synth
    wl = synth.custom_workload(2, 4, 128, 33, 300, 200, n_blocks=5, n_steps=6, ref_drift=0.05,
                               tgt_drift=[0.05, 0.1, 0.2, 0.3, 0.4], theta=0.08, delta_max=3)
    res = _run_both(wl)
    _compare(wl, *res)
    modes = res[0]
    assert (modes == 0).any() and (modes == 1).any() and (modes == 2).any() and (modes == 3).any()


def test_closed_loop_forced_boundary_and_bias(cuda_ok):
    from paper_2609_32415_gb300 import synth
    wl = synth.custom_workload(1, 3, 64, 16, 260, 140, n_blocks=4, n_steps=3, theta=float("inf"),
                               delta_max=8, forced_boundary=2, bias=[-3.0, -1.0, 0.0], mass_rows=1)
    res = _run_both(wl)
    _compare(wl, *res)
    assert list(res[0][1, :, 0]) == [0, 0, 1, 2]


@pytest.mark.parametrize("cue,theta", [("change", 0.15), ("exposure", 0.43), ("anchor_product", 0.1)])
def test_closed_loop_ablation_cues(cuda_ok, cue, theta):
    """The controller ablation's trigger variants (Sec. 5.3, Tab. 4; the anchor
    variant of App. A.2) through the same executor."""
    from paper_2609_32415_gb300 import synth
    wl = synth.custom_workload(2, 4, 128, 33, 300, 200, n_blocks=5, n_steps=6, ref_drift=0.05,
                               tgt_drift=[0.05, 0.1, 0.2, 0.3, 0.4], theta=theta, delta_max=4)
    res = _run_both(wl, cue=cue)
    _compare(wl, *res)


def test_closed_loop_staleness_diagnostics(cuda_ok):
    """Eqs. 7-10 through the executor's diagnostic pass (every second target row)
    against the oracle's closed loop: E_K, E_V exact to the Q-change tolerance,
    the fresh exposure to the mass tolerance, and I_KV within 5e-3 (both
    outputs it compares are rounded to bf16 on the GPU)."""
    from paper_2609_32415_gb300 import synth
    wl = synth.custom_workload(2, 4, 128, 33, 300, 200, n_blocks=3, n_steps=4, ref_drift=0.2,
                               tgt_drift=[0.05, 0.2, 0.4], theta=0.08, delta_max=100)
    *res, diag = _run_both(wl, diagnostics=True, diag_row_stride=2)
    _compare(wl, *res)
    rec = res[-1]
    for t in range(1, wl.n_steps):
        for b in range(wl.n_blocks):
            r = rec[t][b]
            for key in ("E_K", "E_V"):
                want, got = r[key], diag[key][t, b]
                ok = np.where(want > 0, np.abs(got - want) / np.maximum(want, 1e-30) <= D_REL, got <= 1e-6)
                assert ok.all(), (t, b, key, got, want)
            assert np.abs(diag["M_fresh"][t, b] - r["M_fresh"]).max() <= M_ABS, (t, b)
            assert np.abs(diag["I_KV"][t, b] - r["I_KV"]).max() <= 5e-3, (t, b, diag["I_KV"][t, b], r["I_KV"])
    # Eqs. 5-6 over the trajectory, executed and fresh exposure, against the
    # oracle's summaries of its own M (M within M_ABS, so Mbar within M_ABS
    # and Delta within 2 * 100 * M_ABS percentage points)
    for key, src in (("summary", "M"), ("summary_fresh", "M_fresh")):
        Mo = np.stack([np.stack([rec[t][b][src] for b in range(wl.n_blocks)]) for t in range(wl.n_steps)])
        Mbar_o = oracle.head_mean_exposure(Mo)
        Delta_o = oracle.adjacent_ref_mass_change(Mbar_o)
        Mbar, Delta = diag[key]
        assert np.abs(Mbar - Mbar_o).max() <= M_ABS, key
        assert np.abs(Delta - Delta_o).max() <= 200 * M_ABS, (key, Delta, Delta_o)


def test_closed_loop_sampled_target_rows(cuda_ok):
    """D and M over the sampled target rows 0, 4, 8, ... (Algorithm 1's
    sampled target queries and masses) through the executor against the
    oracle's closed loop with the same sample."""
    from paper_2609_32415_gb300 import Executor, roles_from_joint, synth
    wl = synth.custom_workload(2, 4, 128, 33, 300, 200, n_blocks=4, n_steps=5, ref_drift=0.05,
                               tgt_drift=[0.05, 0.1, 0.3, 0.4], theta=0.08, delta_max=3)
    traj = synth.Trajectory(wl, device="cuda")
    ex = Executor(wl.n_blocks, wl.B, wl.H, wl.d, wl.n_text, wl.n_ref, wl.n_tgt, wl.theta, wl.delta_max,
                  wl.eps, log_steps=wl.n_steps, sample_stride=4)
    keep, D = {}, np.zeros((wl.n_steps, wl.n_blocks, wl.B, wl.H))
    for t in range(wl.n_steps):
        xs = []
        for b in range(wl.n_blocks):
            X = traj.get(t, b)
            keep[(t, b)] = X
            xs.append(roles_from_joint(X, wl.offsets(), wl.n))

        def grab(tt, bb):
            D[tt, bb] = ex.D[bb].double().cpu().numpy()

        ex.step(t, xs, after_block=grab)
    torch.cuda.synchronize()
    ex.check()
    modes = ex.modes.cpu().numpy()
    gbar = ex.gbar.double().cpu().numpy()
    off = wl.offsets()

    def raw(t, b):
        X = keep[(t, b)]
        return {r: tuple(bits(X[z, :, :, off[r]:off[r] + wl.n[r], :]) for z in range(3)) for r in ROLES}

    rec = oracle.closed_loop(raw, wl.n_steps, wl.n_blocks, wl.B, theta=wl.theta, delta_max=wl.delta_max,
                             eps=wl.eps, tie=lambda t, b, s: modes[t, b, s] == 1, want_o=False, sample_stride=4)
    for t in range(wl.n_steps):
        for b in range(wl.n_blocks):
            r = rec[t][b]
            assert list(modes[t, b]) == r["mode"], (t, b, modes[t, b], r["mode"])
            if t >= 1:
                assert (np.abs(D[t, b] - r["D"]) / np.abs(r["D"])).max() <= D_REL, (t, b)
                np.testing.assert_allclose(gbar[t, b], r["gbar"], rtol=1e-4, atol=1e-6)
    assert (modes == 1).any() and (modes == 0).any()


def test_gates_first_matches_block_order(cuda_ok):
    """A step's gates enqueued before its attentions (Executor.gate_block for
    every block, then Executor.attend_block; the order bench.py's end-to-end
    timing uses to read the modes before copying reference rows) give the
    same modes, gbar, M, D, mass partials and outputs, bit for bit, as the
    block-by-block order: a gate reads nothing an attention of the same step
    writes. Blocks with no materialising sample (REUSE, BOUNDARY) get garbage
    reference rows here, which they must not read."""
    from paper_2609_32415_gb300 import Executor, roles_from_joint, synth
    wl = synth.custom_workload(2, 4, 128, 33, 300, 200, n_blocks=5, n_steps=6, ref_drift=0.05,
                               tgt_drift=[0.05, 0.1, 0.2, 0.3, 0.4], theta=0.08, delta_max=3)
    traj = synth.Trajectory(wl, device="cuda")

    def run(gates_first):
        ex = Executor(wl.n_blocks, wl.B, wl.H, wl.d, wl.n_text, wl.n_ref, wl.n_tgt, wl.theta, wl.delta_max,
                      wl.eps, mass_rows=wl.mass_rows, forced_boundary=wl.forced_boundary, bias=wl.bias,
                      log_steps=wl.n_steps)
        outs, mass, D = [], [], []
        for t in range(wl.n_steps):
            xs = [roles_from_joint(traj.get(t, b), wl.offsets(), wl.n) for b in range(wl.n_blocks)]
            os_ = [{r: torch.full((wl.B, wl.H, wl.n[r], wl.d), float("nan"), dtype=torch.bfloat16, device="cuda")
                    for r in ROLES} for _ in range(wl.n_blocks)]
            if gates_first:
                for b in range(wl.n_blocks):
                    ex.gate_block(t, b, xs[b]["tgt"][0])
                torch.cuda.synchronize()
                modes = ex.modes[t].cpu()
                for b in range(wl.n_blocks):
                    x = dict(xs[b])
                    if not bool(((modes[b] == 2) | (modes[b] == 3)).any()):
                        x["ref"] = tuple(torch.randn_like(z, dtype=torch.float32).to(torch.bfloat16)
                                         for z in xs[b]["ref"])
                    ex.attend_block(t, b, x, os_[b])
                    D.append(ex.D[b].clone())
                    mass.append(ex.mass[b].clone())
            else:
                for b in range(wl.n_blocks):
                    ex.block(t, b, xs[b], os_[b])
                    D.append(ex.D[b].clone())
                    mass.append(ex.mass[b].clone())
            outs.append(os_)
        torch.cuda.synchronize()
        ex.check()
        return ex.modes.clone(), ex.gbar.clone(), ex.M.clone(), D, mass, outs

    def same(x, y):  # bit-equal, NaN where the other has NaN (gbar has none on a step without a score)
        return torch.equal(torch.isnan(x), torch.isnan(y)) and torch.equal(torch.nan_to_num(x), torch.nan_to_num(y))

    a, b_ = run(False), run(True)
    for x, y in zip(a[:3], b_[:3]):
        assert same(x, y)
    for x, y in zip(a[3] + a[4], b_[3] + b_[4]):
        assert same(x, y)
    for oa, ob in zip(a[5], b_[5]):
        for ba, bb in zip(oa, ob):
            for r in ROLES:
                assert torch.equal(torch.nan_to_num(ba[r], 7.0), torch.nan_to_num(bb[r], 7.0)), r
    assert (a[0] == 0).any() and (a[0] == 3).any()


def test_two_stream_step_matches_one_stream(cuda_ok):
    """Executor.step with overlap (each block's gate and cache update on a
    side stream, consecutive attentions on two streams) gives the same modes,
    gbar, M, D, mass partials and outputs, bit for bit, as the one-stream
    order: no launch of the overlapped schedule reads or writes anything early
    or late."""
    from paper_2609_32415_gb300 import Executor, roles_from_joint, synth
    wl = synth.custom_workload(2, 4, 128, 33, 300, 200, n_blocks=5, n_steps=6, ref_drift=0.05,
                               tgt_drift=[0.05, 0.1, 0.2, 0.3, 0.4], theta=0.08, delta_max=3)
    traj = synth.Trajectory(wl, device="cuda")

    def run(overlap):
        ex = Executor(wl.n_blocks, wl.B, wl.H, wl.d, wl.n_text, wl.n_ref, wl.n_tgt, wl.theta, wl.delta_max,
                      wl.eps, mass_rows=wl.mass_rows, forced_boundary=wl.forced_boundary, bias=wl.bias,
                      log_steps=wl.n_steps, overlap=overlap)
        outs, mass, D = [], [], []
        for t in range(wl.n_steps):
            xs = [roles_from_joint(traj.get(t, b), wl.offsets(), wl.n) for b in range(wl.n_blocks)]
            os_ = [{r: torch.full((wl.B, wl.H, wl.n[r], wl.d), float("nan"), dtype=torch.bfloat16, device="cuda")
                    for r in ROLES} for _ in range(wl.n_blocks)]

            def grab(tt, bb):
                D.append(ex.D[bb].clone())
                mass.append(ex.mass[bb].clone())

            ex.step(t, xs, os_, after_block=grab)
            outs.append(os_)
        torch.cuda.synchronize()
        ex.check()
        return ex.modes.clone(), ex.gbar.clone(), ex.M.clone(), D, mass, outs

    def same(x, y):
        return torch.equal(torch.isnan(x), torch.isnan(y)) and torch.equal(torch.nan_to_num(x), torch.nan_to_num(y))

    a, b_ = run(False), run(True)
    for x, y in zip(a[:3], b_[:3]):
        assert same(x, y)
    for x, y in zip(a[3] + a[4], b_[3] + b_[4]):
        assert same(x, y)
    for oa, ob in zip(a[5], b_[5]):
        for ba, bb in zip(oa, ob):
            for r in ROLES:
                assert same(ba[r].float(), bb[r].float()), r
    assert (a[0] == 0).any() and (a[0] == 3).any()


@pytest.mark.parametrize("overlap", [False, True])
def test_fused_cache_update_matches_separate_update(cuda_ok, overlap):
    """The attention writing the cache slot of materialising blocks (the
    executor's default) and a refadapt_ref_cache_update launch before it give
    the same modes, gbar, M, D, mass partials, outputs, cache slots and a_b,
    bit for bit, over a trajectory that reuses, reactivates at a boundary,
    recomputes and fully refreshes."""
    from paper_2609_32415_gb300 import Executor, roles_from_joint, synth
    wl = synth.custom_workload(2, 4, 128, 33, 300, 200, n_blocks=5, n_steps=6, ref_drift=0.05,
                               tgt_drift=[0.05, 0.1, 0.2, 0.3, 0.4], theta=0.08, delta_max=3)
    traj = synth.Trajectory(wl, device="cuda")

    def run(fused):
        ex = Executor(wl.n_blocks, wl.B, wl.H, wl.d, wl.n_text, wl.n_ref, wl.n_tgt, wl.theta, wl.delta_max,
                      wl.eps, mass_rows=wl.mass_rows, forced_boundary=wl.forced_boundary, bias=wl.bias,
                      log_steps=wl.n_steps, overlap=overlap, fused_cache=fused)
        outs, snap = [], []
        for t in range(wl.n_steps):
            xs = [roles_from_joint(traj.get(t, b), wl.offsets(), wl.n) for b in range(wl.n_blocks)]
            os_ = [{r: torch.full((wl.B, wl.H, wl.n[r], wl.d), float("nan"), dtype=torch.bfloat16, device="cuda")
                    for r in ROLES} for _ in range(wl.n_blocks)]

            def grab(tt, bb):
                snap.extend([ex.D[bb].clone(), ex.mass[bb].clone(), ex.cache_k[bb].clone(),
                             ex.cache_v[bb].clone(), ex.cache_x[bb].clone(), ex.a_b[bb].clone()])

            ex.step(t, xs, os_, after_block=grab)
            outs.append(os_)
        torch.cuda.synchronize()
        ex.check()
        return [ex.modes.clone(), ex.gbar.clone(), ex.M.clone()] + snap, outs

    def same(x, y):
        if x.is_floating_point():
            return torch.equal(torch.isnan(x), torch.isnan(y)) and torch.equal(torch.nan_to_num(x),
                                                                               torch.nan_to_num(y))
        return torch.equal(x, y)

    (ta, oa), (tb, ob) = run(False), run(True)
    assert len(ta) == len(tb)
    for x, y in zip(ta, tb):
        assert same(x, y)
    for sa, sb in zip(oa, ob):
        for ba, bb in zip(sa, sb):
            for r in ROLES:
                assert same(ba[r].float(), bb[r].float()), r
    modes = ta[0]
    assert (modes == 0).any() and (modes == 1).any() and (modes == 2).any() and (modes == 3).any()
