"""Checkpoint / resume and the observation trace of the Executor.

A trajectory interrupted after step 2 (snapshot, a new executor, restore)
continues with the results of the uninterrupted run, bit for bit: outputs,
modes, gbar, M, D, the cache slots, a_b and the controller state. The
trace's records agree with the device logs and serialise as JSON lines."""
import json

import pytest
import torch

pytestmark = pytest.mark.gpu

ROLES = ("text", "ref", "tgt")


def _workload():
    from paper_2609_32415_gb300 import synth
    return synth.custom_workload(2, 4, 128, 33, 300, 200, n_blocks=4, n_steps=6, ref_drift=0.05,
                                 tgt_drift=[0.05, 0.1, 0.3, 0.4], theta=0.08, delta_max=3)


def _make(wl, **kw):
    from paper_2609_32415_gb300 import Executor
    return Executor(wl.n_blocks, wl.B, wl.H, wl.d, wl.n_text, wl.n_ref, wl.n_tgt, wl.theta, wl.delta_max, wl.eps,
                    log_steps=wl.n_steps, **kw)


def _run(ex, wl, traj, t0, t1, outs, keep):
    from paper_2609_32415_gb300 import roles_from_joint
    for t in range(t0, t1):
        xs = [roles_from_joint(traj.get(t, b), wl.offsets(), wl.n) for b in range(wl.n_blocks)]
        keep.append(xs)
        os_ = [{r: torch.full((wl.B, wl.H, wl.n[r], wl.d), float("nan"), dtype=torch.bfloat16, device="cuda")
                for r in ROLES} for _ in range(wl.n_blocks)]
        ex.step(t, xs, os_)
        outs[t] = os_
    torch.cuda.synchronize()
    ex.check()


def _same(x, y):
    if x.is_floating_point():
        return torch.equal(torch.isnan(x), torch.isnan(y)) and torch.equal(x.nan_to_num(), y.nan_to_num())
    return torch.equal(x, y)


def test_snapshot_resume_continues_bit_for_bit(cuda_ok):
    from paper_2609_32415_gb300 import synth
    wl = _workload()
    traj = synth.Trajectory(wl, device="cuda")
    keep = []
    a = _make(wl)
    outs_a = {}
    _run(a, wl, traj, 0, wl.n_steps, outs_a, keep)

    b1 = _make(wl)
    outs_b = {}
    _run(b1, wl, traj, 0, 3, outs_b, keep)
    snap = b1.snapshot()
    del b1
    keep.clear()  # the resumed run holds none of the first run's tensors
    torch.cuda.empty_cache()
    b2 = _make(wl, nvtx=True)
    b2.restore(snap)
    _run(b2, wl, traj, 3, wl.n_steps, outs_b, keep)

    for t in range(3, wl.n_steps):
        for blk in range(wl.n_blocks):
            for r in ROLES:
                assert _same(outs_a[t][blk][r].float(), outs_b[t][blk][r].float()), (t, blk, r)
    for name in ("modes", "gbar", "M", "D", "mass", "cache_k", "cache_v", "cache_x", "a_b", "state"):
        assert _same(getattr(a, name), getattr(b2, name)), name
    m = a.modes.reshape(-1)
    assert (m == 0).any() and (m == 1).any() and (m == 2).any() and (m == 3).any()

    # a snapshot loads only into an executor of the same configuration
    from paper_2609_32415_gb300 import Executor
    other = Executor(wl.n_blocks, wl.B, wl.H, wl.d, wl.n_text, wl.n_ref + 128, wl.n_tgt, wl.theta,
                     wl.delta_max, wl.eps, log_steps=wl.n_steps)
    with pytest.raises(ValueError):
        other.restore(snap)


def test_trace_records_match_the_logs(cuda_ok, tmp_path):
    from paper_2609_32415_gb300 import synth
    wl = _workload()
    traj = synth.Trajectory(wl, device="cuda")
    ex = _make(wl)
    _run(ex, wl, traj, 0, wl.n_steps, {}, [])
    recs = ex.trace(wl.n_steps)
    assert len(recs) == wl.n_steps * wl.n_blocks
    modes = ex.modes.cpu()
    gbar = ex.gbar.double().cpu()
    mbar = ex.M.double().mean(-1).cpu()
    for r in recs:
        t, b = r["t"], r["b"]
        assert r["mode"] == modes[t, b].tolist()
        if t == 0:
            assert r["gbar"] == [None] * wl.B and r["m_bar_read"] is None
        else:
            assert r["gbar"] == gbar[t, b].tolist()
            assert r["m_bar_read"] == mbar[t, b].tolist()
        assert r["a_b"] == ex.a_b[b].tolist()
    path = tmp_path / "trace.jsonl"
    path.write_text("".join(json.dumps(r) + "\n" for r in recs))
    back = [json.loads(line) for line in path.read_text().splitlines()]
    assert back == recs
