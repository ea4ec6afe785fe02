"""GPU parity of refadapt_gate against the oracle's Algorithm 1 controller."""
import math

import numpy as np
import pytest
import torch

import oracle
from _helpers import TIE_BAND

pytestmark = pytest.mark.gpu


CUE_ID = {"product": 0, "change": 1, "exposure": 2}


def _run_gate(D, M, theta, delta_max, forced=-1, L=3, cue="product"):
    """D, M: [T, nb, B, H] arrays. M is spread over L partial tiles. Returns GPU
    modes / gbar [T, nb, B] and the oracle's."""
    from paper_2609_32415_gb300 import api
    T, nb, B, H = D.shape
    state = api.new_state(B)
    rows = 1000
    modes = torch.full((T, nb, B), -1, dtype=torch.int32, device="cuda")
    gbar = torch.zeros((T, nb, B), dtype=torch.float32, device="cuda")
    mparts = []
    for t in range(T):
        for b in range(nb):
            part = np.zeros((B, H, L), dtype=np.float32)
            tot = (M[t, b] * rows).astype(np.float32)
            for i in range(L - 1):
                part[:, :, i] = tot / L
            part[:, :, L - 1] = tot - (L - 1) * (tot / L)
            mparts.append(torch.from_numpy(part).cuda())
    dd = torch.from_numpy(D.astype(np.float32)).cuda()
    for t in range(T):
        for b in range(nb):
            prev = mparts[(t - 1) * nb + b] if t >= 1 else None
            api.refadapt_gate(t, b, state, modes[t, b], theta, delta_max, B, H,
                              q_delta=dd[t, b] if t >= 1 else None, mass_partial_prev=prev,
                              mass_row_count=rows, forced_boundary=forced, gbar_out=gbar[t, b],
                              cue=CUE_ID[cue])
    torch.cuda.synchronize()
    gm = modes.cpu().numpy()
    gg = gbar.double().cpu().numpy()
    # Oracle, using the M the GPU sees (the float32 partial sums) and the float32 D.
    Mq = np.stack([m.double().sum(-1).cpu().numpy() / rows for m in mparts]).reshape(T, nb, B, H)
    gate = oracle.Gate(B, theta, delta_max, forced, cue)
    om = np.zeros((T, nb, B), dtype=np.int32)
    og = np.zeros((T, nb, B))
    for t in range(T):
        gate.begin_step(t)
        for b in range(nb):
            m, g = gate.decide(t, b, D.astype(np.float32).astype(np.float64)[t, b] if t >= 1 else None,
                               Mq[t - 1, b] if t >= 1 else None,
                               tie=lambda tt, bb, s: gm[tt, bb, s] == 1, tie_band=TIE_BAND)
            om[t, b] = m
            og[t, b] = g
    return gm, gg, om, og


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_gate_random_tables(cuda_ok, seed):
    rng = np.random.default_rng(seed)
    T, nb, B, H = 8, 12, 3, 24
    D = rng.uniform(0.0, 0.6, size=(T, nb, B, H))
    M = rng.uniform(0.0, 0.9, size=(T, nb, B, H))
    gm, gg, om, og = _run_gate(D, M, theta=0.1, delta_max=4)
    assert np.array_equal(gm, om)
    fin = np.isfinite(og)
    assert np.all(np.isnan(gg[~fin]))
    np.testing.assert_allclose(gg[fin], og[fin], rtol=1e-6, atol=1e-7)


def test_gate_always_refresh_forced_and_thresholds(cuda_ok):
    rng = np.random.default_rng(5)
    T, nb, B, H = 5, 7, 2, 4
    D = rng.uniform(0, 1, size=(T, nb, B, H))
    M = rng.uniform(0, 1, size=(T, nb, B, H))
    gm, _, om, _ = _run_gate(D, M, theta=0.3, delta_max=1)
    assert np.all(gm == 3) and np.array_equal(gm, om)
    gm, _, om, _ = _run_gate(D, M, theta=math.inf, delta_max=100)
    assert np.all(gm[1:] == 0) and np.array_equal(gm, om)
    gm, _, om, _ = _run_gate(D, M, theta=0.0, delta_max=100)
    assert np.all(gm[1:, 0] == 1) and np.all(gm[1:, 1:] == 2) and np.array_equal(gm, om)
    gm, _, om, _ = _run_gate(D, M, theta=math.inf, delta_max=100, forced=3)
    assert np.array_equal(gm, om)
    assert list(gm[2, :, 0]) == [0, 0, 0, 1, 2, 2, 2]


def test_gate_bounded_age(cuda_ok):
    T, nb, B, H = 9, 3, 1, 2
    D = np.zeros((T, nb, B, H))
    M = np.zeros((T, nb, B, H))
    gm, _, om, _ = _run_gate(D, M, theta=1.0, delta_max=3)
    assert np.array_equal(gm, om)
    for t in range(T):
        assert np.all(gm[t] == (3 if t % 3 == 0 else 0))


@pytest.mark.parametrize("cue,theta", [("change", 0.3), ("exposure", 0.45)])
def test_gate_ablation_cues(cuda_ok, cue, theta):
    """Sec. 5.3 / Tab. 4 trigger variants: D alone or M alone, same controller."""
    rng = np.random.default_rng(7)
    T, nb, B, H = 6, 10, 2, 24
    D = rng.uniform(0.0, 0.6, size=(T, nb, B, H))
    M = rng.uniform(0.0, 0.9, size=(T, nb, B, H))
    gm, gg, om, og = _run_gate(D, M, theta=theta, delta_max=4, cue=cue)
    assert np.array_equal(gm, om)
    fin = np.isfinite(og)
    np.testing.assert_allclose(gg[fin], og[fin], rtol=1e-6, atol=1e-7)
