"""refadapt_q_delta_gate (the Q change with the gate in the same launch) against
refadapt_q_delta followed by refadapt_gate: D, modes, gbar, M and the
controller state bit for bit, over a trajectory of blocks and steps, on both
paths of the Q change, for every cue; and D against the oracle's Eq. 1."""
import numpy as np
import pytest
import torch

import oracle
from _helpers import D_REL, bits

pytestmark = pytest.mark.gpu


def _trajectory(B, H, n, d, T, nb, seed):
    g = torch.Generator().manual_seed(seed)
    sd = 1.0 / d ** 0.5
    q = [[(torch.randn((B, H, n, d), generator=g) * sd).to(torch.bfloat16).cuda()] for _ in range(nb)]
    for b in range(nb):
        for t in range(1, T):
            step = 0.02 + 0.1 * b
            q[b].append((q[b][-1].float() + step * sd * torch.randn((B, H, n, d), generator=g).cuda()
                         ).to(torch.bfloat16))
    return q


def _run(q, B, H, T, nb, L, theta, delta_max, forced, cue, fused, seed=5):
    from paper_2609_32415_gb300 import api
    g = torch.Generator().manual_seed(seed)
    state = api.new_state(B)
    ws = api.q_delta_workspace(B, H)
    rows = 4096
    mass = [(torch.rand((B, H, L), generator=g) * (0.3 * rows / L)).cuda() for _ in range(nb)]
    D = torch.full((T, nb, B, H), float("nan"), device="cuda")
    modes = torch.full((T, nb, B), -1, dtype=torch.int32, device="cuda")
    gbar = torch.zeros((T, nb, B), device="cuda")
    M = torch.zeros((T, nb, B, H), device="cuda")
    states = []
    for t in range(T):
        for b in range(nb):
            if t == 0:
                api.refadapt_gate(t, b, state, modes[t, b], theta, delta_max, B, H, mass_row_count=rows,
                                  forced_boundary=forced, gbar_out=gbar[t, b], m_out=M[t, b], cue=cue)
            elif fused:
                api.refadapt_q_delta_gate(q[b][t], q[b][t - 1], D[t, b], ws, t, b, state, modes[t, b], theta,
                                          delta_max, mass[b], rows, forced_boundary=forced, gbar_out=gbar[t, b],
                                          m_out=M[t, b], cue=cue)
            else:
                api.refadapt_q_delta(q[b][t], q[b][t - 1], D[t, b], ws)
                api.refadapt_gate(t, b, state, modes[t, b], theta, delta_max, B, H, q_delta=D[t, b],
                                  mass_partial_prev=mass[b], mass_row_count=rows, forced_boundary=forced,
                                  gbar_out=gbar[t, b], m_out=M[t, b], cue=cue)
            states.append(state.clone())
    torch.cuda.synchronize()
    return D, modes, gbar, M, states


def _same(x, y):
    if x.is_floating_point():
        return torch.equal(torch.isnan(x), torch.isnan(y)) and torch.equal(x.nan_to_num(), y.nan_to_num())
    return torch.equal(x, y)


CASES = [
    # (B, H, n, d, L): one cluster per slab; several samples; d = 64
    (1, 24, 4096, 128, 33),
    (2, 3, 700, 128, 7),
    (3, 4, 515, 64, 5),
    # slabs too long for one cluster: the multi-block path, the gate as a second launch
    (1, 2, 100000, 128, 4),
    # one row, one head
    (1, 1, 1, 64, 1),
    # more slabs than clusters fit at once: the multi-block path
    (4, 40, 300, 128, 3),
]


@pytest.mark.parametrize("B,H,n,d,L", CASES, ids=["24heads", "B2", "d64", "multiblock", "one-row", "160slabs"])
@pytest.mark.parametrize("cue", [0, 1, 2], ids=["product", "change", "exposure"])
def test_fused_gate_equals_two_calls(cuda_ok, B, H, n, d, L, cue):
    T, nb = 3, 3
    q = _trajectory(B, H, n, d, T, nb, seed=11 + n)
    theta = {0: 0.004, 1: 0.08, 2: 0.05}[cue]
    a = _run(q, B, H, T, nb, L, theta, 100, -1, cue, fused=True)
    b_ = _run(q, B, H, T, nb, L, theta, 100, -1, cue, fused=False)
    for x, y in zip(a[:4], b_[:4]):
        assert _same(x, y)
    for sx, sy in zip(a[4], b_[4]):
        assert torch.equal(sx, sy)
    # D itself against the oracle's Eq. 1 on the same bf16 inputs
    for t in range(1, T):
        for blk in range(nb):
            want = oracle.q_change(oracle.bf16_to_f64(bits(q[blk][t])), oracle.bf16_to_f64(bits(q[blk][t - 1])))
            rel = np.abs(a[0][t, blk].double().cpu().numpy() - want) / want
            assert rel.max() <= D_REL, (t, blk, rel.max())


def test_fused_gate_forced_boundary_and_full_refresh(cuda_ok):
    """A forced boundary at block 1 and delta_max = 2 (step 2 refreshes fully):
    the latch, the boundary and the full-step flag carry across fused calls."""
    B, H, n, d, T, nb = 2, 4, 600, 128, 4, 4
    q = _trajectory(B, H, n, d, T, nb, seed=3)
    a = _run(q, B, H, T, nb, 5, 0.1, 2, 1, 0, fused=True)
    b_ = _run(q, B, H, T, nb, 5, 0.1, 2, 1, 0, fused=False)
    for x, y in zip(a[:4], b_[:4]):
        assert _same(x, y)
    modes = a[1].cpu().numpy()
    assert list(modes[1, :, 0]) == [0, 1, 2, 2] and (modes[2] == 3).all() and list(modes[3, :, 1]) == [0, 1, 2, 2]


def test_fused_gate_rejects_bad_arguments(cuda_ok):
    from paper_2609_32415_gb300 import api
    from paper_2609_32415_gb300._lib import RA_EINVAL, RefAdaptError
    B, H = 1, 2
    q = torch.zeros((B, H, 64, 128), dtype=torch.bfloat16, device="cuda")
    ws = api.q_delta_workspace(B, H)
    D = torch.zeros((B, H), device="cuda")
    state = api.new_state(B)
    mode = torch.zeros(B, dtype=torch.int32, device="cuda")
    mass = torch.zeros((B, H, 2), device="cuda")
    with pytest.raises(RefAdaptError) as e:   # step 0 has no Q change
        api.refadapt_q_delta_gate(q, q, D, ws, 0, 0, state, mode, 0.1, 4, mass, 256)
    assert e.value.status == RA_EINVAL
    with pytest.raises(RefAdaptError) as e:   # workspace of the size before the ticket was added
        api.refadapt_q_delta_gate(q, q, D, ws[:-256], 1, 0, state, mode, 0.1, 4, mass, 256)
    assert e.value.status == RA_EINVAL
    with pytest.raises(RefAdaptError) as e:   # unknown cue (a gate argument)
        api.refadapt_q_delta_gate(q, q, D, ws, 1, 0, state, mode, 0.1, 4, mass, 256, cue=7)
    assert e.value.status == RA_EINVAL
