"""The seeded input generator: determinism, shapes and the drift recipe (CPU)."""
import math

import torch

from paper_2609_32415_gb300 import synth


def test_trajectory_is_deterministic_and_random_access():
    wl = synth.custom_workload(2, 3, 64, 5, 20, 17, n_blocks=2, n_steps=4)
    a = synth.Trajectory(wl)
    b = synth.Trajectory(wl)
    x3 = a.get(3, 1)
    assert torch.equal(x3, b.get(3, 1))
    assert torch.equal(a.get(1, 1), b.get(1, 1))     # earlier step restarts from 0
    assert x3.shape == (3, 2, 3, 42, 64) and x3.dtype == torch.bfloat16
    assert not torch.equal(a.get(0, 0), a.get(0, 1))  # blocks differ


def test_drift_recipe_relative_change():
    wl = synth.custom_workload(1, 4, 128, 0, 2048, 2048, n_blocks=1, n_steps=2, ref_drift=0.02,
                               tgt_drift=0.3)
    tr = synth.Trajectory(wl)
    x0, x1 = tr.get(0, 0).float(), tr.get(1, 0).float()
    for role, delta in (("ref", 0.02), ("tgt", 0.3)):
        a, b = tr.role_view(x0, role), tr.role_view(x1, role)
        rel = (b - a).norm() / a.norm()
        assert abs(rel.item() - delta) < 0.02 * delta + 3e-3
    assert abs(tr.role_view(x0, "tgt").std().item() - 1 / math.sqrt(128)) < 1e-3


def test_named_workloads_shapes():
    c2 = synth.make_workload("c2")
    assert (c2.n_text, c2.n_ref, c2.n_tgt, c2.n_blocks, c2.H, c2.d) == (256, 8192, 4096, 60, 24, 128)
    assert len(c2.ref_drift) == 60 and abs(c2.ref_drift[0] - 0.05) < 1e-12
    assert abs(c2.ref_drift[44] - 0.005) < 1e-12 and abs(c2.ref_drift[59] - 0.010) < 1e-12
    c3 = synth.make_workload("c3")
    assert c3.N == 33272 and all(-3.0 <= b <= 0.0 for b in c3.bias)
    c4 = synth.make_workload("c4")
    assert c4.n_ref == 16384 and len(set(c4.ref_drift)) == 60
    assert c4.theta > 0
    c5 = synth.make_workload("c5", total=16384, ref_frac=0.7, reuse_frac=0.5)
    assert c5.N == 16384 and c5.n_ref % 128 == 0 and c5.forced_boundary == 4
    c1 = synth.make_workload("c1")
    assert (c1.N, c1.d, c1.H, c1.theta) == (544, 64, 8, 0.05)
