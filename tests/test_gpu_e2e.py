"""The end-to-end pipeline bench.py times (inputs copied from page-locked host
memory, a step's gates first, reference rows copied only where a sample
materialises, every executed output row copied back to the host) returns the
oracle's closed-loop results: on a small workload whose schedule has full,
boundary, compute and reuse blocks, every step's modes as the host read them
and every executed output row on the host match Algorithm 1 run by the oracle
on the same inputs."""
import numpy as np
import pytest

import oracle
from _helpers import bits, o_close

pytestmark = pytest.mark.gpu

ROLES = ("text", "ref", "tgt")


def test_e2e_pipeline_host_results_match_oracle(cuda_ok):
    import bench
    from paper_2609_32415_gb300 import synth
    wl = synth.custom_workload(1, 3, 64, 40, 300, 200, n_blocks=4, n_steps=5, ref_drift=0.05,
                               tgt_drift=[0.05, 0.1, 0.2, 0.3], theta=0.06, delta_max=3)
    inputs = bench.make_inputs(wl, "cuda")
    keep = bench.time_e2e(wl, inputs, 0, 0, keep=[])
    assert [k["t"] for k in keep] == list(range(wl.n_steps))
    off = wl.offsets()

    def raw(t, b):
        X = inputs[t][b]
        return {r: tuple(bits(X[z, :, :, off[r]:off[r] + wl.n[r], :]) for z in range(3)) for r in ROLES}

    gpu_modes = np.array([k["modes"].numpy() for k in keep])    # [T, blocks, B]
    rec = oracle.closed_loop(raw, wl.n_steps, wl.n_blocks, wl.B, theta=wl.theta, delta_max=wl.delta_max,
                             eps=wl.eps, tie=lambda t, b, s: gpu_modes[t, b, s] == 1)
    seen = set()
    for t in range(wl.n_steps):
        for b in range(wl.n_blocks):
            r = rec[t][b]
            assert list(gpu_modes[t, b]) == r["mode"], (t, b, gpu_modes[t, b], r["mode"])
            seen.update(r["mode"])
            for role in ROLES:
                ref = r["O"][0][role]
                if ref is None:     # reference rows of a reusing block are not produced
                    continue
                got = keep[t]["out"][b][role][0].double().numpy()
                ok, worst, nw = o_close(got, ref)
                assert ok, (t, b, role, worst, nw)
    assert seen == {0, 1, 2, 3}, seen
