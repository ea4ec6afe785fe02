"""Algorithm 1 driven from plain C through the C ABI alone
(tests/c_client/algorithm1_client.c: the gate, the Q change with the gate,
the joint attention with the fused cache write), against the oracle's closed
loop on the same seeded bf16 inputs: modes, gbar, D, M, O and a_b."""
import os
import subprocess

import numpy as np
import pytest

import oracle
from _helpers import D_REL, M_ABS, TIE_BAND, bits, o_close

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ROLES = ("text", "ref", "tgt")


def _cuda_home():
    for c in (os.environ.get("CUDA_HOME"), "/usr/local/cuda"):
        if c and os.path.exists(os.path.join(c, "include", "cuda_runtime.h")):
            return c
    pytest.skip("no CUDA toolkit headers for the C client")


def test_c_client_runs_algorithm1_against_the_oracle(cuda_ok, tmp_path):
    from paper_2609_32415_gb300 import _lib, synth
    B, H, d, nt, nr, ng, nb, T = 2, 4, 128, 33, 300, 200, 4, 5
    theta, delta_max = 0.08, 3
    wl = synth.custom_workload(B, H, d, nt, nr, ng, n_blocks=nb, n_steps=T, ref_drift=0.05,
                               tgt_drift=[0.05, 0.1, 0.3, 0.4], theta=theta, delta_max=delta_max)
    traj = synth.Trajectory(wl, device="cpu")
    X = {(t, b): traj.get(t, b) for t in range(T) for b in range(nb)}
    inp = tmp_path / "in.bin"
    with open(inp, "wb") as f:
        for t in range(T):
            for b in range(nb):
                f.write(bits(X[(t, b)]).tobytes())

    cuda = _cuda_home()
    exe = tmp_path / "client"
    pkg = os.path.dirname(_lib.LIB_PATH)
    subprocess.run(["gcc", "-std=c99", "-O2", "-I", os.path.join(ROOT, "include"), "-I", os.path.join(cuda, "include"),
                    os.path.join(ROOT, "tests", "c_client", "algorithm1_client.c"), "-o", str(exe),
                    "-L", pkg, "-lrefadapt", "-Wl,-rpath," + pkg,
                    "-L", os.path.join(cuda, "lib64"), "-lcudart", "-Wl,-rpath," + os.path.join(cuda, "lib64")],
                   check=True)
    out = tmp_path / "out.bin"
    res = subprocess.run([str(exe), str(B), str(H), str(d), str(nt), str(nr), str(ng), str(nb), str(T),
                          repr(theta), str(delta_max), str(inp), str(out)], capture_output=True, text=True,
                         timeout=300)
    assert res.returncode == 0, res.stdout + res.stderr

    # parse the client's records
    raw_out = np.fromfile(out, dtype=np.uint8)
    pos = 0

    def take(dtype, count):
        nonlocal pos
        nbytes = np.dtype(dtype).itemsize * count
        a = raw_out[pos:pos + nbytes].view(dtype)
        pos += nbytes
        return a

    recs = {}
    nrole = {"text": nt, "ref": nr, "tgt": ng}
    for t in range(T):
        for b in range(nb):
            r = {"mode": take(np.int32, B).copy(), "gbar": take(np.float32, B).copy(),
                 "D": take(np.float32, B * H).reshape(B, H).astype(np.float64),
                 "M": take(np.float32, B * H).reshape(B, H).astype(np.float64)}
            for role in ROLES:
                r[role] = oracle.bf16_to_f64(take(np.uint16, B * H * nrole[role] * d).copy()).reshape(
                    B, H, nrole[role], d)
            r["a_b"] = take(np.int32, B).copy()
            recs[(t, b)] = r
    assert pos == raw_out.size

    modes = np.array([[recs[(t, b)]["mode"] for b in range(nb)] for t in range(T)])
    off = wl.offsets()

    def raw(t, b):
        x = X[(t, b)]
        return {r: tuple(bits(x[z, :, :, off[r]:off[r] + wl.n[r], :]) for z in range(3)) for r in ROLES}

    rec = oracle.closed_loop(raw, T, nb, B, theta=theta, delta_max=delta_max, eps=wl.eps,
                             tie=lambda t, b, s: modes[t, b, s] == 1)
    last_mat = np.full((nb, B), -1)
    for t in range(T):
        for b in range(nb):
            o, c = rec[t][b], recs[(t, b)]
            assert list(c["mode"]) == o["mode"], (t, b, c["mode"], o["mode"])
            for s in range(B):
                if o["mode"][s] in (2, 3):
                    last_mat[b, s] = t
            assert list(c["a_b"]) == list(last_mat[b]), (t, b, c["a_b"], last_mat[b])
            if t >= 1:
                assert (np.abs(c["D"] - o["D"]) / np.abs(o["D"])).max() <= D_REL, (t, b)
                ok = np.isfinite(o["gbar"]) & (np.abs(np.asarray(o["gbar"]) - theta) >= TIE_BAND)
                np.testing.assert_allclose(c["gbar"][ok], np.asarray(o["gbar"])[ok], rtol=1e-4, atol=1e-6)
                # the gate read the exposure of the previous step's executed attention
                assert np.abs(c["M"] - rec[t - 1][b]["M"]).max() <= M_ABS, (t, b)
            for s in range(B):
                for role in ROLES:
                    want = o["O"][s][role]
                    if want is None:
                        continue
                    good, worst, nw = o_close(c[role][s], want)
                    assert good, (t, b, s, role, worst, nw)
    m = modes.reshape(-1)
    assert (m == 0).any() and (m == 1).any() and (m == 2).any() and (m == 3).any()
