"""Seeded random shapes for refadapt_joint_attn: batch, heads, head dim,
segment lengths (empty text or reference segments, tails of every size),
per-sample modes, with and without the fused cache write. Each sample's O and
M against the oracle on the rows it attends to; the cache slot and a_b after
the call."""
import math

import numpy as np
import pytest
import torch

from _helpers import M_ABS, ROLES, empty_outputs, make_segments, mass_from_partials, o_close, oracle_block

pytestmark = pytest.mark.gpu

REUSE, BOUNDARY, COMPUTE, FULL = 0, 1, 2, 3
STEP = 3


def _case(seed):
    rng = np.random.default_rng(seed)
    B, H = int(rng.integers(1, 4)), int(rng.integers(1, 4))
    d = int(rng.choice([64, 128]))
    n = {"text": int(rng.choice([0, int(rng.integers(1, 300))])),
         "ref": int(rng.choice([0, int(rng.integers(1, 600))])),
         "tgt": int(rng.integers(1, 400))}
    modes = [int(m) for m in rng.integers(0, 4, size=B)]
    fused = bool(rng.integers(0, 2))
    return B, H, d, n, modes, fused


@pytest.mark.parametrize("seed", range(16))
def test_attention_random_shapes(cuda_ok, seed):
    from paper_2609_32415_gb300 import api
    B, H, d, n, modes, fused = _case(seed)
    g = torch.Generator().manual_seed(1000 + seed)
    segs = make_segments(B, H, d, n, gen=g)
    sd = 1.0 / math.sqrt(d)
    slot0 = [(torch.randn((B, H, n["ref"], d), generator=g) * sd).to(torch.bfloat16).cuda() for _ in range(3)]
    slot = [x.clone() for x in slot0]
    a_b = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    out = empty_outputs(B, H, d, n)
    mp = torch.full((B, H, api.refadapt_mass_partial_len(n["text"], n["tgt"])), float("nan"), device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    mode_t = torch.tensor(modes, dtype=torch.int32, device="cuda")
    api.refadapt_joint_attn((segs["text"][0], slot[0], segs["tgt"][0]), (segs["text"][1], slot[1], segs["tgt"][1]),
                            (segs["text"][2], slot[2], segs["tgt"][2]), [out[r] for r in ROLES], mp, mode=mode_t,
                            err_word=err, ref_fresh=segs["ref"] if fused else None,
                            a_b=a_b if fused else None, step=STEP)
    torch.cuda.synchronize()
    api.refadapt_check_error(err)
    M = mass_from_partials(mp, n["tgt"])
    for s in range(B):
        materialise = fused and modes[s] in (COMPUTE, FULL)
        seen = {r: list(segs[r]) for r in ROLES}
        if not materialise:
            seen["ref"] = list(slot0)   # without the fused write every sample reads the slot
        ref = oracle_block(seen, s, modes[s], sd)
        for r in ROLES:
            if ref["O"][r] is None:
                assert torch.isnan(out[r][s].float()).all(), (seed, s, "reuse wrote reference rows")
                continue
            ok, worst, nw = o_close(out[r][s].double().cpu().numpy(), ref["O"][r])
            assert ok, (seed, B, H, d, n, modes, fused, s, r, worst, nw)
        assert np.abs(M[s] - ref["M"]).max() <= M_ABS, (seed, s)
        for z in range(3):
            want = segs["ref"][z][s] if materialise else slot0[z][s]
            assert torch.equal(slot[z][s], want), (seed, s, z)
        assert int(a_b[s]) == (STEP if materialise else -1), (seed, s)
