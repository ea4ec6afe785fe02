"""GPU parity of refadapt_joint_attn's fused reference-cache update (Eq. 11).

Samples in COMPUTE or FULL attend to this step's reference rows and leave them
in the cache slot (bit for bit) with a_b = t; REUSE and BOUNDARY samples attend
to the cache slot and leave it untouched. O and M follow the oracle on the
rows each sample attends to, and equal the unfused path (cache update, then
attention on the slot) bit for bit."""
import math

import pytest
import torch

from _helpers import M_ABS, ROLES, empty_outputs, make_segments, mass_from_partials, o_close, oracle_block

pytestmark = pytest.mark.gpu

REUSE, BOUNDARY, COMPUTE, FULL = 0, 1, 2, 3
STEP = 5


def _stale(B, H, d, n_ref, seed):
    """A cache slot holding older reference Q/K/V."""
    g = torch.Generator().manual_seed(seed)
    sd = 1.0 / math.sqrt(d)
    return [(torch.randn((B, H, n_ref, d), generator=g) * sd).to(torch.bfloat16).cuda() for _ in range(3)]


def _attend(segs, slot, n, modes, B, H, d, fused, a_b):
    from paper_2609_32415_gb300 import api
    out = empty_outputs(B, H, d, n)
    mp = torch.full((B, H, api.refadapt_mass_partial_len(n["text"], n["tgt"])), float("nan"),
                    dtype=torch.float32, device="cuda")
    mode_t = torch.tensor(modes, dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    if not fused:
        api.refadapt_ref_cache_update(segs["ref"][1], segs["ref"][2], slot[1], slot[2], mode_t, STEP, a_b,
                                      x_src=segs["ref"][0], x_cache=slot[0])
    api.refadapt_joint_attn((segs["text"][0], slot[0], segs["tgt"][0]), (segs["text"][1], slot[1], segs["tgt"][1]),
                            (segs["text"][2], slot[2], segs["tgt"][2]), [out[r] for r in ROLES], mp, mode=mode_t,
                            err_word=err, ref_fresh=segs["ref"] if fused else None,
                            a_b=a_b if fused else None, step=STEP)
    torch.cuda.synchronize()
    api.refadapt_check_error(err)
    return out, mp


SHAPES = [
    dict(text=33, ref=300, tgt=200),   # ragged reference tail (2 tiles + 44 rows)
    dict(text=0, ref=129, tgt=130),    # no text: the K/V-storing CTA is a reference-row CTA
    dict(text=130, ref=700, tgt=127),  # six reference tiles, three reference Q-tile pairs
    dict(text=5, ref=1, tgt=1),        # one reference row
]


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("modes", [[COMPUTE, REUSE], [BOUNDARY, FULL], [FULL, COMPUTE]])
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "%d-%d-%d" % (s["text"], s["ref"], s["tgt"]))
def test_fused_cache_update_matches_oracle_and_unfused(cuda_ok, d, modes, shape):
    n = shape
    B, H = 2, 3
    segs = make_segments(B, H, d, n, gen=torch.Generator().manual_seed(21 + d))
    slot0 = _stale(B, H, d, n["ref"], 99)
    slot_f = [x.clone() for x in slot0]
    slot_u = [x.clone() for x in slot0]
    ab_f = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    ab_u = ab_f.clone()
    out_f, mp_f = _attend(segs, slot_f, n, modes, B, H, d, True, ab_f)
    out_u, mp_u = _attend(segs, slot_u, n, modes, B, H, d, False, ab_u)
    sc = 1.0 / math.sqrt(d)
    M = mass_from_partials(mp_f, n["tgt"])
    for s in range(B):
        refresh = modes[s] in (COMPUTE, FULL)
        # rows this sample attends to: fresh reference rows, or the slot's
        seen = {r: list(segs[r]) for r in ROLES}
        if not refresh:
            seen["ref"] = [x for x in slot0]
        ref = oracle_block(seen, s, modes[s], sc)
        for r in ROLES:
            if ref["O"][r] is None:
                assert torch.isnan(out_f[r][s].float()).all(), "reuse wrote reference rows"
                continue
            ok, worst, nw = o_close(out_f[r][s].double().cpu().numpy(), ref["O"][r])
            assert ok, (s, r, worst, nw)
        assert abs(M[s] - ref["M"]).max() <= M_ABS
        for z in range(3):
            want = segs["ref"][z][s] if refresh else slot0[z][s]
            assert torch.equal(slot_f[z][s], want), ("cache slot", s, "qkv"[z])
        assert int(ab_f[s]) == (STEP if refresh else -1)
    # the same arithmetic on the same rows as the unfused path
    for r in ROLES:
        assert torch.equal(out_f[r].nan_to_num(7.0), out_u[r].nan_to_num(7.0)), r
    assert torch.equal(mp_f, mp_u)
    for z in range(3):
        assert torch.equal(slot_f[z], slot_u[z])
    assert torch.equal(ab_f, ab_u)


def test_fused_cache_update_strided_slot_and_joint_inputs(cuda_ok):
    """Fresh rows as slices of joint [B, H, N, d] tensors, the slot a slice of
    a [blocks, B, H, n, d] cache: TMA loads and stores follow the strides and
    write nothing outside the slot."""
    n = dict(text=40, ref=260, tgt=170)
    B, H, d = 2, 2, 128
    segs = make_segments(B, H, d, n, layout="joint", gen=torch.Generator().manual_seed(31))
    g = torch.Generator().manual_seed(32)
    cache = [(torch.randn((3, B, H, n["ref"], d), generator=g) / 11.3).to(torch.bfloat16).cuda() for _ in range(3)]
    before = [c.clone() for c in cache]
    slot = [c[1] for c in cache]
    ab = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    out, mp = _attend(segs, slot, n, [FULL, REUSE], B, H, d, True, ab)
    for z in range(3):
        assert torch.equal(cache[z][1][0], segs["ref"][z][0])
        assert torch.equal(cache[z][1][1], before[z][1][1])
        assert torch.equal(cache[z][0], before[z][0]) and torch.equal(cache[z][2], before[z][2])
    ref = oracle_block(segs, 0, FULL, 1 / math.sqrt(d))
    for r in ROLES:
        assert o_close(out[r][0].double().cpu().numpy(), ref["O"][r])[0], r
    assert ab.tolist() == [STEP, -1]


def test_fused_cache_update_in_place_keys(cuda_ok):
    """Reference K/V already in the slot (the producer wrote them there): read
    in place, nothing copied; the query is still copied; a_b still stamped."""
    from paper_2609_32415_gb300 import api
    n = dict(text=16, ref=200, tgt=150)
    B, H, d = 1, 2, 128
    segs = make_segments(B, H, d, n, gen=torch.Generator().manual_seed(41))
    slot_q = torch.zeros_like(segs["ref"][0])
    out = empty_outputs(B, H, d, n)
    mp = torch.zeros((B, H, api.refadapt_mass_partial_len(16, 150)), device="cuda")
    ab = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    api.refadapt_joint_attn((segs["text"][0], slot_q, segs["tgt"][0]), [segs[r][1] for r in ROLES],
                            [segs[r][2] for r in ROLES], [out[r] for r in ROLES], mp,
                            mode=torch.tensor([COMPUTE], dtype=torch.int32, device="cuda"),
                            ref_fresh=segs["ref"], a_b=ab, step=STEP)
    torch.cuda.synchronize()
    assert torch.equal(slot_q, segs["ref"][0])
    assert ab.tolist() == [STEP]
    ref = oracle_block(segs, 0, COMPUTE, 1 / math.sqrt(d))
    for r in ROLES:
        assert o_close(out[r][0].double().cpu().numpy(), ref["O"][r])[0], r


def test_fused_cache_update_invalid_arguments(cuda_ok):
    from paper_2609_32415_gb300 import api
    from paper_2609_32415_gb300._lib import RA_EINVAL, RefAdaptError
    n = dict(text=8, ref=64, tgt=32)
    B, H, d = 1, 1, 128
    segs = make_segments(B, H, d, n)
    slot = _stale(B, H, d, 64, 1)
    out = empty_outputs(B, H, d, n)
    mp = torch.zeros((B, H, api.refadapt_mass_partial_len(8, 32)), device="cuda")
    q = (segs["text"][0], slot[0], segs["tgt"][0])
    k = (segs["text"][1], slot[1], segs["tgt"][1])
    v = (segs["text"][2], slot[2], segs["tgt"][2])
    o = [out[r] for r in ROLES]
    fq, fk, fv = segs["ref"]
    bad = [
        (fq, fk[:, :, :63], fv[:, :, :63]),     # fewer rows than the slot
        (fq, slot[1], fv),                      # K in place, V copied
        (fq, slot[1].as_strided(slot[1].shape, (2 * 64 * 128, 64 * 128, 128, 1)),
         slot[2].as_strided(slot[2].shape, (2 * 64 * 128, 64 * 128, 128, 1))),  # the slot's pointers, other strides
        (None, fk, fv),                         # query rows run but no fresh query
    ]
    for case in bad:
        with pytest.raises(RefAdaptError) as e:
            api.refadapt_joint_attn(q, k, v, o, mp, ref_fresh=case)
        assert e.value.status == RA_EINVAL
    with pytest.raises(RefAdaptError) as e:  # a fresh query but no reference query rows
        api.refadapt_joint_attn((q[0], None, q[2]), k, v, (o[0], None, o[2]), mp, ref_fresh=(fq, fk, fv))
    assert e.value.status == RA_EINVAL
    with pytest.raises(ValueError):
        api.refadapt_joint_attn(q, k, v, o, mp, a_b=torch.zeros(1, dtype=torch.int32, device="cuda"))
