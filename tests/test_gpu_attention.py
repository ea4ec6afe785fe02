"""GPU parity of refadapt_joint_attn (tcgen05 kernel) against the CPU oracle."""
import math

import numpy as np
import pytest
import torch

from _helpers import (M_ABS, ROLES, empty_outputs, make_segments, mass_from_partials, o_close,
                      oracle_block)

pytestmark = pytest.mark.gpu

REUSE, BOUNDARY, COMPUTE, FULL = 0, 1, 2, 3


def _run(segs, B, H, d, n, modes, bias=None, mass_rows=0, scale=0.0, q_ref=None):
    from paper_2609_32415_gb300 import api
    out = empty_outputs(B, H, d, n)
    mp = torch.full((B, H, api.refadapt_mass_partial_len(n["text"], n["tgt"])), float("nan"),
                    dtype=torch.float32, device="cuda")
    mode_t = None if modes is None else torch.tensor(modes, dtype=torch.int32, device="cuda")
    bias_t = None if bias is None else torch.tensor(bias, dtype=torch.float32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    q = [segs[r][0] for r in ROLES]
    if q_ref is not None:
        q[1] = q_ref
    api.refadapt_joint_attn(q, [segs[r][1] for r in ROLES], [segs[r][2] for r in ROLES],
                            [out[r] for r in ROLES], mp, mode=mode_t, softmax_scale=scale,
                            ref_logit_bias=bias_t, mass_rows=mass_rows, err_word=err)
    torch.cuda.synchronize()
    api.refadapt_check_error(err)
    return out, mp


def _check(segs, out, mp, B, H, d, n, modes, bias=None, mass_rows=0, scale=None, report=None):
    sc = (1.0 / math.sqrt(d)) if not scale else scale
    n_rows = n["tgt"] + (n["text"] if mass_rows else 0)
    M_gpu = mass_from_partials(mp, n_rows)
    worst_m = 0.0
    for s in range(B):
        mode = FULL if modes is None else modes[s]
        ref = oracle_block(segs, s, mode, sc, None if bias is None else np.array(bias), mass_rows)
        for r in ROLES:
            if ref["O"][r] is None:
                # reference rows skipped: their O rows must be untouched (still NaN)
                assert torch.isnan(out[r][s].float()).all(), "reuse wrote reference rows"
                continue
            ok, worst, normwise = o_close(out[r][s].double().cpu().numpy(), ref["O"][r])
            assert ok, "O mismatch role=%s sample=%d worst=%.3g normwise=%.3g" % (r, s, worst, normwise)
        dm = np.abs(M_gpu[s] - ref["M"]).max()
        worst_m = max(worst_m, dm)
        assert dm <= M_ABS, "M mismatch sample=%d max abs err %.3g" % (s, dm)
    if report is not None:
        report.append(worst_m)
    return worst_m


SHAPES = [
    dict(text=32, ref=256, tgt=256),     # the single-block workload
    dict(text=33, ref=300, tgt=127),     # ragged tails everywhere
    dict(text=0, ref=124, tgt=129),      # no text, tails on both sides of 128
    dict(text=1, ref=1, tgt=1),          # degenerate: one row per segment
    dict(text=0, ref=0, tgt=200),        # no reference: M = 0
    dict(text=130, ref=512, tgt=260),    # several tiles per segment
]


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "%d-%d-%d" % (s["text"], s["ref"], s["tgt"]))
def test_attention_refresh_all_rows(cuda_ok, d, shape):
    B, H = 1, 3
    segs = make_segments(B, H, d, shape, gen=torch.Generator().manual_seed(d + shape["ref"]))
    out, mp = _run(segs, B, H, d, shape, None)
    _check(segs, out, mp, B, H, d, shape, None)


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("modes", [[REUSE, BOUNDARY], [COMPUTE, REUSE], [FULL, FULL]])
def test_attention_modes_per_sample(cuda_ok, d, modes):
    n = dict(text=33, ref=300, tgt=200)
    B, H = 2, 2
    segs = make_segments(B, H, d, n, gen=torch.Generator().manual_seed(7))
    out, mp = _run(segs, B, H, d, n, modes)
    _check(segs, out, mp, B, H, d, n, modes)


@pytest.mark.parametrize("layout", ["joint", "token"])
def test_attention_strided_layouts(cuda_ok, layout):
    n = dict(text=40, ref=200, tgt=170)
    B, H, d = 2, 3, 128
    segs = make_segments(B, H, d, n, layout=layout, gen=torch.Generator().manual_seed(11))
    out, mp = _run(segs, B, H, d, n, [REUSE, FULL])
    _check(segs, out, mp, B, H, d, n, [REUSE, FULL])


@pytest.mark.parametrize("d", [64, 128])
def test_attention_sharp_logits_and_bias(cuda_ok, d):
    """Logit std ~4 and +-8 biases: the running max moves across tiles, so the
    lazy O rescale path runs."""
    n = dict(text=64, ref=384, tgt=300)
    B, H = 1, 4
    segs = make_segments(B, H, d, n, std=2.0, gen=torch.Generator().manual_seed(5))
    bias = [-8.0, 8.0, 0.0, -1.5]
    out, mp = _run(segs, B, H, d, n, [BOUNDARY], bias=bias)
    _check(segs, out, mp, B, H, d, n, [BOUNDARY], bias=bias)


def test_attention_mass_rows_text_and_target(cuda_ok):
    n = dict(text=100, ref=300, tgt=150)
    B, H, d = 1, 2, 128
    segs = make_segments(B, H, d, n, gen=torch.Generator().manual_seed(3))
    out, mp = _run(segs, B, H, d, n, [REUSE], mass_rows=1)
    _check(segs, out, mp, B, H, d, n, [REUSE], mass_rows=1)


def test_attention_explicit_scale(cuda_ok):
    n = dict(text=16, ref=130, tgt=140)
    B, H, d = 1, 2, 64
    segs = make_segments(B, H, d, n, gen=torch.Generator().manual_seed(4))
    out, mp = _run(segs, B, H, d, n, None, scale=0.37)
    _check(segs, out, mp, B, H, d, n, None, scale=0.37)


def test_attention_mass_precision_is_far_below_tolerance(cuda_ok):
    """The gate's exactness needs M errors far below the 1e-3 tolerance
    (a 1e-4 band on gbar = D*M): fp32 sums keep them near 1e-6."""
    n = dict(text=256, ref=1024, tgt=512)
    B, H, d = 1, 4, 128
    segs = make_segments(B, H, d, n, gen=torch.Generator().manual_seed(9))
    out, mp = _run(segs, B, H, d, n, None)
    worst = _check(segs, out, mp, B, H, d, n, None)
    assert worst < 2e-5, worst


def test_attention_partials_deterministic(cuda_ok):
    n = dict(text=32, ref=700, tgt=333)
    B, H, d = 1, 4, 128
    segs = make_segments(B, H, d, n, gen=torch.Generator().manual_seed(12))
    out1, mp1 = _run(segs, B, H, d, n, None)
    out2, mp2 = _run(segs, B, H, d, n, None)
    assert torch.equal(mp1, mp2)
    for r in ROLES:
        assert torch.equal(out1[r], out2[r])


def test_attention_no_reference_rows_when_query_absent(cuda_ok):
    """q[ref] = None: reference rows are not computed whatever the mode."""
    n = dict(text=20, ref=140, tgt=100)
    B, H, d = 1, 2, 128
    segs = make_segments(B, H, d, n, gen=torch.Generator().manual_seed(13))
    from paper_2609_32415_gb300 import api
    out = empty_outputs(B, H, d, n)
    mp = torch.zeros((B, H, api.refadapt_mass_partial_len(20, 100)), device="cuda")
    api.refadapt_joint_attn([segs["text"][0], None, segs["tgt"][0]], [segs[r][1] for r in ROLES],
                            [segs[r][2] for r in ROLES], [out["text"], None, out["tgt"]], mp)
    torch.cuda.synchronize()
    ref = oracle_block(segs, 0, REUSE, 1 / math.sqrt(d))
    for r in ("text", "tgt"):
        assert o_close(out[r][0].double().cpu().numpy(), ref["O"][r])[0]


def test_attention_invalid_arguments(cuda_ok):
    from paper_2609_32415_gb300 import api
    from paper_2609_32415_gb300._lib import RA_EINVAL, RefAdaptError
    n = dict(text=8, ref=16, tgt=16)
    segs = make_segments(1, 1, 128, n)
    out = empty_outputs(1, 1, 128, n)
    mp = torch.zeros((1, 1, 2), device="cuda")
    bad_d = [x[..., :96] for x in (segs[r][0] for r in ROLES)]
    with pytest.raises(RefAdaptError) as e:
        api.refadapt_joint_attn(bad_d, [segs[r][1][..., :96] for r in ROLES],
                                [segs[r][2][..., :96] for r in ROLES], [out[r][..., :96] for r in ROLES], mp)
    assert e.value.status == RA_EINVAL
    buf = torch.zeros(16 * 128 + 8, dtype=torch.bfloat16, device="cuda")
    mis = buf[1:1 + 16 * 128].view(1, 1, 16, 128)
    with pytest.raises(RefAdaptError):
        api.refadapt_joint_attn([segs["text"][0], segs["ref"][0], mis], [segs[r][1] for r in ROLES],
                                [segs[r][2] for r in ROLES], [out[r] for r in ROLES], mp)


def test_attention_sampled_query_rows(cuda_ok):
    """Query rows of a role may be a row sample (here every third target row,
    a strided view) while every key row of the role is attended to."""
    from paper_2609_32415_gb300 import api
    n = dict(text=40, ref=260, tgt=301)
    B, H, d = 2, 3, 128
    segs = make_segments(B, H, d, n, gen=torch.Generator().manual_seed(14))
    q_s = segs["tgt"][0][:, :, ::3, :]
    ns = q_s.shape[2]
    o = {"text": torch.full((B, H, 40, d), float("nan"), dtype=torch.bfloat16, device="cuda"),
         "tgt": torch.full((B, H, ns, d), float("nan"), dtype=torch.bfloat16, device="cuda")}
    mp = torch.zeros((B, H, api.refadapt_mass_partial_len(40, ns)), device="cuda")
    api.refadapt_joint_attn([segs["text"][0], None, q_s], [segs[r][1] for r in ROLES], [segs[r][2] for r in ROLES],
                            [o["text"], None, o["tgt"]], mp)
    torch.cuda.synchronize()
    sub = {r: list(segs[r]) for r in ROLES}
    sub["tgt"][0] = q_s
    for s in range(B):
        ref = oracle_block(sub, s, REUSE, 1 / math.sqrt(d))
        for r in ("text", "tgt"):
            ok, worst, nw = o_close(o[r][s].double().cpu().numpy(), ref["O"][r])
            assert ok, (r, worst, nw)
        got_m = mp[s].double().sum(-1).cpu().numpy() / ns
        assert np.abs(got_m - ref["M"]).max() <= M_ABS


@pytest.mark.parametrize("stride,mass_rows", [(3, 0), (4, 1)])
def test_attention_sampled_mass_rows(cuda_ok, stride, mass_rows):
    """Mass partials over the sampled target rows 0, k, 2k, ... (and text rows
    when counted): their sum over the sampled count is the oracle's M with the
    same sample; O is unaffected."""
    import oracle
    from paper_2609_32415_gb300 import api
    n = dict(text=70, ref=300, tgt=333)
    B, H, d = 1, 3, 128
    segs = make_segments(B, H, d, n, gen=torch.Generator().manual_seed(31))
    out = empty_outputs(B, H, d, n)
    mp = torch.full((B, H, api.refadapt_mass_partial_len(n["text"], n["tgt"])), float("nan"),
                    dtype=torch.float32, device="cuda")
    api.refadapt_joint_attn([segs[r][0] for r in ROLES], [segs[r][1] for r in ROLES], [segs[r][2] for r in ROLES],
                            [out[r] for r in ROLES], mp, mass_rows=mass_rows, mass_row_stride=stride)
    torch.cuda.synchronize()
    count = (n["tgt"] + stride - 1) // stride + ((n["text"] + stride - 1) // stride if mass_rows else 0)
    M_gpu = mp.double().sum(-1).cpu().numpy() / count
    from _helpers import f64
    q = {r: f64(segs[r][0][0]) for r in ROLES}
    k = {r: f64(segs[r][1][0]) for r in ROLES}
    v = {r: f64(segs[r][2][0]) for r in ROLES}
    ref = oracle.block_attention(q, k, v, FULL, 1.0 / math.sqrt(d), mass_rows=mass_rows, sample_stride=stride)
    assert np.abs(M_gpu[0] - ref["M"]).max() < 2e-5
    for r in ROLES:
        ok, worst, nw = o_close(out[r][0].double().cpu().numpy(), ref["O"][r])
        assert ok, (r, worst)
