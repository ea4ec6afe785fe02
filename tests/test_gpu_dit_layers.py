"""GPU parity of the DiT block's layers (refadapt_rope_table,
refadapt_ln_modulate, refadapt_gemm and its epilogues) against the oracle's
fp64 layers (oracle/dit.py) on the same seeded bf16 inputs.

Tolerance: every output is one bf16 rounding of a value the GPU forms in fp32
and the oracle in fp64, so the two agree except where the fp32 value lands on
the other side of a bf16 rounding boundary, a difference of one bf16 ulp
(at most 2^-7 |ref|): |got - ref| <= 2^-7 |ref| + 1e-3 rms(ref) (fp32
cancellation in long dot products), and at least 98 % of the elements are
equal."""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import BOUNDARY, COMPUTE, FULL, REUSE
from oracle import dit
from _helpers import bits, f64

pytestmark = pytest.mark.gpu


def _close(got, ref, frac=0.98):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    rms = math.sqrt(float(np.mean(ref ** 2))) + 1e-30
    bad = np.abs(got - ref) > 2.0 ** -7 * np.abs(ref) + 1e-3 * rms
    eq = float(np.mean(got == ref))
    return (not bad.any()) and eq >= frac, int(bad.sum()), eq


def _bf(shape, g, scale=1.0):
    return (torch.randn(shape, generator=g) * scale).to(torch.bfloat16)


def test_rope_table_matches_angles(cuda_ok):
    from paper_2609_32415_gb300 import api
    for n_pos, d in ((33272, 128), (100, 64)):
        t = api.rope_table(n_pos, d).cpu().double().numpy()
        ang = dit.rope_angles(np.arange(n_pos), d)
        assert np.abs(t[..., 0] - np.cos(ang)).max() < 1e-6
        assert np.abs(t[..., 1] - np.sin(ang)).max() < 1e-6


@pytest.mark.parametrize("C", [256, 3072])
def test_ln_modulate_segments_and_gating(cuda_ok, C):
    from paper_2609_32415_gb300 import api
    g = torch.Generator().manual_seed(C)
    B = 2
    rows = {"text": 40, "ref": 130, "tgt": 77}
    mode = torch.tensor([REUSE, BOUNDARY], dtype=torch.int32, device="cuda")
    segs, keep = [], {}
    for r, n in rows.items():
        # strided input: rows of a wider buffer
        wide = (_bf((B, n, C + 64), g) * 2.0 + 0.5).cuda()
        h = wide[:, :, 32:32 + C]
        x = torch.full((B, n, C), float("nan"), dtype=torch.bfloat16, device="cuda")
        shift = (torch.randn((B, C), generator=g) * 0.1).cuda()
        scale = (torch.randn((B, C), generator=g) * 0.1).cuda()
        segs.append({"h": h, "x": x, "shift": shift, "scale": scale, "gated": r == "ref"})
        keep[r] = (h, x, shift, scale)
    api.refadapt_ln_modulate(segs, C, eps=1e-6, mode=mode)
    torch.cuda.synchronize()
    for r, (h, x, shift, scale) in keep.items():
        for s in range(B):
            got = f64(x[s])
            if r == "ref" and s == 0:
                assert np.isnan(got).all()
                continue
            ref = dit.round_bf16(dit.layer_norm_modulate(f64(h[s]), shift[s].double().cpu().numpy(),
                                                         scale[s].double().cpu().numpy(), 1e-6))
            ok, nbad, eq = _close(got, ref, 0.99)
            assert ok, (r, s, nbad, eq)


def _gemm_case(B, K, N, rows_list, epi, g, gated=None, modes=None, inplace=False, tile_mode=0):
    from paper_2609_32415_gb300 import api
    from paper_2609_32415_gb300._lib import RA_EPI_GELU, RA_EPI_RESID, RA_EPI_STORE
    segs, keep = [], []
    for i, rows in enumerate(rows_list):
        a = _bf((B, rows, K), g).cuda()
        w = _bf((N, K), g, 1.0 / math.sqrt(K)).cuda()
        bias = (torch.randn(N, generator=g) * 0.1).cuda() if i != 1 else None
        sd = {"a": a, "w": w, "bias": bias, "gated": bool(gated and gated[i])}
        if epi == RA_EPI_RESID:
            resid = _bf((B, rows, N), g).cuda()
            gate = (0.3 + 0.1 * torch.randn((B, N), generator=g)).cuda()
            sd.update(resid=resid, gate=gate)
            sd["out"] = resid if inplace else torch.full((B, rows, N), float("nan"), dtype=torch.bfloat16,
                                                         device="cuda")
            keep.append((a, w, bias, resid.clone(), gate, sd["out"]))
        else:
            sd["out"] = torch.full((B, rows, N), float("nan"), dtype=torch.bfloat16, device="cuda")
            keep.append((a, w, bias, None, None, sd["out"]))
        segs.append(sd)
    mode = None if modes is None else torch.tensor(modes, dtype=torch.int32, device="cuda")
    api.refadapt_gemm(segs, N, K, epi, mode=mode, tile_mode=tile_mode)
    torch.cuda.synchronize()
    for i, (a, w, bias, resid, gate, out) in enumerate(keep):
        for s in range(B):
            got = f64(out[s])
            if gated and gated[i] and modes[s] == REUSE:
                if epi == RA_EPI_RESID and inplace:
                    np.testing.assert_array_equal(got, f64(resid[s]))
                else:
                    assert np.isnan(got).all()
                continue
            y = dit.linear(f64(a[s]), f64(w), None if bias is None else bias.double().cpu().numpy())
            if epi == RA_EPI_GELU:
                y = dit.gelu_tanh(y)
            elif epi == RA_EPI_RESID:
                y = f64(resid[s]) + gate[s].double().cpu().numpy() * y
            ok, nbad, eq = _close(got, dit.round_bf16(y))
            assert ok, (epi, i, s, nbad, eq)


# tile_mode 1: one CTA per 128 x 256 tile; 2: CTA pairs (cta_group::2) on 256 x 256 tiles.
TILE_MODES = [1, 2]


@pytest.mark.parametrize("tile_mode", TILE_MODES)
@pytest.mark.parametrize("K,N,rows", [(64, 256, [1]), (256, 768, [40, 130, 77]), (3072, 512, [300]),
                                      (512, 2048, [2500]), (128, 512, [4500, 70]), (192, 512, [700])])
def test_gemm_store_matches_oracle(cuda_ok, K, N, rows, tile_mode):
    """Tiles are numbered in bands of 16 tile rows: 4500 rows make a full band
    and a partial one of 256-row tiles (18 = 16 + 2) and of 128-row tiles
    (36 = 16 + 16 + 4), followed by a second segment."""
    from paper_2609_32415_gb300._lib import RA_EPI_STORE
    _gemm_case(2, K, N, rows, RA_EPI_STORE, torch.Generator().manual_seed(K + N), tile_mode=tile_mode)


@pytest.mark.parametrize("tile_mode", TILE_MODES)
def test_gemm_gelu_matches_oracle(cuda_ok, tile_mode):
    from paper_2609_32415_gb300._lib import RA_EPI_GELU
    _gemm_case(1, 256, 1024, [129, 200], RA_EPI_GELU, torch.Generator().manual_seed(5), tile_mode=tile_mode)


@pytest.mark.parametrize("tile_mode", TILE_MODES)
@pytest.mark.parametrize("inplace", [False, True])
def test_gemm_gated_residual_matches_oracle(cuda_ok, inplace, tile_mode):
    from paper_2609_32415_gb300._lib import RA_EPI_RESID
    _gemm_case(2, 1024, 256, [40, 256, 200], RA_EPI_RESID, torch.Generator().manual_seed(6),
               gated=[False, True, False], modes=[REUSE, COMPUTE], inplace=inplace, tile_mode=tile_mode)


@pytest.mark.parametrize("tile_mode", TILE_MODES)
def test_gemm_skips_gated_tiles_in_a_long_schedule(cuda_ok, tile_mode):
    """Three segments, the middle one gated off for one sample, enough tiles
    that every CTA walks several (both accumulators, several phases)."""
    from paper_2609_32415_gb300._lib import RA_EPI_STORE
    _gemm_case(2, 192, 1024, [700, 1500, 900], RA_EPI_STORE, torch.Generator().manual_seed(7),
               gated=[False, True, False], modes=[COMPUTE, REUSE], tile_mode=tile_mode)


@pytest.mark.parametrize("tile_mode", TILE_MODES)
@pytest.mark.parametrize("H,d,modes", [(4, 64, [FULL, BOUNDARY]), (2, 128, [REUSE, COMPUTE])])
def test_gemm_qkv_epilogue_matches_oracle(cuda_ok, H, d, modes, tile_mode):
    """QKV projection with per-head RMS norm and RoPE at the rows' joint
    positions; the reference segment is gated: REUSE writes nothing,
    BOUNDARY writes only its query (K/V stay the cached ones)."""
    from paper_2609_32415_gb300 import api
    from paper_2609_32415_gb300._lib import RA_EPI_QKV
    g = torch.Generator().manual_seed(H * d)
    B, C = 2, H * d
    n = {"text": 37, "ref": 256, "tgt": 300}
    pos0 = {"text": 0, "ref": n["text"], "tgt": n["text"] + n["ref"]}
    rope = api.rope_table(sum(n.values()), d)
    mode = torch.tensor(modes, dtype=torch.int32, device="cuda")
    segs, keep = [], {}
    for i, (r, rows) in enumerate(n.items()):
        x = _bf((B, rows, C), g).cuda()
        w = _bf((3 * C, C), g, 1.0 / math.sqrt(C)).cuda()
        bias = (torch.randn(3 * C, generator=g) * 0.02).cuda()
        qn = (1.0 + 0.1 * torch.randn(d, generator=g)).cuda()
        kn = (1.0 + 0.1 * torch.randn(d, generator=g)).cuda()
        out = [torch.full((B, H, rows, d), float("nan"), dtype=torch.bfloat16, device="cuda") for _ in range(3)]
        segs.append({"a": x, "w": w, "bias": bias, "q": out[0], "k": out[1], "v": out[2], "q_norm": qn,
                     "k_norm": kn, "pos_offset": pos0[r], "gated": r == "ref"})
        keep[r] = (x, w, bias, qn, kn, out)
    api.refadapt_gemm(segs, 3 * C, C, RA_EPI_QKV, mode=mode, rope=rope, H=H, d=d, norm_eps=1e-6,
                      tile_mode=tile_mode)
    torch.cuda.synchronize()
    for r, (x, w, bias, qn, kn, out) in keep.items():
        pos = pos0[r] + np.arange(n[r])
        for s in range(B):
            y = dit.linear(f64(x[s]), f64(w), bias.double().cpu().numpy())
            parts = [y[:, z * C:(z + 1) * C].reshape(n[r], H, d).transpose(1, 0, 2) for z in range(3)]
            want = [dit.round_bf16(dit.apply_rope(dit.rms_norm(parts[0], qn.double().cpu().numpy()), pos)),
                    dit.round_bf16(dit.apply_rope(dit.rms_norm(parts[1], kn.double().cpu().numpy()), pos)),
                    dit.round_bf16(parts[2])]
            for z in range(3):
                got = f64(out[z][s])
                skip = r == "ref" and (modes[s] == REUSE or (modes[s] == BOUNDARY and z > 0))
                if skip:
                    assert np.isnan(got).all(), (r, s, z)
                    continue
                ok, nbad, eq = _close(got, want[z])
                assert ok, (r, s, z, nbad, eq)


def test_gemm_rejects_bad_shapes(cuda_ok):
    from paper_2609_32415_gb300 import api
    from paper_2609_32415_gb300._lib import RA_EINVAL, RA_EPI_STORE, RefAdaptError
    a = torch.zeros((1, 10, 96), dtype=torch.bfloat16, device="cuda")
    w = torch.zeros((256, 96), dtype=torch.bfloat16, device="cuda")
    out = torch.zeros((1, 10, 256), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(RefAdaptError) as e:
        api.refadapt_gemm([{"a": a, "w": w, "out": out}], 256, 96, RA_EPI_STORE)   # K not a multiple of 64
    assert e.value.status == RA_EINVAL
    w2 = torch.zeros((128, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(RefAdaptError) as e:
        api.refadapt_gemm([{"a": a[:, :, :64], "w": w2, "out": out[:, :, :128]}], 128, 64,
                          RA_EPI_STORE)                                         # N not a multiple of 256
    assert e.value.status == RA_EINVAL
