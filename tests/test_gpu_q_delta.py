"""GPU parity of refadapt_q_delta (paper Eq. 1 on the target query) against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from _helpers import D_REL, f64

pytestmark = pytest.mark.gpu


def _d(q_cur, q_prev, eps=1e-6, ws=None):
    from paper_2609_32415_gb300 import api
    B, H = q_cur.shape[:2]
    out = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
    ws = api.q_delta_workspace(B, H) if ws is None else ws
    api.refadapt_q_delta(q_cur, q_prev, out, ws, eps)
    torch.cuda.synchronize()
    return out.double().cpu().numpy(), ws


@pytest.mark.parametrize("B,H,n,d", [(1, 8, 256, 64), (2, 3, 1, 128), (1, 24, 4096, 128),
                                     (2, 4, 127, 128), (1, 2, 129, 64), (3, 5, 1000, 64),
                                     (1, 24, 16380, 128), (2, 20, 700, 128), (8, 25, 130, 64),
                                     (1, 1, 100000, 128), (2, 1, 200000, 64), (1, 2, 20000, 128)])
def test_q_delta_matches_oracle(cuda_ok, B, H, n, d):
    """The shapes span both unit sizes of the cluster path (8 KB units for
    slabs up to 2 MB, 12 KB beyond: (1, 24, 16380, 128)), several cluster
    sizes and both stage counts, ragged last units, and, in the last three
    (slabs too long for a cluster, or too few slabs to fill the GPU), the
    workspace path with per-slab tickets."""
    g = torch.Generator().manual_seed(n + d)
    prev = (torch.randn((B, H, n, d), generator=g) / d ** 0.5).to(torch.bfloat16)
    cur = (prev.float() + 0.3 * torch.randn((B, H, n, d), generator=g) / d ** 0.5).to(torch.bfloat16)
    got, _ = _d(cur.cuda(), prev.cuda())
    want = oracle.q_change(f64(cur), f64(prev), 1e-6)
    rel = np.abs(got - want) / np.abs(want)
    assert rel.max() <= D_REL, rel.max()


def test_q_delta_strided_views_and_workspace_reuse(cuda_ok):
    B, H, N, d = 2, 6, 700, 128
    g = torch.Generator().manual_seed(1)
    X = (torch.randn((B, N, H, d), generator=g) / d ** 0.5).to(torch.bfloat16).cuda()
    Y = (X.float() + 0.05 * torch.randn((B, N, H, d), generator=g).cuda() / d ** 0.5).to(torch.bfloat16)
    cur = Y.permute(0, 2, 1, 3)[:, :, 300:, :]
    prev = X.permute(0, 2, 1, 3)[:, :, 300:, :]
    got1, ws = _d(cur, prev)
    got2, _ = _d(cur, prev, ws=ws)
    assert np.array_equal(got1, got2)
    want = oracle.q_change(f64(cur), f64(prev), 1e-6)
    assert (np.abs(got1 - want) / want).max() <= D_REL


def test_q_delta_closed_forms(cuda_ok):
    g = torch.Generator().manual_seed(2)
    q = (torch.randn((1, 4, 333, 128), generator=g)).to(torch.bfloat16).cuda()
    got, _ = _d(q, q)
    assert np.all(got == 0.0)
    q2 = (q.float() * 2.0).to(torch.bfloat16)   # exact in bf16: D = 1 / (1 + eps/||q||)
    got, _ = _d(q2, q, eps=0.0)
    np.testing.assert_allclose(got, 1.0, rtol=1e-6)
