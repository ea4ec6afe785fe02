"""refadapt_q_delta_noalloc: the Q change for callers that cannot allocate
device memory (for example a plugin whose host framework owns the device
memory pool, or a latency-critical loop that must not pay cudaMalloc's implicit
synchronisation). Its scratch is a static array inside the library; the result
must equal refadapt_q_delta with a caller-owned workspace bit for bit, call
after call (both run the same fixed-order reduction on the same inputs), and
Eq. 1 as the oracle computes it within the Q-change tolerance.

This file sorts last so that a run stopping at the first failure has already
run every other test; it also passes on its own in a fresh process."""
import numpy as np
import pytest
import torch

import oracle
from _helpers import D_REL, f64

pytestmark = pytest.mark.gpu


def _pair(g, B, H, n, d, drift):
    prev = (torch.randn((B, H, n, d), generator=g) / d ** 0.5).to(torch.bfloat16)
    cur = (prev.float() + drift * torch.randn((B, H, n, d), generator=g) / d ** 0.5).to(torch.bfloat16)
    return cur.cuda(), prev.cuda()


def _both(cur, prev, ws):
    from paper_2609_32415_gb300 import api
    B, H = cur.shape[:2]
    want = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
    got = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
    api.refadapt_q_delta(cur, prev, want, ws, 1e-6)
    api.refadapt_q_delta_noalloc(cur, prev, got, 1e-6)
    torch.cuda.synchronize()
    return got, want


def test_noalloc_matches_workspace_entry_point_twice(cuda_ok):
    from paper_2609_32415_gb300 import api
    B, H, d = 2, 24, 128
    g = torch.Generator().manual_seed(21)
    ws = api.q_delta_workspace(B, H)
    for call, (n, drift) in enumerate([(1000, 0.3), (4096, 0.05)]):
        cur, prev = _pair(g, B, H, n, d, drift)
        got, want = _both(cur, prev, ws)
        assert torch.isfinite(got).all(), call
        assert torch.equal(got, want), call
        ref = oracle.q_change(f64(cur), f64(prev), 1e-6)
        assert (np.abs(got.double().cpu().numpy() - ref) / np.abs(ref)).max() <= D_REL, call


def test_noalloc_rejects_sizes_beyond_its_scratch(cuda_ok):
    from paper_2609_32415_gb300 import api
    from paper_2609_32415_gb300._lib import RA_EINVAL, RA_Q_DELTA_NOALLOC_MAX_BH, RefAdaptError
    B, H, n, d = 1, RA_Q_DELTA_NOALLOC_MAX_BH + 1, 16, 64
    x = torch.zeros((B, H, n, d), dtype=torch.bfloat16, device="cuda")
    out = torch.zeros((B, H), dtype=torch.float32, device="cuda")
    with pytest.raises(RefAdaptError) as e:
        api.refadapt_q_delta_noalloc(x, x, out)
    assert e.value.status == RA_EINVAL


def test_noalloc_long_slab_uses_the_static_scratch(cuda_ok):
    """Slabs too long for one cluster of CTAs go through the path that needs
    scratch (per-slab tickets and partial sums): the static array serves it,
    on two calls in a row with different slab counts and lengths."""
    from paper_2609_32415_gb300 import api
    d = 128
    g = torch.Generator().manual_seed(22)
    for B, H, n in ((1, 2, 100000), (2, 3, 120000)):
        cur, prev = _pair(g, B, H, n, d, 0.2)
        got, want = _both(cur, prev, api.q_delta_workspace(B, H))
        assert torch.isfinite(got).all(), n
        assert torch.equal(got, want), n
        ref = oracle.q_change(f64(cur), f64(prev), 1e-6)
        assert (np.abs(got.double().cpu().numpy() - ref) / np.abs(ref)).max() <= D_REL, n
