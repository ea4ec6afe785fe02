"""refadapt_ref_cache_update: bit-exact materialisation per sample mode (Eq. 11)."""
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("d", [64, 128])
def test_cache_update_per_mode(cuda_ok, d):
    from paper_2609_32415_gb300 import api
    B, H, n = 4, 3, 300
    g = torch.Generator().manual_seed(d)
    src = [torch.randn((B, H, n, d), generator=g).to(torch.bfloat16).cuda() for _ in range(3)]
    dst = [torch.randn((B, H, n, d), generator=g).to(torch.bfloat16).cuda() for _ in range(3)]
    before = [x.clone() for x in dst]
    mode = torch.tensor([0, 1, 2, 3], dtype=torch.int32, device="cuda")
    a_b = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    api.refadapt_ref_cache_update(src[0], src[1], dst[0], dst[1], mode, 5, a_b, x_src=src[2], x_cache=dst[2])
    torch.cuda.synchronize()
    assert a_b.tolist() == [-7, -7, 5, 5]
    for i in range(3):
        for s in range(B):
            want = src[i][s] if s >= 2 else before[i][s]
            assert torch.equal(dst[i][s], want)


def test_cache_update_strided_and_in_place(cuda_ok):
    from paper_2609_32415_gb300 import api
    B, H, N, d = 2, 4, 900, 128
    g = torch.Generator().manual_seed(3)
    joint = torch.randn((B, N, H, d), generator=g).to(torch.bfloat16).cuda().permute(0, 2, 1, 3)
    k_src, v_src = joint[:, :, 100:600], joint[:, :, 300:800]
    k_c = torch.zeros((B, H, 500, d), dtype=torch.bfloat16, device="cuda")
    v_c = torch.zeros_like(k_c)
    mode = torch.tensor([3, 0], dtype=torch.int32, device="cuda")
    api.refadapt_ref_cache_update(k_src, v_src, k_c, v_c, mode, 2)
    torch.cuda.synchronize()
    assert torch.equal(k_c[0], k_src[0]) and torch.equal(v_c[0], v_src[0])
    assert torch.count_nonzero(k_c[1]) == 0
    a_b = torch.zeros(B, dtype=torch.int32, device="cuda")
    api.refadapt_ref_cache_update(k_c, v_c, k_c, v_c, mode, 9, a_b)   # in place: only a_b moves
    torch.cuda.synchronize()
    assert a_b.tolist() == [9, 0]
    assert torch.equal(k_c[0], k_src[0])


def test_cache_update_empty_reference(cuda_ok):
    from paper_2609_32415_gb300 import api
    e = torch.zeros((1, 2, 0, 64), dtype=torch.bfloat16, device="cuda")
    a_b = torch.zeros(1, dtype=torch.int32, device="cuda")
    api.refadapt_ref_cache_update(e, e, e, e, torch.tensor([2], dtype=torch.int32, device="cuda"), 4, a_b)
    torch.cuda.synchronize()
    assert a_b.item() == 4


def test_cache_update_bulk_path_long_slabs(cuda_ok):
    """Contiguous slabs (the executor's layout) take the bulk-copy path: video-
    sized reference slabs (16,380 rows x 24 heads), so every CTA streams many
    32 KB chunks through its ring, plus a hidden-state-like third tensor of one
    3072-wide row per token; copied bit for bit for the materialising sample
    only, a_b stamped for it only."""
    from paper_2609_32415_gb300 import api
    B, H, n, d, C = 2, 24, 16380, 128, 3072
    g = torch.Generator(device="cuda").manual_seed(11)
    src = [torch.randn((B, H, n, d), generator=g, device="cuda").to(torch.bfloat16) for _ in range(2)]
    dst = [torch.zeros((B, H, n, d), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    xs = torch.randn((B, 1, n, C), generator=g, device="cuda").to(torch.bfloat16)
    xd = torch.zeros_like(xs)
    mode = torch.tensor([2, 0], dtype=torch.int32, device="cuda")
    a_b = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    api.refadapt_ref_cache_update(src[0], src[1], dst[0], dst[1], mode, 3, a_b, x_src=xs, x_cache=xd)
    torch.cuda.synchronize()
    assert a_b.tolist() == [3, -1]
    for i in range(2):
        assert torch.equal(dst[i][0], src[i][0])
        assert torch.count_nonzero(dst[i][1]) == 0
    assert torch.equal(xd[0], xs[0]) and torch.count_nonzero(xd[1]) == 0
