"""The allocation-free local-loss entry point against the allocating one (GPU).

zl_op_local_loss_noalloc serves callers that cannot allocate device memory (their own
allocator holds the device budget, or their loop must not take the synchronisation an
allocation can imply); its scratch is a static device array shared by all calls. Two calls
in a row, with different sizes and label patterns, must each match zl_op_local_loss, which
shows that no state of the previous call leaks into the next.
"""
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    import paper_2608_07974_gb300 as pkg
    pkg.build()
    from paper_2608_07974_gb300 import binding
    return binding


def _inputs(seed, N, V, alpha, masked_every):
    g = torch.Generator(device="cuda").manual_seed(seed)
    ldz = (V + 127) // 128 * 128
    z = (3 * torch.randn(N, ldz, device="cuda", generator=g, dtype=torch.float32)).to(torch.bfloat16)
    t = (3 * torch.randn(N, ldz, device="cuda", generator=g, dtype=torch.float32)).to(torch.bfloat16)
    labels = torch.randint(0, V, (N,), device="cuda", generator=g, dtype=torch.int32)
    labels[::masked_every] = -1
    return z, t if alpha < 1 else None, labels, ldz


def test_noalloc_matches_allocating_entry_point_two_calls_in_a_row(B):
    for seed, N, V, alpha, kl_dir, every in ((1, 300, 50257, 0.5, 0, 4), (2, 37, 32000, 0.7, 1, 2)):
        z, t, labels, ldz = _inputs(seed, N, V, alpha, every)
        dz_ref = torch.empty_like(z)
        rl = torch.empty(N, device="cuda", dtype=torch.float32)
        loss_ref = torch.empty(1, device="cuda", dtype=torch.float32)
        B.zl_op_local_loss(B.ZL_DTYPE_BF16, z, t, labels, N, V, ldz, alpha, kl_dir, dz_ref, rl, loss_ref)
        dz = torch.full_like(z, float("nan"))
        loss = torch.full((1,), float("nan"), device="cuda", dtype=torch.float32)
        B.zl_op_local_loss_noalloc(B.ZL_DTYPE_BF16, z, t, labels, N, V, ldz, alpha, kl_dir, dz, loss)
        torch.cuda.synchronize()
        assert abs(float(loss) - float(loss_ref)) <= 1e-5 * max(1.0, abs(float(loss_ref)))
        assert torch.allclose(dz.float(), dz_ref.float(), rtol=1e-5, atol=1e-7)


def test_noalloc_rejects_rows_beyond_its_scratch(B):
    V, N = 512, 65537
    z = torch.zeros(1, V, device="cuda", dtype=torch.float32)
    labels = torch.zeros(1, device="cuda", dtype=torch.int32)
    with pytest.raises(B.ZLError) as e:
        B.zl_op_local_loss_noalloc(B.ZL_DTYPE_F32, z, None, labels, N, V, V, 1.0, 0, z, labels.float())
    assert e.value.status == B.ZL_ERR_ARG and "65536" in str(e.value)
