"""The allocation-free local-loss entry point against the allocating one (GPU).

zl_op_local_loss_noalloc serves callers that cannot allocate device memory (their own
allocator holds the device budget, or their loop must not take the synchronisation an
allocation can imply); its scratch is a static device array shared by all calls. Two calls
in a row, with different sizes and label patterns, must each match zl_op_local_loss, which
shows that no state of the previous call leaks into the next. The same calls are checked
against the oracle's loss and its autograd gradient, in fp32 and bf16, and around them the
device's default memory pool and torch's allocator must not move.
"""
import ctypes
import os

import pytest
import torch

import oracle

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


def _oracle_loss(z, t, labels, V, alpha, kl_dir):
    """Loss and dL/dz of the local objective (Eq. 3-5) by the oracle, in fp64 on the same values."""
    zz = z[:, :V].double().cpu().requires_grad_(True)
    tt = None if t is None else t[:, :V].double().cpu()
    L = oracle.local_objective(zz, tt, labels.cpu(), alpha, kl_dir)
    (dz,) = torch.autograd.grad(L, zz)
    return float(L.detach()), dz


def _default_pool():
    """(get, reset_high) over the current device's default memory pool through the CUDA runtime, or None
    where the toolkit's runtime library is not at its usual place."""
    path = "/usr/local/cuda/lib64/libcudart.so"
    if not os.path.exists(path):
        return None
    rt = ctypes.CDLL(path)
    pool = ctypes.c_void_p()
    assert rt.cudaDeviceGetDefaultMemPool(ctypes.byref(pool), torch.cuda.current_device()) == 0
    RESERVED_CUR, USED_CUR, USED_HIGH = 0x5, 0x7, 0x8

    def get(attr):
        v = ctypes.c_uint64()
        assert rt.cudaMemPoolGetAttribute(pool, attr, ctypes.byref(v)) == 0
        return v.value

    def reset_high():
        z = ctypes.c_uint64(0)
        assert rt.cudaMemPoolSetAttribute(pool, USED_HIGH, ctypes.byref(z)) == 0

    return get, reset_high, (RESERVED_CUR, USED_CUR, USED_HIGH)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_noalloc_matches_oracle_and_allocates_nothing(B, dtype):
    """fp32 without a teacher (alpha = 1, t = NULL) and bf16 with one, each twice in a row: loss and dz
    against the oracle (the tolerances of the allocating kernel's own oracle test), and no allocation."""
    torch.manual_seed(7)
    td, code = (torch.float32, B.ZL_DTYPE_F32) if dtype == "f32" else (torch.bfloat16, B.ZL_DTYPE_BF16)
    cases = [(96, 1000, 1.0, 0), (41, 32000, 0.5, 1)] if dtype == "f32" else [(50, 50257, 0.5, 0), (7, 512, 1.0, 0)]
    ins = []
    for N, V, alpha, kl_dir in cases:
        ldz = (V + 127) // 128 * 128
        z = (3 * torch.randn(N, ldz)).to(td).cuda()
        t = (3 * torch.randn(N, ldz)).to(td).cuda() if alpha < 1 else None
        labels = torch.randint(0, V, (N,), dtype=torch.int32)
        labels[1::3] = -1
        ins.append((N, V, ldz, alpha, kl_dir, z, t, labels.cuda(), torch.empty_like(z),
                    torch.full((1,), float("nan"), device="cuda")))
    torch.cuda.synchronize()
    pool = _default_pool()
    if pool:
        get, reset_high, (RES, CUR, HIGH) = pool
        reset_high()
        before = (get(RES), get(CUR))
    alloc0 = torch.cuda.memory_allocated()
    for N, V, ldz, alpha, kl_dir, z, t, labels, dz, loss in ins:
        B.zl_op_local_loss_noalloc(code, z, t, labels, N, V, ldz, alpha, kl_dir, dz, loss)
    torch.cuda.synchronize()
    assert torch.cuda.memory_allocated() == alloc0
    if pool:
        assert (get(RES), get(CUR)) == before and get(HIGH) == before[1]
    for N, V, ldz, alpha, kl_dir, z, t, labels, dz, loss in ins:
        L, dref = _oracle_loss(z.float(), None if t is None else t.float(), labels, V, alpha, kl_dir)
        assert abs(float(loss) - L) <= 1e-5 * max(1.0, abs(L)), (N, V, float(loss), L)
        out = dz.float().cpu().double()
        assert float(out[:, V:].abs().max()) == 0.0 if ldz > V else True
        err = float((out[:, :V] - dref).abs().max())
        assert err <= (2e-5 if dtype == "f32" else 1e-2) * float(dref.abs().max()) + 1e-9, (N, V, err)
