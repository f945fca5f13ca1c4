"""Single kernels through the C ABI against the oracle's definitions (GPU)."""
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    import paper_2608_07974_gb300 as pkg
    pkg.build()
    from paper_2608_07974_gb300 import binding
    return binding


def _loss_ref(z, t, labels, V, alpha, kl_dir):
    zz = z[:, :V].double().cpu().requires_grad_(True)
    tt = None if t is None else t[:, :V].double().cpu()
    L = oracle.local_objective(zz, tt, labels.cpu(), alpha, kl_dir)
    rows = oracle.local_objective_rows(zz.detach(), tt, labels.cpu(), alpha, kl_dir)
    (dz,) = torch.autograd.grad(L, zz)
    return float(L), rows, dz


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("N,V,alpha,kl_dir", [(37, 512, 0.5, 0), (64, 1000, 0.3, 1), (5, 50257, 0.5, 0),
                                               (300, 32000, 1.0, 0), (1, 2, 0.7, 0)])
def test_local_loss_matches_oracle(B, dtype, N, V, alpha, kl_dir):
    torch.manual_seed(N + V)
    ldz = (V + 127) // 128 * 128
    td = torch.float32 if dtype == "f32" else torch.bfloat16
    z = (torch.randn(N, ldz) * 3).to(td).cuda()
    t = (torch.randn(N, ldz) * 3).to(td).cuda()
    labels = torch.randint(0, V, (N,), dtype=torch.int32)
    if N > 3:
        labels[::4] = -1                        # holes in Omega
    labels = labels.cuda()
    dz = torch.empty_like(z)
    rl = torch.empty(N, dtype=torch.float32, device="cuda")
    loss = torch.empty(1, dtype=torch.float32, device="cuda")
    B.zl_op_local_loss(B.ZL_DTYPE_F32 if dtype == "f32" else B.ZL_DTYPE_BF16, z, t if alpha < 1 else None, labels,
                       N, V, ldz, alpha, kl_dir, dz, rl, loss)
    torch.cuda.synchronize()
    L, rows, dref = _loss_ref(z.float(), t.float() if alpha < 1 else None, labels, V, alpha, kl_dir)
    tol = 1e-5 if dtype == "f32" else 1e-5   # math is fp32 in both cases; inputs are the same values
    assert abs(float(loss) - L) <= tol * max(1.0, abs(L))
    assert torch.allclose(rl.cpu().double(), rows, rtol=1e-5, atol=1e-5)
    out = dz.float().cpu().double()
    assert float(out[:, V:].abs().max() if ldz > V else 0.0) == 0.0           # padding columns
    err = (out[:, :V] - dref).abs().max()
    scale = dref.abs().max()
    assert float(err) <= (2e-5 if dtype == "f32" else 1e-2) * float(scale) + 1e-9


def test_loss_all_rows_outside_omega(B):
    N, V = 8, 512
    z = torch.randn(N, V, device="cuda")
    labels = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    dz = torch.empty_like(z)
    rl = torch.empty(N, device="cuda")
    loss = torch.full((1,), 7.0, device="cuda")
    B.zl_op_local_loss(0, z, None, labels, N, V, V, 1.0, 0, dz, rl, loss)
    torch.cuda.synchronize()
    assert float(loss) == 0.0 and float(dz.abs().max()) == 0.0


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("M,N,K", [(256, 384, 128), (130, 70, 50), (1, 1, 1), (512, 768, 320)])
def test_gemm_matches_matmul(B, dtype, mode, M, N, K):
    torch.manual_seed(M * 7 + N * 3 + K)
    td = torch.float32 if dtype == "f32" else torch.bfloat16
    if mode == 0:
        a, b = torch.randn(M, K).to(td), torch.randn(N, K).to(td)
        ref = a.double() @ b.double().T
    elif mode == 1:
        a, b = torch.randn(M, K).to(td), torch.randn(K, N).to(td)
        ref = a.double() @ b.double()
    else:
        a, b = torch.randn(K, M).to(td), torch.randn(K, N).to(td)
        ref = a.double().T @ b.double()
    c0 = torch.randn(M, N) if mode == 2 else None
    c = c0.clone().cuda() if mode == 2 else torch.empty(M, N, dtype=td, device="cuda")
    B.zl_op_gemm(0 if dtype == "f32" else 1, mode, M, N, K, a.cuda(), b.cuda(), c)
    torch.cuda.synchronize()
    out = c.double().cpu()
    if mode == 2:
        ref = ref + c0.double()
    tol = 1e-5 if dtype == "f32" or mode == 2 else 8e-3
    err = float((out - ref).abs().max()) / max(float(ref.abs().max()), 1.0)
    assert err <= tol, err
