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
    return float(L.detach()), rows, dz


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("N,V,alpha,kl_dir", [(37, 512, 0.5, 0), (64, 1000, 0.3, 1), (5, 50257, 0.5, 0),
                                               (300, 32000, 1.0, 0), (1, 2, 0.7, 0), (6, 50257, 0.4, 1),
                                               (3, 65536, 0.5, 0), (3, 100000, 0.5, 1)])
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
    c0 = torch.randn(M, N, dtype=torch.float32) if mode == 2 else None
    c = c0.clone().cuda() if mode == 2 else torch.empty(M, N, dtype=td, device="cuda")
    B.zl_op_gemm(0 if dtype == "f32" else 1, mode, M, N, K, a.cuda(), b.cuda(), c)
    torch.cuda.synchronize()
    out = c.double().cpu()
    if mode == 2:
        ref = ref + c0.double()
    tol = 1e-5 if dtype == "f32" or mode == 2 else 8e-3
    err = float((out - ref).abs().max()) / max(float(ref.abs().max()), 1.0)
    assert err <= tol, err


def _gelu_tanh_grad(u):
    """d/du of the tanh-form GELU, by autograd through PyTorch's own GELU (fp64)."""
    u = u.detach().double().requires_grad_(True)
    (g,) = torch.autograd.grad(torch.nn.functional.gelu(u, approximate="tanh").sum(), u)
    return g


# The fused epilogue of modes 0 / 1 (zl_op_gemm_ex): bias, residual add, and the GELU-gradient product
# the GPT-2 FFN backward uses; on the tensor-core path with and without split-K ("BN:SPLITS" forces the
# tile), and on the CUDA-core path (fp32).
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("r_mode,with_bias", [(0, True), (0, False), (1, False)])
@pytest.mark.parametrize("tile", [None, "128:3"])
@pytest.mark.parametrize("M,N,K", [(256, 384, 512), (130, 136, 200)])
def test_gemm_fused_epilogue(B, monkeypatch, dtype, mode, r_mode, with_bias, tile, M, N, K):
    if dtype == "f32" and tile:
        pytest.skip("the tile override applies to the tensor-core path")
    if tile:
        monkeypatch.setenv("ZL_GEMM_TILE", tile)
    g = torch.Generator(device="cuda").manual_seed(M + 5 * N + 11 * K + mode + 3 * r_mode)
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    a = torch.randn(M, K, device="cuda", generator=g).to(td)
    b = (torch.randn(N, K, device="cuda", generator=g) if mode == 0 else
         torch.randn(K, N, device="cuda", generator=g)).to(td)
    R = (2.5 * torch.randn(M, N, device="cuda", generator=g)).to(td)
    bias = torch.randn(N, device="cuda", generator=g) if with_bias else None
    prod = a.double() @ (b.double().T if mode == 0 else b.double())
    if r_mode == 0:
        ref = prod + R.double() + (bias.double() if with_bias else 0.0)
    else:
        ref = prod * _gelu_tanh_grad(R)
    c = torch.full((M, N), float("nan"), device="cuda", dtype=td)
    B.zl_op_gemm_ex(1 if dtype == "bf16" else 0, mode, M, N, K, a, b, c, bias=bias, R=R, r_mode=r_mode)
    torch.cuda.synchronize()
    err = float((c.double() - ref).abs().max()) / float(ref.abs().max())
    assert err <= (1e-2 if dtype == "bf16" else 1e-5), err


# dW with the bias gradient: C += A^T B (tensor-core GEMM for bf16 under the default and forced tiles,
# CUDA cores for fp32) and db += column sums of A (the column-sum kernel of the bias gradients).
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("tile", [None, "64:1", "256:1", "128:3"])
@pytest.mark.parametrize("M,N,K", [(768, 768, 4096), (2304, 768, 512), (136, 264, 333)])
def test_gemm_dw_with_bias_gradient(B, monkeypatch, dtype, tile, M, N, K):
    if dtype == "f32" and tile:
        pytest.skip("the tile override applies to the tensor-core path")
    if tile:
        monkeypatch.setenv("ZL_GEMM_TILE", tile)
    g = torch.Generator(device="cuda").manual_seed(M + 7 * N + 13 * K)
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    a = torch.randn(K, M, device="cuda", generator=g).to(td)
    b = torch.randn(K, N, device="cuda", generator=g).to(td)
    c0 = torch.randn(M, N, device="cuda", generator=g)
    db0 = torch.randn(M, device="cuda", generator=g)
    c, db = c0.clone(), db0.clone()
    B.zl_op_gemm_ex(1 if dtype == "bf16" else 0, 2, M, N, K, a, b, c, bias=db)
    torch.cuda.synchronize()
    ref = c0.double() + a.double().T @ b.double()
    ref_db = db0.double() + a.double().sum(0)
    assert float((c.double() - ref).abs().max()) / float(ref.abs().max()) <= 1e-5
    assert float((db.double() - ref_db).abs().max()) / float(ref_db.abs().max()) <= 1e-5


def test_gemm_fused_epilogue_rejects_bad_arguments(B):
    a = torch.zeros(16, 16, device="cuda")
    with pytest.raises(B.ZLError):
        B.zl_op_gemm_ex(0, 2, 16, 16, 16, a, a, a, R=a, r_mode=0)    # mode 2 takes no R
    with pytest.raises(B.ZLError):
        B.zl_op_gemm_ex(0, 0, 16, 16, 16, a, a, a, r_mode=1)         # r_mode 1 needs R


# Shapes of the layer GEMMs (GPT-2 and Llama workloads) plus ragged tiles; the tensor-core path
# takes every bf16 case here. Reference: fp32 torch.matmul of the same bf16 values.
TC_SHAPES = [(0, 256, 384, 128), (0, 4096, 2304, 768), (1, 4096, 768, 3072), (2, 2304, 768, 4096),
             (0, 1024, 50304, 768), (1, 1024, 768, 50304), (0, 200, 136, 72), (1, 333, 264, 200),
             (2, 136, 264, 333), (0, 4096, 8640, 512), (1, 512, 8640, 3200), (2, 3200, 8640, 256),
             (2, 768, 768, 4096), (1, 4096, 768, 50304)]


@pytest.mark.parametrize("mode,M,N,K", TC_SHAPES)
def test_gemm_tensor_core_matches_fp32(B, mode, M, N, K):
    g = torch.Generator(device="cuda").manual_seed(M + 3 * N + 7 * K + mode)
    bf = torch.bfloat16
    if mode == 0:
        a = torch.randn(M, K, device="cuda", generator=g).to(bf)
        b = torch.randn(N, K, device="cuda", generator=g).to(bf)
        ref = a.float() @ b.float().T
    elif mode == 1:
        a = torch.randn(M, K, device="cuda", generator=g).to(bf)
        b = torch.randn(K, N, device="cuda", generator=g).to(bf)
        ref = a.float() @ b.float()
    else:
        a = torch.randn(K, M, device="cuda", generator=g).to(bf)
        b = torch.randn(K, N, device="cuda", generator=g).to(bf)
        ref = a.float().T @ b.float()
    if mode == 2:
        c0 = torch.randn(M, N, device="cuda", generator=g, dtype=torch.float32)
        c = c0.clone()
        ref = ref + c0
    else:
        c = torch.full((M, N), float("nan"), device="cuda", dtype=bf)
    B.zl_op_gemm(1, mode, M, N, K, a, b, c)
    torch.cuda.synchronize()
    err = float((c.float() - ref).abs().max()) / float(ref.abs().max())
    assert err <= (1e-5 if mode == 2 else 8e-3), err


@pytest.mark.parametrize("tile", ["64:1", "128:1:0", "256:1:0", "64:3", "128:4:0", "256:2:0",
                                  "128:1:1", "256:1:1", "128:4:1", "256:2:1"])
@pytest.mark.parametrize("mode,M,N,K", [(0, 384, 200, 1024), (1, 260, 136, 3000), (2, 136, 264, 2100),
                                        (0, 1000, 520, 777), (2, 904, 392, 640)])
def test_gemm_every_tile_and_split(B, monkeypatch, tile, mode, M, N, K):
    """Each tile width, split-K count and CTA-pair choice (forced: BN:SPLITS:PAIR) agrees with the fp32
    reference on ragged shapes, including an odd number of tile rows (the last pair's second tile lies past M)."""
    monkeypatch.setenv("ZL_GEMM_TILE", tile)
    test_gemm_tensor_core_matches_fp32(B, mode, M, N, K)


def test_gemm_tensor_core_throughput(B):
    """A 4096 x 4096 x 4096 bf16 GEMM runs far above what CUDA cores can do (tcgen05 path taken)."""
    M = N = K = 4096
    a = torch.randn(M, K, device="cuda").to(torch.bfloat16)
    b = torch.randn(N, K, device="cuda").to(torch.bfloat16)
    c = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
    for _ in range(3):
        B.zl_op_gemm(1, 0, M, N, K, a, b, c)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(10):
        B.zl_op_gemm(1, 0, M, N, K, a, b, c)
    t1.record()
    torch.cuda.synchronize()
    tflops = 2 * M * N * K * 10 / (t0.elapsed_time(t1) / 1e3) / 1e12
    print(f"tcgen05 GEMM 4096^3: {tflops:.1f} TFLOP/s")
    assert tflops > 150, tflops


# Causal attention with grouped KV heads against PyTorch's fp32 SDPA / autograd on the same values.
ATTN_SHAPES = [(2, 512, 12, 12, 64), (1, 1024, 32, 4, 64), (1, 200, 4, 4, 32), (2, 130, 4, 2, 100),
               (1, 300, 8, 8, 128), (3, 1, 4, 2, 64), (1, 64, 2, 1, 32), (2, 1500, 4, 2, 128),
               (2, 333, 6, 3, 64), (1, 130, 2, 2, 64), (1, 65, 2, 2, 128),
               # head dims the tcgen05 kernels take zero-padded to 128 or 64 (the 3B workload's is 100)
               (1, 2048, 4, 4, 100), (2, 257, 4, 2, 96), (1, 700, 2, 2, 80), (1, 300, 4, 4, 48),
               # more tiles than SMs: the persistent forward runs several tiles per CTA (O in both buffers)
               (4, 1024, 32, 4, 64), (2, 1024, 32, 32, 128), (8, 300, 16, 16, 128)]


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("Bb,S,H,Hkv,hd", ATTN_SHAPES)
def test_attention_matches_sdpa(B, dtype, Bb, S, H, Hkv, hd):
    if dtype == "f32" and S * H > 4096:
        pytest.skip("the CUDA-core path is checked on the small shapes")
    g = torch.Generator(device="cuda").manual_seed(S * 31 + H * 7 + hd)
    td = torch.bfloat16 if dtype == "bf16" else torch.float32
    W = (H + 2 * Hkv) * hd
    qkv = torch.randn(Bb * S, W, device="cuda", generator=g, dtype=torch.float32).to(td)
    dout = torch.randn(Bb * S, H * hd, device="cuda", generator=g, dtype=torch.float32).to(td)
    out = torch.empty(Bb * S, H * hd, device="cuda", dtype=td)
    lse = torch.empty(Bb, H, S, device="cuda", dtype=torch.float32)
    dq = torch.full_like(qkv, float("nan"))
    dt = B.ZL_DTYPE_BF16 if dtype == "bf16" else B.ZL_DTYPE_F32
    B.zl_op_attention(dt, qkv, out, lse, Bb, S, H, Hkv, hd)
    B.zl_op_attention_bwd(dt, qkv, out, dout, lse, dq, Bb, S, H, Hkv, hd)
    torch.cuda.synchronize()
    x = qkv.float().view(Bb, S, W).requires_grad_(True)
    q = x[..., : H * hd].view(Bb, S, H, hd).transpose(1, 2)
    k = x[..., H * hd: (H + Hkv) * hd].view(Bb, S, Hkv, hd).transpose(1, 2)
    v = x[..., (H + Hkv) * hd:].view(Bb, S, Hkv, hd).transpose(1, 2)
    rep = H // Hkv
    k, v = k.repeat_interleave(rep, 1), v.repeat_interleave(rep, 1)
    s = (q @ k.transpose(-1, -2)) / hd ** 0.5
    s = s.masked_fill(torch.triu(torch.ones(S, S, dtype=torch.bool, device="cuda"), 1), float("-inf"))
    ref_lse = torch.logsumexp(s, -1)
    ref = (torch.softmax(s, -1) @ v).transpose(1, 2).reshape(Bb * S, H * hd)
    (gx,) = torch.autograd.grad(ref, x, dout.float().view(Bb * S, H * hd), retain_graph=False)
    ref_lse = ref_lse.detach()
    tol = 2e-2 if dtype == "bf16" else 1e-5
    ref = ref.detach()
    assert float((out.float() - ref).abs().max()) <= tol * max(1.0, float(ref.abs().max()))
    assert float((lse - ref_lse).abs().max()) <= (1e-3 if dtype == "bf16" else 1e-5)
    gx = gx.view(Bb * S, W)
    err = float((dq.float() - gx).abs().max()) / max(1.0, float(gx.abs().max()))
    assert err <= (3e-2 if dtype == "bf16" else 1e-5), err
    # sections: cosine per q / k / v block must be tight
    for lo, hi in ((0, H * hd), (H * hd, (H + Hkv) * hd), ((H + Hkv) * hd, W)):
        a, r = dq.float()[:, lo:hi].reshape(-1).double(), gx[:, lo:hi].reshape(-1).double()
        if float(r.norm()) <= 1e-3 * max(1.0, float(gx.norm())):   # dQ and dK are exactly 0 when S = 1
            assert float(a.abs().max()) <= 1e-2, (lo, float(a.abs().max()))
            continue
        cos = float(a @ r / (a.norm() * r.norm() + 1e-30))
        assert cos >= 0.9995, (lo, cos)


# Scores that grow along the sequence (keys aligned with a shared direction, scaled by position): every
# 128-key block's maximum exceeds the previous one by far more than the rescale threshold, so the
# one-pass forward rescales O in TMEM at every block; outputs, log-sum-exp and gradients against the
# fp32 reference as in test_attention_matches_sdpa.
@pytest.mark.parametrize("Bb,S,H,Hkv,hd", [(1, 700, 2, 2, 64), (2, 520, 4, 2, 64), (1, 600, 2, 2, 128),
                                            (16, 520, 16, 8, 64)])
def test_attention_rescales_on_growing_scores(B, Bb, S, H, Hkv, hd):
    g = torch.Generator(device="cuda").manual_seed(S + hd)
    W = (H + 2 * Hkv) * hd
    u = torch.ones(hd, device="cuda") / hd ** 0.5
    qkv = torch.randn(Bb * S, W, device="cuda", generator=g)
    qkv[:, : (H + Hkv) * hd] *= 0.05          # small noise on queries and keys; values stay N(0, 1)
    pos = torch.arange(S, device="cuda", dtype=torch.float32).repeat(Bb)
    for hh in range(H):                       # queries ~ 4 u
        qkv[:, hh * hd:(hh + 1) * hd] += 4.0 * u
    ramp = 0.08 * hd ** 0.5 / 4.0            # keys ~ ramp pos u: scores grow by ~ 0.08 per key, ~ 15 (log2) per block
    for kk in range(Hkv):
        c = (H + kk) * hd
        qkv[:, c:c + hd] += (ramp * pos)[:, None] * u
    qkv = qkv.to(torch.bfloat16)
    dout = torch.randn(Bb * S, H * hd, device="cuda", generator=g).to(torch.bfloat16)
    out = torch.empty(Bb * S, H * hd, device="cuda", dtype=torch.bfloat16)
    lse = torch.empty(Bb, H, S, device="cuda", dtype=torch.float32)
    dq = torch.full_like(qkv, float("nan"))
    B.zl_op_attention(B.ZL_DTYPE_BF16, qkv, out, lse, Bb, S, H, Hkv, hd)
    B.zl_op_attention_bwd(B.ZL_DTYPE_BF16, qkv, out, dout, lse, dq, Bb, S, H, Hkv, hd)
    torch.cuda.synchronize()
    x = qkv.float().view(Bb, S, W).requires_grad_(True)
    q = x[..., : H * hd].view(Bb, S, H, hd).transpose(1, 2)
    k = x[..., H * hd: (H + Hkv) * hd].view(Bb, S, Hkv, hd).transpose(1, 2)
    v = x[..., (H + Hkv) * hd:].view(Bb, S, Hkv, hd).transpose(1, 2)
    rep = H // Hkv
    k, v = k.repeat_interleave(rep, 1), v.repeat_interleave(rep, 1)
    sc = (q @ k.transpose(-1, -2)) / hd ** 0.5
    sc = sc.masked_fill(torch.triu(torch.ones(S, S, dtype=torch.bool, device="cuda"), 1), float("-inf"))
    ref_lse = torch.logsumexp(sc, -1)
    ref = (torch.softmax(sc, -1) @ v).transpose(1, 2).reshape(Bb * S, H * hd)
    (gx,) = torch.autograd.grad(ref, x, dout.float().view(Bb * S, H * hd))
    # the scores really grow: maxima of the last query row over full 128-key blocks rise by more than 8
    # (log2 units)
    last = sc[0, 0, S - 1].detach() * 1.4426950408889634
    bm = torch.stack([last[j:j + 128].max() for j in range(0, S - 127, 128)])
    assert float((bm[1:] - bm[:-1]).min()) > 8.0
    ref, ref_lse = ref.detach(), ref_lse.detach()
    assert float((out.float() - ref).abs().max()) <= 2e-2 * max(1.0, float(ref.abs().max()))
    assert float((lse - ref_lse).abs().max()) <= 1e-3 * max(1.0, float(ref_lse.abs().max()))
    # Gradients: a sanity bound only. With keys sharing a large aligned component, dQ = sum_k dS K is a
    # small residue of large, mostly cancelling terms, so the bf16 rounding of dS (as in any bf16
    # backward) costs a few 1e-3 of cosine here; the forward checks above are the point of this test.
    gx = gx.view(Bb * S, W)
    for lo, hi in ((0, H * hd), (H * hd, (H + Hkv) * hd), ((H + Hkv) * hd, W)):
        a, r = dq.float()[:, lo:hi].reshape(-1).double(), gx[:, lo:hi].reshape(-1).double()
        cos = float(a @ r / (a.norm() * r.norm() + 1e-30))
        assert cos >= 0.99, (lo, cos)


@pytest.mark.parametrize("mode,M,N,K", [(0, 4096, 16, 768), (1, 4096, 2304, 16), (2, 16, 2304, 4096),
                                        (2, 16, 768, 4096), (0, 512, 16, 3072), (1, 300, 768, 16)])
def test_gemm_rank16_shapes(B, mode, M, N, K):
    """The LoRA products: one of M, N, K is the padded rank 16 (tensor-core path, partial tiles)."""
    test_gemm_tensor_core_matches_fp32(B, mode, M, N, K)
