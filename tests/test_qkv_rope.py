"""The QKV projection with rotate-half RoPE in one pass (GPU; the chunk function f_k of Eq. 1).

zl_op_qkv_rope forms C = A B^T (+ bias) and rotates the query and key heads of every row by the angles
of its position. Checked
  (1) bit for bit against the two-pass composition: the product alone (zl_op_gemm_ex, rounded to the
      dtype), then each pair rotated with every product and sum rounded in fp32 (torch ops on the same
      table), rounded again;
  (2) against the oracle's RoPE on the fp64 product within the rounding of the output dtype;
  (3) in one kernel launch where the bf16 tensor-core path applies (head dims 64 and 128), and through
      the product-then-RoPE path otherwise (fp32, head dim 100).
Shapes: ragged row counts, grouped KV heads, a bias, and the Llama-7B-shaped projection of 2 x 1024
tokens (4096 -> 12288) that the chunk forward runs.
"""
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu

THETA = 10000.0


@pytest.fixture(scope="module")
def B():
    import paper_2608_07974_gb300 as pkg
    pkg.build()
    from paper_2608_07974_gb300 import binding
    return binding


def _table(S, hd):
    """(cos, sin) of position s and pair i, angle s * theta^(-2i/hd), computed in fp64, stored fp32."""
    i = torch.arange(hd // 2, dtype=torch.float64)
    ang = torch.arange(S, dtype=torch.float64)[:, None] * (THETA ** (-2.0 * i / hd))[None, :]
    return torch.stack([torch.cos(ang), torch.sin(ang)], dim=-1).float()


def _two_pass(C0, cs, S, hd, rot_cols, dt):
    """The product C0 (already rounded to dt) rotated pair by pair in fp32, then rounded to dt."""
    M, N = C0.shape
    x = C0.float().clone()
    half = hd // 2
    pos = torch.arange(M, device=C0.device) % S
    c = cs[pos, :, 0][:, None, :]   # [M, 1, half]
    s = cs[pos, :, 1][:, None, :]
    h = x[:, :rot_cols].view(M, rot_cols // hd, hd)
    x1, x2 = h[..., :half].clone(), h[..., half:].clone()
    h[..., :half] = x1 * c - x2 * s    # each torch op rounds in fp32, as the kernels' explicit rounding
    h[..., half:] = x2 * c + x1 * s
    return x.to(dt)


CASES = [  # dtype, B, S, H, Hkv, hd, K, bias, fused
    ("bf16", 2, 150, 4, 2, 128, 256, False, True),
    ("bf16", 3, 111, 8, 2, 64, 192, True, True),
    ("bf16", 1, 1000, 2, 1, 128, 64, True, True),
    ("f32", 2, 64, 4, 2, 32, 128, False, False),
    ("bf16", 1, 70, 4, 4, 100, 160, False, False),
]


def _product(B, code, M, N, K, A, W, C0, bias, monkeypatch):
    """The product alone, in one split (the K order of the rotating product's single pass)."""
    with monkeypatch.context() as mp:
        mp.setenv("ZL_GEMM_TILE", "256:1")
        B.zl_op_gemm_ex(code, 0, M, N, K, A, W, C0, bias=bias)


@pytest.mark.parametrize("dts,Bt,S,H,Hkv,hd,K,use_bias,fused", CASES)
def test_qkv_rope_matches_two_pass_and_oracle(B, monkeypatch, dts, Bt, S, H, Hkv, hd, K, use_bias, fused):
    torch.manual_seed(7)
    dt = torch.bfloat16 if dts == "bf16" else torch.float32
    code = B.ZL_DTYPE_BF16 if dts == "bf16" else B.ZL_DTYPE_F32
    M, N, rot = Bt * S, (H + 2 * Hkv) * hd, (H + Hkv) * hd
    A = (torch.randn(M, K, device="cuda") / K ** 0.5).to(dt)
    W = torch.randn(N, K, device="cuda").to(dt)
    bias = torch.randn(N, device="cuda") * 0.1 if use_bias else None
    cs = _table(S, hd).cuda()
    C0 = torch.empty(M, N, device="cuda", dtype=dt)
    if fused:
        _product(B, code, M, N, K, A, W, C0, bias, monkeypatch)
    else:   # the same plan as the op's own product
        B.zl_op_gemm_ex(code, 0, M, N, K, A, W, C0, bias=bias)
    C = torch.full((M, N), float("nan"), device="cuda", dtype=dt)
    n0 = B.zl_kernel_launches()
    B.zl_op_qkv_rope(code, M, N, K, A, W, C, cs, S, hd, rot, bias=bias)
    torch.cuda.synchronize()
    launches = B.zl_kernel_launches() - n0
    assert (launches == 1) if fused else (launches >= 2), launches
    ref = _two_pass(C0, cs, S, hd, rot, dt)
    assert torch.equal(C.view(torch.int16 if dts == "bf16" else torch.int32),
                       ref.view(torch.int16 if dts == "bf16" else torch.int32)), \
        f"{(C.float() != ref.float()).sum().item()} elements differ from the two-pass composition"
    # the oracle's RoPE on the exact product, rows as B sequences of S positions
    P = A.double().cpu() @ W.double().cpu().T
    if bias is not None:
        P += bias.double().cpu()
    q = oracle.rope(P[:, :rot].reshape(Bt, S, rot // hd, hd), THETA).reshape(M, rot)
    Y = torch.cat([q, P[:, rot:]], dim=1)
    # bound per element: the product's rounding (its dot-product scale sum_k |a_k w_k|), the product
    # rounded to the dtype before the rotation, the rotation's result rounded again
    half = hd // 2
    Pa = A.double().cpu().abs() @ W.double().cpu().abs().T
    if bias is not None:
        Pa += bias.double().cpu().abs()
    ha = Pa[:, :rot].reshape(M, rot // hd, hd)
    pair = torch.cat([ha[..., :half] + ha[..., half:], ha[..., half:] + ha[..., :half]], dim=-1).reshape(M, rot)
    scale = torch.cat([pair, Pa[:, rot:]], dim=1) + Y.abs()
    u = 2.0 ** -8 if dts == "bf16" else K * 2.0 ** -23
    err = (C.double().cpu() - Y).abs()
    bad = err > u * scale + 1e-6
    assert not bad.any(), f"{bad.sum().item()} elements off the oracle; worst {(err - u * scale).max().item():.3g}"


def test_qkv_rope_llama7b_projection(B, monkeypatch):
    """The 7B-shaped projection (2 x 1024 tokens, d 4096, 32 + 32 + 32 heads of 128) in one launch,
    bit for bit the two-pass composition; the oracle on 48 sampled rows (both sequences, early and late
    positions)."""
    torch.manual_seed(3)
    Bt, S, H, hd, K = 2, 1024, 32, 128, 4096
    M, N, rot = Bt * S, 3 * H * hd, 2 * H * hd
    A = (torch.randn(M, K, device="cuda") / K ** 0.5).bfloat16()
    W = (torch.randn(N, K, device="cuda") * 0.02).bfloat16()
    cs = _table(S, hd).cuda()
    C0 = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
    _product(B, B.ZL_DTYPE_BF16, M, N, K, A, W, C0, None, monkeypatch)
    C = torch.empty_like(C0)
    n0 = B.zl_kernel_launches()
    B.zl_op_qkv_rope(B.ZL_DTYPE_BF16, M, N, K, A, W, C, cs, S, hd, rot)
    torch.cuda.synchronize()
    assert B.zl_kernel_launches() - n0 == 1
    ref = _two_pass(C0, cs, S, hd, rot, torch.bfloat16)
    assert torch.equal(C.view(torch.int16), ref.view(torch.int16))
    rows = torch.tensor(list(range(0, 8)) + list(range(1016, 1032)) + list(range(2024, 2048)))
    P = A[rows].double().cpu() @ W.double().cpu().T
    pos = rows % S
    i = torch.arange(hd // 2, dtype=torch.float64)
    ang = pos.double()[:, None] * (THETA ** (-2.0 * i / hd))[None, :]
    c, s = torch.cos(ang)[:, None, :], torch.sin(ang)[:, None, :]
    h = P[:, :rot].reshape(len(rows), rot // hd, hd)
    x1, x2 = h[..., :hd // 2], h[..., hd // 2:]
    Y = torch.cat([torch.cat([x1 * c - x2 * s, x2 * c + x1 * s], dim=-1).reshape(len(rows), rot), P[:, rot:]], 1)
    pair = torch.cat([(x1.abs() + x2.abs()), (x1.abs() + x2.abs())], dim=-1).reshape(len(rows), rot)
    scale = torch.cat([pair, P[:, rot:].abs()], 1) + Y.abs()
    err = (C[rows.cuda()].double().cpu() - Y).abs()
    assert (err <= 2.0 ** -8 * scale + 1e-6).all()


def test_qkv_rope_rejects_bad_heads(B):
    A = torch.zeros(4, 16, device="cuda", dtype=torch.bfloat16)
    W = torch.zeros(96, 16, device="cuda", dtype=torch.bfloat16)
    C = torch.zeros(4, 96, device="cuda", dtype=torch.bfloat16)
    cs = _table(4, 32).cuda()
    with pytest.raises(B.ZLError):
        B.zl_op_qkv_rope(B.ZL_DTYPE_BF16, 4, 96, 16, A, W, C, cs, 4, 32, 80)   # not whole heads
    with pytest.raises(B.ZLError):
        B.zl_op_qkv_rope(B.ZL_DTYPE_BF16, 4, 96, 16, A, W, C, cs, 4, 32, 128)  # beyond N
