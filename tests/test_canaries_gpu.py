"""Guard-band canaries around every single-kernel entry point's outputs (GPU).

compute-sanitizer is closed on this machine, so out-of-bounds writes are caught the plain way: each
output buffer is the interior of a larger allocation whose bands before and after hold a sentinel bit
pattern, and after the call (and a synchronize) the bands must still hold it. Shapes are odd and
ragged on purpose (N not a multiple of 128, V = 50257 with padding, head dims 64 / 100 / 128,
sequence tails), so every tile edge and clipped TMA store is crossed.
"""
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu
GUARD = 4096   # elements in each band (keeps the interior 16-byte aligned)
# sentinel bit patterns (NaNs no kernel writes: a NaN result would carry other payload bits)
SENT = {torch.float32: (torch.int32, 0x7FC0DEAD), torch.bfloat16: (torch.int16, 0x7FA5)}


@pytest.fixture(scope="module")
def B():
    import paper_2608_07974_gb300 as pkg
    pkg.build()
    from paper_2608_07974_gb300 import binding
    return binding


class Guarded:
    """A device buffer of n elements with sentinel bands on both sides."""

    def __init__(self, n, dtype, init=None):
        self.n, self.dtype = n, dtype
        self.full = torch.empty(n + 2 * GUARD, dtype=dtype, device="cuda")
        it, pat = SENT[dtype]
        self.full.view(it).fill_(pat)
        self.inner = self.full[GUARD:GUARD + n]
        if init is not None:
            self.inner.copy_(init.reshape(-1))

    def view(self, *shape):
        return self.inner.view(*shape)

    def check(self, what):
        torch.cuda.synchronize()
        it, pat = SENT[self.dtype]
        bits = self.full.view(it)
        assert bool((bits[:GUARD] == pat).all()), f"{what}: write before the buffer"
        assert bool((bits[GUARD + self.n:] == pat).all()), f"{what}: write past the buffer"


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("N,V,alpha", [(37, 50257, 0.5), (129, 1000, 1.0), (1, 2, 0.3)])
def test_local_loss_outputs_stay_in_bounds(B, dtype, N, V, alpha):
    td = torch.float32 if dtype == "f32" else torch.bfloat16
    code = B.ZL_DTYPE_F32 if dtype == "f32" else B.ZL_DTYPE_BF16
    ldz = (V + 127) // 128 * 128 if V > 8 else 8
    z = (3 * torch.randn(N, ldz, device="cuda")).to(td)
    t = (3 * torch.randn(N, ldz, device="cuda")).to(td) if alpha < 1 else None
    labels = torch.randint(-1, V, (N,), dtype=torch.int32, device="cuda")
    dz, rl, loss = Guarded(N * ldz, td), Guarded(N, torch.float32), Guarded(1, torch.float32)
    B.zl_op_local_loss(code, z, t, labels, N, V, ldz, alpha, 0, dz.view(N, ldz), rl.inner, loss.inner)
    for g, n in ((dz, "dz"), (rl, "row_loss"), (loss, "loss")):
        g.check(n)
    dz2, loss2 = Guarded(N * ldz, td), Guarded(1, torch.float32)
    B.zl_op_local_loss_noalloc(code, z, t, labels, N, V, ldz, alpha, 0, dz2.view(N, ldz), loss2.inner)
    dz2.check("noalloc dz")
    loss2.check("noalloc loss")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("mode", [0, 1, 2])
@pytest.mark.parametrize("M,N,K", [(130, 72, 50), (257, 200, 96), (1000, 136, 776), (4100, 264, 128)])
def test_gemm_output_stays_in_bounds(B, dtype, mode, M, N, K):
    td = torch.float32 if dtype == "f32" else torch.bfloat16
    code = B.ZL_DTYPE_F32 if dtype == "f32" else B.ZL_DTYPE_BF16
    a = torch.randn(K, M) if mode == 2 else torch.randn(M, K)
    b = torch.randn(N, K) if mode == 0 else torch.randn(K, N)
    a, b = a.to(td).cuda(), b.to(td).cuda()
    cdt = torch.float32 if mode == 2 else td
    c = Guarded(M * N, cdt, torch.zeros(M * N, dtype=cdt) if mode == 2 else None)
    B.zl_op_gemm(code, mode, M, N, K, a, b, c.view(M, N))
    c.check(f"gemm mode {mode}")
    if mode < 2:
        bias = Guarded(N, torch.float32, torch.randn(N))
        r = torch.randn(M, N, device="cuda").to(td)
        c2 = Guarded(M * N, td)
        B.zl_op_gemm_ex(code, mode, M, N, K, a, b, c2.view(M, N), bias.inner, r, 0)
        c2.check("gemm_ex bias + residual")
        bias.check("gemm_ex bias (read only)")
    elif M % 8 == 0:
        bias = Guarded(M, torch.float32, torch.zeros(M))
        c3 = Guarded(M * N, torch.float32, torch.zeros(M * N))
        B.zl_op_gemm_ex(code, 2, M, N, K, a, b, c3.view(M, N), bias.inner, None, 0)
        c3.check("gemm_ex dW")
        bias.check("gemm_ex column sums")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("Bb,S,H,Hkv,hd", [(2, 100, 4, 2, 64), (1, 300, 2, 1, 128), (1, 77, 2, 2, 100),
                                           (3, 129, 2, 2, 32)])
def test_attention_outputs_stay_in_bounds(B, dtype, Bb, S, H, Hkv, hd):
    td = torch.float32 if dtype == "f32" else torch.bfloat16
    code = B.ZL_DTYPE_F32 if dtype == "f32" else B.ZL_DTYPE_BF16
    W, N = (H + 2 * Hkv) * hd, Bb * S
    qkv = torch.randn(N, W, device="cuda").to(td)
    out, lse = Guarded(N * H * hd, td), Guarded(Bb * H * S, torch.float32)
    B.zl_op_attention(code, qkv, out.view(N, H * hd), lse.inner, Bb, S, H, Hkv, hd)
    out.check("attention out")
    lse.check("attention lse")
    dout = torch.randn(N, H * hd, device="cuda").to(td)
    dqkv = Guarded(N * W, td)
    B.zl_op_attention_bwd(code, qkv, out.view(N, H * hd), dout, lse.inner, dqkv.view(N, W), Bb, S, H, Hkv, hd)
    dqkv.check("attention dqkv")


@pytest.mark.parametrize("w", [synth.TINY, synth.Workload("canary-gpt2", synth.ModelDims(
    synth.ARCH_GPT2, 2, 192, 3, 3, 768, 1000, 200), "bf16", batch=3, seq=133, K=2, steps=1)], ids=["tiny", "gpt2"])
def test_forward_chunk_and_embedding_outputs_stay_in_bounds(w):
    from tests.gpu_common import engine_for
    eng = engine_for(w)
    eng.load({n: (synth.round_bf16(t) if (w.dtype == "bf16" and t.dim() == 2) else t)
              for n, t in synth.make_params(w.dims, w.seed).items()})
    td = torch.float32 if w.dtype == "f32" else torch.bfloat16
    ids, _ = synth.make_batch(w, 0)
    ids = ids.cuda()
    N, d = w.batch * w.seq, w.dims.d_model
    from paper_2608_07974_gb300 import binding as b
    h0 = Guarded(N * d, td)
    b.zl_embed(eng.ctx, ids, w.batch, w.seq, h0.view(N, d))
    eng.synchronize()
    h0.check("embedding")
    h1 = Guarded(N * d, td)
    b.zl_forward_chunk(eng.ctx, 1, h0.view(N, d), None, h1.view(N, d), w.batch, w.seq)
    eng.synchronize()
    h1.check("chunk forward")
    eng.close()
