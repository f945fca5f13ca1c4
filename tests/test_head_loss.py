"""The frozen head fused with the local objective over row slices (GPU; Eq. 2-5).

zl_op_head_loss forms z = n W^T and the teacher t = tn W^T for a slice of rows at a time, the fused
loss writes dz in place of z, and dn = dz W follows; vocab-sized buffers hold one slice only. The op
is checked element by element against the oracle (logits, local objective and its gradient at n by
autograd, fp64) on ragged row counts and slice sizes; the engine's row-sliced readout (cfg.loss_rows)
is checked against the oracle over training steps (fp32: 1e-4; bf16 GPT-2 at full size: the bf16
bars), and it must cut the GPT-2 step's peak HBM by at least 0.9 GB.
"""
import pytest
import torch

import oracle
import synth
from tests.gpu_common import cosine, engine_for, fro_rel, oracle_for, rel

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    import paper_2608_07974_gb300 as pkg
    pkg.build()
    from paper_2608_07974_gb300 import binding
    return binding


def _oracle(n, tn, W, labels, V, alpha, kl_dir):
    """Loss, per-row losses, dL/dn (autograd) and, per element of dn, the dot-product scale |dz| |W|
    (the sum of magnitudes that bounds the rounding error of dn_j = sum_v dz_v W_vj)."""
    nn = n.double().cpu().requires_grad_(True)
    Wd = W[:V].double().cpu()
    z = nn @ Wd.T
    t = None if tn is None else tn.double().cpu() @ Wd.T
    L = oracle.local_objective(z, t, labels.cpu(), alpha, kl_dir)
    rows = oracle.local_objective_rows(z.detach(), t, labels.cpu(), alpha, kl_dir)
    (dn, dz) = torch.autograd.grad(L, [nn, z])
    return float(L.detach()), rows, dn, dz.abs() @ Wd.abs(), float(z.detach().abs().max())


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("N,d,V,R,alpha,kl_dir", [(300, 64, 1000, 128, 0.5, 0), (300, 64, 1000, 300, 0.3, 1),
                                                  (129, 256, 50257, 64, 0.5, 0), (77, 128, 512, 1000, 1.0, 0),
                                                  (1, 64, 2, 1, 0.5, 0)])
def test_head_loss_matches_oracle(B, dtype, N, d, V, R, alpha, kl_dir):
    torch.manual_seed(N + d + V + R)
    td = torch.float32 if dtype == "f32" else torch.bfloat16
    code = B.ZL_DTYPE_F32 if dtype == "f32" else B.ZL_DTYPE_BF16
    ldw = (V + 127) // 128 * 128
    n = torch.randn(N, d).to(td)
    tn = torch.randn(N, d).to(td) if alpha < 1 else None
    W = torch.zeros(ldw, d)
    W[:V] = (2.0 / d ** 0.5) * torch.randn(V, d)   # logits of a few units, as a trained head gives
    W = W.to(td)
    labels = torch.randint(0, V, (N,), dtype=torch.int32)
    if N > 3:
        labels[::5] = -1
    dn = torch.full((N, d), float("nan"), dtype=td, device="cuda")
    rl = torch.empty(N, device="cuda")
    loss = torch.empty(1, device="cuda")
    B.zl_op_head_loss(code, n.cuda(), None if tn is None else tn.cuda(), W.cuda(), labels.cuda(), N, d, V, ldw, alpha,
                      kl_dir, R, dn, rl, loss)
    torch.cuda.synchronize()
    L, rows, dref, scale, zmax = _oracle(n.float(), None if tn is None else tn.float(), W.float(), labels, V, alpha,
                                         kl_dir)
    # fp32: the products round in fp32 (1e-4 of the dot-product scale sum_v |dz_v W_vj|). bf16: the logits
    # are rounded to bf16 before the loss, which moves p_v by up to |z_v| 2^-9 relative, and dz is rounded
    # again (2^-9): dn_j is held to 2^-8 (1 + max |z|) of its scale
    ltol, gtol = (1e-5, 1e-4) if dtype == "f32" else (2e-2, 2.0 ** -8 * (1.0 + zmax))
    assert abs(float(loss) - L) <= ltol * max(1.0, abs(L)), (float(loss), L)
    assert torch.allclose(rl.cpu().double(), rows, rtol=ltol, atol=ltol * max(1.0, abs(L)))
    got = dn.double().cpu()
    excess = (got - dref).abs() - gtol * scale
    assert float(excess.max()) <= 1e-12, float(((got - dref).abs() / (scale + 1e-30)).max())
    assert cosine(got, dref) >= 0.9999 if dtype == "f32" else cosine(got, dref) >= 0.999


def test_head_loss_rejects_bad_arguments(B):
    z = torch.zeros(8, 8, device="cuda")
    lab = torch.zeros(8, dtype=torch.int32, device="cuda")
    one = torch.zeros(1, device="cuda")
    rl = torch.zeros(8, device="cuda")
    for args in [(8, 8, 8, 8, 0.5, 0, 4, None), (8, 8, 8, 12, 1.0, 0, 4, None), (8, 8, 8, 8, 1.0, 0, 0, None)]:
        N, d, V, ldw, alpha, kl, R, tn = args
        with pytest.raises(B.ZLError) as e:
            B.zl_op_head_loss(B.ZL_DTYPE_F32, z, tn, z, lab, N, d, V, ldw, alpha, kl, R, z, rl, one)
        assert e.value.status == B.ZL_ERR_ARG


W_TINY = synth.TINY


@pytest.mark.parametrize("rows", [96, 256, 1000])
def test_sliced_readout_ten_steps_match_oracle(rows):
    """The tiny fp32 workload with its readout in row slices (96: ragged, 256: one slice, 1000: wider than
    the micro-batch) over 10 steps, then a backpropagation step and the global loss."""
    P = synth.make_params(W_TINY.dims, W_TINY.seed)
    eng = engine_for(W_TINY, loss_rows=rows)
    eng.load(P)
    orc = oracle_for(W_TINY, P)
    for s in range(W_TINY.steps):
        ids, labels = synth.make_batch(W_TINY, s)
        lg = eng.step(ids.cuda(), labels.cuda())
        lo = orc.step(ids, labels)
        for a, b in zip(lg, lo):
            assert rel(a, b) <= 1e-4, (s, lg, lo)
    ids, labels = synth.make_batch(W_TINY, 20)
    assert rel(eng.bp_step(ids.cuda(), labels.cuda()), orc.bp_step(ids, labels)) <= 1e-4
    ids, labels = synth.make_batch(W_TINY, 21)
    assert rel(eng.global_loss(ids.cuda(), labels.cuda()), orc.global_loss(ids, labels)) <= 1e-4
    for n in orc.trainable_names():
        assert fro_rel(eng.get(n), orc.P[n]) <= 1e-4, n
    eng.close()


def test_sliced_local_steps_match_oracle():
    P = synth.make_params(W_TINY.dims, W_TINY.seed)
    eng = engine_for(W_TINY, loss_rows=80, kl_dir=1)
    eng.load(P)
    orc = oracle_for(W_TINY, P, kl_dir=1)
    ids, labels = synth.make_batch(W_TINY, 0)
    h = None
    ho = orc.embed(ids)
    for k in range(1, W_TINY.K + 1):
        out = torch.empty(W_TINY.batch * W_TINY.seq, W_TINY.dims.d_model, device="cuda")
        lg = eng.local_step(k, h, ids.cuda(), labels.cuda(), h_out=out)
        lo, ho = orc.local_step(k, ho, labels)
        assert rel(lg, lo) <= 1e-4, (k, lg, lo)
        h = out
    eng.close()


def test_adapters_with_sliced_readout_are_unsupported():
    from paper_2608_07974_gb300 import binding as b
    with pytest.raises(b.ZLError) as e:
        engine_for(W_TINY, loss_rows=64, adapter_dim=16)
    assert e.value.status == b.ZL_ERR_UNSUPPORTED


G2 = synth.GPT2_SMALL


def test_gpt2_sliced_readout_full_size_and_memory():
    """GPT-2-small bf16, K = 4, the full 8 x 512 micro-batch with 512-row slices: every chunk's loss and
    gradients against the fp32 oracle on the same bf16-rounded weights (gradients read with accum_m = 2),
    and the concurrent step's peak HBM at least 0.9 GB below the unsliced step's."""
    P = {n: (synth.round_bf16(t) if t.dim() == 2 else t) for n, t in synth.make_params(G2.dims, G2.seed).items()}
    ids, labels = synth.make_batch(G2, 0)
    eng = engine_for(G2, accum_m=2, loss_rows=512)
    eng.load(P)
    lg = eng.step(ids.cuda(), labels.cuda())
    orc = oracle_for(G2, P, dtype=torch.float32)
    h = orc.embed(ids)
    for k in range(1, G2.K + 1):
        L, g, h = orc.local_grad(k, h, labels)
        assert rel(lg[k - 1], L) <= 2e-2, (k, lg, L)
        for n in orc.chunk_names(k):
            c = cosine(eng.get(n, 1), g[n])
            assert c >= 0.999, (k, n, c)
    eng.close()
    peaks = {}
    for rows in (0, 512):
        e2 = engine_for(G2, max_live_chunks=2, loss_rows=rows)
        e2.load(P)
        e2.reset_peak()
        e2.step(ids.cuda(), labels.cuda())
        peaks[rows] = e2.peak_bytes()[0]
        e2.close()
    assert peaks[0] - peaks[512] >= 0.9e9, peaks
