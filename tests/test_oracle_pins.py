"""Pins of the CPU oracle to facts outside itself (no GPU).

Each test checks the oracle against something it does not contain: central
finite differences, PyTorch library routines, closed forms, the identities of
Lemmas 1-3 of Section II, and the alpha = 1 / K = 1 reduction to backpropagation.
"""
import math

import pytest
import torch
import torch.nn.functional as F

import oracle
from oracle.model import Oracle, OracleConfig
import synth
from synth import ARCH_GPT2, ARCH_LLAMA, ModelDims



@pytest.fixture(autouse=True)
def float64_default():
    """The pins run in float64; the default dtype is restored for the other test modules."""
    old = torch.get_default_dtype()
    torch.set_default_dtype(torch.float64)
    yield
    torch.set_default_dtype(old)


LLAMA_T = ModelDims(ARCH_LLAMA, n_layers=2, d_model=16, n_heads=4, n_kv_heads=2, d_ff=24,
                    vocab=37, max_seq=8)
GPT2_T = ModelDims(ARCH_GPT2, n_layers=2, d_model=16, n_heads=2, n_kv_heads=2, d_ff=32,
                   vocab=37, max_seq=8)


def tiny_params(d, seed=7, std=0.3):
    """Larger-than-default weights so every term of the model matters numerically."""
    P = synth.make_params(d, seed)
    out = {}
    for n, t in P.items():
        if t.dim() == 2:
            out[n] = synth.normal(synth.stream_key(seed, n), t.numel(), std).view(t.shape)
        else:   # gains around 1, biases around 0, both non-trivial
            base = 1.0 if "weight" in n else 0.0
            out[n] = base + synth.normal(synth.stream_key(seed + 1, n), t.numel(), 0.2).view(t.shape)
    return out


def tiny_batch(d, B=2, S=8, seed=3):
    ids = synth.zipf_ids(seed, B, S, d.vocab)
    return ids, synth.next_token_labels(ids)


# ---------------------------------------------------------------------------------------
# Gradients: central finite differences (fp64)
# ---------------------------------------------------------------------------------------

@pytest.mark.parametrize("d", [LLAMA_T, GPT2_T], ids=["llama", "gpt2"])
@pytest.mark.parametrize("alpha,kl_dir", [(0.5, 0), (0.3, 1), (1.0, 0)])
def test_local_gradient_matches_finite_differences(d, alpha, kl_dir):
    P = tiny_params(d)
    ids, labels = tiny_batch(d)
    labels[0, 3] = -1                              # a hole in Omega
    cfg = OracleConfig(dims=d, bounds=[0, 1, 2], alpha=alpha, kl_dir=kl_dir)
    orc = Oracle(cfg, P)
    h = orc.embed(ids)
    gen = torch.Generator().manual_seed(0)
    for k in (1, 2):
        L, grads, h_next = orc.local_grad(k, h, labels)
        a = orc.alpha_k(k)

        def Lk(Pp):
            t = oracle.readout(Pp, h, d) if a < 1 else None
            hk = oracle.chunk_forward(Pp, cfg.bounds, k, h, d)
            return float(oracle.local_objective(oracle.readout(Pp, hk, d), t, labels, a, kl_dir))

        assert abs(Lk(orc.P) - L) < 1e-12
        for name, g in grads.items():
            flat = orc.P[name].view(-1)
            for idx in torch.randint(0, flat.numel(), (4,), generator=gen).tolist():
                eps = 1e-6
                old = float(flat[idx])
                flat[idx] = old + eps
                lp = Lk(orc.P)
                flat[idx] = old - eps
                lm = Lk(orc.P)
                flat[idx] = old
                fd = (lp - lm) / (2 * eps)
                ag = float(g.view(-1)[idx])
                assert abs(fd - ag) <= 1e-7 + 1e-6 * abs(fd), (name, idx, fd, ag)
        h = h_next


# ---------------------------------------------------------------------------------------
# Building blocks against library routines
# ---------------------------------------------------------------------------------------

def test_blocks_match_library_routines():
    g = torch.Generator().manual_seed(1)
    x = torch.randn(3, 5, 16, generator=g)
    w = torch.randn(16, generator=g)
    b = torch.randn(16, generator=g)
    assert torch.allclose(oracle.rmsnorm(x, w, 1e-5), F.rms_norm(x, (16,), w, 1e-5), atol=1e-13, rtol=0)
    assert torch.allclose(oracle.layernorm(x, w, b, 1e-5), F.layer_norm(x, (16,), w, b, 1e-5),
                          atol=1e-13, rtol=0)
    assert torch.allclose(oracle.gelu_tanh(x), F.gelu(x, approximate="tanh"), atol=1e-14, rtol=0)
    assert torch.allclose(oracle.silu(x), F.silu(x), atol=1e-14, rtol=0)


@pytest.mark.parametrize("H,Hkv,hd", [(4, 4, 8), (4, 2, 8), (8, 1, 6)])
def test_attention_matches_sdpa(H, Hkv, hd):
    g = torch.Generator().manual_seed(2)
    B, S = 2, 9
    q = torch.randn(B, S, H, hd, generator=g)
    k = torch.randn(B, S, Hkv, hd, generator=g)
    v = torch.randn(B, S, Hkv, hd, generator=g)
    ref = F.scaled_dot_product_attention(q.transpose(1, 2), k.transpose(1, 2), v.transpose(1, 2),
                                         is_causal=True, enable_gqa=(H != Hkv)).transpose(1, 2)
    assert torch.allclose(oracle.attention(q, k, v), ref, atol=1e-12, rtol=0)


def test_rope_is_the_complex_rotation():
    """RoPE (Su et al.) as a complex product: (x_i + i x_{i+hd/2}) * exp(i s theta^(-2i/hd))."""
    g = torch.Generator().manual_seed(3)
    B, S, H, hd = 2, 7, 3, 10
    x = torch.randn(B, S, H, hd, generator=g)
    half = hd // 2
    c = torch.complex(x[..., :half], x[..., half:])
    freq = 10000.0 ** (-torch.arange(half) * 2.0 / hd)
    rot = torch.polar(torch.ones(S, half), torch.arange(S)[:, None] * freq[None])
    y = c * rot[None, :, None, :]
    ref = torch.cat([y.real, y.imag], dim=-1)
    out = oracle.rope(x, 10000.0)
    assert torch.allclose(out, ref, atol=1e-13, rtol=0)
    assert torch.equal(out[:, 0], x[:, 0])                      # position 0: identity
    # relative position: <R_m q, R_n k> depends on m - n only
    q = torch.randn(hd, generator=g)
    k = torch.randn(hd, generator=g)
    seq = lambda v: v[None, None, None, :].expand(1, S, 1, hd).contiguous()
    rq, rk = oracle.rope(seq(q), 10000.0)[0, :, 0], oracle.rope(seq(k), 10000.0)[0, :, 0]
    assert abs(float(rq[4] @ rk[2]) - float(rq[3] @ rk[1])) < 1e-12


def test_layer_matches_library_composition():
    """A whole block written with F.linear / rms_norm / layer_norm / sdpa / silu / gelu."""
    for d in (LLAMA_T, GPT2_T):
        P = tiny_params(d)
        ids, _ = tiny_batch(d)
        x = oracle.embed(P, ids, d)
        assert torch.equal(oracle.embed(P, ids, d)[..., :],
                           F.embedding(ids.long(), P["tok_emb"]) +
                           (P["pos_emb"][: ids.shape[1]] if d.arch == ARCH_GPT2 else 0))
        B, S, D = x.shape
        H, Hkv, hd = d.n_heads, d.n_kv_heads, d.head_dim
        p = lambda s: P[f"layers.0.{s}"]
        if d.arch == ARCH_LLAMA:
            a = F.rms_norm(x, (D,), p("attn_norm.weight"), d.norm_eps)
            qkv = F.linear(a, p("wqkv"))
        else:
            a = F.layer_norm(x, (D,), p("attn_norm.weight"), p("attn_norm.bias"), d.norm_eps)
            qkv = F.linear(a, p("wqkv"), p("bqkv"))
        q, k, v = qkv.split([H * hd, Hkv * hd, Hkv * hd], dim=-1)
        q, k, v = q.view(B, S, H, hd), k.view(B, S, Hkv, hd), v.view(B, S, Hkv, hd)
        if d.arch == ARCH_LLAMA:
            half = hd // 2
            freq = d.rope_theta ** (-torch.arange(half) * 2.0 / hd)
            rot = torch.polar(torch.ones(S, half), torch.arange(S)[:, None] * freq[None])[None, :, None]
            cq = torch.complex(q[..., :half], q[..., half:]) * rot
            ck = torch.complex(k[..., :half], k[..., half:]) * rot
            q = torch.cat([cq.real, cq.imag], -1)
            k = torch.cat([ck.real, ck.imag], -1)
        o = F.scaled_dot_product_attention(q.transpose(1, 2), k.transpose(1, 2), v.transpose(1, 2),
                                           is_causal=True, enable_gqa=(H != Hkv))
        o = o.transpose(1, 2).reshape(B, S, H * hd)
        if d.arch == ARCH_LLAMA:
            x2 = x + F.linear(o, p("wo"))
            b = F.rms_norm(x2, (D,), p("ffn_norm.weight"), d.norm_eps)
            g, u = F.linear(b, p("w1")).split([d.d_ff, d.d_ff], -1)
            y = x2 + F.linear(F.silu(g) * u, p("w2"))
            zref = F.linear(F.rms_norm(y, (D,), P["norm_f.weight"], d.norm_eps), P["lm_head"])
        else:
            x2 = x + F.linear(o, p("wo"), p("bo"))
            b = F.layer_norm(x2, (D,), p("ffn_norm.weight"), p("ffn_norm.bias"), d.norm_eps)
            y = x2 + F.linear(F.gelu(F.linear(b, p("w1"), p("b1")), approximate="tanh"),
                              p("w2"), p("b2"))
            zref = F.linear(F.layer_norm(y, (D,), P["norm_f.weight"], P["norm_f.bias"], d.norm_eps),
                            P["tok_emb"])
        out = oracle.layer_forward(P, 0, x, d)
        assert torch.allclose(out, y, atol=1e-12, rtol=0)
        assert torch.allclose(oracle.readout(P, out, d), zref, atol=1e-12, rtol=0)


def test_adamw_matches_torch_optim():
    g = torch.Generator().manual_seed(4)
    theta0 = torch.randn(50, generator=g)
    grads = [torch.randn(50, generator=g) for _ in range(6)]
    p = torch.nn.Parameter(theta0.clone())
    opt = torch.optim.AdamW([p], lr=1e-2, betas=(0.9, 0.999), eps=1e-8, weight_decay=0.01)
    th, m, v = theta0.clone(), torch.zeros(50), torch.zeros(50)
    for t, gr in enumerate(grads, start=1):
        p.grad = gr.clone()
        opt.step()
        oracle.adamw_update(th, gr, m, v, t, 1e-2, 0.9, 0.999, 1e-8, 0.01)
    assert torch.allclose(th, p.detach(), atol=1e-14, rtol=1e-12)
    # step-1 closed form: theta (1 - lr wd) - lr g / (|g| + eps)
    th1, m1, v1 = theta0.clone(), torch.zeros(50), torch.zeros(50)
    oracle.adamw_update(th1, grads[0], m1, v1, 1, 1e-2, 0.9, 0.999, 1e-8, 0.01)
    ref = theta0 * (1 - 1e-2 * 0.01) - 1e-2 * grads[0] / (grads[0].abs() + 1e-8)
    assert torch.allclose(th1, ref, atol=1e-15, rtol=0)


# ---------------------------------------------------------------------------------------
# Local objective: closed forms and the lemmas of Section II
# ---------------------------------------------------------------------------------------

def test_loss_closed_forms():
    V = 37
    lab = torch.tensor([3, 0, -1, 36])
    z0 = torch.zeros(4, V)
    for a in (1.0, 0.5, 0.2):
        assert abs(float(oracle.local_objective(z0, z0, lab, a)) - a * math.log(V)) < 1e-14
    g = torch.Generator().manual_seed(5)
    z = torch.randn(4, V, generator=g)
    shift = torch.randn(4, 1, generator=g)
    # softmax is shift invariant: KL(p || softmax(z + c)) = 0 for either direction
    for kd in (0, 1):
        assert float(oracle.kl_rows(z, z + shift, kd).abs().max()) < 1e-14
    # against library cross-entropy / kl_div
    t = torch.randn(4, V, generator=g)
    ce = F.cross_entropy(z, lab.long(), ignore_index=-1, reduction="sum") / 3
    klr = F.kl_div(F.log_softmax(t, -1), F.log_softmax(z, -1), log_target=True,
                   reduction="none").sum(-1)       # KL(p || q), p = softmax(z)
    klr = klr[lab >= 0].sum() / 3
    for a in (1.0, 0.5):
        val = float(oracle.local_objective(z, t, lab, a, 0))
        assert abs(val - float(a * ce + (1 - a) * klr)) < 1e-13
    # two classes: CE = log(1 + e^(z1 - z0)) for y = 0; Bernoulli KL
    z2 = torch.tensor([[0.3, -1.1]])
    t2 = torch.tensor([[-0.4, 0.9]])
    sp = 1 / (1 + math.exp(-(0.3 + 1.1)))
    sq = 1 / (1 + math.exp(-(-0.4 - 0.9)))
    ce2 = math.log(1 + math.exp(-1.1 - 0.3))
    kl2 = sp * math.log(sp / sq) + (1 - sp) * math.log((1 - sp) / (1 - sq))
    got = float(oracle.local_objective(z2, t2, torch.tensor([0]), 0.25, 0))
    assert abs(got - (0.25 * ce2 + 0.75 * kl2)) < 1e-14


@pytest.mark.parametrize("kl_dir", [0, 1])
def test_logit_gradient_rows_sum_to_zero_and_alpha1_textbook(kl_dir):
    g = torch.Generator().manual_seed(6)
    V = 29
    lab = torch.tensor([1, 28, -1, 5, 0])
    z = torch.randn(5, V, generator=g).requires_grad_(True)
    t = torch.randn(5, V, generator=g)
    L = oracle.local_objective(z, t, lab, 0.4, kl_dir)
    (dz,) = torch.autograd.grad(L, z)
    assert float(dz.sum(-1).abs().max()) < 1e-16 * V + 1e-17     # proof of Lemma 3: sum_l dp(l) = 0
    assert float(dz[2].abs().max()) == 0.0                       # row outside Omega
    L1 = oracle.local_objective(z, t, lab, 1.0, kl_dir)
    (dz1,) = torch.autograd.grad(L1, z)
    ref = torch.softmax(z.detach(), -1) - F.one_hot(lab.clamp(min=0).long(), V)
    ref[2] = 0
    assert torch.allclose(dz1, ref / 4, atol=1e-16, rtol=0)
    # the consistency gradient vanishes when the teacher equals the student
    L2 = oracle.local_objective(z, z.detach(), lab, 0.0, kl_dir)
    (dz2,) = torch.autograd.grad(L2, z)
    assert float(dz2.abs().max()) < 1e-16


def test_lemma2_geometric_mixture():
    """alpha KL(p||r) + (1-alpha) KL(p||q) = KL(p||p*) - log Z, p* ∝ r^alpha q^(1-alpha)."""
    g = torch.Generator().manual_seed(8)
    V = 11
    for a in (0.1, 0.5, 0.9):
        zp, zr, zq = (torch.randn(6, V, generator=g) for _ in range(3))
        lr_, lq = torch.log_softmax(zr, -1), torch.log_softmax(zq, -1)
        lstar_un = a * lr_ + (1 - a) * lq
        logZ = torch.logsumexp(lstar_un, -1)
        lhs = a * oracle.kl_rows(zp, zr) + (1 - a) * oracle.kl_rows(zp, zq)
        rhs = oracle.kl_rows(zp, lstar_un) - logZ
        assert torch.allclose(lhs, rhs, atol=1e-13, rtol=0)
        # p* minimises the left side: its logit gradient vanishes there
        zs = lstar_un.clone().requires_grad_(True)
        obj = (a * oracle.kl_rows(zs, zr) + (1 - a) * oracle.kl_rows(zs, zq)).sum()
        (gz,) = torch.autograd.grad(obj, zs)
        assert float(gz.abs().max()) < 1e-14


def test_lemma1_three_point_identity():
    """D(p,y) = D(p',y) + <grad L(p'), p - p'> + D(p,p') for the KL (negative entropy) case."""
    g = torch.Generator().manual_seed(9)
    V = 13
    zp, zpp, zy = (torch.randn(5, V, generator=g) for _ in range(3))
    p, pp, y = (torch.softmax(t, -1) for t in (zp, zpp, zy))
    gradL = torch.log(pp) - torch.log(y)          # d/du KL(u||y) at u = p', up to +1 (mean-zero pairing)
    lhs = oracle.kl_rows(zp, zy)
    rhs = oracle.kl_rows(zpp, zy) + ((p - pp) * gradL).sum(-1) + oracle.kl_rows(zp, zpp)
    assert torch.allclose(lhs, rhs, atol=1e-13, rtol=0)


# ---------------------------------------------------------------------------------------
# Structure: stop-gradient (Lemma 3), alpha = 1 mapping, K = 1 == BP
# ---------------------------------------------------------------------------------------

@pytest.mark.parametrize("d", [LLAMA_T, GPT2_T], ids=["llama", "gpt2"])
def test_k1_alpha1_is_backprop_bit_for_bit(d):
    P = tiny_params(d)
    cfg = OracleConfig(dims=d, bounds=[0, 2], alpha=1.0, lr=1e-2)
    a, b = Oracle(cfg, P), Oracle(cfg, P)
    for s in range(3):
        ids, labels = tiny_batch(d, seed=10 + s)
        la = a.step(ids, labels)[0]
        lb = b.bp_step(ids, labels)
        assert la == lb
    for n in a.trainable_names():
        assert torch.equal(a.P[n], b.P[n]), n


@pytest.mark.parametrize("d", [LLAMA_T, GPT2_T], ids=["llama", "gpt2"])
def test_last_chunk_alpha1_equals_bp_gradient_and_global_loss(d):
    P = tiny_params(d)
    ids, labels = tiny_batch(d)
    cfg = OracleConfig(dims=d, bounds=[0, 1, 2], alpha=1.0)
    orc = Oracle(cfg, P)
    Lbp, gbp = orc.bp_grad(ids, labels)
    h1 = orc.forward_chunk(1, orc.embed(ids))
    LK, gK, _ = orc.local_grad(2, h1, labels)
    assert abs(LK - Lbp) < 1e-13
    assert abs(orc.global_loss(ids, labels) - LK) < 1e-13
    for n, g in gK.items():
        assert torch.allclose(g, gbp[n], atol=1e-14, rtol=1e-12), n
    # and the first chunk's local gradient is NOT the BP gradient (decoupled update)
    _, g1, _ = orc.local_grad(1, orc.embed(ids), labels)
    n0 = orc.chunk_names(1)[1]
    assert not torch.allclose(g1[n0], gbp[n0], rtol=0)


def test_stop_gradient_block_structure():
    """Lemma 3: chunk k's gradient is a function of (h_{k-1}, theta_k) only."""
    d = LLAMA_T
    P = tiny_params(d)
    ids, labels = tiny_batch(d)
    cfg = OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5)
    orc = Oracle(cfg, P)
    h1 = orc.forward_chunk(1, orc.embed(ids))
    _, g2, _ = orc.local_grad(2, h1, labels)
    for n in orc.chunk_names(1):                   # perturb chunk 1 after h_1 is fixed
        orc.P[n] += 0.1
    _, g2b, _ = orc.local_grad(2, h1, labels)
    for n in g2:
        assert torch.equal(g2[n], g2b[n])


def test_zero_layers_are_identity_and_kl_vanishes():
    """Zero matrices make every block the identity, so h_k = h_0 and p_k = p_0 (KL = 0)."""
    d = LLAMA_T
    P = tiny_params(d)
    for n in list(P):
        if n.startswith("layers.") and P[n].dim() == 2:
            P[n] = torch.zeros_like(P[n])
    ids, labels = tiny_batch(d)
    orc = Oracle(OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5), P)
    h0 = orc.embed(ids)
    h1 = orc.forward_chunk(1, h0)
    assert torch.equal(h1, h0)
    L, _, _ = orc.local_grad(1, h0, labels)
    ce = float(oracle.local_objective(orc.readout(h0), None, labels, 1.0))
    assert abs(L - 0.5 * ce) < 1e-14


def test_causality():
    d = GPT2_T
    P = tiny_params(d)
    ids, _ = tiny_batch(d)
    orc = Oracle(OracleConfig(dims=d, bounds=[0, 2]), P)
    h = orc.forward_chunk(1, orc.embed(ids))
    ids2 = ids.clone()
    ids2[:, -1] = (ids2[:, -1] + 1) % d.vocab
    h2 = orc.forward_chunk(1, orc.embed(ids2))
    assert torch.equal(h[:, :-1], h2[:, :-1])
    assert not torch.equal(h[:, -1], h2[:, -1])


def test_accumulation_window_is_the_mean():
    """With m = 2 the window gradient is the mean of two micro-batch gradients (step S3)."""
    d = LLAMA_T
    P = tiny_params(d)
    b1, b2 = tiny_batch(d, seed=21), tiny_batch(d, seed=22)
    cfg2 = OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5, accum_m=2, lr=1e-2)
    a = Oracle(cfg2, P)
    a.step(*b1)
    assert a.t[1] == 0
    a.step(*b2)
    assert a.t[1] == 1 and a.t[2] == 1
    ref = Oracle(OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5, lr=1e-2), P)
    h = ref.embed(b1[0])
    _, ga, _ = ref.local_grad(1, h, b1[1])
    _, gb, _ = ref.local_grad(1, ref.embed(b2[0]), b2[1])
    n = ref.chunk_names(1)[1]
    th, m, v = ref.P[n].clone(), torch.zeros_like(ref.P[n]), torch.zeros_like(ref.P[n])
    oracle.adamw_update(th, (ga[n] + gb[n]) / 2, m, v, 1, 1e-2, 0.9, 0.999, 1e-8, 0.01)
    assert torch.allclose(a.P[n], th, atol=1e-15, rtol=0)


# ---------------------------------------------------------------------------------------
# LoRA chunks (the paper's setting: frozen w_l, trainable A_l, B_l, Delta w_l = s B_l A_l)
# ---------------------------------------------------------------------------------------

def _lora_setup(d, rank=3, scale=2.0, b_std=0.3):
    P = tiny_params(d)
    P.update({n: t * 15.0 if n.endswith("lora_a") else t
              for n, t in synth.make_lora_params(d, 11, rank, b_std=b_std).items()})
    cfg = OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5, lora_rank=rank, lora_scale=scale)
    return P, cfg


@pytest.mark.parametrize("d", [LLAMA_T, GPT2_T], ids=["llama", "gpt2"])
def test_lora_gradient_matches_finite_differences(d):
    P, cfg = _lora_setup(d)
    ids, labels = tiny_batch(d)
    orc = Oracle(cfg, P)
    h = orc.embed(ids)
    gen = torch.Generator().manual_seed(5)
    for k in (1, 2):
        L, grads, h_next = orc.local_grad(k, h, labels)
        assert set(grads) == set(orc.chunk_names(k)) and all("lora_" in n for n in grads)

        def Lk(Pp):
            t = oracle.readout(Pp, h, d)
            hk = oracle.chunk_forward(Pp, cfg.bounds, k, h, d, cfg.lora_scale)
            return float(oracle.local_objective(oracle.readout(Pp, hk, d), t, labels, 0.5))

        for name, g in grads.items():
            flat = orc.P[name].view(-1)
            for idx in torch.randint(0, flat.numel(), (3,), generator=gen).tolist():
                old = float(flat[idx])
                flat[idx] = old + 1e-6
                lp = Lk(orc.P)
                flat[idx] = old - 1e-6
                lm = Lk(orc.P)
                flat[idx] = old
                fd = (lp - lm) / 2e-6
                assert abs(fd - float(g.view(-1)[idx])) <= 1e-7 + 1e-6 * abs(fd), (name, idx)
        h = h_next


def test_lora_zero_b_is_the_base_model_and_chain_rule():
    """B = 0 gives the base model exactly; dL/dB = s G A^T and dL/dA = s B^T G, G = dL/dW_eff."""
    d = LLAMA_T
    P, cfg = _lora_setup(d, b_std=0.0)
    ids, labels = tiny_batch(d)
    base = Oracle(OracleConfig(dims=d, bounds=[0, 1, 2]), {n: t for n, t in P.items() if "lora_" not in n})
    lora = Oracle(cfg, P)
    h0 = base.embed(ids)
    assert torch.equal(lora.forward_chunk(1, h0), base.forward_chunk(1, h0))
    # chain rule with a non-zero B: full fine-tune gradients of the merged weights
    P, cfg = _lora_setup(d)
    lora = Oracle(cfg, P)
    merged = {n: t for n, t in lora.P.items() if "lora_" not in n}
    for l in range(d.n_layers):
        for s in synth.LORA_TARGETS:
            merged[f"layers.{l}.{s}"] = oracle.model.lora_weight(lora.P, l, s, cfg.lora_scale)
    full = Oracle(OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5), merged)
    h0 = full.embed(ids)
    _, gl, _ = lora.local_grad(1, h0, labels)
    _, gf, _ = full.local_grad(1, h0, labels)
    for s in synth.LORA_TARGETS:
        G = gf[f"layers.0.{s}"]
        A, Bm = lora.P[f"layers.0.{s}.lora_a"], lora.P[f"layers.0.{s}.lora_b"]
        assert torch.allclose(gl[f"layers.0.{s}.lora_b"], cfg.lora_scale * G @ A.T, atol=1e-12, rtol=1e-9)
        assert torch.allclose(gl[f"layers.0.{s}.lora_a"], cfg.lora_scale * Bm.T @ G, atol=1e-12, rtol=1e-9)


# ---------------------------------------------------------------------------------------
# Readout adapters (Section III-B, option (b)): a_k(h) = h + GELU(h D^T) U^T before the frozen head
# ---------------------------------------------------------------------------------------

def _adapter_setup(d, dim=4, up_std=0.3):
    P = tiny_params(d)
    A = synth.make_adapter_params(d, 2, 13, dim, up_std=up_std)
    P.update({n: t * 15.0 if n.endswith("down") else t for n, t in A.items()})
    return P, OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5, adapter_dim=dim)


def _library_adapter(P, k, h):
    """The adapter written with torch.nn.functional's linear and tanh-GELU."""
    F = torch.nn.functional
    return h + F.linear(F.gelu(F.linear(h, P[f"adapters.{k}.down"]), approximate="tanh"), P[f"adapters.{k}.up"])


@pytest.mark.parametrize("d", [LLAMA_T, GPT2_T], ids=["llama", "gpt2"])
def test_adapter_gradient_matches_finite_differences(d):
    """L_k with chunk k's adapter on its own readout, the teacher the frozen head on h_{k-1}: autograd
    gradients of every chunk tensor (layers and adapter) against central differences of the loss
    composed from library routines."""
    P, cfg = _adapter_setup(d)
    ids, labels = tiny_batch(d)
    orc = Oracle(cfg, P)
    h = orc.embed(ids)
    gen = torch.Generator().manual_seed(9)
    for k in (1, 2):
        L, grads, h_next = orc.local_grad(k, h, labels)
        assert {n for n in grads if n.startswith("adapters.")} == {f"adapters.{k}.down", f"adapters.{k}.up"}

        def Lk(Pp):
            t = oracle.readout(Pp, h, d)
            hk = oracle.chunk_forward(Pp, cfg.bounds, k, h, d)
            z = oracle.readout(Pp, _library_adapter(Pp, k, hk), d)
            return float(oracle.local_objective(z, t, labels, 0.5))

        assert abs(Lk(orc.P) - L) < 1e-12
        for name, g in grads.items():
            flat = orc.P[name].view(-1)
            for idx in torch.randint(0, flat.numel(), (3,), generator=gen).tolist():
                old = float(flat[idx])
                flat[idx] = old + 1e-6
                lp = Lk(orc.P)
                flat[idx] = old - 1e-6
                lm = Lk(orc.P)
                flat[idx] = old
                fd = (lp - lm) / 2e-6
                assert abs(fd - float(g.view(-1)[idx])) <= 1e-7 + 1e-6 * abs(fd), (name, idx)
        h = h_next


def test_adapter_zero_up_is_identity_and_chain_rule():
    """U = 0: the loss and every layer gradient equal the static-head ones exactly, dL/dD = 0, and
    dL/dU = G^T GELU(h_k D^T) with G = dL/dh_k of the static-head objective (chain rule)."""
    d = GPT2_T
    P, cfg = _adapter_setup(d, up_std=0.0)
    ids, labels = tiny_batch(d)
    static = Oracle(OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5),
                    {n: t for n, t in P.items() if not n.startswith("adapters.")})
    ad = Oracle(cfg, P)
    h0 = static.embed(ids)
    Ls, gs, h1 = static.local_grad(1, h0, labels)
    La, ga, _ = ad.local_grad(1, h0, labels)
    assert La == Ls
    for n, g in gs.items():
        assert torch.equal(ga[n], g), n
    assert torch.count_nonzero(ga["adapters.1.down"]) == 0
    hk = h1.clone().requires_grad_(True)
    t = oracle.readout(static.P, h0, d)
    G, = torch.autograd.grad(oracle.local_objective(oracle.readout(static.P, hk, d), t, labels, 0.5), hk)
    act = oracle.gelu_tanh(h1 @ ad.P["adapters.1.down"].T)
    ref = torch.einsum("bsd,bsr->dr", G, act)
    assert torch.allclose(ga["adapters.1.up"], ref, atol=1e-13, rtol=1e-10)


def test_adapter_teacher_is_the_frozen_head_and_bp_ignores_adapters():
    """Chunk 2's loss, with h_1 fixed, does not depend on chunk 1's adapter (its teacher is the frozen
    head on h_1); the global objective and the backpropagation step leave every adapter untouched."""
    d = LLAMA_T
    P, cfg = _adapter_setup(d)
    ids, labels = tiny_batch(d)
    orc = Oracle(cfg, P)
    h1 = orc.forward_chunk(1, orc.embed(ids))
    L2, _, _ = orc.local_grad(2, h1, labels)
    orc.P["adapters.1.down"].mul_(3.0)
    orc.P["adapters.1.up"].add_(0.5)
    assert orc.local_grad(2, h1, labels)[0] == L2
    base = Oracle(OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5),
                  {n: t for n, t in P.items() if not n.startswith("adapters.")})
    bp = Oracle(cfg, P)
    assert bp.global_loss(ids, labels) == base.global_loss(ids, labels)
    before = {n: t.clone() for n, t in bp.P.items() if n.startswith("adapters.")}
    bp.bp_step(ids, labels)
    base.bp_step(ids, labels)
    for n, t in before.items():
        assert torch.equal(bp.P[n], t), n
    for n, t in base.P.items():
        assert torch.equal(bp.P[n], t), n


# ---------------------------------------------------------------------------------------
# Options of the update rule: the step-size schedule of Theorem 1, chunk 1 without a
# consistency term, and the reverse distillation direction
# ---------------------------------------------------------------------------------------

def test_lr_schedule_matches_torch_lambda_lr():
    """lr_schedule = 1 is eta_t = eta_0 / sqrt(t + gamma), t = 0, 1, .. counting each chunk's own
    updates (Theorem 1's step size): the oracle's parameters follow torch.optim.AdamW driven by a
    LambdaLR with that factor, fed the oracle's own gradients (so only the update rule is pinned)."""
    d = LLAMA_T
    P = tiny_params(d)
    lr, gamma = 3e-2, 2.0
    cfg = OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5, lr=lr, lr_schedule=1, lr_gamma=gamma)
    orc = Oracle(cfg, P)
    names = orc.chunk_names(1)
    ps = [torch.nn.Parameter(orc.P[n].clone()) for n in names]
    opt = torch.optim.AdamW(ps, lr=lr, betas=(0.9, 0.999), eps=1e-8, weight_decay=0.01)
    sched = torch.optim.lr_scheduler.LambdaLR(opt, lambda t: 1.0 / math.sqrt(t + gamma))
    for s in range(4):
        ids, labels = tiny_batch(d, seed=40 + s)
        _, grads, _ = orc.local_grad(1, orc.embed(ids), labels)
        for p, n in zip(ps, names):
            p.grad = grads[n].clone()
        opt.step()
        sched.step()
        orc.step(ids, labels)
        assert orc.t[1] == s + 1
        for p, n in zip(ps, names):
            assert torch.allclose(orc.P[n], p.detach(), atol=1e-14, rtol=1e-12), (s, n)
    # the schedule really changed the step: a constant-lr run ends elsewhere
    const = Oracle(OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5, lr=lr), P)
    for s in range(4):
        const.step(*tiny_batch(d, seed=40 + s))
    assert not torch.allclose(const.P[names[1]], orc.P[names[1]], atol=1e-6, rtol=0)


def test_consis_first_zero_is_plain_cross_entropy():
    """consis_first = 0 gives chunk 1 the task term alone (alpha_1 = 1): its local loss is the
    library cross-entropy of its readout over Omega; chunk 2 keeps the consistency term."""
    d = GPT2_T
    P = tiny_params(d)
    ids, labels = tiny_batch(d)
    labels[1, 2] = -1
    cfg = OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5, consis_first=0)
    orc = Oracle(cfg, P)
    h0 = orc.embed(ids)
    L1, _, h1 = orc.local_grad(1, h0, labels)
    z1 = oracle.readout(orc.P, h1, d).reshape(-1, d.vocab)
    ce = F.cross_entropy(z1, labels.reshape(-1).long(), ignore_index=-1)
    assert abs(L1 - float(ce)) < 1e-13
    L2, _, h2 = orc.local_grad(2, h1, labels)
    z2 = oracle.readout(orc.P, h2, d).reshape(-1, d.vocab)
    ce2 = F.cross_entropy(z2, labels.reshape(-1).long(), ignore_index=-1)
    assert abs(L2 - float(ce2)) > 1e-6          # 0.5 CE + 0.5 KL(p_2 || p_1), not CE
    with_first = Oracle(OracleConfig(dims=d, bounds=[0, 1, 2], alpha=0.5), P)
    L1b, _, _ = with_first.local_grad(1, h0, labels)
    assert abs(L1b - float(ce)) > 1e-6


def test_reverse_kl_direction_matches_library():
    """kl_dir = 1 is KL(p_{k-1} || p_k) (forward distillation): the library kl_div with the student
    as input and the teacher as target; its logit gradient is (p - q) / |Omega| per row at alpha 0."""
    g = torch.Generator().manual_seed(12)
    V = 23
    lab = torch.tensor([4, -1, 0, 22, 9])
    z = torch.randn(5, V, generator=g).requires_grad_(True)
    t = torch.randn(5, V, generator=g)
    with torch.no_grad():
        kl = F.kl_div(F.log_softmax(z, -1), F.log_softmax(t, -1), log_target=True, reduction="none").sum(-1)
        ref = kl[lab >= 0].sum() / 4
        ce = F.cross_entropy(z, lab.long(), ignore_index=-1)
    for a in (0.5, 0.0):
        val = oracle.local_objective(z, t, lab, a, 1).detach()
        assert abs(float(val) - float(a * ce + (1 - a) * ref)) < 1e-13
    (dz,) = torch.autograd.grad(oracle.local_objective(z, t, lab, 0.0, 1), z)
    pq = (torch.softmax(z.detach(), -1) - torch.softmax(t, -1)) / 4
    pq[1] = 0
    assert torch.allclose(dz, pq, atol=1e-16, rtol=0)


def test_proposition1_chunkwise_bound():
    """Proposition 1 in the token-level geometry it is stated in: with psi the negative entropy
    (D_psi = the oracle's KL), a soft target r and L(p) = KL(p || r) (smooth relative to psi with
    beta = 1), p_k* the minimiser of the oracle's local objective alpha KL(p || r) + (1 - alpha)
    KL(p || p_{k-1}) and any p_k with delta_k = KL(p_k || p_k*), the global loss obeys
    L(p_K) <= L(p_0) - sum_k (1/alpha - 1) KL(p_k || p_{k-1}) + (1/alpha) sum_k delta_k."""
    g = torch.Generator().manual_seed(21)
    V, K = 9, 4
    for a in (0.1, 0.3, 0.5, 0.8, 0.95):
        for trial in range(300):
            zr = 2 * torch.randn(1, V, generator=g)
            zs = [torch.log_softmax(2 * torch.randn(1, V, generator=g), -1)]
            stars = []
            for k in range(K):
                zstar = torch.log_softmax(a * torch.log_softmax(zr, -1) + (1 - a) * zs[-1], -1)
                if trial == 0:   # p_k* is where the oracle's local objective is stationary
                    zz = zstar.clone().requires_grad_(True)
                    obj = a * oracle.kl_rows(zz, zr) + (1 - a) * oracle.kl_rows(zz, zs[-1])
                    (gz,) = torch.autograd.grad(obj.sum(), zz)
                    assert float(gz.abs().max()) < 1e-14
                noise = 0.0 if trial % 5 == 0 else 0.3   # every fifth trial: p_k = p_k* (delta_k = 0)
                stars.append(zstar)
                zs.append(torch.log_softmax(zstar + noise * torch.randn(1, V, generator=g), -1))
            L = lambda z: float(oracle.kl_rows(z, zr))
            D = lambda u, v: float(oracle.kl_rows(u, v))
            bound = (L(zs[0]) - sum((1 / a - 1) * D(zs[k + 1], zs[k]) for k in range(K))
                     + sum(D(zs[k + 1], stars[k]) for k in range(K)) / a)
            assert L(zs[-1]) <= bound + 1e-12, (a, trial, L(zs[-1]), bound)


def test_global_update_equivalence_gradient_is_jacobian_times_log_gap():
    """Lemma 3 (global update equivalence, Section II-C): the gradient of the local objective
    alpha KL(p || r) + (1 - alpha) KL(p || p_{k-1}) (the oracle's KL) is J^T e with
    e = log p - log p*, p* the geometric mixture of Lemma 2. At the logits
    J = diag(p) - p p^T, so dL/dz = p (e - <p, e>); and through a linear readout z = h W^T the chain
    rule carries the same J^T e to the parameters."""
    g = torch.Generator().manual_seed(31)
    V, Dm = 11, 5
    for a in (0.2, 0.5, 0.9):
        zr, zq = torch.randn(4, V, generator=g), torch.randn(4, V, generator=g)
        h = torch.randn(4, Dm, generator=g)
        W = torch.randn(V, Dm, generator=g).requires_grad_(True)
        z = h @ W.T
        L = (a * oracle.kl_rows(z, zr) + (1 - a) * oracle.kl_rows(z, zq)).sum()
        (gW,) = torch.autograd.grad(L, W)
        with torch.no_grad():
            lp = torch.log_softmax(z, -1)
            lstar = torch.log_softmax(a * torch.log_softmax(zr, -1) + (1 - a) * torch.log_softmax(zq, -1), -1)
            e = lp - lstar
            p = lp.exp()
            dz = p * (e - (p * e).sum(-1, keepdim=True))
        assert torch.allclose(gW, dz.T @ h, atol=1e-13, rtol=1e-11)
