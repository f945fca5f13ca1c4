"""Autograd-free forward and backward of the chunked decoder in numpy float64 (test infrastructure).

A second statement of the model, written independently of the oracle: numpy instead of torch, and
every backward formula derived by hand instead of taken from autograd. It covers Eq. 1 (blocks and
chunks), Eq. 2 (readout through the frozen final norm and head), the logit gradient of the local
objective of Eq. 3-5 in closed form, and backpropagation through a chunk or through the whole model.
The tests use it to pin the oracle's gradients element by element at float64 rounding.

Closed forms used (one row i of logits z, teacher t, label y, p = softmax(z), q = softmax(t)):
  CE_i = lse(z) - z_y,                       dCE_i/dz = p - onehot(y)
  KL(p || q) = sum p (log p - log q),        d/dz = p * (z - t - (lse(z) - lse(t)) - KL(p || q))
  KL(q || p) = sum q (log q - log p),        d/dz = p - q
and L_k = (1/|Omega|) sum over rows with y >= 0 of alpha CE_i + (1 - alpha) KL_i.
"""
from __future__ import annotations

import math
from typing import Dict, Tuple

import numpy as np

ARCH_LLAMA, ARCH_GPT2 = 0, 1


# ----------------------------------------------------------------------------------------------
# Row-wise pieces with their hand-derived backward
# ----------------------------------------------------------------------------------------------

def rms_fwd(x, g, eps):
    r = 1.0 / np.sqrt((x * x).mean(-1, keepdims=True) + eps)
    xh = x * r
    return xh * g, (xh, r, g)


def rms_bwd(dy, cache):
    """y = x r g, r = (mean x^2 + eps)^(-1/2): dx = r (dxh - xh mean(dxh xh)), dxh = dy g."""
    xh, r, g = cache
    dxh = dy * g
    dx = r * (dxh - xh * (dxh * xh).mean(-1, keepdims=True))
    return dx, (dy * xh).reshape(-1, xh.shape[-1]).sum(0)


def ln_fwd(x, g, b, eps):
    mu = x.mean(-1, keepdims=True)
    r = 1.0 / np.sqrt(((x - mu) ** 2).mean(-1, keepdims=True) + eps)
    xh = (x - mu) * r
    return xh * g + b, (xh, r, g)


def ln_bwd(dy, cache):
    """y = xh g + b, xh = (x - mu) r: dx = r (dxh - mean(dxh) - xh mean(dxh xh))."""
    xh, r, g = cache
    dxh = dy * g
    dx = r * (dxh - dxh.mean(-1, keepdims=True) - xh * (dxh * xh).mean(-1, keepdims=True))
    D = xh.shape[-1]
    return dx, (dy * xh).reshape(-1, D).sum(0), dy.reshape(-1, D).sum(0)


GELU_C = math.sqrt(2.0 / math.pi)


def gelu_fwd(x):
    u = np.tanh(GELU_C * (x + 0.044715 * x ** 3))
    return 0.5 * x * (1.0 + u), (x, u)


def gelu_bwd(dy, cache):
    """d/dx 0.5 x (1 + tanh a(x)) = 0.5 (1 + tanh a) + 0.5 x (1 - tanh^2 a) a'(x)."""
    x, u = cache
    da = GELU_C * (1.0 + 3 * 0.044715 * x * x)
    return dy * (0.5 * (1.0 + u) + 0.5 * x * (1.0 - u * u) * da)


def sigmoid(x):
    return 1.0 / (1.0 + np.exp(-x))


def rope_tables(S, hd, theta):
    half = hd // 2
    inv = theta ** (-2.0 * np.arange(half) / hd)
    ang = np.arange(S)[:, None] * inv[None, :]
    return np.cos(ang)[None, :, None, :], np.sin(ang)[None, :, None, :]


def rope_fwd(x, cos, sin):
    """Rotate-half: pair (j, j + hd/2) turned by the angle s theta^(-2j/hd)."""
    half = x.shape[-1] // 2
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], -1)


def rope_bwd(dy, cos, sin):
    """The transpose of a rotation turns by the opposite angle."""
    half = dy.shape[-1] // 2
    d1, d2 = dy[..., :half], dy[..., half:]
    return np.concatenate([d1 * cos + d2 * sin, d2 * cos - d1 * sin], -1)


def attn_fwd(q, k, v):
    """Causal attention per (batch, query head); query head h reads KV head h // (H / Hkv).
    q [B,S,H,hd], k, v [B,S,Hkv,hd] -> o [B,S,H,hd]."""
    B, S, H, hd = q.shape
    rep = H // k.shape[2]
    kv = np.arange(H) // rep
    qh = q.transpose(0, 2, 1, 3)
    kh = k.transpose(0, 2, 1, 3)[:, kv]
    vh = v.transpose(0, 2, 1, 3)[:, kv]
    s = qh @ kh.transpose(0, 1, 3, 2) / math.sqrt(hd)
    s = np.where(np.triu(np.ones((S, S), bool), 1), -np.inf, s)
    s = s - s.max(-1, keepdims=True)
    p = np.exp(s)
    p /= p.sum(-1, keepdims=True)
    o = p @ vh
    return o.transpose(0, 2, 1, 3), (qh, kh, vh, p, rep)


def attn_bwd(do, cache):
    """o = p v, p = softmax(q k^T / sqrt(hd)): dv = p^T do, dp = do v^T,
    ds = p (dp - rowsum(dp p)), dq = ds k / sqrt(hd), dk = ds^T q / sqrt(hd); a KV head's gradient
    is the sum over the query heads that read it."""
    qh, kh, vh, p, rep = cache
    B, H, S, hd = qh.shape
    doh = do.transpose(0, 2, 1, 3)
    dvh = p.transpose(0, 1, 3, 2) @ doh
    dp = doh @ vh.transpose(0, 1, 3, 2)
    ds = p * (dp - (dp * p).sum(-1, keepdims=True))
    sc = 1.0 / math.sqrt(hd)
    dq = (ds @ kh) * sc
    dkh = (ds.transpose(0, 1, 3, 2) @ qh) * sc
    Hkv = H // rep
    dk = dkh.reshape(B, Hkv, rep, S, hd).sum(2)
    dv = dvh.reshape(B, Hkv, rep, S, hd).sum(2)
    return dq.transpose(0, 2, 1, 3), dk.transpose(0, 2, 1, 3), dv.transpose(0, 2, 1, 3)


def lin_bwd(dy, x, w):
    """y = x w^T: dx = dy w, dw = dy^T x over every row."""
    D_out, D_in = w.shape
    return dy @ w, dy.reshape(-1, D_out).T @ x.reshape(-1, D_in)


# ----------------------------------------------------------------------------------------------
# Blocks, chunks and the readout
# ----------------------------------------------------------------------------------------------

class Dims:
    def __init__(self, d):
        self.arch, self.D, self.H, self.Hkv = d.arch, d.d_model, d.n_heads, d.n_kv_heads
        self.f, self.V, self.eps, self.theta = d.d_ff, d.vocab, d.norm_eps, d.rope_theta
        self.hd = self.D // self.H


def layer_fwd(P, l, x, m: Dims):
    w = lambda s: P[f"layers.{l}.{s}"]
    B, S, _ = x.shape
    H, Hkv, hd = m.H, m.Hkv, m.hd
    c = {"x": x}
    if m.arch == ARCH_LLAMA:
        a, c["n1"] = rms_fwd(x, w("attn_norm.weight"), m.eps)
        qkv = a @ w("wqkv").T
    else:
        a, c["n1"] = ln_fwd(x, w("attn_norm.weight"), w("attn_norm.bias"), m.eps)
        qkv = a @ w("wqkv").T + w("bqkv")
    c["a"] = a
    q = qkv[..., :H * hd].reshape(B, S, H, hd)
    k = qkv[..., H * hd:(H + Hkv) * hd].reshape(B, S, Hkv, hd)
    v = qkv[..., (H + Hkv) * hd:].reshape(B, S, Hkv, hd)
    if m.arch == ARCH_LLAMA:
        c["rope"] = rope_tables(S, hd, m.theta)
        q, k = rope_fwd(q, *c["rope"]), rope_fwd(k, *c["rope"])
    o, c["attn"] = attn_fwd(q, k, v)
    o = o.reshape(B, S, H * hd)
    c["o"] = o
    x2 = x + o @ w("wo").T + (w("bo") if m.arch == ARCH_GPT2 else 0.0)
    c["x2"] = x2
    if m.arch == ARCH_LLAMA:
        b, c["n2"] = rms_fwd(x2, w("ffn_norm.weight"), m.eps)
        gu = b @ w("w1").T
        gate, up = gu[..., :m.f], gu[..., m.f:]
        sg = sigmoid(gate)
        act = gate * sg * up
        c.update(b=b, gate=gate, up=up, sg=sg, act=act)
        return x2 + act @ w("w2").T, c
    b, c["n2"] = ln_fwd(x2, w("ffn_norm.weight"), w("ffn_norm.bias"), m.eps)
    pre = b @ w("w1").T + w("b1")
    act, c["gelu"] = gelu_fwd(pre)
    c.update(b=b, act=act)
    return x2 + act @ w("w2").T + w("b2"), c


def layer_bwd(P, l, dy, c, m: Dims) -> Tuple[np.ndarray, Dict[str, np.ndarray]]:
    """Gradient at the block input and of every block tensor, from dy at the block output."""
    w = lambda s: P[f"layers.{l}.{s}"]
    n = lambda s: f"layers.{l}.{s}"
    g = {}
    B, S, D = dy.shape
    H, Hkv, hd = m.H, m.Hkv, m.hd
    # FFN (residual: dy reaches x2 directly and through the FFN)
    dact, g[n("w2")] = lin_bwd(dy, c["act"], w("w2"))
    if m.arch == ARCH_LLAMA:
        sg, gate, up = c["sg"], c["gate"], c["up"]
        silu = gate * sg
        dgate = dact * up * sg * (1.0 + gate * (1.0 - sg))
        dup = dact * silu
        dgu = np.concatenate([dgate, dup], -1)
        db, g[n("w1")] = lin_bwd(dgu, c["b"], w("w1"))
        dx2, g[n("ffn_norm.weight")] = rms_bwd(db, c["n2"])
    else:
        g[n("b2")] = dy.reshape(-1, D).sum(0)
        dpre = gelu_bwd(dact, c["gelu"])
        g[n("b1")] = dpre.reshape(-1, dpre.shape[-1]).sum(0)
        db, g[n("w1")] = lin_bwd(dpre, c["b"], w("w1"))
        dx2, g[n("ffn_norm.weight")], g[n("ffn_norm.bias")] = ln_bwd(db, c["n2"])
    dx2 = dx2 + dy
    # attention
    do, g[n("wo")] = lin_bwd(dx2, c["o"], w("wo"))
    if m.arch == ARCH_GPT2:
        g[n("bo")] = dx2.reshape(-1, D).sum(0)
    dq, dk, dv = attn_bwd(do.reshape(B, S, H, hd), c["attn"])
    if m.arch == ARCH_LLAMA:
        dq, dk = rope_bwd(dq, *c["rope"]), rope_bwd(dk, *c["rope"])
    dqkv = np.concatenate([dq.reshape(B, S, -1), dk.reshape(B, S, -1), dv.reshape(B, S, -1)], -1)
    da, g[n("wqkv")] = lin_bwd(dqkv, c["a"], w("wqkv"))
    if m.arch == ARCH_LLAMA:
        dx, g[n("attn_norm.weight")] = rms_bwd(da, c["n1"])
    else:
        g[n("bqkv")] = dqkv.reshape(-1, dqkv.shape[-1]).sum(0)
        dx, g[n("attn_norm.weight")], g[n("attn_norm.bias")] = ln_bwd(da, c["n1"])
    return dx + dx2, g


def embed(P, ids, m: Dims):
    h = P["tok_emb"][ids]
    if m.arch == ARCH_GPT2:
        h = h + P["pos_emb"][: ids.shape[1]][None]
    return h


def readout_fwd(P, h, m: Dims):
    if m.arch == ARCH_LLAMA:
        nrm, c = rms_fwd(h, P["norm_f.weight"], m.eps)
        return nrm @ P["lm_head"].T, c
    nrm, c = ln_fwd(h, P["norm_f.weight"], P["norm_f.bias"], m.eps)
    return nrm @ P["tok_emb"].T, c


def readout_bwd(P, dz, c, m: Dims):
    """dh through the frozen head and final norm (their own gradients are not needed)."""
    head = P["lm_head"] if m.arch == ARCH_LLAMA else P["tok_emb"]
    dn = dz @ head
    return rms_bwd(dn, c)[0] if m.arch == ARCH_LLAMA else ln_bwd(dn, c)[0]


# ----------------------------------------------------------------------------------------------
# Local objective (Eq. 3-5) and its logit gradient in closed form
# ----------------------------------------------------------------------------------------------

def lse(z):
    mx = z.max(-1, keepdims=True)
    return (mx + np.log(np.exp(z - mx).sum(-1, keepdims=True)))[..., 0]


def objective_and_dz(z, t, labels, alpha, kl_dir):
    V = z.shape[-1]
    zf = z.reshape(-1, V)
    y = labels.reshape(-1)
    valid = y >= 0
    n_valid = max(int(valid.sum()), 1)
    lz = lse(zf)
    p = np.exp(zf - lz[:, None])
    onehot = np.zeros_like(zf)
    onehot[np.arange(len(y)), np.maximum(y, 0)] = 1.0
    ce = lz - zf[np.arange(len(y)), np.maximum(y, 0)]
    row = alpha * ce
    dz = alpha * (p - onehot)
    if alpha < 1.0:
        tf = t.reshape(-1, V)
        lt = lse(tf)
        q = np.exp(tf - lt[:, None])
        if kl_dir == 0:
            diff = (zf - lz[:, None]) - (tf - lt[:, None])     # log p - log q
            kl = (p * diff).sum(-1)
            dz = dz + (1.0 - alpha) * p * (diff - kl[:, None])
        else:
            kl = (q * ((tf - lt[:, None]) - (zf - lz[:, None]))).sum(-1)
            dz = dz + (1.0 - alpha) * (p - q)
        row = row + (1.0 - alpha) * kl
    row = np.where(valid, row, 0.0)
    dz = np.where(valid[:, None], dz, 0.0) / n_valid
    return row.sum() / n_valid, dz.reshape(z.shape)


# ----------------------------------------------------------------------------------------------
# Gradients: one chunk's local objective, and backpropagation through every chunk
# ----------------------------------------------------------------------------------------------

def chunk_fwd(P, bounds, k, h, m: Dims):
    caches = []
    for l in range(bounds[k - 1], bounds[k]):
        h, c = layer_fwd(P, l, h, m)
        caches.append((l, c))
    return h, caches


def chunk_bwd(P, dh, caches, m: Dims):
    grads = {}
    for l, c in reversed(caches):
        dh, g = layer_bwd(P, l, dh, c, m)
        grads.update(g)
    return dh, grads


LORA_LINEARS = ("wqkv", "wo", "w1", "w2")


def merge_lora(P, n_layers, scale):
    """Weights with their low-rank updates folded in: w + scale * B A (Section II-A)."""
    Q = dict(P)
    for l in range(n_layers):
        for s in LORA_LINEARS:
            a = P.get(f"layers.{l}.{s}.lora_a")
            if a is not None:
                Q[f"layers.{l}.{s}"] = P[f"layers.{l}.{s}"] + scale * (P[f"layers.{l}.{s}.lora_b"] @ a)
    return Q


def lora_grads(P, grads, scale):
    """y = x (w + s B A)^T: with G = dL/d(w + s B A), dL/dB = s G A^T and dL/dA = s B^T G; the base
    weights, norms and biases are frozen."""
    out = {}
    for n, G in grads.items():
        a = P.get(n + ".lora_a")
        if a is not None:
            out[n + ".lora_b"] = scale * G @ a.T
            out[n + ".lora_a"] = scale * P[n + ".lora_b"].T @ G
    return out


def adapter_fwd(P, k, h):
    """a_k(h) = h + GELU(h D^T) U^T (readout adapter of chunk k, Section III-B (b))."""
    D, U = P[f"adapters.{k}.down"], P[f"adapters.{k}.up"]
    act, gc = gelu_fwd(h @ D.T)
    return h + act @ U.T, (h, act, gc)


def adapter_bwd(P, k, da, cache):
    """dU = da^T GELU(u), du = (da U) GELU'(u), dD = du^T h, dh = da + du D."""
    h, act, gc = cache
    D, U = P[f"adapters.{k}.down"], P[f"adapters.{k}.up"]
    r, dm = D.shape
    dU = da.reshape(-1, dm).T @ act.reshape(-1, r)
    du = gelu_bwd(da @ U, gc)
    dD = du.reshape(-1, r).T @ h.reshape(-1, dm)
    return da + du @ D, {f"adapters.{k}.down": dD, f"adapters.{k}.up": dU}


def local_grad(P, d, bounds, k, h_prev, labels, alpha, kl_dir=0, lora_scale=None, adapters=False):
    """(L_k, dL_k/dtheta_k, h_k): teacher and input held constant (Eq. 5, Remark 1). lora_scale: only
    the low-rank factors train; adapters: chunk k's readout goes through its adapter (the teacher is
    the frozen head on h_{k-1})."""
    m = Dims(d)
    W = merge_lora(P, d.n_layers, lora_scale) if lora_scale is not None else P
    t = readout_fwd(W, h_prev, m)[0] if alpha < 1.0 else None
    h, caches = chunk_fwd(W, bounds, k, h_prev, m)
    x, ac = adapter_fwd(P, k, h) if adapters else (h, None)
    z, rc = readout_fwd(W, x, m)
    L, dz = objective_and_dz(z, t, labels, alpha, kl_dir)
    dh = readout_bwd(W, dz, rc, m)
    extra = {}
    if adapters:
        dh, extra = adapter_bwd(P, k, dh, ac)
    _, grads = chunk_bwd(W, dh, caches, m)
    if lora_scale is not None:
        grads = lora_grads(P, grads, lora_scale)
    grads.update(extra)
    return L, grads, h


def bp_grad(P, d, bounds, ids, labels):
    """Cross-entropy of the last readout and its gradient through all chunks (backpropagation)."""
    m = Dims(d)
    h = embed(P, ids, m)
    all_caches = []
    for k in range(1, len(bounds)):
        h, caches = chunk_fwd(P, bounds, k, h, m)
        all_caches.append(caches)
    z, rc = readout_fwd(P, h, m)
    L, dz = objective_and_dz(z, None, labels, 1.0, 0)
    dh = readout_bwd(P, dz, rc, m)
    grads = {}
    for caches in reversed(all_caches):
        dh, g = chunk_bwd(P, dh, caches, m)
        grads.update(g)
    return L, grads
