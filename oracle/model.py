"""Plain CPU restatement of ZeroLock (Section II-A, Eq. 1-6) -- test infrastructure only.

Only tests, ``__graft_entry__.smoke()`` and bench.py's CPU-baseline leg use this
module; the CUDA library never does.

Notation follows the paper: h_0 = E(x), h_k = f_k(h_{k-1}) (Eq. 1);
z_k = Norm(h_k) W_lm^T, p_k = softmax(z_k) (Eq. 2);
L_k = alpha * L_Task(p_k) + (1 - alpha) * L_Consis(p_k, sg(p_{k-1})) (Eq. 3),
with L_Task read as token cross-entropy (Eq. 4 and the sentence after it) and
L_Consis as KL(p_k || p_{k-1}) (Eq. 5 with the KL choice of Section II-C);
both are means over the loss set Omega (positions with label >= 0).
Chunk k's gradient is the gradient of L_k with respect to chunk k's own
parameters with h_{k-1} and p_{k-1} held constant (stop-gradient, Eq. 5;
Remark 1); the update is AdamW (the paper's on-device optimizer, Section
III-C) in its decoupled form, the gradient of a window being the mean of its
m micro-batch gradients (step S3).

Readings where the paper is silent (the same readings are listed in the design
notes of the repository):
  * Eq. 4's leading minus sign is a typo (it would maximise the divergence); the
    task term is +CE.
  * p_0 (the consistency target of chunk 1) is the readout of h_0 = E(x);
    ``consis_first=0`` drops it (alpha_1 = 1).
  * Llama blocks: RMSNorm (eps 1e-5), rotate-half RoPE with theta 10000 and
    positions 0..S-1 per sequence, causal attention with scale 1/sqrt(hd),
    grouped KV heads (query head h reads KV head h // (H / H_kv)), SwiGLU FFN
    silu(gate) * up. GPT-2 blocks: LayerNorm with bias, learned positions,
    GELU (tanh form), biased linears, LM head tied to the token embedding.
  * The readout reuses the model's final norm and LM head, frozen (Eq. 2,
    "static model head" of Section III-B). The embedding is frozen.
  * Every layer tensor of a chunk is trainable (full fine-tune); weight decay
    applies to all of them; no clipping.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Sequence, Tuple

import torch

from synth import (ARCH_GPT2, ARCH_LLAMA, LORA_TARGETS, ModelDims, adapter_param_shapes, layer_param_shapes,
                   lora_param_shapes)

Tensor = torch.Tensor


# ----------------------------------------------------------------------------------------
# Building blocks (each is the textbook definition)
# ----------------------------------------------------------------------------------------

def rmsnorm(x: Tensor, g: Tensor, eps: float) -> Tensor:
    """x / sqrt(mean(x^2) + eps) * g over the last axis."""
    return x / torch.sqrt((x * x).mean(-1, keepdim=True) + eps) * g


def layernorm(x: Tensor, g: Tensor, b: Tensor, eps: float) -> Tensor:
    """(x - mean) / sqrt(var + eps) * g + b, biased variance, over the last axis."""
    mu = x.mean(-1, keepdim=True)
    var = ((x - mu) ** 2).mean(-1, keepdim=True)
    return (x - mu) / torch.sqrt(var + eps) * g + b


def gelu_tanh(x: Tensor) -> Tensor:
    """GELU, tanh approximation: 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))."""
    return 0.5 * x * (1.0 + torch.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def silu(x: Tensor) -> Tensor:
    """x * sigmoid(x)."""
    return x / (1.0 + torch.exp(-x))


def rope(x: Tensor, theta: float) -> Tensor:
    """Rotate-half rotary embedding of x [B, S, H, hd] at positions 0..S-1.

    Pair (i, i + hd/2) is rotated by the angle s * theta^(-2i/hd).
    """
    S, hd = x.shape[1], x.shape[3]
    half = hd // 2
    i = torch.arange(half, dtype=torch.float64)
    inv = theta ** (-2.0 * i / hd)
    ang = torch.arange(S, dtype=torch.float64)[:, None] * inv[None, :]
    cos = torch.cos(ang).to(x.dtype)[None, :, None, :]
    sin = torch.sin(ang).to(x.dtype)[None, :, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return torch.cat([x1 * cos - x2 * sin, x2 * cos + x1 * sin], dim=-1)


def attention(q: Tensor, k: Tensor, v: Tensor) -> Tensor:
    """Causal softmax attention; q [B,S,H,hd], k/v [B,S,Hkv,hd] -> [B,S,H,hd]."""
    B, S, H, hd = q.shape
    Hkv = k.shape[2]
    rep = H // Hkv
    kk = k.repeat_interleave(rep, dim=2)          # query head h reads kv head h // rep
    vv = v.repeat_interleave(rep, dim=2)
    qh, kh, vh = (t.permute(0, 2, 1, 3) for t in (q, kk, vv))   # [B,H,S,hd]
    s = qh @ kh.transpose(-1, -2) / math.sqrt(hd)
    mask = torch.triu(torch.ones(S, S, dtype=torch.bool), diagonal=1)
    s = s.masked_fill(mask, float("-inf"))
    p = torch.softmax(s, dim=-1)
    return (p @ vh).permute(0, 2, 1, 3)


# ----------------------------------------------------------------------------------------
# Model (Eq. 1, Eq. 2)
# ----------------------------------------------------------------------------------------

def embed(P: Dict[str, Tensor], ids: Tensor, d: ModelDims) -> Tensor:
    """h_0 = E(x): token embedding rows (+ learned positions for GPT-2). [B,S,d]."""
    h = P["tok_emb"][ids.long()]
    if d.arch == ARCH_GPT2:
        S = ids.shape[1]
        h = h + P["pos_emb"][:S][None]
    return h


def lora_weight(P: Dict[str, Tensor], l: int, name: str, scale: float) -> Tensor:
    """w_l + Delta w_l with Delta w_l = scale * B_l A_l when the layer carries LoRA factors (Section II-A)."""
    w = P[f"layers.{l}.{name}"]
    a = P.get(f"layers.{l}.{name}.lora_a")
    if a is None:
        return w
    return w + scale * (P[f"layers.{l}.{name}.lora_b"] @ a)


def layer_forward(P: Dict[str, Tensor], l: int, x: Tensor, d: ModelDims, lora_scale: float = 1.0) -> Tensor:
    """One transformer block (pre-norm residual) on x [B,S,d]; linear weights include LoRA updates."""
    g = lambda s: lora_weight(P, l, s, lora_scale) if s in LORA_TARGETS else P[f"layers.{l}.{s}"]
    B, S, _ = x.shape
    H, Hkv, hd = d.n_heads, d.n_kv_heads, d.head_dim
    if d.arch == ARCH_LLAMA:
        a = rmsnorm(x, g("attn_norm.weight"), d.norm_eps)
        qkv = a @ g("wqkv").T
    else:
        a = layernorm(x, g("attn_norm.weight"), g("attn_norm.bias"), d.norm_eps)
        qkv = a @ g("wqkv").T + g("bqkv")
    q = qkv[..., : H * hd].reshape(B, S, H, hd)
    k = qkv[..., H * hd: (H + Hkv) * hd].reshape(B, S, Hkv, hd)
    v = qkv[..., (H + Hkv) * hd:].reshape(B, S, Hkv, hd)
    if d.arch == ARCH_LLAMA:
        q, k = rope(q, d.rope_theta), rope(k, d.rope_theta)
    o = attention(q, k, v).reshape(B, S, H * hd)
    if d.arch == ARCH_LLAMA:
        x = x + o @ g("wo").T
        b = rmsnorm(x, g("ffn_norm.weight"), d.norm_eps)
        gu = b @ g("w1").T
        act = silu(gu[..., : d.d_ff]) * gu[..., d.d_ff:]
        return x + act @ g("w2").T
    x = x + o @ g("wo").T + g("bo")
    b = layernorm(x, g("ffn_norm.weight"), g("ffn_norm.bias"), d.norm_eps)
    act = gelu_tanh(b @ g("w1").T + g("b1"))
    return x + act @ g("w2").T + g("b2")


def chunk_forward(P: Dict[str, Tensor], bounds: Sequence[int], k: int, h: Tensor,
                  d: ModelDims, lora_scale: float = 1.0) -> Tensor:
    """h_k = f_k(h_{k-1}; W_k + Delta W_k) over layers bounds[k-1] .. bounds[k]-1 (Eq. 1)."""
    for l in range(bounds[k - 1], bounds[k]):
        h = layer_forward(P, l, h, d, lora_scale)
    return h


def readout(P: Dict[str, Tensor], h: Tensor, d: ModelDims) -> Tensor:
    """z = Norm(h) W_lm^T with the model's frozen final norm and head (Eq. 2)."""
    if d.arch == ARCH_LLAMA:
        n = rmsnorm(h, P["norm_f.weight"], d.norm_eps)
        return n @ P["lm_head"].T
    n = layernorm(h, P["norm_f.weight"], P["norm_f.bias"], d.norm_eps)
    return n @ P["tok_emb"].T


def adapter(P: Dict[str, Tensor], k: int, h: Tensor) -> Tensor:
    """Readout adapter of chunk k (Section III-B, Local Update Interface, option (b)): a small residual
    MLP before the frozen head, a_k(h) = h + GELU(h D_k^T) U_k^T, which is the identity while U_k = 0."""
    return h + gelu_tanh(h @ P[f"adapters.{k}.down"].T) @ P[f"adapters.{k}.up"].T


# ----------------------------------------------------------------------------------------
# Local objective (Eq. 3-5)
# ----------------------------------------------------------------------------------------

def kl_rows(z: Tensor, t: Tensor, kl_dir: int = 0) -> Tensor:
    """Per-row KL between softmax(z) = p and softmax(t) = q.

    kl_dir 0: KL(p || q) = sum p (log p - log q)  (Eq. 5, the paper's direction);
    kl_dir 1: KL(q || p) (forward distillation, an option).
    """
    lp = torch.log_softmax(z, dim=-1)
    lq = torch.log_softmax(t, dim=-1)
    if kl_dir == 0:
        return (lp.exp() * (lp - lq)).sum(-1)
    return (lq.exp() * (lq - lp)).sum(-1)


def local_objective_rows(z: Tensor, t: Optional[Tensor], labels: Tensor, alpha: float,
                         kl_dir: int = 0) -> Tensor:
    """alpha * CE_i + (1 - alpha) * KL_i per row i; 0 on rows outside Omega.

    z, t: [..., V] logits of this chunk and of the stop-gradient teacher;
    labels: [...] int with -1 marking rows outside Omega.
    """
    V = z.shape[-1]
    zf = z.reshape(-1, V)
    lab = labels.reshape(-1).long()
    valid = lab >= 0
    lse = torch.logsumexp(zf, dim=-1)
    zy = zf.gather(1, lab.clamp(min=0)[:, None])[:, 0]
    ce = lse - zy
    row = alpha * ce
    if alpha < 1.0:
        row = row + (1.0 - alpha) * kl_rows(zf, t.reshape(-1, V), kl_dir)
    return torch.where(valid, row, torch.zeros_like(row))


def local_objective(z: Tensor, t: Optional[Tensor], labels: Tensor, alpha: float,
                    kl_dir: int = 0) -> Tensor:
    """L_k = (1/|Omega|) sum_{i in Omega} [alpha CE_i + (1 - alpha) KL_i] (Eq. 3)."""
    n_valid = int((labels >= 0).sum())
    return local_objective_rows(z, t, labels, alpha, kl_dir).sum() / max(n_valid, 1)


# ----------------------------------------------------------------------------------------
# Update rule
# ----------------------------------------------------------------------------------------

def adamw_update(theta: Tensor, g: Tensor, m: Tensor, v: Tensor, step: int, lr: float,
                 beta1: float, beta2: float, eps: float, wd: float) -> None:
    """One decoupled AdamW step (Loshchilov and Hutter), in place; `step` counts from 1.

    theta <- theta (1 - lr wd); m <- b1 m + (1-b1) g; v <- b2 v + (1-b2) g^2;
    theta <- theta - lr * (m / (1 - b1^step)) / (sqrt(v / (1 - b2^step)) + eps).
    """
    theta.mul_(1.0 - lr * wd)
    m.mul_(beta1).add_((1.0 - beta1) * g)
    v.mul_(beta2).add_((1.0 - beta2) * g * g)
    mhat = m / (1.0 - beta1 ** step)
    vhat = v / (1.0 - beta2 ** step)
    theta.sub_(lr * mhat / (torch.sqrt(vhat) + eps))


# ----------------------------------------------------------------------------------------
# The stateful oracle
# ----------------------------------------------------------------------------------------

@dataclasses.dataclass
class OracleConfig:
    dims: ModelDims
    bounds: List[int]              # K + 1 layer boundaries, bounds[0] = 0, bounds[K] = n_layers
    alpha: float = 0.5
    kl_dir: int = 0
    consis_first: int = 1
    lr: float = 1e-3
    beta1: float = 0.9
    beta2: float = 0.999
    eps: float = 1e-8
    weight_decay: float = 0.01
    accum_m: int = 1
    lr_schedule: int = 0            # 0: constant; 1: lr / sqrt(t + lr_gamma) (Theorem 1)
    lr_gamma: float = 1.0
    lora_rank: int = 0              # 0: every layer tensor trainable; r > 0: only the LoRA factors
    lora_scale: float = 1.0         # Delta w = lora_scale * B A
    adapter_dim: int = 0            # > 0: chunk k's own readout goes through its adapter a_k

    @property
    def K(self) -> int:
        return len(self.bounds) - 1


class Oracle:
    """ZeroLock state (parameters, AdamW moments, per-chunk counters) and its steps."""

    def __init__(self, cfg: OracleConfig, params: Dict[str, Tensor],
                 dtype: torch.dtype = torch.float64):
        self.cfg = cfg
        self.d = cfg.dims
        self.dtype = dtype
        self.P = {n: t.detach().to(dtype).clone() for n, t in params.items()}
        self.m = {}
        self.v = {}
        self.acc = {}
        for n in self.trainable_names():
            self.m[n] = torch.zeros_like(self.P[n])
            self.v[n] = torch.zeros_like(self.P[n])
            self.acc[n] = torch.zeros_like(self.P[n])
        K = cfg.K
        self.micro = [0] * (K + 1)       # micro-batches seen in the current window, per chunk
        self.t = [0] * (K + 1)           # optimizer steps taken, per chunk

    # -- parameter sets ------------------------------------------------------------------
    def chunk_names(self, k: int) -> List[str]:
        """The trainable tensors of chunk k: all layer tensors, or only the LoRA factors A_l, B_l."""
        shapes = (lora_param_shapes(self.d, self.cfg.lora_rank) if self.cfg.lora_rank > 0
                  else layer_param_shapes(self.d))
        out = []
        for l in range(self.cfg.bounds[k - 1], self.cfg.bounds[k]):
            out += [f"layers.{l}.{s}" for s, _ in shapes]
        if self.cfg.adapter_dim > 0:
            out += [f"adapters.{k}.{s}" for s, _ in adapter_param_shapes(self.d, self.cfg.adapter_dim)]
        return out

    def trainable_names(self) -> List[str]:
        out = []
        for k in range(1, self.cfg.K + 1):
            out += self.chunk_names(k)
        return out

    def alpha_k(self, k: int) -> float:
        return 1.0 if (k == 1 and not self.cfg.consis_first) else self.cfg.alpha

    # -- forward pieces ------------------------------------------------------------------
    def embed(self, ids: Tensor) -> Tensor:
        return embed(self.P, ids, self.d)

    def forward_chunk(self, k: int, h_prev: Tensor) -> Tensor:
        with torch.no_grad():
            return chunk_forward(self.P, self.cfg.bounds, k, h_prev.to(self.dtype), self.d, self.cfg.lora_scale)

    def readout(self, h: Tensor) -> Tensor:
        with torch.no_grad():
            return readout(self.P, h.to(self.dtype), self.d)

    def student_readout(self, P: Dict[str, Tensor], k: int, h: Tensor) -> Tensor:
        """Chunk k's own readout z_k: through its adapter when adapters are on. The teacher p_{k-1} is
        always the frozen head on h_{k-1} (chunk k builds it from its input hidden state alone)."""
        if self.cfg.adapter_dim > 0:
            h = adapter(P, k, h)
        return readout(P, h, self.d)

    # -- one chunk's local objective and gradient -----------------------------------------
    def local_grad(self, k: int, h_prev: Tensor, labels: Tensor
                   ) -> Tuple[float, Dict[str, Tensor], Tensor]:
        """(L_k, dL_k/dtheta_k, h_k) with h_{k-1} and the teacher p_{k-1} held constant."""
        names = self.chunk_names(k)
        leaves = {n: self.P[n].clone().requires_grad_(True) for n in names}
        P = dict(self.P)
        P.update(leaves)
        h_in = h_prev.detach().to(self.dtype)                      # sg(h_{k-1})
        a = self.alpha_k(k)
        t = readout(self.P, h_in, self.d).detach() if a < 1.0 else None   # sg(p_{k-1})
        h = chunk_forward(P, self.cfg.bounds, k, h_in, self.d, self.cfg.lora_scale)
        z = self.student_readout(P, k, h)
        L = local_objective(z, t, labels, a, self.cfg.kl_dir)
        grads = torch.autograd.grad(L, [leaves[n] for n in names])
        return float(L.detach()), dict(zip(names, grads)), h.detach()

    def _apply_window(self, k: int, adapters: bool = True) -> None:
        c = self.cfg
        self.t[k] += 1
        lr = c.lr if c.lr_schedule == 0 else c.lr / math.sqrt(self.t[k] - 1 + c.lr_gamma)
        for n in self.chunk_names(k):
            if not adapters and n.startswith("adapters."):
                continue
            g = self.acc[n] / c.accum_m
            adamw_update(self.P[n], g, self.m[n], self.v[n], self.t[k], lr,
                         c.beta1, c.beta2, c.eps, c.weight_decay)
            self.acc[n].zero_()
        self.micro[k] = 0

    def local_step(self, k: int, h_prev: Tensor, labels: Tensor) -> Tuple[float, Tensor]:
        """Chunk k's step on one micro-batch: accumulate its gradient, update at window end."""
        L, grads, h = self.local_grad(k, h_prev, labels)
        for n, g in grads.items():
            self.acc[n] += g
        self.micro[k] += 1
        if self.micro[k] == self.cfg.accum_m:
            self._apply_window(k)
        return L, h

    def step(self, ids: Tensor, labels: Tensor) -> List[float]:
        """One micro-batch through all K chunks (synchronous order, Eq. 1-6).

        Chunk k+1 reads h_k computed with chunk k's parameters before chunk k's
        own update of this micro-batch; the concurrent schedule must reach the
        same values.
        """
        h = self.embed(ids)
        losses = []
        for k in range(1, self.cfg.K + 1):
            L, h = self.local_step(k, h, labels)
            losses.append(L)
        return losses

    # -- backpropagation baseline and the global objective ------------------------------
    def bp_grad(self, ids: Tensor, labels: Tensor) -> Tuple[float, Dict[str, Tensor]]:
        """Global CE of the last readout and its gradient through all chunks (no adapters: they only
        serve the local objectives)."""
        names = [n for n in self.trainable_names() if not n.startswith("adapters.")]
        leaves = {n: self.P[n].clone().requires_grad_(True) for n in names}
        P = dict(self.P)
        P.update(leaves)
        h = embed(P, ids, self.d)
        for k in range(1, self.cfg.K + 1):
            h = chunk_forward(P, self.cfg.bounds, k, h, self.d, self.cfg.lora_scale)
        z = readout(P, h, self.d)
        L = local_objective(z, None, labels, 1.0)
        grads = torch.autograd.grad(L, [leaves[n] for n in names])
        return float(L.detach()), dict(zip(names, grads))

    def bp_step(self, ids: Tensor, labels: Tensor) -> float:
        L, grads = self.bp_grad(ids, labels)
        for n, g in grads.items():
            self.acc[n] += g
        for k in range(1, self.cfg.K + 1):
            self.micro[k] += 1
            if self.micro[k] == self.cfg.accum_m:
                self._apply_window(k, adapters=False)
        return L

    def global_loss(self, ids: Tensor, labels: Tensor) -> float:
        """L(p_K) = L_Task(p_K): CE of the last chunk's readout over Omega."""
        with torch.no_grad():
            h = self.embed(ids)
            for k in range(1, self.cfg.K + 1):
                h = chunk_forward(self.P, self.cfg.bounds, k, h, self.d, self.cfg.lora_scale)
            return float(local_objective(readout(self.P, h, self.d), None, labels, 1.0))
