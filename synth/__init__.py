"""Seeded synthetic inputs shared by the CUDA path's tests/bench and the CPU oracle's tests.

This module holds no arithmetic of the method itself: it only draws numbers.
Everything is counter based, so any tensor (or any slice of one) can be drawn
independently of the others and on any device with bit-identical integers.

Generator definitions (each is a published construction):

* SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom number
  generators", OOPSLA 2014): ``mix(z)`` below is its finaliser, applied to the
  counter ``key + (i + 1) * GOLDEN`` (the SplitMix64 state after i + 1 steps).
* Uniforms in (0, 1): the top 53 bits, ``((x >> 11) + 0.5) * 2**-53``.
* Normals: Box-Muller (Box and Muller 1958) in float64 from uniform pairs
  ``(u[2i], u[2i+1])``: ``r = sqrt(-2 ln u1)``, outputs ``r cos(2 pi u2)``
  and ``r sin(2 pi u2)`` interleaved.
* Token ids: Zipf(s) over ``[0, V)`` with rank r = id + 1,
  ``P(id) = r**-s / sum_r r**-s``, drawn by inverse-CDF search on a float64
  cumulative table.
* Labels: next-token shift inside each sequence, ``-1`` on the last position
  (``-1`` marks a position outside the loss set Omega).

Workload recipe of the model configurations (weights ~ N(0, 0.02), norm gains
1, biases 0, ids ~ Zipf(1.1)) follows the configurations listed in
``CONFIGS`` below.
"""
from __future__ import annotations

import dataclasses
import math
import zlib
from typing import Dict, Iterable, List, Optional, Tuple

import torch

GOLDEN = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB


def _s64(c: int) -> int:
    """Python int (0 <= c < 2**64) -> the int64 with the same bits."""
    c &= (1 << 64) - 1
    return c - (1 << 64) if c >= (1 << 63) else c


def _srl(z: torch.Tensor, s: int) -> torch.Tensor:
    """Logical right shift of int64 bit patterns."""
    return (z >> s) & ((1 << (64 - s)) - 1)


def mix64(z: torch.Tensor) -> torch.Tensor:
    """SplitMix64 finaliser on int64 bit patterns (wrapping arithmetic)."""
    z = (z ^ _srl(z, 30)) * _s64(_M1)
    z = (z ^ _srl(z, 27)) * _s64(_M2)
    return z ^ _srl(z, 31)


def mix64_int(z: int) -> int:
    """Scalar SplitMix64 finaliser on a Python int."""
    m = (1 << 64) - 1
    z &= m
    z = ((z ^ (z >> 30)) * _M1) & m
    z = ((z ^ (z >> 27)) * _M2) & m
    return z ^ (z >> 31)


def stream_key(seed: int, name: str) -> int:
    """Key of the named stream: mixes the seed and a CRC-32 of the name."""
    return mix64_int((seed * GOLDEN) ^ (zlib.crc32(name.encode()) << 17) ^ 0x5DEECE66D)


def raw_u64(key: int, start: int, n: int, device="cpu") -> torch.Tensor:
    """n SplitMix64 outputs (int64 bit patterns) at counters start..start+n-1."""
    i = torch.arange(start + 1, start + n + 1, dtype=torch.int64, device=device)
    return mix64(i * _s64(GOLDEN) + _s64(key))


def uniform(key: int, n: int, start: int = 0, device="cpu") -> torch.Tensor:
    """n float64 uniforms in (0, 1)."""
    x = _srl(raw_u64(key, start, n, device), 11).to(torch.float64)
    return (x + 0.5) * (2.0 ** -53)


def normal(key: int, n: int, std: float = 1.0, device="cpu") -> torch.Tensor:
    """n float64 N(0, std^2) draws by Box-Muller."""
    pairs = (n + 1) // 2
    u = uniform(key, 2 * pairs, 0, device).view(pairs, 2)
    r = torch.sqrt(-2.0 * torch.log(u[:, 0]))
    a = (2.0 * math.pi) * u[:, 1]
    out = torch.stack([r * torch.cos(a), r * torch.sin(a)], dim=1).reshape(-1)[:n]
    return out * std


def zipf_ids(seed: int, B: int, S: int, V: int, s: float = 1.1, device="cpu") -> torch.Tensor:
    """[B, S] int32 token ids, Zipf(s) over [0, V) with id = rank - 1."""
    r = torch.arange(1, V + 1, dtype=torch.float64)
    w = r ** (-s)
    cdf = torch.cumsum(w, 0)
    cdf = cdf / cdf[-1]
    u = uniform(stream_key(seed, "token_ids"), B * S)
    ids = torch.searchsorted(cdf, u, right=True).clamp_(max=V - 1)
    return ids.to(torch.int32).view(B, S).to(device)


def next_token_labels(ids: torch.Tensor) -> torch.Tensor:
    """labels[b, i] = ids[b, i + 1]; the last position of each row is -1 (not in Omega)."""
    lab = torch.full_like(ids, -1)
    lab[:, :-1] = ids[:, 1:]
    return lab


# ----------------------------------------------------------------------------------------
# Model configurations and parameter layout
# ----------------------------------------------------------------------------------------

ARCH_LLAMA = 0
ARCH_GPT2 = 1


@dataclasses.dataclass(frozen=True)
class ModelDims:
    arch: int
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    d_ff: int
    vocab: int
    max_seq: int
    norm_eps: float = 1e-5
    rope_theta: float = 10000.0

    @property
    def head_dim(self) -> int:
        return self.d_model // self.n_heads


@dataclasses.dataclass(frozen=True)
class Workload:
    """One model configuration with its batch, chunking and training settings."""
    name: str
    dims: ModelDims
    dtype: str            # "f32" or "bf16" (compute dtype of the CUDA path)
    batch: int
    seq: int
    K: int
    steps: int
    lr: float = 1e-3
    beta1: float = 0.9
    beta2: float = 0.999
    eps: float = 1e-8
    weight_decay: float = 0.01
    alpha: float = 0.5
    seed: int = 1234


def chunk_bounds(n_layers: int, K: int) -> List[int]:
    """Near-equal consecutive splits; the remainder goes to the last chunks.

    22 layers: K=2 -> 11,11; K=4 -> 5,5,6,6; K=8 -> 2,2,3,3,3,3,3,3 (the paper's
    TinyLlama split 7/7/8 also puts the remainder last).
    """
    base, rem = divmod(n_layers, K)
    sizes = [base + (1 if k >= K - rem else 0) for k in range(K)]
    b = [0]
    for sz in sizes:
        b.append(b[-1] + sz)
    return b


TINY = Workload("tiny-llama-f32", ModelDims(ARCH_LLAMA, 4, 128, 4, 4, 344, 512, 64),
                "f32", batch=4, seq=64, K=2, steps=10, seed=1234 + 0)
GPT2_SMALL = Workload("gpt2-small-bf16", ModelDims(ARCH_GPT2, 12, 768, 12, 12, 3072, 50257, 1024),
                      "bf16", batch=8, seq=512, K=4, steps=50, seed=1234 + 1)
LLAMA_1B = Workload("llama-1.1b-bf16", ModelDims(ARCH_LLAMA, 22, 2048, 32, 4, 5632, 32000, 2048),
                    "bf16", batch=4, seq=1024, K=8, steps=10, seed=1234 + 2)
LLAMA_3B = Workload("llama-3b-bf16", ModelDims(ARCH_LLAMA, 26, 3200, 32, 32, 8640, 32000, 2048),
                    "bf16", batch=2, seq=2048, K=4, steps=20, seed=1234 + 3)
LLAMA_7B = Workload("llama-7b-bf16", ModelDims(ARCH_LLAMA, 32, 4096, 32, 32, 11008, 32000, 4096),
                    "bf16", batch=2, seq=1024, K=8, steps=10, seed=1234 + 4)
CONFIGS = [TINY, GPT2_SMALL, LLAMA_1B, LLAMA_3B, LLAMA_7B]


def layer_param_shapes(d: ModelDims) -> List[Tuple[str, Tuple[int, ...]]]:
    """Per-layer tensors (suffix, shape). Weights are [out, in] row-major (y = x W^T).

    Llama: attn_norm.weight, wqkv = [Wq; Wk; Wv], wo, ffn_norm.weight,
    w1 = [W_gate; W_up] ([2f, d]), w2 = W_down ([d, f]).
    GPT-2 adds LayerNorm biases and linear biases; w1 = W_fc ([f, d]).
    """
    hd = d.head_dim
    qkv = (d.n_heads + 2 * d.n_kv_heads) * hd
    if d.arch == ARCH_LLAMA:
        return [("attn_norm.weight", (d.d_model,)),
                ("wqkv", (qkv, d.d_model)),
                ("wo", (d.d_model, d.n_heads * hd)),
                ("ffn_norm.weight", (d.d_model,)),
                ("w1", (2 * d.d_ff, d.d_model)),
                ("w2", (d.d_model, d.d_ff))]
    return [("attn_norm.weight", (d.d_model,)), ("attn_norm.bias", (d.d_model,)),
            ("wqkv", (qkv, d.d_model)), ("bqkv", (qkv,)),
            ("wo", (d.d_model, d.n_heads * hd)), ("bo", (d.d_model,)),
            ("ffn_norm.weight", (d.d_model,)), ("ffn_norm.bias", (d.d_model,)),
            ("w1", (d.d_ff, d.d_model)), ("b1", (d.d_ff,)),
            ("w2", (d.d_model, d.d_ff)), ("b2", (d.d_model,))]


LORA_TARGETS = ("wqkv", "wo", "w1", "w2")


def lora_param_shapes(d: ModelDims, rank: int) -> List[Tuple[str, Tuple[int, ...]]]:
    """Per-layer LoRA tensors: for each linear W [out, in], lora_a [rank, in] and lora_b [out, rank]."""
    out = []
    for s, (o, i) in ((s, shp) for s, shp in layer_param_shapes(d) if s in LORA_TARGETS):
        out += [(f"{s}.lora_a", (rank, i)), (f"{s}.lora_b", (o, rank))]
    return out


def make_lora_params(d: ModelDims, seed: int, rank: int, b_std: float = 0.0,
                     layers: Optional[Iterable[int]] = None) -> Dict[str, torch.Tensor]:
    """LoRA factors: A ~ N(0, 0.02^2); B = 0 (the usual start, so the model begins at its base
    weights) unless b_std > 0 (tests use a non-zero B to exercise every gradient)."""
    layers = range(d.n_layers) if layers is None else layers
    out = {}
    for l in layers:
        for s, shp in lora_param_shapes(d, rank):
            name = f"layers.{l}.{s}"
            n = shp[0] * shp[1]
            if s.endswith("lora_a"):
                out[name] = normal(stream_key(seed, name), n, 0.02).to(torch.float32).view(shp)
            elif b_std > 0:
                out[name] = normal(stream_key(seed, name), n, b_std).to(torch.float32).view(shp)
            else:
                out[name] = torch.zeros(shp, dtype=torch.float32)
    return out


def adapter_param_shapes(d: ModelDims, dim: int) -> List[Tuple[str, Tuple[int, ...]]]:
    """Readout adapter of one chunk (residual bottleneck MLP a(h) = h + up(GELU(down(h)))):
    down [dim, d_model], up [d_model, dim]."""
    return [("down", (dim, d.d_model)), ("up", (d.d_model, dim))]


def make_adapter_params(d: ModelDims, K: int, seed: int, dim: int, up_std: float = 0.0) -> Dict[str, torch.Tensor]:
    """Adapters of chunks 1..K: down ~ N(0, 0.02^2); up = 0 (the adapter starts as the identity map)
    unless up_std > 0 (tests use a non-zero up to exercise every gradient)."""
    out = {}
    for k in range(1, K + 1):
        for s, shp in adapter_param_shapes(d, dim):
            name = f"adapters.{k}.{s}"
            n = shp[0] * shp[1]
            if s == "down":
                out[name] = normal(stream_key(seed, name), n, 0.02).to(torch.float32).view(shp)
            elif up_std > 0:
                out[name] = normal(stream_key(seed, name), n, up_std).to(torch.float32).view(shp)
            else:
                out[name] = torch.zeros(shp, dtype=torch.float32)
    return out


def frozen_param_shapes(d: ModelDims) -> List[Tuple[str, Tuple[int, ...]]]:
    """Frozen tensors: embedding (+ learned positions), final norm, LM head (GPT-2: tied to tok_emb)."""
    out = [("tok_emb", (d.vocab, d.d_model))]
    if d.arch == ARCH_GPT2:
        out += [("pos_emb", (d.max_seq, d.d_model)),
                ("norm_f.weight", (d.d_model,)), ("norm_f.bias", (d.d_model,))]
    else:
        out += [("norm_f.weight", (d.d_model,)), ("lm_head", (d.vocab, d.d_model))]
    return out


def param_names(d: ModelDims, layers: Optional[Iterable[int]] = None) -> List[Tuple[str, Tuple[int, ...]]]:
    layers = range(d.n_layers) if layers is None else layers
    out = []
    for l in layers:
        out += [(f"layers.{l}.{s}", shp) for s, shp in layer_param_shapes(d)]
    return out


def init_tensor(seed: int, name: str, shape: Tuple[int, ...], std: float = 0.02,
                device="cpu") -> torch.Tensor:
    """The fp32 initial value of one named tensor: gains 1, biases 0, matrices N(0, std^2)."""
    n = 1
    for s in shape:
        n *= s
    last = name.split(".")[-1]
    if name.endswith("norm.weight") or name == "norm_f.weight":
        return torch.ones(shape, dtype=torch.float32, device=device)
    if last == "bias" or last.startswith("b"):
        return torch.zeros(shape, dtype=torch.float32, device=device)
    return normal(stream_key(seed, name), n, std, device).to(torch.float32).view(shape)


def make_params(d: ModelDims, seed: int, layers: Optional[Iterable[int]] = None,
                frozen: bool = True, device="cpu") -> Dict[str, torch.Tensor]:
    """fp32 tensors of the named layers (all by default) and the frozen tensors."""
    out = {}
    if frozen:
        for name, shp in frozen_param_shapes(d):
            out[name] = init_tensor(seed, name, shp, device=device)
    for name, shp in param_names(d, layers):
        out[name] = init_tensor(seed, name, shp, device=device)
    return out


def round_bf16(t: torch.Tensor) -> torch.Tensor:
    """Round-to-nearest-even to bfloat16, returned as float32."""
    return t.to(torch.bfloat16).to(torch.float32)


def make_batch(w: Workload, step: int, device="cpu") -> Tuple[torch.Tensor, torch.Tensor]:
    """(ids [B,S] int32, labels [B,S] int32) of micro-batch `step` of a workload."""
    ids = zipf_ids(w.seed * 1_000_003 + step, w.batch, w.seq, w.dims.vocab)
    return ids.to(device), next_token_labels(ids).to(device)
