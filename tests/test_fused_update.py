"""The optimizer step fused into the weight-gradient products (GPU).

At the last micro-batch of an update window the backward's dW products of the chunk's matrices apply
AdamW (Eq. 6 as AdamW) in their epilogue instead of storing a gradient; norm gains, biases and adapters
get a range update after the backward. Every kernel applies the same explicitly rounded AdamW step, and
the fused gradient is formed with the same additions as the stored one, so the fused and unfused
engines must agree bit for bit: parameters, both moments, the (zeroed) gradient accumulators and the
losses, over several windows, for ZeroLock steps, local steps and the backpropagation baseline, on the
tensor-core path (with and without split-K) and on the CUDA-core fp32 path.
"""
import os

import pytest
import torch

import synth
from tests.gpu_common import engine_for

pytestmark = pytest.mark.gpu
GPT2S = synth.Workload("fused-gpt2-bf16", synth.ModelDims(synth.ARCH_GPT2, 4, 256, 4, 4, 1024, 1000, 256), "bf16",
                       batch=2, seq=256, K=2, steps=4, seed=1234 + 1)
LLAMAS = synth.Workload("fused-llama-bf16", synth.ModelDims(synth.ARCH_LLAMA, 2, 256, 4, 2, 704, 512, 256), "bf16",
                        batch=2, seq=128, K=2, steps=4, seed=1234 + 2)
# the down projection [256, 344] keeps row-major state (344 % 32 != 0), the other matrices take the blocked one
MIXED = synth.Workload("fused-llama-mixed", synth.ModelDims(synth.ARCH_LLAMA, 2, 256, 4, 2, 344, 512, 128), "bf16",
                       batch=2, seq=128, K=2, steps=4, seed=1234 + 4)
# ragged everywhere: d 200 (head dim 50, padded to 64 in attention), gate/up 688 rows, FFN 344 columns
ODD = synth.Workload("fused-llama-odd", synth.ModelDims(synth.ARCH_LLAMA, 2, 200, 4, 2, 344, 500, 192), "bf16",
                     batch=3, seq=96, K=2, steps=4, seed=1234 + 3)


def _params(w):
    P = synth.make_params(w.dims, w.seed)
    return {n: (synth.round_bf16(t) if (w.dtype == "bf16" and t.dim() == 2) else t) for n, t in P.items()}


def _state(eng, w):
    names = [n for n, _ in synth.param_names(w.dims)]
    if eng_adapter(eng):
        names += [f"adapters.{k}.{s}" for k in range(1, w.K + 1) for s in ("down", "up")]
    return {(n, i): eng.get(n, i) for n in names for i in range(4)}


def eng_adapter(eng):
    return getattr(eng, "adapter_dim", 0) > 0


def _run(w, P, kind, steps, **kw):
    eng = engine_for(w, **kw)
    eng.load(P)
    losses = []
    for s in range(steps):
        ids, labels = (t.cuda() for t in synth.make_batch(w, s))
        if kind == "zl":
            losses.append(eng.step(ids, labels))
        elif kind == "bp":
            losses.append(eng.bp_step(ids, labels))
        else:
            h = None
            for k in range(1, w.K + 1):
                out = torch.empty(w.batch * w.seq, w.dims.d_model, device="cuda", dtype=eng.torch_dtype)
                losses.append(eng.local_step(k, h, ids, labels, h_out=out))
                h = out
    st = _state(eng, w)
    eng.close()
    return losses, st


@pytest.mark.parametrize("w", [GPT2S, LLAMAS, MIXED, ODD, synth.TINY],
                         ids=["gpt2s-bf16", "llama-bf16", "mixed-bf16", "odd-bf16", "tiny-f32"])
@pytest.mark.parametrize("kind", ["zl", "bp", "local"])
@pytest.mark.parametrize("accum_m", [1, 2])
def test_fused_update_equals_unfused_bitwise(w, kind, accum_m):
    P = _params(w)
    a = _run(w, P, kind, 4, accum_m=accum_m)
    b = _run(w, P, kind, 4, accum_m=accum_m, unfused_update=True)
    assert a[0] == b[0]
    for key in b[1]:
        assert torch.equal(a[1][key], b[1][key]), key


@pytest.mark.parametrize("tile", ["128:2", "256:3", "64:1", "128:1:0", "128:1:1", "128:3:1"])
def test_fused_update_with_forced_tiles_and_split_k(tile, monkeypatch):
    """The fused step in the split-K reduction and under every tile width (the test hook ZL_GEMM_TILE
    forces the tile and split count of every product, fused and unfused alike)."""
    monkeypatch.setenv("ZL_GEMM_TILE", tile)
    P = _params(GPT2S)
    for accum_m in (1, 2):
        a = _run(GPT2S, P, "zl", 2 * accum_m, accum_m=accum_m)
        b = _run(GPT2S, P, "zl", 2 * accum_m, accum_m=accum_m, unfused_update=True)
        assert a[0] == b[0]
        for key in b[1]:
            assert torch.equal(a[1][key], b[1][key]), (tile, accum_m, key)


def test_fused_update_with_adapters():
    """Readout adapters ride the range update after a fused backward."""
    P = _params(GPT2S)
    P.update(synth.make_adapter_params(GPT2S.dims, GPT2S.K, GPT2S.seed, 32, up_std=0.02))
    a = _run(GPT2S, P, "zl", 3, adapter_dim=32)
    b = _run(GPT2S, P, "zl", 3, adapter_dim=32, unfused_update=True)
    assert a[0] == b[0]
    for key in b[1]:
        assert torch.equal(a[1][key], b[1][key]), key


def test_checkpoints_move_between_blocked_and_row_major_state():
    """With the fused update the matrices' master and moments are held in a blocked layout (16 x 32 pieces)
    where the shape allows it; the unfused engine keeps them row-major. Checkpoints are row-major either
    way: a chunk saved by one engine and loaded into the other continues exactly like an uninterrupted run
    of either (parameters, moments and losses bit for bit)."""
    from paper_2608_07974_gb300 import binding as b
    w = MIXED
    P = _params(w)
    ref = _run(w, P, "zl", 4)
    for src_kw, dst_kw in (({}, {"unfused_update": True}), ({"unfused_update": True}, {})):
        src, dst = engine_for(w, **src_kw), engine_for(w, **dst_kw)
        src.load(P)
        dst.load(P)   # the frozen tensors (embedding, head, final norm) are not part of a chunk checkpoint
        losses = []
        for s in range(2):
            ids, labels = (t.cuda() for t in synth.make_batch(w, s))
            losses.append(src.step(ids, labels))
        for k in range(1, w.K + 1):
            b.zl_chunk_load(dst.ctx, k, b.zl_chunk_save(src.ctx, k))
        src.close()
        for s in range(2, 4):
            ids, labels = (t.cuda() for t in synth.make_batch(w, s))
            losses.append(dst.step(ids, labels))
        st = _state(dst, w)
        dst.close()
        assert losses == ref[0], (src_kw, dst_kw)
        for key in ref[1]:
            assert torch.equal(st[key], ref[1][key]), (src_kw, dst_kw, key)
