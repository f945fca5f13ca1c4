"""Readout adapters (Section III-B, local update interface (b)) through the C ABI against the oracle.

Chunk k's own readout goes through a_k(h) = h + GELU(h D_k^T) U_k^T; its teacher stays the frozen head
on h_{k-1}. The adapters here start away from the identity (U drawn with std 0.05) so every gradient
term is exercised. fp32 workloads: losses and parameters after the steps within 1e-4 relative.
GPT-2 bf16 at full size: loss within 2e-2 and per-tensor gradient cosine >= 0.999 (oracle in fp32 on
the same bf16-rounded weights).
"""
import dataclasses

import pytest
import torch

import synth
from tests.gpu_common import cosine, engine_for, fro_rel, oracle_for, rel
from tests.test_parity_widths import WIDE

pytestmark = pytest.mark.gpu
DIM = 16


def _params(w, up_std=0.05, dim=DIM, K=None):
    P = synth.make_params(w.dims, w.seed)
    P.update(synth.make_adapter_params(w.dims, K or w.K, w.seed, dim, up_std=up_std))
    return P


@pytest.mark.parametrize("w", [synth.TINY, WIDE["gpt2-d1280"]], ids=["tiny-llama", "gpt2-d1280"])
def test_adapter_steps_match_oracle(w):
    P = _params(w)
    eng = engine_for(w, adapter_dim=DIM)
    eng.load(P)
    orc = oracle_for(w, P, adapter_dim=DIM)
    for s in range(min(w.steps, 5)):
        ids, labels = synth.make_batch(w, s)
        lg = eng.step(ids.cuda(), labels.cuda())
        lo = orc.step(ids, labels)
        for a, b in zip(lg, lo):
            assert rel(a, b) <= 1e-4, (s, lg, lo)
    for n in orc.trainable_names():
        got, ref = eng.get(n), orc.P[n]
        if n.endswith(".bqkv"):   # key bias: zero exact gradient, compared on the query and value thirds
            d, kv = w.dims.d_model, w.dims.n_kv_heads * w.dims.head_dim
            keep = list(range(d)) + list(range(d + kv, d + 2 * kv))
            got, ref = got[keep], ref[keep]
        assert fro_rel(got, ref) <= 1e-4, n
    eng.close()


def test_adapter_local_step_and_backprop_leave_the_rest_unchanged():
    """zl_local_step builds the same loss as the oracle's isolated chunk step; the backpropagation
    step does not touch the adapters and matches the adapter-free backpropagation step."""
    w = synth.TINY
    P = _params(w)
    eng = engine_for(w, adapter_dim=DIM)
    eng.load(P)
    orc = oracle_for(w, P, adapter_dim=DIM)
    ids, labels = synth.make_batch(w, 0)
    h1 = orc.forward_chunk(1, orc.embed(ids))
    got = eng.local_step(2, h1.float().reshape(-1, w.dims.d_model).contiguous().cuda(), None, labels.cuda())
    ref, _ = orc.local_step(2, h1, labels)
    assert rel(got, ref) <= 1e-4
    for n in orc.chunk_names(2):
        assert fro_rel(eng.get(n), orc.P[n]) <= 1e-4, n
    eng.close()
    bp = engine_for(w, adapter_dim=DIM)
    base = engine_for(w)
    bp.load(P)
    base.load({n: t for n, t in P.items() if not n.startswith("adapters.")})
    lb = bp.bp_step(ids.cuda(), labels.cuda())
    l0 = base.bp_step(ids.cuda(), labels.cuda())
    assert lb == l0
    for n, t in P.items():
        if n.startswith("adapters."):
            assert torch.equal(bp.get(n), t.reshape(-1)), n
        elif not n.startswith(("tok_emb", "pos_emb", "lm_head", "norm_f")):
            assert torch.equal(bp.get(n), base.get(n)), n
    bp.close()
    base.close()


def test_gpt2_adapter_chunk_full_size():
    """Chunk 2 of the GPT-2 bf16 workload at 8 x 512 with adapter width 64: gradients of its layers
    and of its adapter against the oracle on the engine's own h_1."""
    w = synth.GPT2_SMALL
    P = _params(w, dim=64)
    P = {n: (synth.round_bf16(t) if t.dim() == 2 else t) for n, t in P.items()}
    eng = engine_for(w, accum_m=2, adapter_dim=64)
    eng.load(P)
    ids, labels = synth.make_batch(w, 0)
    h1 = eng.forward_chunk(1, None, ids.cuda(), w.batch, w.seq)
    lg = eng.step(ids.cuda(), labels.cuda())
    orc = oracle_for(w, P, dtype=torch.float32, adapter_dim=64)
    L, g, _ = orc.local_grad(2, h1.float().cpu().view(w.batch, w.seq, -1), labels)
    assert rel(lg[1], L) <= 2e-2, (lg, L)
    for n in orc.chunk_names(2):
        c = cosine(eng.get(n, 1), g[n])
        assert c >= 0.999, (n, c)
    eng.close()
