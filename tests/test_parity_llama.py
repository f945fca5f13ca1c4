"""Llama-style bf16 workloads (1.1B with grouped KV heads, 3B with head_dim 100, 7B-shaped) against
the oracle, at full width and the full micro-batch of each workload.

The oracle runs in fp32 on the same bf16-rounded weights. Bars: loss relative error <= 2e-2, per-
tensor gradient cosine >= 0.999 (gradients read before the optimizer step: accum_m = 2).
Chunks are checked in isolation (input h_{k-1} taken from the engine), which is exact for the
method: chunk k's step depends on the rest of the model only through h_{k-1} (Lemma 3).
For 3B and 7B the engine holds just the first chunk's layers (a K = 1 model over them): its
input is h_0 and its teacher readout(h_0), the same computation as chunk 1 of the full model.

Steps 1 and 2 of the optimizer: with accum_m = 2, micro-batch 1's gradient is read from the
accumulator (step 1, at the loaded weights), micro-batch 2 ends the window (AdamW), and micro-batch
3's gradient is read again (step 2) and checked against the oracle at the engine's updated weights
rounded to bf16 (what the refreshed bf16 compute copy must hold), from the engine's own h_{k-1}.
"""
import dataclasses
import functools

import pytest
import torch

import synth
from tests.gpu_common import cosine, engine_for, fro_rel, oracle_for, rel

pytestmark = pytest.mark.gpu
LOSS_TOL, COS_MIN = 2e-2, 0.999


@functools.lru_cache(maxsize=1)
def _params(name, n_layers):
    w = {"1b": synth.LLAMA_1B, "3b": synth.LLAMA_3B, "7b": synth.LLAMA_7B}[name]
    P = synth.make_params(w.dims, w.seed, layers=range(n_layers))
    return {n: (synth.round_bf16(t) if t.dim() == 2 else t) for n, t in P.items()}


def _check_chunk(eng, orc, k, h_prev, labels, got_loss):
    L, g, _ = orc.local_grad(k, h_prev, labels)
    assert rel(got_loss, L) <= LOSS_TOL, (k, got_loss, L)
    for n in orc.chunk_names(k):
        c = cosine(eng.get(n, 1), g[n])
        assert c >= COS_MIN, (k, n, c)


def test_llama_1b_isolated_chunks_full_size():
    w = synth.LLAMA_1B
    P = _params("1b", w.dims.n_layers)
    eng = engine_for(w, accum_m=2)
    eng.load(P)
    ids, labels = synth.make_batch(w, 0)
    ids_d = ids.cuda()
    hs = {0: None}
    h = None
    for k in range(1, 5):
        h = eng.forward_chunk(k, h, ids_d if k == 1 else None, w.batch, w.seq)
        hs[k] = h
    losses = eng.step(ids_d, labels.cuda())
    orc = oracle_for(w, P, dtype=torch.float32)
    view = lambda t: t.float().cpu().view(w.batch, w.seq, -1)
    _check_chunk(eng, orc, 1, orc.embed(ids), labels, losses[0])
    _check_chunk(eng, orc, 5, view(hs[4]), labels, losses[4])
    eng.close()


def test_llama_1b_sampled_sequence_full_chain():
    """All 8 chunks forward at 4 x 1024; sequence 2 recomputed alone by the oracle."""
    w = synth.LLAMA_1B
    P = _params("1b", w.dims.n_layers)
    eng = engine_for(w)
    eng.load(P)
    orc = oracle_for(w, P, dtype=torch.float32)
    ids, _ = synth.make_batch(w, 1)
    hg = None
    ho = orc.embed(ids[2:3])
    for k in range(1, w.K + 1):
        hg = eng.forward_chunk(k, hg, ids.cuda() if k == 1 else None, w.batch, w.seq)
        ho = orc.forward_chunk(k, ho)
    got = hg.view(w.batch, w.seq, -1)[2].float().cpu()
    assert fro_rel(got, ho[0]) <= LOSS_TOL
    eng.close()


@pytest.mark.parametrize("name", ["3b", "7b"])
def test_first_chunk_full_width(name):
    w = {"3b": synth.LLAMA_3B, "7b": synth.LLAMA_7B}[name]
    nl = synth.chunk_bounds(w.dims.n_layers, w.K)[1]
    sub = dataclasses.replace(w, dims=dataclasses.replace(w.dims, n_layers=nl), K=1)
    P = _params(name, nl)
    eng = engine_for(sub, accum_m=2)
    eng.load(P)
    ids, labels = synth.make_batch(w, 0)
    losses = eng.step(ids.cuda(), labels.cuda())
    orc = oracle_for(sub, P, dtype=torch.float32)
    _check_chunk(eng, orc, 1, orc.embed(ids), labels, losses[0])
    eng.close()


def _reanchored(w, eng, P, names, **kw):
    Q = dict(P)
    for n in names:
        t = eng.get(n, 0).view(P[n].shape)
        Q[n] = synth.round_bf16(t) if t.dim() == 2 else t
    return oracle_for(w, Q, dtype=torch.float32, **kw)


def _two_steps_of_chunk(w, P, K, k, **okw):
    """Chunk k of a K-chunk engine over w, isolated, at optimizer steps 1 and 2 (module docstring)."""
    eng = engine_for(w, K=K, accum_m=2)
    eng.load(P)
    orc = oracle_for(w, P, K=K, dtype=torch.float32, accum_m=2, **okw)
    names = orc.chunk_names(k)
    view = lambda t: t.float().cpu().view(w.batch, w.seq, -1)

    def h_in(ids):
        h = None
        for j in range(1, k):
            h = eng.forward_chunk(j, h, ids.cuda() if j == 1 else None, w.batch, w.seq)
        return orc.embed(ids) if k == 1 else view(h)

    for mb in range(3):
        ids, labels = synth.make_batch(w, mb)
        h = h_in(ids) if mb != 1 else None
        losses = eng.step(ids.cuda(), labels.cuda())
        if mb == 0:
            _check_chunk(eng, orc, k, h, labels, losses[k - 1])
        elif mb == 2:
            ref = _reanchored(w, eng, P, names, K=K, **okw)
            _check_chunk(eng, ref, k, h if k > 1 else ref.embed(ids), labels, losses[k - 1])
    eng.close()


@pytest.mark.parametrize("K", [1, 2, 4])
def test_llama_1b_deepest_chunk_two_steps(K):
    """The deepest (last) chunk of the 1.1B model split into K = 1, 2 or 4 chunks (22, 11 or 6 layers),
    full micro-batch (4 x 1024), optimizer steps 1 and 2."""
    w = synth.LLAMA_1B
    P = _params("1b", w.dims.n_layers)
    _two_steps_of_chunk(w, P, K, K)


@pytest.mark.parametrize("name", ["3b", "7b"])
def test_first_chunk_full_width_step_two(name):
    """Chunk 1 of the 3B and 7B-shaped models (a K = 1 model over its layers) at optimizer steps 1 and 2."""
    w = {"3b": synth.LLAMA_3B, "7b": synth.LLAMA_7B}[name]
    nl = synth.chunk_bounds(w.dims.n_layers, w.K)[1]
    sub = dataclasses.replace(w, dims=dataclasses.replace(w.dims, n_layers=nl), K=1)
    P = _params(name, nl)
    _two_steps_of_chunk(sub, P, 1, 1)
