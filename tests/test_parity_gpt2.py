"""GPT-2-small-shaped bf16 workload (12 layers, d 768, vocab 50257, seq 512, K = 4) against the oracle.

The oracle runs in fp32 on the same bf16-rounded weights. Bars: loss relative error <= 2e-2 and
per-tensor gradient cosine >= 0.999. Gradients are read before the optimizer step (accum_m = 2
keeps the first micro-batch's gradient in the accumulator).
"""
import functools

import pytest
import torch

import synth
from tests.gpu_common import cosine, engine_for, fro_rel, oracle_for, rel

pytestmark = pytest.mark.gpu
W = synth.GPT2_SMALL
LOSS_TOL, COS_MIN = 2e-2, 0.999


@functools.lru_cache(maxsize=1)
def _params():
    P = synth.make_params(W.dims, W.seed)
    return {n: (synth.round_bf16(t) if t.dim() == 2 else t) for n, t in P.items()}


def _check_grads(eng, orc, grads, names):
    for n in names:
        c = cosine(eng.get(n, 1), grads[n])
        assert c >= COS_MIN, (n, c)


def test_full_chain_small_batch():
    """All K chunks, own chains on both sides, B = 2 sequences of 512."""
    P = _params()
    eng = engine_for(W, accum_m=2)
    eng.load(P)
    orc = oracle_for(W, P, dtype=torch.float32)
    ids = synth.zipf_ids(11, 2, W.seq, W.dims.vocab)
    labels = synth.next_token_labels(ids)
    lg = eng.step(ids.cuda(), labels.cuda())
    h = orc.embed(ids)
    for k in range(1, W.K + 1):
        L, g, h = orc.local_grad(k, h, labels)
        assert rel(lg[k - 1], L) <= LOSS_TOL, (k, lg, L)
        _check_grads(eng, orc, g, orc.chunk_names(k))
    eng.close()


def test_isolated_chunk_full_size():
    """Chunk 2 at the full micro-batch (8 x 512) from the engine's own h_1 (per-chunk isolation)."""
    P = _params()
    eng = engine_for(W, accum_m=2)
    eng.load(P)
    ids, labels = synth.make_batch(W, 0)
    h1 = eng.forward_chunk(1, None, ids.cuda(), W.batch, W.seq)
    lg = eng.step(ids.cuda(), labels.cuda())
    orc = oracle_for(W, P, dtype=torch.float32)
    L, g, _ = orc.local_grad(2, h1.float().cpu().view(W.batch, W.seq, -1), labels)
    assert rel(lg[1], L) <= LOSS_TOL, (lg, L)
    _check_grads(eng, orc, g, orc.chunk_names(2))
    eng.close()


def test_sampled_sequences_forward_full_size():
    """Forward of every chunk at 8 x 512; sequences 0 and 7 recomputed alone by the oracle."""
    P = _params()
    eng = engine_for(W)
    eng.load(P)
    orc = oracle_for(W, P, dtype=torch.float32)
    ids, _ = synth.make_batch(W, 3)
    hg = None
    hs = {b: orc.embed(ids[b:b + 1]) for b in (0, 7)}
    for k in range(1, W.K + 1):
        hg = eng.forward_chunk(k, hg, ids.cuda() if k == 1 else None, W.batch, W.seq)
        for b in hs:
            hs[b] = orc.forward_chunk(k, hs[b])
            got = hg.view(W.batch, W.seq, -1)[b].float().cpu()
            assert fro_rel(got, hs[b][0]) <= LOSS_TOL, (k, b)
    eng.close()


def test_zerolock_peak_memory_below_backprop():
    """Peak HBM of the concurrent step (2 live chunks) is below same-engine backprop at K = 4."""
    P = _params()
    ids, labels = synth.make_batch(W, 0)
    ids, labels = ids.cuda(), labels.cuda()
    peaks = {}
    for mode in ("zl", "bp"):
        eng = engine_for(W, max_live_chunks=2)
        eng.load(P)
        eng.reset_peak()
        if mode == "zl":
            eng.step(ids, labels)
        else:
            eng.bp_step(ids, labels)
        peaks[mode] = eng.peak_bytes()[0]
        eng.close()
    assert peaks["zl"] < peaks["bp"], peaks
