"""CUDA-graph steps (cfg.graph = 1): zl_step and zl_bp_step captured once per micro-batch shape and
replayed. A replay runs the same kernels in the same order, so every value must equal the eager run
bit for bit, across shape changes (re-capture), and the host bookkeeping (step counts in checkpoints,
the launch counter) must follow the replays."""
import pytest
import torch

import synth
from paper_2608_07974_gb300 import binding as zb
from tests.gpu_common import engine_for

pytestmark = pytest.mark.gpu
W = synth.TINY


def _engine(w=W, **kw):
    eng = engine_for(w, **kw)
    eng.load(synth.make_params(w.dims, w.seed))
    return eng


def _batch(w, s, B=None, S=None):
    ids, labels = synth.make_batch(w, s)
    if B is not None:
        ids, labels = ids[:B, :S].contiguous(), synth.next_token_labels(ids[:B, :S].contiguous())
    return ids.cuda(), labels.cuda()


def _params(eng, w=W):
    return {n: eng.get(n) for n, _ in synth.param_names(w.dims)}


# (B, S) per step: a shape change forces a re-capture, and the first call at a shape runs eagerly
SHAPES = [(4, 64)] * 3 + [(2, 48)] * 3 + [(4, 64)] * 2


def test_graph_steps_equal_eager_bit_for_bit():
    g = _engine(graph=True)
    e = _engine()
    for s, (B, S) in enumerate(SHAPES):
        b = _batch(W, s, B, S)
        assert g.step(*b) == e.step(*b), s
    pg, pe = _params(g), _params(e)
    for n in pg:
        assert torch.equal(pg[n], pe[n]), n
    g.close()
    e.close()


def test_graph_backprop_steps_equal_eager():
    g = _engine(graph=True)
    e = _engine()
    for s in range(4):
        b = _batch(W, s)
        assert g.bp_step(*b) == e.bp_step(*b), s
    pg, pe = _params(g), _params(e)
    for n in pg:
        assert torch.equal(pg[n], pe[n]), n
    g.close()
    e.close()


def test_graph_replays_count_launches_and_keep_step_counts():
    g = _engine(graph=True)
    b = _batch(W, 0)
    counts = []
    for _ in range(4):   # eager, capture + first launch, then two replays
        n0 = zb.zl_kernel_launches()
        g.step(*b, want_losses=False)
        g.synchronize()
        counts.append(zb.zl_kernel_launches() - n0)
    assert counts[0] == counts[1] == counts[2] == counts[3] > 0, counts
    # a checkpoint taken after the replays resumes in an eager engine exactly where the graph engine is
    blobs = [zb.zl_chunk_save(g.ctx, k) for k in range(1, W.K + 1)]
    e = _engine()
    for k, blob in enumerate(blobs, start=1):
        zb.zl_chunk_load(e.ctx, k, blob)
    for s in range(1, 4):
        b = _batch(W, s)
        assert g.step(*b) == e.step(*b), s
    pg, pe = _params(g), _params(e)
    for n in pg:
        assert torch.equal(pg[n], pe[n]), n
    g.close()
    e.close()


def test_graph_gpt2_small_batch_equals_eager():
    """GPT-2 bf16 (tensor-core GEMMs with split-K workspaces, attention, the vocab-sized loss) on 2 x 512."""
    w = synth.GPT2_SMALL
    P = synth.make_params(w.dims, w.seed)
    g = engine_for(w, graph=True, max_live_chunks=2)
    e = engine_for(w, max_live_chunks=2)
    g.load(P)
    e.load(P)
    for s in range(3):
        ids = synth.zipf_ids(100 + s, 2, w.seq, w.dims.vocab)
        labels = synth.next_token_labels(ids)
        assert g.step(ids.cuda(), labels.cuda()) == e.step(ids.cuda(), labels.cuda()), s
    for n in ("layers.0.wqkv", "layers.5.w1", "layers.11.b2", "layers.11.ffn_norm.weight"):
        assert torch.equal(g.get(n), e.get(n)), n
    g.close()
    e.close()
