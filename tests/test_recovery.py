"""Per-chunk checkpoints and replay from the hidden-state buffer (Section III-B-3), on the GPU.

Failures are made on the host (a chunk's state is thrown away and restored); nothing faults the
GPU. Replaying a chunk from its buffered inputs must reproduce the uninterrupted run bit for bit,
and the other chunks keep their state; the recovered parameters also match the oracle's uninterrupted
trajectory (fp64, Eq. 1-6) within the fp32 bar of 1e-4 (per-tensor Frobenius relative error).
"""
import pytest
import torch

import synth
from tests.gpu_common import engine_for, fro_rel, oracle_for

pytestmark = pytest.mark.gpu
W = synth.TINY
BOUNDS = [0, 1, 2, 3, 4]     # K = 4 one-layer chunks


def _engine(**kw):
    eng = engine_for(W, K=4, bounds=BOUNDS, **kw)
    eng.load(synth.make_params(W.dims, W.seed))
    return eng


def _steps(eng, lo, hi):
    for s in range(lo, hi):
        ids, labels = synth.make_batch(W, s)
        eng.step(ids.cuda(), labels.cuda())


def _all_params(eng):
    return {n: eng.get(n) for n, _ in synth.param_names(W.dims)}


@pytest.mark.parametrize("accum_m", [1, 2])
def test_failed_chunk_recovers_by_replay(accum_m):
    from paper_2608_07974_gb300 import binding as b
    ref = _engine(accum_m=accum_m)
    _steps(ref, 0, 7)
    eng = _engine(accum_m=accum_m, replay_depth=4)
    _steps(eng, 0, 3)
    ckpt = b.zl_chunk_save(eng.ctx, 2)                 # proactive checkpoint of chunk 2 (mid-window if m = 2)
    _steps(eng, 3, 7)
    before = _all_params(eng)
    junk = torch.randn(b.zl_param_numel(eng.ctx, "layers.1.wqkv"))
    b.zl_set_param(eng.ctx, "layers.1.wqkv", junk)     # chunk 2 "fails": its state is lost
    b.zl_chunk_load(eng.ctx, 2, ckpt)                  # restore from the checkpoint ...
    n, _ = b.zl_replay(eng.ctx, 2)                     # ... and replay the buffered micro-batches
    assert n == 4
    after = _all_params(eng)
    want = _all_params(ref)
    for name in want:
        assert torch.equal(after[name], want[name]), name
        if not name.startswith("layers.1."):
            assert torch.equal(after[name], before[name]), name    # other chunks kept their state
    eng.close(); ref.close()
    orc = oracle_for(W, synth.make_params(W.dims, W.seed), K=4, bounds=BOUNDS, accum_m=accum_m)
    for s in range(7):                                 # the uninterrupted run, by the oracle
        ids, labels = synth.make_batch(W, s)
        orc.step(ids, labels)
    for name in want:
        assert fro_rel(after[name], orc.P[name]) <= 1e-4, name


def test_checkpoint_round_trip_and_rejections():
    from paper_2608_07974_gb300 import binding as b
    eng = _engine(replay_depth=2)
    _steps(eng, 0, 2)
    blob = b.zl_chunk_save(eng.ctx, 3)
    snap = _all_params(eng)
    _steps(eng, 2, 5)
    b.zl_chunk_load(eng.ctx, 3, blob)
    assert torch.equal(eng.get("layers.2.w1"), snap["layers.2.w1"])
    with pytest.raises(b.ZLError) as e:                # 3 micro-batches behind, the ring keeps 2
        b.zl_replay(eng.ctx, 3)
    assert e.value.status == b.ZL_ERR_ARG
    with pytest.raises(b.ZLError):                     # a blob of another chunk
        b.zl_chunk_load(eng.ctx, 4, blob)
    assert b.zl_replay(eng.ctx, 1)[0] == 0             # an up-to-date chunk has nothing to replay
    eng.close()


def test_timed_out_poll_leaves_the_context_usable():
    from paper_2608_07974_gb300 import binding as b
    w = synth.GPT2_SMALL
    eng = engine_for(w)
    ids, labels = synth.make_batch(w, 0)
    ids, labels = ids.cuda(), labels.cuda()
    for _ in range(4):
        eng.step(ids, labels, want_losses=False)
    with pytest.raises(b.ZLError) as e:
        b.zl_synchronize(eng.ctx, 0)                   # gives up at once: the work is still queued
    assert e.value.status == b.ZL_ERR_TIMEOUT
    b.zl_synchronize(eng.ctx, -1)
    assert len(eng.step(ids, labels)) == w.K
    eng.close()
