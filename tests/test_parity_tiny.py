"""The tiny fp32 Llama-style workload: the CUDA path through the C ABI against the float64 oracle.

Tolerances: per-step loss relative error <= 1e-4 and per-tensor relative Frobenius error of the
parameters <= 1e-4 after 10 AdamW steps (elementwise comparison is not used: an AdamW update of
a coordinate whose gradient is ~0 is sign-unstable under rounding).
"""
import pytest
import torch

import synth
from tests.gpu_common import engine_for, fro_rel, oracle_for, rel

pytestmark = pytest.mark.gpu
W = synth.TINY
TOL = 1e-4


def _params():
    return synth.make_params(W.dims, W.seed)


def _cuda(b):
    return b[0].cuda(), b[1].cuda()


def test_ten_steps_match_oracle():
    P = _params()
    eng = engine_for(W)
    eng.load(P)
    orc = oracle_for(W, P)
    for s in range(W.steps):
        ids, labels = synth.make_batch(W, s)
        lg = eng.step(*_cuda((ids, labels)))
        lo = orc.step(ids, labels)
        for a, b in zip(lg, lo):
            assert rel(a, b) <= TOL, (s, lg, lo)
    for n in orc.trainable_names():
        assert fro_rel(eng.get(n), orc.P[n]) <= TOL, n
        assert fro_rel(eng.get(n, 2), orc.m[n]) <= 1e-3, n      # AdamW first moment
    ids, labels = synth.make_batch(W, W.steps)
    assert rel(eng.global_loss(*_cuda((ids, labels))), orc.global_loss(ids, labels)) <= TOL
    eng.close()


@pytest.mark.parametrize("cap", [1, 2, 0])
def test_schedule_does_not_change_results(cap):
    """Any bound on live chunks (1 = serial, 0 = all K) gives bit-identical parameters."""
    P = _params()
    ref = engine_for(W, max_live_chunks=1)
    eng = engine_for(W, max_live_chunks=cap)
    ref.load(P)
    eng.load(P)
    for s in range(3):
        b = _cuda(synth.make_batch(W, s))
        ref.step(*b, want_losses=False)
        eng.step(*b, want_losses=False)     # no host sync between steps: streams overlap across steps
    eng.synchronize()
    ref.synchronize()
    for n in synth.param_names(W.dims):
        assert torch.equal(eng.get(n[0]), ref.get(n[0])), n[0]
    eng.close(); ref.close()


def test_local_steps_equal_concurrent_step_bitwise():
    """K zl_local_step calls (teacher recomputed from h_{k-1}) == one zl_step (teacher reused)."""
    P = _params()
    a = engine_for(W)
    b = engine_for(W)
    a.load(P)
    b.load(P)
    N = W.batch * W.seq
    for s in range(2):
        ids, labels = _cuda(synth.make_batch(W, s))
        la = a.step(ids, labels)
        h = None
        lb = []
        for k in range(1, W.K + 1):
            out = torch.empty(N, W.dims.d_model, device="cuda")
            lb.append(b.local_step(k, h, ids, labels, h_out=out))
            h = out
        assert la == lb
    for n, _ in synth.param_names(W.dims):
        assert torch.equal(a.get(n), b.get(n)), n


def test_bp_step_matches_oracle_backprop():
    P = _params()
    eng = engine_for(W)
    eng.load(P)
    orc = oracle_for(W, P)
    for s in range(3):
        ids, labels = synth.make_batch(W, s)
        assert rel(eng.bp_step(*_cuda((ids, labels))), orc.bp_step(ids, labels)) <= TOL
    for n in orc.trainable_names():
        assert fro_rel(eng.get(n), orc.P[n]) <= TOL, n


def test_forward_chunks_and_embedding():
    P = _params()
    eng = engine_for(W)
    eng.load(P)
    orc = oracle_for(W, P)
    ids, _ = synth.make_batch(W, 0)
    h0 = eng.embed(ids.cuda())
    assert torch.equal(h0.cpu(), P["tok_emb"][ids.long()].view(-1, W.dims.d_model))   # bit-exact gather
    h = orc.embed(ids)
    hg = None
    for k in range(1, W.K + 1):
        hg = eng.forward_chunk(k, hg, ids.cuda() if k == 1 else None, W.batch, W.seq)
        h = orc.forward_chunk(k, h)
        assert fro_rel(hg.cpu(), h.reshape(-1, W.dims.d_model)) <= 1e-5


@pytest.mark.parametrize("opts", [dict(kl_dir=1), dict(consis_first=0), dict(accum_m=2), dict(alpha=1.0),
                                  dict(lr_schedule=1, lr_gamma=2.0)])
def test_variants_match_oracle(opts):
    P = _params()
    alpha = opts.pop("alpha", None)
    eng = engine_for(W, alpha=alpha, **opts)
    eng.load(P)
    orc = oracle_for(W, P, alpha=alpha, **opts)
    for s in range(4):
        ids, labels = synth.make_batch(W, s)
        lg = eng.step(*_cuda((ids, labels)))
        lo = orc.step(ids, labels)
        for x, y in zip(lg, lo):
            assert rel(x, y) <= TOL, (opts, s, lg, lo)
    for n in orc.trainable_names():
        assert fro_rel(eng.get(n), orc.P[n]) <= TOL, (opts, n)


def test_ragged_batch_empty_omega_and_short_sequences():
    P = _params()
    eng = engine_for(W)
    eng.load(P)
    orc = oracle_for(W, P)
    for (Bb, S) in [(3, 37), (1, 1), (5, 64)]:
        ids = synth.zipf_ids(99 + S, Bb, S, W.dims.vocab)
        labels = synth.next_token_labels(ids)
        if S == 37:
            labels[1, :] = -1
        lg = eng.step(ids.cuda(), labels.cuda())
        lo = orc.step(ids, labels)
        for x, y in zip(lg, lo):
            assert abs(x - y) <= TOL * max(abs(y), 1.0), (Bb, S, lg, lo)
    for n in orc.trainable_names():
        assert fro_rel(eng.get(n), orc.P[n]) <= TOL, n


def test_out_of_range_ids_and_labels_are_reported():
    from paper_2608_07974_gb300 import binding as b
    eng = engine_for(W)
    eng.load(_params())
    ids, labels = synth.make_batch(W, 0)
    bad = ids.clone()
    bad[0, 3] = W.dims.vocab + 5
    with pytest.raises(b.ZLError) as e:
        eng.step(bad.cuda(), labels.cuda())
    assert e.value.status == b.ZL_ERR_ARG and "token id" in str(e.value)
    badl = labels.clone()
    badl[1, 2] = W.dims.vocab
    with pytest.raises(b.ZLError) as e:
        eng.step(ids.cuda(), badl.cuda())
    assert "label" in str(e.value)
    # the context stays usable
    eng.step(*_cuda((ids, labels)))
    with pytest.raises(b.ZLError) as e:
        eng.step(ids[:, :0].contiguous().cuda(), labels[:, :0].contiguous().cuda())
    assert e.value.status == b.ZL_ERR_ARG


def test_load_weights_is_set_param():
    """zl_load_weights stores a tensor exactly as zl_set_param does, from host or device memory, and
    rejects an unknown name or a wrong byte count."""
    from paper_2608_07974_gb300 import binding as b
    eng = engine_for(W)
    eng.load(_params())
    g = torch.Generator().manual_seed(7)
    for name, dev in (("layers.0.wqkv", False), ("layers.3.w2", True), ("layers.1.ffn_norm.weight", True)):
        t = torch.randn(eng.get(name).shape, generator=g)
        b.zl_load_weights(eng.ctx, name, t.cuda() if dev else t)
        assert torch.equal(eng.get(name).cpu(), t), name
    with pytest.raises(b.ZLError) as e:
        b.zl_load_weights(eng.ctx, "layers.0.no_such", torch.zeros(4))
    assert e.value.status == b.ZL_ERR_ARG
    with pytest.raises(b.ZLError) as e:
        b.zl_load_weights(eng.ctx, "layers.0.wqkv", torch.zeros(4))
    assert e.value.status == b.ZL_ERR_ARG
    eng.close()
