"""Scheduler fuzz (GPU): host-side sleeps between enqueues must not change any result.

With cfg.fuzz_delay_us the engine sleeps a seeded pseudo-random time at every phase boundary of its
enqueues (forward, readout, loss, backward, AdamW of each chunk), so the GPU runs ahead of the host in
a different interleaving of the K chunk streams, their column-sum side streams and the auxiliary
stream on every run. The concurrent schedule (Section III-A/B: early forwarding, readiness events,
no update locking, also across steps) must reach bit-identical parameters and losses to a serialised
run (every chunk on one stream), for several seeds and live-chunk bounds.
"""
import pytest
import torch

import synth
from tests.gpu_common import engine_for

pytestmark = pytest.mark.gpu

# a small GPT-2-style bf16 model: tcgen05 GEMMs and attention, side-stream column sums, K = 4
GPT2S = synth.Workload("fuzz-gpt2-bf16", synth.ModelDims(synth.ARCH_GPT2, 4, 256, 4, 4, 1024, 1024, 256), "bf16",
                       batch=2, seq=256, K=4, steps=3, seed=1234 + 1)


def _params(w):
    P = synth.make_params(w.dims, w.seed)
    return {n: (synth.round_bf16(t) if (w.dtype == "bf16" and t.dim() == 2) else t) for n, t in P.items()}


def _run(w, P, steps, **kw):
    eng = engine_for(w, **kw)
    eng.load(P)
    losses = []
    for s in range(steps):
        ids, labels = synth.make_batch(w, s)
        eng.step(ids.cuda(), labels.cuda(), want_losses=False)   # no host sync between steps
        if s == steps - 1:
            losses = eng.read_losses()
    eng.synchronize()
    params = {n: eng.get(n) for n, _ in synth.param_names(w.dims)}
    moments = {n: eng.get(n, 3) for n, _ in synth.param_names(w.dims)}
    eng.close()
    return losses, params, moments


@pytest.mark.parametrize("w", [synth.TINY, GPT2S], ids=["tiny-f32", "gpt2s-bf16"])
def test_fuzzed_schedules_equal_the_serialised_run(w):
    P = _params(w)
    K = 4 if w is GPT2S else 2
    ref = _run(w, P, 3, K=K, serialize=True)
    for seed, cap, delay in ((1, 0, 200), (2, 2, 500), (3, 1, 50), (4, 0, 1000)):
        got = _run(w, P, 3, K=K, max_live_chunks=cap, fuzz_delay_us=delay, fuzz_seed=seed)
        assert got[0] == ref[0], (seed, got[0], ref[0])
        for n in ref[1]:
            assert torch.equal(got[1][n], ref[1][n]), (seed, n)
            assert torch.equal(got[2][n], ref[2][n]), (seed, n)


def test_fuzz_delay_is_validated():
    from paper_2608_07974_gb300 import binding as b
    with pytest.raises(b.ZLError) as e:
        engine_for(synth.TINY, fuzz_delay_us=-1)
    assert e.value.status == b.ZL_ERR_ARG
