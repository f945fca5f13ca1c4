"""The oracle against an independent, autograd-free statement of the model and its gradients (no GPU).

tests/manual_backprop.py restates the blocks, the readout, the closed-form logit gradient of the
local objective (Eq. 3-5) and backpropagation in numpy with hand-derived backward formulas. The
oracle (torch autograd over its own forward) must agree with it on every element of every gradient
at float64 rounding: for backpropagation through the whole model, for K = 1 with alpha = 1 (where the
local update is backpropagation), and for every chunk's local gradient in both KL directions.
A separately written backward adds in another order, so agreement is to rounding, not bit for bit;
the bit-for-bit K = 1 check is against the oracle's own backpropagation step (test_oracle_pins).
"""
import numpy as np
import pytest
import torch

import tests.manual_backprop as mb
from oracle.model import Oracle, OracleConfig
from tests.test_oracle_pins import GPT2_T, LLAMA_T, float64_default, tiny_batch, tiny_params  # noqa: F401

REL = 1e-13


def _np(P):
    return {n: t.detach().double().numpy() for n, t in P.items()}


def _close(got, ref, what):
    got = got.detach().double().numpy() if isinstance(got, torch.Tensor) else np.asarray(got)
    scale = max(float(np.abs(ref).max()), 1e-300)
    err = float(np.abs(got - ref).max())
    assert err <= REL * scale, (what, err, scale)


def _batch(d, seed=3):
    ids, labels = tiny_batch(d, seed=seed)
    labels[0, 2] = -1                              # a hole in Omega
    return ids, labels


@pytest.mark.parametrize("d", [LLAMA_T, GPT2_T], ids=["llama", "gpt2"])
@pytest.mark.parametrize("bounds", [[0, 2], [0, 1, 2]], ids=["K1", "K2"])
def test_backprop_gradient_matches_manual_backward(d, bounds):
    P = tiny_params(d)
    ids, labels = _batch(d)
    orc = Oracle(OracleConfig(dims=d, bounds=bounds, alpha=1.0), P)
    L, g = orc.bp_grad(ids, labels)
    Lm, gm = mb.bp_grad(_np(P), d, bounds, ids.numpy(), labels.numpy())
    assert abs(L - Lm) <= REL * abs(Lm)
    assert set(g) == set(gm)
    for n in gm:
        _close(g[n], gm[n], n)


@pytest.mark.parametrize("d", [LLAMA_T, GPT2_T], ids=["llama", "gpt2"])
def test_single_chunk_alpha1_local_update_is_manual_backprop(d):
    """K = 1, alpha = 1: the local gradient of the one chunk is the backpropagation gradient."""
    P = tiny_params(d)
    ids, labels = _batch(d, seed=5)
    orc = Oracle(OracleConfig(dims=d, bounds=[0, 2], alpha=1.0), P)
    L, g, _ = orc.local_grad(1, orc.embed(ids), labels)
    Lm, gm = mb.bp_grad(_np(P), d, [0, 2], ids.numpy(), labels.numpy())
    assert abs(L - Lm) <= REL * abs(Lm)
    for n in gm:
        _close(g[n], gm[n], n)


@pytest.mark.parametrize("d", [LLAMA_T, GPT2_T], ids=["llama", "gpt2"])
@pytest.mark.parametrize("alpha,kl_dir", [(0.5, 0), (0.3, 1), (1.0, 0)])
def test_every_chunk_local_gradient_matches_manual_backward(d, alpha, kl_dir):
    """Each chunk's L_k, dL_k/dtheta_k and h_k, with the teacher and h_{k-1} held constant."""
    P = tiny_params(d)
    ids, labels = _batch(d, seed=9)
    bounds = [0, 1, 2]
    orc = Oracle(OracleConfig(dims=d, bounds=bounds, alpha=alpha, kl_dir=kl_dir), P)
    Pn = _np(P)
    h = orc.embed(ids)
    hm = mb.embed(Pn, ids.numpy(), mb.Dims(d))
    _close(h, hm, "h_0")
    for k in (1, 2):
        L, g, h_next = orc.local_grad(k, h, labels)
        Lm, gm, hm_next = mb.local_grad(Pn, d, bounds, k, hm, labels.numpy(), alpha, kl_dir)
        assert abs(L - Lm) <= REL * abs(Lm), (k, L, Lm)
        assert set(g) == set(gm)
        for n in gm:
            _close(g[n], gm[n], (k, n))
        _close(h_next, hm_next, f"h_{k}")
        h, hm = h_next, hm_next


def test_manual_backward_agrees_with_its_own_finite_differences():
    """The independent statement is itself checked against central differences of its forward."""
    d = LLAMA_T
    Pn = _np(tiny_params(d))
    ids, labels = _batch(d, seed=13)
    m = mb.Dims(d)
    h0 = mb.embed(Pn, ids.numpy(), m)
    t = mb.readout_fwd(Pn, h0, m)[0]

    def L_of(Q):
        h, _ = mb.chunk_fwd(Q, [0, 2], 1, h0, m)
        return mb.objective_and_dz(mb.readout_fwd(Q, h, m)[0], t, labels.numpy(), 0.5, 0)[0]

    _, gm, _ = mb.local_grad(Pn, d, [0, 2], 1, h0, labels.numpy(), 0.5, 0)
    rng = np.random.default_rng(0)
    for n, gr in gm.items():
        flat = Pn[n].reshape(-1)
        for idx in rng.integers(0, flat.size, 3):
            old = flat[idx]
            flat[idx] = old + 1e-6
            lp = L_of(Pn)
            flat[idx] = old - 1e-6
            lm = L_of(Pn)
            flat[idx] = old
            fd = (lp - lm) / 2e-6
            assert abs(fd - gr.reshape(-1)[idx]) <= 1e-7 + 1e-6 * abs(fd), (n, idx)


@pytest.mark.parametrize("d", [LLAMA_T, GPT2_T], ids=["llama", "gpt2"])
def test_lora_local_gradients_match_manual_backward(d):
    """LoRA chunks (only A and B train, Delta w = s B A): every factor's gradient element by element."""
    from tests.test_oracle_pins import _lora_setup
    P, cfg = _lora_setup(d)
    ids, labels = _batch(d, seed=17)
    orc = Oracle(cfg, P)
    Pn = _np(P)
    h = orc.embed(ids)
    hm = h.numpy().copy()
    for k in (1, 2):
        L, g, h_next = orc.local_grad(k, h, labels)
        Lm, gm, hm_next = mb.local_grad(Pn, d, cfg.bounds, k, hm, labels.numpy(), cfg.alpha,
                                        lora_scale=cfg.lora_scale)
        assert abs(L - Lm) <= REL * abs(Lm)
        assert set(g) == set(gm) and all("lora_" in n for n in gm)
        for n in g:
            _close(g[n], gm[n], (k, n))
        _close(h_next, hm_next, f"h_{k}")
        h, hm = h_next, hm_next


@pytest.mark.parametrize("d", [LLAMA_T, GPT2_T], ids=["llama", "gpt2"])
def test_adapter_local_gradients_match_manual_backward(d):
    """Readout adapters: every layer tensor and both adapter matrices of chunk k, element by element."""
    from tests.test_oracle_pins import _adapter_setup
    P, cfg = _adapter_setup(d)
    ids, labels = _batch(d, seed=19)
    orc = Oracle(cfg, P)
    Pn = _np(P)
    h = orc.embed(ids)
    hm = h.numpy().copy()
    for k in (1, 2):
        L, g, h_next = orc.local_grad(k, h, labels)
        Lm, gm, hm_next = mb.local_grad(Pn, d, cfg.bounds, k, hm, labels.numpy(), cfg.alpha, adapters=True)
        assert abs(L - Lm) <= REL * abs(Lm)
        assert set(g) == set(gm)
        for n in g:
            _close(g[n], gm[n], (k, n))
        h, hm = h_next, hm_next
