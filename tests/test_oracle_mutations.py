"""Plant plausible mistakes in the oracle (on the CPU) and check that a pin catches each."""
import math

import pytest
import torch

import oracle
import oracle.model as om
import tests.test_oracle_pins as pins
from tests.test_oracle_pins import float64_default  # noqa: F401  (autouse fixture)


def _patch(monkeypatch, name, fn):
    monkeypatch.setattr(om, name, fn)
    monkeypatch.setattr(oracle, name, fn)


def bad_rope(x, theta):            # wrong rotation sign
    S, hd = x.shape[1], x.shape[3]
    half = hd // 2
    inv = theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / hd)
    ang = torch.arange(S, dtype=torch.float64)[:, None] * inv[None, :]
    c, s = torch.cos(ang)[None, :, None, :], torch.sin(ang)[None, :, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return torch.cat([x1 * c + x2 * s, x2 * c - x1 * s], dim=-1)


def bad_attention(q, k, v):        # missing 1/sqrt(hd)
    return om.attention.__wrapped__(q * math.sqrt(q.shape[-1]), k, v)


def bad_kl(z, t, kl_dir=0):        # lse of the teacher dropped
    lp = torch.log_softmax(z, -1)
    return (lp.exp() * (lp - t)).sum(-1)


def bad_rmsnorm(x, g, eps):        # eps outside the square root
    return x / (torch.sqrt((x * x).mean(-1, keepdim=True)) + eps) * g


def bad_adamw(theta, g, m, v, step, lr, b1, b2, eps, wd):   # no bias correction
    theta.mul_(1 - lr * wd)
    m.mul_(b1).add_((1 - b1) * g)
    v.mul_(b2).add_((1 - b2) * g * g)
    theta.sub_(lr * m / (torch.sqrt(v) + eps))


def bad_gelu(x):                   # erf-GELU instead of the tanh form
    return torch.nn.functional.gelu(x)


MUTATIONS = [
    ("rope", bad_rope, [pins.test_rope_is_the_complex_rotation, pins.test_layer_matches_library_composition]),
    ("kl_rows", bad_kl, [pins.test_loss_closed_forms]),
    ("rmsnorm", bad_rmsnorm, [pins.test_blocks_match_library_routines]),
    ("adamw_update", bad_adamw, [pins.test_adamw_matches_torch_optim]),
    ("gelu_tanh", bad_gelu, [pins.test_blocks_match_library_routines]),
]


@pytest.mark.parametrize("name,fn,tests", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_pins_catch_planted_mistake(monkeypatch, name, fn, tests):
    _patch(monkeypatch, name, fn)
    for t in tests:
        with pytest.raises(AssertionError):
            t()


def test_pins_catch_unscaled_attention(monkeypatch):
    orig = om.attention
    _patch(monkeypatch, "attention", lambda q, k, v: orig(q * math.sqrt(q.shape[-1]), k, v))
    with pytest.raises(AssertionError):
        pins.test_attention_matches_sdpa(4, 2, 8)


def test_pins_catch_wrong_gqa_grouping(monkeypatch):
    orig = om.attention

    def tiled(q, k, v):            # kv head h % Hkv instead of h // (H / Hkv)
        rep = q.shape[2] // k.shape[2]
        return orig(q, k.repeat(1, 1, rep, 1), v.repeat(1, 1, rep, 1))
    _patch(monkeypatch, "attention", tiled)
    with pytest.raises(AssertionError):
        pins.test_attention_matches_sdpa(4, 2, 8)


def test_pins_catch_dropped_residual(monkeypatch):
    orig = om.layer_forward
    _patch(monkeypatch, "layer_forward", lambda P, l, x, d: orig(P, l, x, d) - x)
    with pytest.raises(AssertionError):
        pins.test_layer_matches_library_composition()


def test_pins_catch_unscaled_lora(monkeypatch):
    orig = om.lora_weight
    monkeypatch.setattr(om, "lora_weight", lambda P, l, name, scale: orig(P, l, name, 1.0))
    with pytest.raises(AssertionError):
        pins.test_lora_zero_b_is_the_base_model_and_chain_rule()


def test_pins_catch_adapter_without_residual(monkeypatch):
    def bad_adapter(P, k, h):      # the residual connection dropped
        return oracle.gelu_tanh(h @ P[f"adapters.{k}.down"].T) @ P[f"adapters.{k}.up"].T
    _patch(monkeypatch, "adapter", bad_adapter)
    with pytest.raises(AssertionError):
        pins.test_adapter_gradient_matches_finite_differences(pins.LLAMA_T)


def test_pins_catch_adapter_on_the_teacher(monkeypatch):
    real = om.readout

    def readout_through_adapter(P, h, d):   # an upstream chunk's adapter leaks into the teacher
        return real(P, om.adapter(P, 1, h) if "adapters.1.down" in P else h, d)
    _patch(monkeypatch, "readout", readout_through_adapter)
    with pytest.raises(AssertionError):
        pins.test_adapter_teacher_is_the_frozen_head_and_bp_ignores_adapters()


def test_pins_catch_schedule_off_by_one(monkeypatch):
    def apply_window(self, k, adapters=True):   # eta_0 / sqrt(t + 1 + gamma): the schedule one step late
        c = self.cfg
        self.t[k] += 1
        lr = c.lr if c.lr_schedule == 0 else c.lr / math.sqrt(self.t[k] + c.lr_gamma)
        for n in self.chunk_names(k):
            g = self.acc[n] / c.accum_m
            om.adamw_update(self.P[n], g, self.m[n], self.v[n], self.t[k], lr, c.beta1, c.beta2, c.eps,
                            c.weight_decay)
            self.acc[n].zero_()
        self.micro[k] = 0
    monkeypatch.setattr(om.Oracle, "_apply_window", apply_window)
    with pytest.raises(AssertionError):
        pins.test_lr_schedule_matches_torch_lambda_lr()


def test_pins_catch_ignored_consis_first(monkeypatch):
    monkeypatch.setattr(om.Oracle, "alpha_k", lambda self, k: self.cfg.alpha)
    with pytest.raises(AssertionError):
        pins.test_consis_first_zero_is_plain_cross_entropy()


def test_pins_catch_swapped_kl_direction(monkeypatch):
    orig = om.kl_rows
    _patch(monkeypatch, "kl_rows", lambda z, t, kl_dir=0: orig(z, t, 1 - kl_dir))
    with pytest.raises(AssertionError):
        pins.test_reverse_kl_direction_matches_library()
    with pytest.raises(AssertionError):
        pins.test_loss_closed_forms()
    with pytest.raises(AssertionError):
        pins.test_proposition1_chunkwise_bound()


def test_independent_backward_catches_swapped_swiglu_halves(monkeypatch):
    import tests.test_oracle_independent_bp as ib

    def swapped(P, l, x, d, lora_scale=1.0):   # silu applied to the up half instead of the gate half
        Q = dict(P)
        w1 = P[f"layers.{l}.w1"]
        Q[f"layers.{l}.w1"] = torch.cat([w1[d.d_ff:], w1[:d.d_ff]])
        return orig(Q, l, x, d, lora_scale)
    orig = om.layer_forward
    _patch(monkeypatch, "layer_forward", lambda P, l, x, d, lora_scale=1.0:
           swapped(P, l, x, d, lora_scale) if d.arch == 0 else orig(P, l, x, d, lora_scale))
    with pytest.raises(AssertionError):
        ib.test_backprop_gradient_matches_manual_backward(pins.LLAMA_T, [0, 2])


def test_independent_backward_catches_unbiased_layernorm_variance(monkeypatch):
    import tests.test_oracle_independent_bp as ib

    def ln_unbiased(x, g, b, eps):
        mu = x.mean(-1, keepdim=True)
        var = ((x - mu) ** 2).sum(-1, keepdim=True) / (x.shape[-1] - 1)
        return (x - mu) / torch.sqrt(var + eps) * g + b
    _patch(monkeypatch, "layernorm", ln_unbiased)
    with pytest.raises(AssertionError):
        ib.test_backprop_gradient_matches_manual_backward(pins.GPT2_T, [0, 1, 2])


def test_independent_backward_catches_detached_lora_update(monkeypatch):
    import tests.test_oracle_independent_bp as ib
    orig = om.lora_weight

    def merged_constant(P, l, name, scale):   # the merged weight built outside autograd: no factor gradient
        return orig(P, l, name, scale).detach()
    monkeypatch.setattr(om, "lora_weight", merged_constant)
    with pytest.raises((AssertionError, RuntimeError)):
        ib.test_lora_local_gradients_match_manual_backward(pins.LLAMA_T)


def test_pins_catch_mask_hiding_the_diagonal(monkeypatch):
    def attention_no_self(q, k, v):   # each position may not attend to itself (mask one too wide)
        B, S, H, hd = q.shape
        rep = H // k.shape[2]
        kk, vv = k.repeat_interleave(rep, dim=2), v.repeat_interleave(rep, dim=2)
        qh, kh, vh = (t.permute(0, 2, 1, 3) for t in (q, kk, vv))
        s = qh @ kh.transpose(-1, -2) / math.sqrt(hd)
        mask = torch.triu(torch.ones(S, S, dtype=torch.bool), diagonal=0)
        mask[0, 0] = False                # keep row 0 defined
        p = torch.softmax(s.masked_fill(mask, float("-inf")), dim=-1)
        return (p @ vh).permute(0, 2, 1, 3)
    _patch(monkeypatch, "attention", attention_no_self)
    with pytest.raises(AssertionError):
        pins.test_attention_matches_sdpa(4, 2, 8)


def test_pins_catch_mean_over_all_rows(monkeypatch):
    orig = om.local_objective_rows
    _patch(monkeypatch, "local_objective",   # |Omega| replaced by the row count
           lambda z, t, labels, alpha, kl_dir=0: orig(z, t, labels, alpha, kl_dir).sum() / labels.numel())
    with pytest.raises(AssertionError):
        pins.test_loss_closed_forms()


def test_pins_catch_summed_window(monkeypatch):
    orig = om.Oracle._apply_window

    def summed(self, k, adapters=True):   # the window gradient summed instead of averaged
        for n in self.chunk_names(k):
            self.acc[n] *= self.cfg.accum_m
        orig(self, k, adapters)
    monkeypatch.setattr(om.Oracle, "_apply_window", summed)
    with pytest.raises(AssertionError):
        pins.test_accumulation_window_is_the_mean()


def test_pins_catch_decay_after_the_adam_step(monkeypatch):
    def late_decay(theta, g, m, v, step, lr, b1, b2, eps, wd):
        m.mul_(b1).add_((1 - b1) * g)
        v.mul_(b2).add_((1 - b2) * g * g)
        theta.sub_(lr * (m / (1 - b1 ** step)) / (torch.sqrt(v / (1 - b2 ** step)) + eps))
        theta.mul_(1 - lr * wd)
    _patch(monkeypatch, "adamw_update", late_decay)
    with pytest.raises(AssertionError):
        pins.test_adamw_matches_torch_optim()
