"""LoRA chunks (the paper's fine-tuning setting, Section II-A) through the C ABI against the oracle.

Only A_l and B_l train (Delta w_l = s B_l A_l on the QKV, output and FFN linears); base weights,
norms and biases are frozen. Tiny fp32 workload: losses and parameters after 10 AdamW steps
within 1e-4 relative. GPT-2 bf16 at full size: loss within 2e-2, gradient cosine >= 0.999.
"""
import pytest
import torch

import synth
from tests.gpu_common import cosine, engine_for, fro_rel, oracle_for, rel

pytestmark = pytest.mark.gpu
RANK, SCALE = 4, 4.0     # rank 4, lora_alpha 16 -> scale 16 / 4


def _params(w, b_std):
    P = synth.make_params(w.dims, w.seed)
    P.update(synth.make_lora_params(w.dims, w.seed, RANK, b_std=b_std))
    return P


@pytest.mark.parametrize("b_std", [0.0, 0.05])
def test_tiny_lora_ten_steps(b_std):
    w = synth.TINY
    P = _params(w, b_std)
    eng = engine_for(w, lora_rank=RANK, lora_scale=SCALE)
    eng.load(P)
    orc = oracle_for(w, P, lora_rank=RANK, lora_scale=SCALE)
    for s in range(w.steps):
        ids, labels = synth.make_batch(w, s)
        lg = eng.step(ids.cuda(), labels.cuda())
        lo = orc.step(ids, labels)
        for a, b in zip(lg, lo):
            assert rel(a, b) <= 1e-4, (s, lg, lo)
    for n in orc.trainable_names():
        assert "lora_" in n
        assert fro_rel(eng.get(n), orc.P[n]) <= 1e-4, n
    # frozen tensors did not move
    for n in ("layers.0.wqkv", "layers.1.ffn_norm.weight", "layers.3.w2"):
        assert torch.equal(eng.get(n), P[n].reshape(-1)), n
    eng.close()


def test_gpt2_lora_chunk_full_size():
    w = synth.GPT2_SMALL
    P = {n: (synth.round_bf16(t) if t.dim() == 2 else t) for n, t in _params(w, 0.02).items()}
    eng = engine_for(w, accum_m=2, lora_rank=RANK, lora_scale=SCALE)
    eng.load(P)
    ids, labels = synth.make_batch(w, 0)
    h1 = eng.forward_chunk(1, None, ids.cuda(), w.batch, w.seq)
    lg = eng.step(ids.cuda(), labels.cuda())
    orc = oracle_for(w, P, dtype=torch.float32, lora_rank=RANK, lora_scale=SCALE)
    L, g, _ = orc.local_grad(2, h1.float().cpu().view(w.batch, w.seq, -1), labels)
    assert rel(lg[1], L) <= 2e-2, (lg, L)
    for n in orc.chunk_names(2):
        c = cosine(eng.get(n, 1), g[n])
        assert c >= 0.999, (n, c)
    eng.close()
