"""Writes tests/golden/*.json from the CPU oracle only (run: python tests/golden/make_golden.py).

tiny_f32_oracle_losses.json: the 10-step ZeroLock trajectory of the tiny
fp32 Llama-style workload (4 layers, d 128, 4 heads, FFN 344, vocab 512,
seq 64, batch 4, K = 2, alpha 0.5, AdamW lr 1e-3, betas 0.9/0.999, wd 0.01),
computed by the float64 oracle on the seeded synthetic inputs.
"""
import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import torch  # noqa: E402

import synth  # noqa: E402
from oracle import Oracle, OracleConfig  # noqa: E402


def tiny_trajectory():
    w = synth.TINY
    cfg = OracleConfig(dims=w.dims, bounds=synth.chunk_bounds(w.dims.n_layers, w.K), alpha=w.alpha,
                       lr=w.lr, beta1=w.beta1, beta2=w.beta2, eps=w.eps, weight_decay=w.weight_decay)
    orc = Oracle(cfg, synth.make_params(w.dims, w.seed), dtype=torch.float64)
    losses = []
    for s in range(w.steps):
        ids, labels = synth.make_batch(w, s)
        losses.append(orc.step(ids, labels))
    ids, labels = synth.make_batch(w, w.steps)
    return {"workload": w.name, "K": w.K, "alpha": w.alpha, "steps": w.steps,
            "local_losses": losses, "global_loss_after": orc.global_loss(ids, labels)}


if __name__ == "__main__":
    out = tiny_trajectory()
    with open(os.path.join(HERE, "tiny_f32_oracle_losses.json"), "w") as f:
        json.dump(out, f, indent=1)
    print(json.dumps(out)[:300])
