"""CPU oracle of ZeroLock's decoupled per-chunk update (test infrastructure).

This package is test infrastructure. Only ``tests/``, ``__graft_entry__.smoke()``
and the ``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import
it. The CUDA library never calls into it, and it shares no code with the CUDA
path; the only common module is ``synth`` (seeded input draws).

It is a plain, slow, float64 (by default) PyTorch-CPU restatement of Section
II-A of the paper (Eq. 1-6) with the readings listed in ``model.py``.
Gradients come from autograd over the chunk's own parameters, which is the
plain definition of "backpropagate inside the chunk only" (Remark 1).

Pins (``tests/test_oracle_pins.py``): central finite differences, library
routines (scaled_dot_product_attention, rms_norm, layer_norm, gelu, AdamW),
closed forms of the loss, Lemma 1 (three-point identity), Lemma 2 (geometric
mixture), Lemma 3 (stop-gradient block structure), K=1, alpha=1 == BP, an
independent autograd-free backward (tests/manual_backprop.py), and Proposition 1's
chunk-wise bound in its token-level geometry (random soft targets and chains).
Parity unpinned: Theorem 1 (a convergence rate over training) and Proposition 1
for whole trained models need trained weights and data and are not checked.
"""
from .model import (Oracle, OracleConfig, embed, layer_forward, chunk_forward, readout, adapter,
                    local_objective, local_objective_rows, rmsnorm, layernorm, rope,
                    attention, gelu_tanh, silu, kl_rows, adamw_update)

__all__ = ["Oracle", "OracleConfig", "embed", "layer_forward", "chunk_forward", "readout", "adapter",
           "local_objective", "local_objective_rows", "rmsnorm", "layernorm", "rope",
           "attention", "gelu_tanh", "silu", "kl_rows", "adamw_update"]
