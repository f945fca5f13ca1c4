"""Helpers shared by the GPU tests: engine construction from a workload and comparisons."""
import torch

import synth
from oracle import Oracle, OracleConfig


def engine_for(w, K=None, bounds=None, alpha=None, **kw):
    import paper_2608_07974_gb300 as pkg
    pkg.build()
    from paper_2608_07974_gb300.binding import ZeroLock
    K = K or w.K
    bounds = bounds or synth.chunk_bounds(w.dims.n_layers, K)
    a = w.alpha if alpha is None else alpha
    return ZeroLock(w.dims, K, bounds, dtype=w.dtype, alpha=a, lr=w.lr, beta1=w.beta1, beta2=w.beta2,
                    eps=w.eps, weight_decay=w.weight_decay, **kw)


def oracle_for(w, params, K=None, bounds=None, alpha=None, dtype=torch.float64, **kw):
    K = K or w.K
    bounds = bounds or synth.chunk_bounds(w.dims.n_layers, K)
    a = w.alpha if alpha is None else alpha
    cfg = OracleConfig(dims=w.dims, bounds=bounds, alpha=a, lr=w.lr, beta1=w.beta1, beta2=w.beta2, eps=w.eps,
                       weight_decay=w.weight_decay, **kw)
    return Oracle(cfg, params, dtype=dtype)


def rel(a, b):
    return abs(a - b) / max(abs(b), 1e-30)


def fro_rel(x, ref):
    x, ref = x.double().view(-1), ref.double().view(-1)
    return float((x - ref).norm() / max(float(ref.norm()), 1e-30))


def cosine(x, ref):
    x, ref = x.double().view(-1), ref.double().view(-1)
    return float(x @ ref / max(float(x.norm() * ref.norm()), 1e-300))
