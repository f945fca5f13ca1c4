"""Single-kernel timings through the C ABI (CUDA events, after warm-up), for tuning and profiling.

    python -m paper_2608_07974_gb300.microbench loss [--rows 1024] [--vocab 50257] [--reps 4]
    python -m paper_2608_07974_gb300.microbench gemm [--workload gpt2|llama-1b|llama-7b]
    python -m paper_2608_07974_gb300.microbench attention [--batch 8 --seq 512 --heads 12 --kv-heads 12 --head-dim 64]
    python -m paper_2608_07974_gb300.microbench layer-step [--width 4096 --ffn 11008 --steps 2 --unfused]

`loss` runs the fused local objective on random bf16 logits; `gemm` times the GEMM shapes of the
GPT-2-small workload (12 layers, d 768, FFN 3072, vocab 50304 padded, 4096 tokens) or of the
Llama-style 1.1B one, each with the tile width and split-K count the library's planner picks;
`attention` the causal attention forward and backward.
"""
from __future__ import annotations

import argparse
import os
import sys

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))


def _lib():
    import paper_2608_07974_gb300 as pkg
    pkg.build()
    from paper_2608_07974_gb300 import binding
    return binding


def _time(fn, reps):
    for _ in range(3):
        fn()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        fn()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


def loss(args):
    B = _lib()
    N, V = args.rows, args.vocab
    ldz = (V + 127) // 128 * 128
    g = torch.Generator(device="cuda").manual_seed(0)
    z = (3 * torch.randn(N, ldz, device="cuda", generator=g)).to(torch.bfloat16)
    t = (3 * torch.randn(N, ldz, device="cuda", generator=g)).to(torch.bfloat16)
    lab = torch.randint(0, V, (N,), device="cuda", generator=g, dtype=torch.int32)
    dz = torch.empty_like(z)
    rl = torch.empty(N, device="cuda")
    out = torch.empty(1, device="cuda")
    ms = _time(lambda: B.zl_op_local_loss(1, z, t, lab, N, V, ldz, args.alpha, 0, dz, rl, out), args.reps)
    gb = 3 * N * ldz * 2 / 1e9
    print(f"local loss N={N} V={V}: {ms * 1e3:.1f} us, {gb / (ms / 1e3):.0f} GB/s of {gb * 1e3:.0f} MB algorithmic")


GPT2_SHAPES = [("qkv fwd", 0, 4096, 2304, 768), ("o fwd", 0, 4096, 768, 768), ("fc fwd", 0, 4096, 3072, 768),
               ("proj fwd", 0, 4096, 768, 3072), ("head fwd", 0, 4096, 50304, 768), ("qkv dX", 1, 4096, 768, 2304),
               ("o dX", 1, 4096, 768, 768), ("fc dX", 1, 4096, 768, 3072), ("proj dX", 1, 4096, 3072, 768),
               ("head dX", 1, 4096, 768, 50304), ("qkv dW", 2, 2304, 768, 4096), ("o dW", 2, 768, 768, 4096),
               ("fc dW", 2, 3072, 768, 4096), ("proj dW", 2, 768, 3072, 4096), ("4096^3", 0, 4096, 4096, 4096)]


def _shapes_of(d, d_qkv, f1, f, V, n=4096):
    return [("qkv fwd", 0, n, d_qkv, d), ("o fwd", 0, n, d, d), ("ffn-in fwd", 0, n, f1, d), ("ffn-out fwd", 0, n, d, f),
            ("head fwd", 0, n, V, d), ("qkv dX", 1, n, d, d_qkv), ("o dX", 1, n, d, d), ("ffn-in dX", 1, n, d, f1),
            ("ffn-out dX", 1, n, f, d), ("head dX", 1, n, d, V), ("qkv dW", 2, d_qkv, d, n), ("o dW", 2, d, d, n),
            ("ffn-in dW", 2, f1, d, n), ("ffn-out dW", 2, d, f, n), ("4096^3", 0, 4096, 4096, 4096)]


# Llama-style 1.1B: d 2048, 32 query / 4 key-value heads of 64, SwiGLU 5632 (gate and up fused), vocab 32000
LLAMA1B_SHAPES = _shapes_of(2048, 2560, 11264, 5632, 32000)
# Llama-2-7B-shaped: d 4096, 32 heads of 128, SwiGLU 11008, vocab 32000, 2 x 1024 tokens
LLAMA7B_SHAPES = _shapes_of(4096, 12288, 22016, 11008, 32000, n=2048)


def gemm(args):
    B = _lib()
    shapes = {"gpt2": GPT2_SHAPES, "llama-1b": LLAMA1B_SHAPES, "llama-7b": LLAMA7B_SHAPES}[args.workload]
    if args.only and args.only not in [sh[0] for sh in shapes]:
        raise SystemExit(f"no shape named {args.only!r}")
    for name, mode, M, N, K in shapes:
        if args.only and name != args.only:
            continue
        bf = torch.bfloat16
        if mode == 0:
            a, b = torch.randn(M, K, device="cuda").to(bf), torch.randn(N, K, device="cuda").to(bf)
        elif mode == 1:
            a, b = torch.randn(M, K, device="cuda").to(bf), torch.randn(K, N, device="cuda").to(bf)
        else:
            a, b = torch.randn(K, M, device="cuda").to(bf), torch.randn(K, N, device="cuda").to(bf)
        c = torch.zeros(M, N, device="cuda", dtype=torch.float32 if mode == 2 else bf)
        ms = _time(lambda: B.zl_op_gemm(1, mode, M, N, K, a, b, c), args.reps)
        print(f"{name:9s} M={M:5d} N={N:6d} K={K:6d} {ms * 1e3:7.1f} us {2 * M * N * K / ms / 1e9:7.1f} TFLOP/s",
              flush=True)


def attention(args):
    B = _lib()
    Bb, S, H, Hkv, hd = args.batch, args.seq, args.heads, args.kv_heads, args.head_dim
    W = (H + 2 * Hkv) * hd
    qkv = torch.randn(Bb * S, W, device="cuda").to(torch.bfloat16)
    out = torch.empty(Bb * S, H * hd, device="cuda", dtype=torch.bfloat16)
    dout = torch.randn_like(out)
    dq = torch.empty_like(qkv)
    lse = torch.empty(Bb, H, S, device="cuda")
    f = _time(lambda: B.zl_op_attention(1, qkv, out, lse, Bb, S, H, Hkv, hd), args.reps)
    b = _time(lambda: B.zl_op_attention_bwd(1, qkv, out, dout, lse, dq, Bb, S, H, Hkv, hd), args.reps)
    fl = 2.0 * Bb * H * S * S * hd   # causal: half of 4 B H S^2 hd
    print(f"attention B={Bb} S={S} H={H}/{Hkv} hd={hd}: fwd {f * 1e3:.1f} us ({fl / f / 1e9:.0f} TFLOP/s), "
          f"bwd {b * 1e3:.1f} us ({2 * fl / b / 1e9:.0f} TFLOP/s, 4 matmuls counted)")


def layer_step(args):
    """Concurrent steps of one Llama-style layer as a one-chunk model (small enough for a full ncu capture
    of every kernel of a step, with the optimizer step fused into the dW products unless --unfused)."""
    _lib()
    import synth
    from paper_2608_07974_gb300.binding import ZeroLock
    d = synth.ModelDims(synth.ARCH_LLAMA, 1, args.width, args.heads, args.heads, args.ffn, args.vocab, args.seq)
    w = synth.Workload("layer", d, "bf16", batch=args.batch, seq=args.seq, K=1, steps=args.steps)
    eng = ZeroLock(d, 1, [0, 1], dtype="bf16", alpha=0.5, unfused_update=args.unfused)
    eng.load(synth.make_params(d, 1, device="cuda"))
    ids, labels = (t.cuda() for t in synth.make_batch(w, 0))
    from paper_2608_07974_gb300.binding import zl_join

    def step():
        eng.step(ids, labels, want_losses=False)
        zl_join(eng.ctx)   # every stream of the engine back into the timing stream
    ms = _time(step, args.steps)
    eng.synchronize()
    print(f"layer step d={args.width} ffn={args.ffn} {args.batch}x{args.seq} tokens: {ms * 1e3:.1f} us per step")


def main():
    ap = argparse.ArgumentParser()
    sub = ap.add_subparsers(dest="cmd", required=True)
    p = sub.add_parser("loss")
    p.add_argument("--rows", type=int, default=1024)
    p.add_argument("--vocab", type=int, default=50257)
    p.add_argument("--alpha", type=float, default=0.5)
    p.add_argument("--reps", type=int, default=4)
    p = sub.add_parser("gemm")
    p.add_argument("--workload", choices=["gpt2", "llama-1b", "llama-7b"], default="gpt2")
    p.add_argument("--reps", type=int, default=20)
    p.add_argument("--only", default="", help="run this shape only (its name, e.g. 'qkv fwd')")
    p = sub.add_parser("attention")
    p.add_argument("--batch", type=int, default=8)
    p.add_argument("--seq", type=int, default=512)
    p.add_argument("--heads", type=int, default=12)
    p.add_argument("--kv-heads", type=int, default=12)
    p.add_argument("--head-dim", type=int, default=64)
    p.add_argument("--reps", type=int, default=10)
    p = sub.add_parser("layer-step")
    p.add_argument("--width", type=int, default=4096)
    p.add_argument("--ffn", type=int, default=11008)
    p.add_argument("--heads", type=int, default=32)
    p.add_argument("--vocab", type=int, default=1024)
    p.add_argument("--batch", type=int, default=2)
    p.add_argument("--seq", type=int, default=1024)
    p.add_argument("--steps", type=int, default=2)
    p.add_argument("--unfused", action="store_true")
    args = ap.parse_args()
    {"loss": loss, "gemm": gemm, "attention": attention, "layer-step": layer_step}[args.cmd](args)


if __name__ == "__main__":
    main()
