#!/usr/bin/env python
"""Throughput of ZeroLock's concurrent per-chunk update on GB300 (one JSON line on stdout).

A step is one micro-batch through all K chunks (forward, readout, local objective, local
backward, AdamW) via zl_step. Default workload: the largest configuration, the Llama-2-7B-shaped
bf16 full fine-tune (32 layers, d 4096, SwiGLU 11008, vocab 32000, micro-batch 2 x 1024 tokens,
K = 8 chunks of 4 layers); --workload gpt2|llama1b|llama3b|tiny selects the others. Also reported: the same-engine
backpropagation baseline (zl_bp_step), peak HBM of both, the GEMM roofline fraction measured
live with CUDA events, the CPU oracle on a bounded sample, an end-to-end figure through the
public API with host buffers, and SM clocks sampled during the timed region.

Multi-GPU (torchrun): the path does not shard; every rank trains an independent replica on
its own micro-batches ("replicas only"), value = tokens of all ranks / max rank time.

--impl reference times the CPU oracle (the only reference implementation there is) on
bounded samples of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import torch  # noqa: E402

import synth  # noqa: E402

WORKLOADS = {"gpt2": synth.GPT2_SMALL, "tiny": synth.TINY, "llama1b": synth.LLAMA_1B, "llama3b": synth.LLAMA_3B,
             "llama7b": synth.LLAMA_7B}
METRIC = "training tokens/s on 1 GB300 (ZeroLock vs same-engine BP), peak HBM GB, % roofline"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama7b", choices=list(WORKLOADS))
    ap.add_argument("--K", type=int, default=0, help="chunk count (default: the workload's)")
    ap.add_argument("--max-live", type=int, default=2, help="chunks whose activations may be alive at once")
    ap.add_argument("--lora", type=int, default=0, help="LoRA rank (0: full fine-tune); scale 16 / rank")
    ap.add_argument("--graph", action="store_true",
                    help="replay each step as a captured CUDA graph (same GPU time here; more peak memory)")
    ap.add_argument("--adapter", type=int, default=0,
                    help="readout adapter width per chunk (0: static head; a multiple of 16)")
    ap.add_argument("--loss-rows", type=int, default=0,
                    help="readout, local objective and head backward in row slices of this many rows (0: whole)")
    ap.add_argument("--no-bp", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    return ap.parse_args()


def max_over_ranks(ms: float, world: int, device: str = "cuda") -> float:
    """The slowest rank's time (all_reduce MAX over the default process group)."""
    if world <= 1:
        return ms
    import torch.distributed as dist
    x = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(x, op=dist.ReduceOp.MAX)
    return float(x)


def job_tokens_per_s(tokens_per_step: int, steps: int, world: int, max_ms: float) -> float:
    """Whole-job throughput: every rank's tokens over the slowest rank's time."""
    return tokens_per_step * steps * world / (max_ms / 1e3)


def class_ideal_s(v, pk):
    """Ideal time of one kernel class: the larger of its algorithmic FLOPs at the measured sustained bf16
    peak and its algorithmic bytes at the measured HBM copy rate (a GEMM with the optimizer step fused
    into its epilogue is bound by the second)."""
    return max(v["flops"] / (pk["bf16_tflops_sustained"] * 1e12), v["bytes"] / (pk["hbm_gbs"] * 1e9))


def step_roofline(prof, steps: int, ms_per_step: float):
    """Whole-step roofline: the step time if every class ran at its bound (class_ideal_s; algorithmic FLOPs
    and bytes per step from the live profile), split into tensor-bound and HBM-bound classes, and the
    measured step's fraction of it."""
    pk, pk_kind = peaks()
    t_tensor = t_hbm = 0.0
    for v in prof.values():
        t = class_ideal_s(v, pk) / steps
        if v["flops"] / (pk["bf16_tflops_sustained"] * 1e12) >= v["bytes"] / (pk["hbm_gbs"] * 1e9):
            t_tensor += t
        else:
            t_hbm += t
    ideal_ms = (t_tensor + t_hbm) * 1e3
    return {"ideal_ms": ideal_ms, "tensor_ms": t_tensor * 1e3, "hbm_ms": t_hbm * 1e3, "measured_ms": ms_per_step,
            "frac": ideal_ms / ms_per_step if ms_per_step > 0 else None,
            "peak_kind": f"{pk_kind} bf16 sustained / HBM copy"}


def roofline_of(prof, workload="llama7b"):
    """Roofline entry of the kernel class with the largest time share in a zl_profile_read result."""
    pk, pk_kind = peaks()
    tot_ms = sum(v["ms"] for v in prof.values())
    dom = max(prof, key=lambda k: prof[k]["ms"])
    g = prof[dom]
    tensor = g["flops"] / (pk["bf16_tflops_sustained"] * 1e12) >= g["bytes"] / (pk["hbm_gbs"] * 1e9)
    if tensor:
        achieved = g["flops"] / (g["ms"] / 1e3) / 1e12
        peak_v, unit, kind = pk["bf16_tflops_sustained"], "TFLOP/s", f"{pk_kind} bf16 sustained"
    else:
        achieved = g["bytes"] / (g["ms"] / 1e3) / 1e9
        peak_v, unit, kind = pk["hbm_gbs"], "GB/s", f"{pk_kind} HBM copy"
    traffic = measured_traffic(dom, workload)
    return {"bound": "tensor" if tensor else "hbm", "kernel": dom, "achieved": achieved, "peak": peak_v,
            "unit": unit, "frac": achieved / peak_v, "peak_kind": kind, "traffic": traffic,
            "launches": g["launches"],
            "work_per_launch": (g["flops"] if tensor else g["bytes"]) / max(g["launches"], 1),
            "share_of_kernel_time": g["ms"] / tot_ms if tot_ms else None}


# DRAM bytes per launch (read + write) from ncu captures, valid only for the kernel sources they were
# taken on (sha256 prefix over the listed files, in order) and for the workload named; any change to the
# sources makes the figure null. Llama-7B-shaped step (profiles/gemm_tc_llama7b_shapes.md and
# profiles/gemm_update_llama7b_layer.md): layer GEMMs are the mean over the eight forward and dX shapes of
# a layer (each once per layer and step); head GEMMs weight nine forwards (eight students and the first
# teacher) against eight dX products; the fused dW + AdamW products are the mean over a layer's four.
GEMM_SOURCES = ["gemm_tc.cu", "tcgen05.cuh"]
TRAFFIC = {
    "llama7b": {
        "gemm_layer": {"sources": GEMM_SOURCES, "sha256": "d63ff40f8b5a50fe", "bytes_per_launch": 182011136.0},
        "gemm_head": {"sources": GEMM_SOURCES, "sha256": "d63ff40f8b5a50fe", "bytes_per_launch": 467916107.3},
        "gemm_update": {"sources": GEMM_SOURCES, "sha256": "d63ff40f8b5a50fe", "bytes_per_launch": 1408223168.0},
    },
}


def sources_sha(names):
    import hashlib
    h = hashlib.sha256()
    for n in names:
        with open(os.path.join(ROOT, "paper_2608_07974_gb300", "csrc", n), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def measured_traffic(cls, workload="llama7b"):
    ent = TRAFFIC.get(workload, {}).get(cls)
    if not ent or ent["bytes_per_launch"] is None:
        return None
    if sources_sha(ent["sources"]) != ent["sha256"]:
        return None
    return ent["bytes_per_launch"]


def rank_batch_ids(rank: int, n: int):
    """Micro-batch indices of one replica (distinct per rank)."""
    return [1000 * rank + i for i in range(n)]


def workload_desc(w, K, lora=0, adapter=0):
    d = w.dims
    arch = "llama" if d.arch == synth.ARCH_LLAMA else "gpt2"
    tune = f"LoRA rank {lora} scale {16 / lora:g} on QKV/O/FFN" if lora else "full fine-tune"
    return (f"{w.name}: {arch}-style decoder, {d.n_layers} layers, d_model {d.d_model}, {d.n_heads} heads "
            f"({d.n_kv_heads} kv), ffn {d.d_ff}, vocab {d.vocab}, micro-batch {w.batch} x seq {w.seq}, "
            f"K={K} chunks, alpha {w.alpha}, AdamW, {tune}" + (f", readout adapters of width {adapter}" if adapter else ""))


def run_config(args, w, K, world):
    """The `config` object of both arms' JSON lines (the workload they measure)."""
    return {"workload": workload_desc(w, K, args.lora, args.adapter), "K": K,
            "bounds": synth.chunk_bounds(w.dims.n_layers, K), "global_batch": w.batch * world, "seq_len": w.seq,
            "max_live_chunks": args.max_live, "cuda_graph": args.graph, "loss_rows": args.loss_rows,
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU, K streams",
            "l2": "no flush: every step's working set (weights, AdamW state, logits) exceeds L2"}


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return json.load(f), "measured"
    return FALLBACK_PEAKS, "fallback"


# ---------------------------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, local_rank: int):
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        self.gpu = vis.split(",")[local_rank] if vis else str(local_rank)
        self.proc = None
        self.out = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.out, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.flush()
        self.out.seek(0)
        text = self.out.read()
        os.unlink(self.out.name)
        return parse_clocks(text)


def parse_clocks(text: str):
    """Summary of nvidia-smi samples in ClockSampler.FIELDS order (csv, no header, no units): median SM
    clock, the maximum SM clock, and every throttle reason seen Active in any sample."""
    rows = [r.split(",") for r in text.strip().splitlines() if r.strip()]
    sm, mx, reasons = [], 0.0, set()
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    for r in rows:
        try:
            sm.append(float(r[1]))
            mx = max(mx, float(r[2]))
            for n, v in zip(names, r[5:9]):
                if v.strip() == "Active":
                    reasons.add(n)
        except (ValueError, IndexError):
            continue
    if not sm:
        return None
    return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------------------------
# CPU oracle on a bounded sample
# ---------------------------------------------------------------------------------------------
ORACLE_SAMPLE_FLOP = 0.5e12      # about the oracle work of one CPU-baseline sample
ORACLE_WHOLE_MODEL_PARAMS = 3e9  # above this the sample runs chunk 1 alone (every chunk costs about the same)


def oracle_sample_plan(w, K):
    """(chunks sampled, tokens per sample sequence) of the CPU-baseline sample.

    One sample is chunk k's local step on one sequence. Its length is the longest power of two up to
    the workload's sequence length whose estimated cost (6 FLOP per chunk parameter and token for the
    forward and backward, plus the student and teacher heads) stays near ORACLE_SAMPLE_FLOP, at least
    64. Models above ORACLE_WHOLE_MODEL_PARAMS sample chunk 1 only (as a one-chunk model of its own
    layers, whose teacher is the readout of h_0 exactly as in the full model); smaller ones go
    round-robin over all K chunks.
    """
    d = w.dims
    layer = sum(int(torch.tensor(shp).prod()) for _, shp in synth.layer_param_shapes(d))
    per_tok = 6.0 * layer * d.n_layers / K + 6.0 * d.d_model * d.vocab
    seq = 64
    while seq * 2 <= w.seq and seq * 2 * per_tok <= ORACLE_SAMPLE_FLOP:
        seq *= 2
    seq = min(seq, w.seq)
    chunks = list(range(1, K + 1)) if layer * d.n_layers <= ORACLE_WHOLE_MODEL_PARAMS else [1]
    return chunks, seq


def oracle_params(w, K, chunks, params=None):
    """fp32 CPU tensors the oracle needs for the sampled chunks (drawn on the GPU when one is present)."""
    import dataclasses
    bounds = synth.chunk_bounds(w.dims.n_layers, K)
    if chunks == list(range(1, K + 1)):
        dims, layers = w.dims, None
    else:
        dims, layers = dataclasses.replace(w.dims, n_layers=bounds[1]), range(bounds[1])
    if params is None:
        dev = "cuda" if torch.cuda.is_available() else "cpu"
        params = synth.make_params(w.dims, w.seed, layers=layers, device=dev)
    keep = set(n for n, _ in synth.frozen_param_shapes(w.dims)) | set(n for n, _ in synth.param_names(dims))
    return dims, {n: t.cpu() for n, t in params.items() if n in keep}


def oracle_sample(w, K, params, n_samples: int, min_seconds: float = 0.0):
    """Times the oracle on local steps of one chunk on one sequence each (oracle_sample_plan: the
    chunks, round-robin, and the sequence length): `n_samples` of them, or, with `min_seconds` > 0, as
    many as it takes for the samples after the first to add up to min_seconds (at least one per sampled
    chunk after the first sample, at most n_samples). `params` may be None (drawn here) or the
    workload's tensors on any device.

    One local step of one chunk costs about 1/K of a full ZeroLock step of the same tokens, so the
    equivalent rate is (sequence length / K) tokens per sample time. Returns (times, tokens per
    sample, intra-op threads, a description of the sample).
    """
    from oracle import Oracle, OracleConfig
    chunks, seq = oracle_sample_plan(w, K)
    dims, P = oracle_params(w, K, chunks, params)
    bounds = synth.chunk_bounds(dims.n_layers, K) if dims is w.dims else [0, dims.n_layers]
    P = {n: (synth.round_bf16(t) if (w.dtype == "bf16" and t.dim() == 2) else t) for n, t in P.items()}
    dt = torch.float32 if w.dtype == "bf16" else torch.float64
    orc = Oracle(OracleConfig(dims=dims, bounds=bounds, alpha=w.alpha, lr=w.lr), P, dtype=dt)
    ids = synth.zipf_ids(w.seed + 77, 1, seq, w.dims.vocab)
    labels = synth.next_token_labels(ids)
    h0 = orc.embed(ids)
    times = []
    for i in range(n_samples):
        if min_seconds > 0 and i > len(chunks) and sum(times[1:]) >= min_seconds:
            break
        k = chunks[i % len(chunks)]
        t0 = time.perf_counter()
        orc.local_grad(k, h0, labels)
        times.append(time.perf_counter() - t0)
    which = "round-robin over the K chunks" if len(chunks) == K else "of chunk 1 (every chunk has about its size)"
    desc = f"local steps of one chunk on 1 x {seq} tokens, {which}; rate = ({seq}/K) tokens per sample time"
    return times, (seq / K), torch.get_num_threads(), desc


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    w = WORKLOADS[args.workload]
    K = args.K or w.K
    times, tok, cores, desc = oracle_sample(w, K, None, args.warmup + args.steps)
    t = sum(times[args.warmup:])
    value = tok * args.steps / t
    sample = f"{args.steps} {desc}"
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32" if w.dtype == "bf16" else "f64", "data": "synthetic",
            "config": run_config(args, w, K, int(os.environ.get("WORLD_SIZE", "1"))),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "nproc": os.cpu_count(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------------------------
def run_ours(args):
    import torch.distributed as dist
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")
    import paper_2608_07974_gb300 as pkg
    pkg.build()
    from paper_2608_07974_gb300 import binding as zb

    w = WORKLOADS[args.workload]
    K = args.K or w.K
    bounds = synth.chunk_bounds(w.dims.n_layers, K)
    # drawn on the device (the same counter-based draws as on the host; the 7B-shaped model has 6.7 B)
    params = synth.make_params(w.dims, w.seed, device="cuda")
    if args.lora:
        params.update({n: t.cuda() for n, t in synth.make_lora_params(w.dims, w.seed, args.lora).items()})
    if args.adapter:
        params.update({n: t.cuda() for n, t in synth.make_adapter_params(w.dims, K, w.seed, args.adapter).items()})

    def make_engine(max_live, serialize=False):
        e = zb.ZeroLock(w.dims, K, bounds, dtype=w.dtype, alpha=w.alpha, lr=w.lr, beta1=w.beta1, beta2=w.beta2,
                        eps=w.eps, weight_decay=w.weight_decay, max_live_chunks=max_live, serialize=serialize,
                        lora_rank=args.lora, lora_scale=16.0 / args.lora if args.lora else 1.0,
                        adapter_dim=args.adapter, graph=args.graph, loss_rows=args.loss_rows)
        e.load(params)
        return e

    nb = 4   # distinct resident micro-batches, per rank
    batches = [synth.make_batch(w, i) for i in rank_batch_ids(rank, nb)]
    dev_batches = [(a.cuda(), b.cuda()) for a, b in batches]
    tokens = w.batch * w.seq
    stream = torch.cuda.current_stream()

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()

    def timed(fn, steps, finish=None):
        """Device time of `steps` calls of fn: the steps are queued back to back (no host sync between
        them), then `finish` joins every stream of the engine into the timing stream."""
        barrier()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for i in range(steps):
            fn(i)
        if finish is not None:
            finish()
        t1.record(stream)
        barrier()
        return max_over_ranks(t0.elapsed_time(t1), world)

    # ---- ZeroLock: device-resident inputs -----------------------------------------------------
    eng = make_engine(args.max_live)

    # Steps are queued as a training loop queues them: chunk k of step i+1 waits only for its own update
    # of step i and for chunk k-1's output of step i+1, so it may start while later chunks of step i
    # still run (no update locking across steps either). One join at the end covers all of them.
    def zl(i):
        ids, lab = dev_batches[i % nb]
        zb.zl_step(eng.ctx, ids, lab, w.batch, w.seq, K, want_losses=False)

    for i in range(args.warmup):
        zl(i)
    zb.zl_join(eng.ctx)
    eng.synchronize()
    eng.reset_peak()
    clocks = ClockSampler(local)
    clocks.start()
    n0 = zb.zl_kernel_launches()
    ms = timed(zl, args.steps, finish=lambda: zb.zl_join(eng.ctx))
    launches = zb.zl_kernel_launches() - n0
    clk = clocks.stop()
    zl_peak = eng.peak_bytes()[0]
    value = job_tokens_per_s(tokens, args.steps, world, ms)

    # ---- live per-kernel-class timing (CUDA events on the launching streams) ------------------
    zb.zl_profile(eng.ctx, True)
    prof_steps = min(args.steps, 5)
    for i in range(prof_steps):
        zl(i)
    prof = zb.zl_profile_read(eng.ctx)
    zb.zl_profile(eng.ctx, False)
    roof = roofline_of(prof, args.workload if not (args.K or args.lora or args.adapter or args.loss_rows) else "")
    step_roof = step_roofline(prof, prof_steps, ms / args.steps)
    classes = {k: {"launches": v["launches"], "ms_per_step": v["ms"] / prof_steps,
                   "TFLOP/s" if v["flops"] else "GB/s":
                       (v["flops"] / (v["ms"] / 1e3) / 1e12) if v["flops"] else (v["bytes"] / (v["ms"] / 1e3) / 1e9)
                       if v["ms"] > 0 else 0.0}
               for k, v in prof.items() if v["launches"]}

    # ---- end to end through the public API with host buffers ---------------------------------
    e2e = None
    if not args.no_e2e:
        host = [(a.pin_memory(), b.pin_memory()) for a, b in batches]
        dids = torch.empty_like(dev_batches[0][0])
        dlab = torch.empty_like(dev_batches[0][1])
        out = torch.empty(K, dtype=torch.float32)

        def e2e_step(i):
            hi, hl = host[i % nb]
            dids.copy_(hi, non_blocking=True)
            dlab.copy_(hl, non_blocking=True)
            zb.zl_step(eng.ctx, dids, dlab, w.batch, w.seq, K, want_losses=False)
            out[:] = torch.tensor(zb.zl_read_losses(eng.ctx, K))
        for i in range(2):
            e2e_step(i)
        ems = timed(e2e_step, args.steps)
        e2e = {"value": job_tokens_per_s(tokens, args.steps, world, ems), "unit": "tokens/s",
               "h2d_bytes_per_step": 2 * tokens * 4, "d2h_bytes_per_step": K * 4}
    eng.close()
    del eng
    torch.cuda.empty_cache()

    # ---- same-engine backpropagation ----------------------------------------------------------
    bp = None
    if not args.no_bp:
        beng = make_engine(args.max_live)

        def bps(i):   # each backprop step waits for the previous one's update on the engine's streams
            ids, lab = dev_batches[i % nb]
            zb.zl_bp_step(beng.ctx, ids, lab, w.batch, w.seq, want_loss=False)
        for i in range(args.warmup):
            bps(i)
        beng.synchronize()
        beng.reset_peak()
        bms = timed(bps, args.steps, finish=lambda: zb.zl_join(beng.ctx))
        bp = {"value": job_tokens_per_s(tokens, args.steps, world, bms), "unit": "tokens/s",
              "peak_hbm_gb": beng.peak_bytes()[0] / 1e9, "ms_per_step": bms / args.steps}
        beng.close()
        del beng
        torch.cuda.empty_cache()

    # ---- the same step with every chunk on one stream: per-launch times without the other chunks' kernels
    seng = make_engine(args.max_live, serialize=True)
    for i in range(2):
        zb.zl_step(seng.ctx, dev_batches[i % nb][0], dev_batches[i % nb][1], w.batch, w.seq, K, want_losses=False)
    zb.zl_profile(seng.ctx, True)
    for i in range(prof_steps):
        zb.zl_step(seng.ctx, dev_batches[i % nb][0], dev_batches[i % nb][1], w.batch, w.seq, K, want_losses=False)
    sprof = zb.zl_profile_read(seng.ctx)
    seng.close()
    del seng
    torch.cuda.empty_cache()
    roof_serial = roofline_of(sprof, args.workload if not (args.K or args.lora or args.adapter or args.loss_rows) else "")
    classes_serial = {k: {"launches": v["launches"], "ms_per_step": v["ms"] / prof_steps}
                      for k, v in sprof.items() if v["launches"]}

    # ---- CPU oracle on a bounded sample (rank 0, one GPU only) --------------------------------
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu and not args.lora and not args.adapter:
        times, tok, cores, desc = oracle_sample(w, K, params, 64, min_seconds=15.0)
        n, secs = len(times) - 1, sum(times[1:])
        cpu = {"value": tok * n / secs, "unit": "tokens/s", "cores": cores, "nproc": os.cpu_count(),
               "kind": "oracle", "sample": f"{n} {desc} ({secs:.1f} s of oracle work after one warm-up sample)"}

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
                "config": run_config(args, w, K, world),
                "peak_hbm_gb": zl_peak / 1e9, "bp": bp,
                "zl_vs_bp": {"throughput": value / bp["value"], "peak_hbm": (zl_peak / 1e9) / bp["peak_hbm_gb"]}
                if bp else None,
                "roofline": roof, "roofline_serial": roof_serial, "step_roofline": step_roof, "kernel_classes": classes,
                "kernel_classes_serial": classes_serial, "cpu_baseline": cpu, "e2e": e2e,
                "gpu_launches": launches, "clocks": clk}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
