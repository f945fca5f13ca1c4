"""bench.py's CPU-baseline sampling (no GPU): a time-bounded, round-robin sample of oracle local steps."""
import bench
import synth


def test_oracle_sample_runs_until_the_time_budget_and_covers_every_chunk():
    w = bench.WORKLOADS["tiny"]
    P = synth.make_params(w.dims, w.seed)
    times, tok, cores, desc = bench.oracle_sample(w, 2, P, 200, min_seconds=0.3)
    assert len(times) > 2 + 1                      # the warm-up sample plus at least one per chunk
    assert sum(times[1:]) >= 0.3 or len(times) == 200
    assert sum(times[1:-1]) < 0.3                  # stopped at the first sample past the budget
    assert tok == w.seq / 2 and cores >= 1 and "round-robin" in desc
    fixed, _, _, _ = bench.oracle_sample(w, 2, P, 3)
    assert len(fixed) == 3                         # without a budget: exactly the requested count


def test_oracle_sample_plan_bounds_the_work_of_one_sample():
    """Every workload's sample is a few hundred GFLOP at most; the largest models sample chunk 1 alone,
    as a one-chunk model of its own layers."""
    for name, w in bench.WORKLOADS.items():
        chunks, seq = bench.oracle_sample_plan(w, w.K)
        assert 64 <= seq <= w.seq or seq == w.seq
        assert chunks == list(range(1, w.K + 1)) or chunks == [1]
    assert bench.oracle_sample_plan(bench.WORKLOADS["llama7b"], 8)[0] == [1]
    assert bench.oracle_sample_plan(bench.WORKLOADS["gpt2"], 4) == ([1, 2, 3, 4], 512)


def test_one_chunk_sample_model_is_chunk_one_of_the_full_model():
    """The sub-model the large workloads sample has exactly chunk 1's layers and the frozen tensors."""
    w = bench.WORKLOADS["tiny"]
    dims, P = bench.oracle_params(w, 2, [1])
    assert dims.n_layers == synth.chunk_bounds(w.dims.n_layers, 2)[1]
    full = synth.make_params(w.dims, w.seed)
    assert set(P) == {n for n, _ in synth.frozen_param_shapes(w.dims)} | {n for n, _ in synth.param_names(dims)}
    for n, t in P.items():
        assert t.equal(full[n]), n
