"""bench.py's CPU-baseline sampling (no GPU): a time-bounded, round-robin sample of oracle local steps."""
import bench
import synth


def test_oracle_sample_runs_until_the_time_budget_and_covers_every_chunk():
    w = bench.WORKLOADS["tiny"]
    P = synth.make_params(w.dims, w.seed)
    times, tok, cores = bench.oracle_sample(w, 2, P, 200, min_seconds=0.3)
    assert len(times) > 2 + 1                      # the warm-up sample plus at least one per chunk
    assert sum(times[1:]) >= 0.3 or len(times) == 200
    assert sum(times[1:-1]) < 0.3                  # stopped at the first sample past the budget
    assert tok == w.seq / 2 and cores >= 1
    fixed, _, _ = bench.oracle_sample(w, 2, P, 3)
    assert len(fixed) == 3                         # without a budget: exactly the requested count
