"""The seeded input generator against its published definitions (no GPU)."""
import math

import torch

import synth


def test_splitmix64_published_vector():
    # SplitMix64 from state 0: the first outputs are 0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4
    out = synth.raw_u64(0, 0, 2).numpy().view("uint64")
    assert int(out[0]) == 0xE220A8397B1DCDAF
    assert int(out[1]) == 0x6E789E6AA1B965F4
    assert synth.mix64_int(0x9E3779B97F4A7C15) == 0xE220A8397B1DCDAF


def test_counter_based_slices_agree():
    key = synth.stream_key(5, "x")
    full = synth.uniform(key, 1000)
    part = synth.uniform(key, 100, start=300)
    assert torch.equal(full[300:400], part)
    assert float(full.min()) > 0 and float(full.max()) < 1


def test_normal_moments():
    x = synth.normal(synth.stream_key(1, "n"), 200_000, 0.02)
    assert abs(float(x.mean())) < 3 * 0.02 / math.sqrt(2e5)
    assert abs(float(x.std()) - 0.02) < 0.02 * 0.01


def test_zipf_frequencies_and_labels():
    V = 50
    ids = synth.zipf_ids(3, 64, 512, V)
    assert ids.dtype == torch.int32 and int(ids.min()) >= 0 and int(ids.max()) < V
    cnt = torch.bincount(ids.view(-1).long(), minlength=V).double()
    r = torch.arange(1, V + 1, dtype=torch.float64)
    p = r ** -1.1 / (r ** -1.1).sum()
    # rank-1 vs rank-2 frequency ratio is 2^1.1 under Zipf(1.1)
    assert abs(float(cnt[0] / cnt[1]) - 2 ** 1.1) < 0.15   # ~4 sigma at this sample size
    chi = float(((cnt - p * cnt.sum()) ** 2 / (p * cnt.sum())).sum())
    assert chi < 150          # 49 degrees of freedom
    lab = synth.next_token_labels(ids)
    assert torch.equal(lab[:, :-1], ids[:, 1:]) and bool((lab[:, -1] == -1).all())


def test_chunk_bounds_put_remainder_last():
    assert synth.chunk_bounds(22, 4) == [0, 5, 10, 16, 22]
    assert synth.chunk_bounds(22, 8) == [0, 2, 4, 7, 10, 13, 16, 19, 22]
    assert synth.chunk_bounds(22, 2) == [0, 11, 22]
    assert synth.chunk_bounds(12, 4) == [0, 3, 6, 9, 12]
