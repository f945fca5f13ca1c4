"""The oracle still reproduces its stored tiny-workload trajectory (no GPU)."""
import json
import os

import tests.golden.make_golden as mg

HERE = os.path.dirname(os.path.abspath(__file__))


def test_tiny_trajectory_is_reproducible():
    with open(os.path.join(HERE, "golden", "tiny_f32_oracle_losses.json")) as f:
        ref = json.load(f)
    out = mg.tiny_trajectory()
    assert out["local_losses"] == ref["local_losses"]
    assert out["global_loss_after"] == ref["global_loss_after"]
    # the local losses decrease over the 10 AdamW steps
    first, last = ref["local_losses"][0], ref["local_losses"][-1]
    assert all(l < f for f, l in zip(first, last))
