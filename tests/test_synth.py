"""The seeded generators produce the shapes, densities and row-length mixes
the workloads call for (they hold no training arithmetic)."""

import numpy as np

from paper_1905_07931_gb300 import synth


def test_zipf_lengths_sum_clip_and_skew():
    lengths = synth.zipf_row_lengths(4096, 4096, int(round(0.05 * 4096 * 4096)))
    assert lengths.sum() == round(0.05 * 4096 * 4096)
    assert lengths.max() == 4096 and lengths.min() >= 0
    assert (np.diff(lengths) <= 0).all()          # non-increasing in rank


def test_masks_density_and_determinism():
    a = synth.masked_weights(synth.rng_for(0), 300, 784, 0.10, std=0.05)
    b = synth.masked_weights(synth.rng_for(0), 300, 784, 0.10, std=0.05)
    np.testing.assert_array_equal(a, b)
    assert abs((a != 0).mean() - 0.10) < 0.01
    z = synth.masked_weights(synth.rng_for(1), 64, 128, 0.2, zipf=True)
    assert (z != 0).sum() == round(0.2 * 64 * 128)


def test_workload_shapes():
    c1 = synth.single_fc()
    assert c1["W"].shape == (300, 784) and c1["X"].shape == (784, 64) and c1["dY"].shape == (300, 64)
    c2 = synth.mlp()
    assert [w.shape for w in c2["W"]] == [(300, 784), (100, 300), (10, 100)]
    c3 = synth.lenet()
    assert [w.shape for w in c3["W"]] == [(20, 25), (50, 500), (500, 800), (10, 500)]
    assert c3["X"].shape == (1, 128, 28, 28)
