"""Host-side checks of the bench's device-drawn activations (the recipe of the
large prefill inputs), run here on the CPU device: the outlier channels, their
per-token jitter, the bulk distributions and the seeding."""

import os
import sys

import numpy as np
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
import workloads as W  # noqa: E402

CPU = torch.device("cpu")


def test_outlier_channels_carry_the_jittered_amplitude():
    w = bench.workload_by_name("llama2_70b")
    T, K = 256, 2048
    x = bench.device_activations(T, K, w, seed=3, device=CPU)
    assert x.shape == (T, K) and x.dtype == torch.bfloat16
    xf = x.float().numpy()
    chans = W.outlier_channels(K, w.n_out)
    assert len(chans) == w.n_out and chans[0] == 0
    # Every outlier channel of a token holds the same amplitude mult * (1 + 0.1 z_t).
    amp = xf[:, chans[0]]
    for c in chans[1:]:
        np.testing.assert_array_equal(xf[:, c], amp)
    rel = amp / w.mult - 1.0
    assert abs(rel.mean()) < 0.03 and 0.07 < rel.std() < 0.13
    assert np.all(amp > 0)


def test_bulk_distributions():
    T, K = 512, 1024
    normal = bench.device_activations(T, K, bench.workload_by_name("llama2_70b"), seed=4, device=CPU).float()
    heavy = bench.device_activations(T, K, bench.workload_by_name("llama3_8b_mlp"), seed=4, device=CPU).float()
    keep = torch.ones(K, dtype=torch.bool)
    keep[W.outlier_channels(K, 6)] = False
    keep[W.outlier_channels(K, 3)] = False
    nb = normal[:, keep].flatten()
    hb = heavy[:, keep].flatten()
    assert abs(nb.mean().item()) < 0.02 and abs(nb.std().item() - 1.0) < 0.02
    # Student-t with 3 degrees of freedom: variance 3 and much heavier tails than N(0, 1).
    assert 2.0 < hb.var().item() < 4.5
    assert (hb.abs() > 6).float().mean().item() > 20 * (nb.abs() > 6).float().mean().item() + 1e-4


def test_seeded_and_distinct_per_seed():
    w = bench.workload_by_name("llama3_8b_mlp")
    a = bench.device_activations(64, 512, w, seed=7, device=CPU)
    b = bench.device_activations(64, 512, w, seed=7, device=CPU)
    c = bench.device_activations(64, 512, w, seed=8, device=CPU)
    assert torch.equal(a, b)
    assert not torch.equal(a, c)
