"""Seeded synthetic inputs shaped like the paper's workloads.

This module draws random numbers and nothing else: masks, initial weights,
inputs, upstream gradients and labels. It holds none of the training step's
arithmetic and imports neither the CUDA binding nor the CPU oracle, so both
sides can be fed from it.

MNIST and CIFAR-10 (Section 4) are not available; these arrays stand in for
them with the same shapes: 28x28 single-channel images with values U[0, 1],
10 classes; AlexNet's 9216-dim pooled features as half-normal values.
Weights use N(0, 0.05^2) (single FC layer) or He normal N(0, 2/fan_in)
(Section 4: the He initialisation), masked by a Bernoulli(density) draw.
"""

from __future__ import annotations

import numpy as np


def rng_for(seed: int) -> np.random.Generator:
    return np.random.default_rng(seed)


def bernoulli_mask(rng, m: int, k: int, density: float) -> np.ndarray:
    return rng.random((m, k)) < density


def zipf_row_lengths(m: int, k: int, nnz: int, s: float = 1.2) -> np.ndarray:
    """Row lengths proportional to rank^-s, summing to ``nnz``, each <= k.

    Rank r (1-based) gets weight r^-s. Rows that would exceed k are clipped
    to k and the excess is shared among the other rows in proportion to
    their weights, repeatedly; the rounding remainder goes one entry at a
    time to the highest-ranked rows that still have room.
    """
    nnz = min(nnz, m * k)
    weights = np.arange(1, m + 1, dtype=np.float64) ** (-s)
    lengths = np.zeros(m, dtype=np.int64)
    free = np.ones(m, dtype=bool)
    remaining = nnz
    while remaining > 0 and free.any():
        share = remaining * weights[free] / weights[free].sum()
        cap = k - lengths[free]
        take = np.minimum(np.floor(share).astype(np.int64), cap)
        lengths[free] += take
        remaining -= int(take.sum())
        newly_full = lengths >= k
        if not (free & newly_full).any():
            break
        free &= ~newly_full
    order = np.arange(m)
    while remaining > 0:
        for r in order:
            if remaining == 0:
                break
            if lengths[r] < k:
                lengths[r] += 1
                remaining -= 1
    return lengths


def zipf_mask(rng, m: int, k: int, density: float, s: float = 1.2) -> np.ndarray:
    """Power-law row lengths over a random row permutation; columns of each
    row drawn uniformly without replacement."""
    lengths = zipf_row_lengths(m, k, int(round(density * m * k)), s)
    perm = rng.permutation(m)
    mask = np.zeros((m, k), dtype=bool)
    for rank, row in enumerate(perm):
        n = int(lengths[rank])
        if n:
            mask[row, rng.choice(k, size=n, replace=False)] = True
    return mask


def he_normal(rng, m: int, k: int) -> np.ndarray:
    return rng.normal(0.0, np.sqrt(2.0 / k), size=(m, k))


def masked_weights(rng, m: int, k: int, density: float, std: float | None = None,
                   zipf: bool = False) -> np.ndarray:
    """Dense float32 M x K matrix, zero off a random mask."""
    mask = zipf_mask(rng, m, k, density) if zipf else bernoulli_mask(rng, m, k, density)
    vals = rng.normal(0.0, std, size=(m, k)) if std is not None else he_normal(rng, m, k)
    return np.where(mask, vals, 0.0).astype(np.float32)


def uniform01(rng, *shape) -> np.ndarray:
    return rng.random(shape).astype(np.float32)


def std_normal(rng, *shape) -> np.ndarray:
    return rng.standard_normal(shape).astype(np.float32)


def half_normal(rng, *shape) -> np.ndarray:
    return np.abs(rng.standard_normal(shape)).astype(np.float32)


def labels(rng, n: int, classes: int) -> np.ndarray:
    return rng.integers(0, classes, size=n).astype(np.int32)


# ---------------------------------------------------------------------------
# The five workloads. Each returns plain numpy arrays and scalars.
# ---------------------------------------------------------------------------

ETA = 0.01
LAMBDA = 1e-4


def single_fc(seed: int = 0, m: int = 300, k: int = 784, n: int = 64, density: float = 0.10):
    """FC 784->300 at 10%, W ~ N(0, 0.05^2), X ~ U[0,1] (K x N), dY ~ N(0,1)."""
    rng = rng_for(seed)
    w = masked_weights(rng, m, k, density, std=0.05)
    x = uniform01(rng, k, n)
    dy = std_normal(rng, m, n)
    return {"W": w, "X": x, "dY": dy, "eta": ETA, "lambda": LAMBDA}


def mlp(seed: int = 0, batch: int = 256, sizes=(784, 300, 100, 10),
        densities=(0.08, 0.09, 0.26)):
    """MLP 784-300-100-10, He init, inputs U[0,1] (784 x B), labels 0..9."""
    rng = rng_for(seed)
    ws, bs = [], []
    for (k, m), d in zip(zip(sizes[:-1], sizes[1:]), densities):
        ws.append(masked_weights(rng, m, k, d))
        bs.append(np.zeros(m, dtype=np.float32))
    x = uniform01(rng, sizes[0], batch)
    y = labels(rng, batch, sizes[-1])
    return {"W": ws, "b": bs, "X": x, "labels": y, "eta": ETA, "lambda": LAMBDA}


def lenet(seed: int = 0, batch: int = 128, conv_density: float = 0.30, fc_density: float = 0.08):
    """LeNet-5 style: conv 20x(1*5*5), pool, conv 50x(20*5*5), pool,
    fc 800->500, fc 500->10. Inputs U[0,1] as (1, B, 28, 28)."""
    rng = rng_for(seed)
    shapes = [(20, 25), (50, 500), (500, 800), (10, 500)]
    dens = [conv_density, conv_density, fc_density, fc_density]
    ws = [masked_weights(rng, m, k, d) for (m, k), d in zip(shapes, dens)]
    bs = [np.zeros(m, dtype=np.float32) for m, _ in shapes]
    x = uniform01(rng, 1, batch, 28, 28)
    y = labels(rng, batch, 10)
    return {"W": ws, "b": bs, "X": x, "labels": y, "eta": ETA, "lambda": LAMBDA}


def fc_head(seed: int = 0, batch: int = 256, sizes=(9216, 4096, 4096, 1000),
            densities=(0.05, 0.05, 0.15)):
    """AlexNet-sized classifier head on half-normal 9216-dim features."""
    rng = rng_for(seed)
    ws, bs = [], []
    for (k, m), d in zip(zip(sizes[:-1], sizes[1:]), densities):
        ws.append(masked_weights(rng, m, k, d))
        bs.append(np.zeros(m, dtype=np.float32))
    x = half_normal(rng, sizes[0], batch)
    y = labels(rng, batch, sizes[-1])
    return {"W": ws, "b": bs, "X": x, "labels": y, "eta": ETA, "lambda": LAMBDA}


def sweep_layer(seed: int = 0, density: float = 0.05, n: int = 256, zipf: bool = False,
                m: int = 4096, k: int = 4096):
    """One 4096 x 4096 layer for the density / row-length / batch sweep."""
    rng = rng_for(seed)
    w = masked_weights(rng, m, k, density, zipf=zipf)
    x = std_normal(rng, k, n)
    dy = std_normal(rng, m, n)
    g = std_normal(rng, m, k)
    return {"W": w, "X": x, "dY": dy, "G": g, "eta": ETA, "lambda": LAMBDA}
