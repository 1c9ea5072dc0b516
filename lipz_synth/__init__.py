"""Seeded synthetic inputs shared by the CUDA path's tests/bench and the CPU oracle.

This module holds no arithmetic of the coevolutionary method itself: it only makes the
"real data" pool that both sides read. The paper trains on MNIST (784-dim images scaled to
[-1, 1]); that dataset is not available, so a seeded mixture of Gaussian blobs with the same
shape and value range stands in for it.

Recipe (one pool of ``n`` rows, ``dim`` columns):
  * ``k`` blob centres mu_k drawn i.i.d. U(-1, 1)^dim,
  * each row picks a blob uniformly and is ``clip(mu_k + sigma * N(0, I), -1, 1)``.
Generated with numpy's PCG64 stream from ``seed``; stored as float32.
"""

import numpy as np

__all__ = ["blob_pool", "host_batch"]


def blob_pool(seed: int, n: int = 60000, dim: int = 784, k: int = 10, sigma: float = 0.3,
              chunk: int = 8192) -> np.ndarray:
    """Return a float32 [n, dim] pool of blob-mixture samples in [-1, 1]."""
    if n < 1 or dim < 1 or k < 1:
        raise ValueError("blob_pool: n, dim and k must be >= 1")
    rng = np.random.Generator(np.random.PCG64(seed))
    centres = rng.uniform(-1.0, 1.0, size=(k, dim)).astype(np.float32)
    labels = rng.integers(0, k, size=n)
    out = np.empty((n, dim), dtype=np.float32)
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        noise = rng.standard_normal(size=(e - s, dim), dtype=np.float32)
        np.clip(centres[labels[s:e]] + np.float32(sigma) * noise, -1.0, 1.0, out=out[s:e])
    return out


def host_batch(seed: int, cells: int, batch: int, dim: int = 784, k: int = 10,
               sigma: float = 0.3) -> np.ndarray:
    """A float32 [cells, batch, dim] block of blob samples: one caller-supplied minibatch
    per cell, the shape a host-side data loader hands to the engine each iteration."""
    return blob_pool(seed, n=cells * batch, dim=dim, k=k, sigma=sigma).reshape(cells, batch, dim)
