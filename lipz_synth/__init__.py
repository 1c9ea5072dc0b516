"""Seeded synthetic inputs shared by the CUDA path's tests/bench and the CPU oracle.

This module holds no arithmetic of the coevolutionary method itself: it only makes the
"real data" pool that both sides read. The paper trains on MNIST (784-dim images scaled to
[-1, 1]); that dataset is not available, so a seeded mixture of Gaussian blobs with the same
shape and value range stands in for it.

The DCGAN setting (CelebA, 3 x 64 x 64 colour images in [-1, 1]) gets ``field_pool``: each
sample is, per channel, white noise smoothed by a periodic Gaussian filter (sigma 4 pixels,
applied in the Fourier domain) and scaled by its largest magnitude into [-1, 1]; rows are the
images flattened channel-major (C, H, W).

Blob recipe (one pool of ``n`` rows, ``dim`` columns):
  * ``k`` blob centres mu_k drawn i.i.d. U(-1, 1)^dim,
  * each row picks a blob uniformly and is ``clip(mu_k + sigma * N(0, I), -1, 1)``.
Generated with numpy's PCG64 stream from ``seed``; stored as float32.
"""

import numpy as np

__all__ = ["blob_pool", "host_batch", "field_pool"]


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


def field_pool(seed: int, n: int = 10000, size: int = 64, channels: int = 3,
               sigma: float = 4.0, chunk: int = 512) -> np.ndarray:
    """Return a float32 [n, channels * size * size] pool of smooth Gaussian random fields."""
    if n < 1 or size < 2 or channels < 1:
        raise ValueError("field_pool: n, size and channels must be positive")
    rng = np.random.Generator(np.random.PCG64(seed))
    f = np.fft.fftfreq(size)
    filt = np.exp(-2.0 * (np.pi * sigma) ** 2 * (f[:, None] ** 2 + f[None, :] ** 2))
    out = np.empty((n, channels * size * size), dtype=np.float32)
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        w = rng.standard_normal(size=(e - s, channels, size, size))
        sm = np.real(np.fft.ifft2(np.fft.fft2(w) * filt))
        sm /= np.max(np.abs(sm), axis=(2, 3), keepdims=True)
        out[s:e] = sm.reshape(e - s, -1).astype(np.float32)
    return out
