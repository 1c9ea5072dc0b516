"""The generator output's tanh in the tensor-core forward is computed from its definition,
tanh(x) = 1 - 2 / (1 + e^(2x)) for |x| >= 1/4, and from its Taylor series through x^9 below. This checks that formula, evaluated in float32 as the kernel does (with an exact 2^x in
place of the hardware's, whose relative error is about 2^-22), against float64 tanh: relative
error below 2e-6 everywhere, so that its bf16 rounding almost never differs from that of an
exact tanh."""

import numpy as np


def tanh_fast_f32(x):
    x = np.asarray(x, np.float32)
    ax = np.minimum(np.abs(x), np.float32(16))
    e = np.exp2(np.float32(2.8853900817779268) * ax).astype(np.float32)
    t = np.float32(1) - np.float32(2) / (np.float32(1) + e)
    x2 = ax * ax
    q = x2 * np.float32(0.021869488536155203) + np.float32(-0.053968253968253971)
    q = x2 * q + np.float32(0.13333333333333333)
    q = x2 * q + np.float32(-0.33333333333333333)
    s = ax * (x2 * q + np.float32(1))
    return np.copysign(np.where(ax < np.float32(0.25), s, t), x).astype(np.float32)


def test_tanh_formula_relative_error():
    x = np.concatenate([np.linspace(-20, 20, 400001), np.geomspace(1e-30, 20, 200001),
                        -np.geomspace(1e-30, 20, 200001), [0.25, -0.25, 0.0]])
    x = x.astype(np.float32)
    got = tanh_fast_f32(x).astype(np.float64)
    ref = np.tanh(x.astype(np.float64))
    nz = ref != 0
    rel = np.abs(got[nz] - ref[nz]) / np.abs(ref[nz])
    assert rel.max() < 2e-6, (rel.max(), x[nz][np.argmax(rel)])
    assert np.all(got[~nz] == 0)
    assert np.all(np.abs(got) <= 1)
