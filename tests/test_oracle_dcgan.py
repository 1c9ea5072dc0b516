"""Pins for the oracle's DCGAN networks: convolutions, transposed convolutions and training-mode
batch normalisation against torch.nn.functional (an independent implementation, float64 on the
CPU), a whole generator-discriminator pair's gradients against torch autograd and central
finite differences, the ln 2 loss of an undecided discriminator, and the initialisation's
moments."""

import math

import numpy as np
import pytest

from oracle import dcgan as C
from oracle import lipz_oracle as O

torch = pytest.importorskip("torch")
F = torch.nn.functional

TINY = dict(kind="dcgan", z_dim=3, ngf=2, ndf=2, x_dim=12288, batch=3)


def _t(a, grad=False):
    return torch.tensor(np.asarray(a, np.float64), requires_grad=grad)


@pytest.mark.parametrize("s,p,H", [(2, 1, 8), (1, 0, 4), (2, 1, 5)])
def test_conv_and_transposed_conv_match_torch(s, p, H):
    rng = np.random.default_rng(H + s)
    x = rng.normal(size=(2, 3, H, H))
    w = rng.normal(size=(4, 3, 4, 4))
    assert np.allclose(C.conv2d(x, w, s, p), F.conv2d(_t(x), _t(w), stride=s, padding=p).numpy(),
                       rtol=1e-12, atol=1e-12)
    wt = rng.normal(size=(3, 4, 4, 4))
    assert np.allclose(C.conv_transpose2d(x, wt, s, p),
                       F.conv_transpose2d(_t(x), _t(wt), stride=s, padding=p).numpy(),
                       rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("s,p", [(2, 1), (1, 0)])
def test_conv_backward_matches_autograd(s, p):
    rng = np.random.default_rng(7)
    x, w = rng.normal(size=(2, 3, 8, 8)), rng.normal(size=(5, 3, 4, 4))
    xt, wtt = _t(x, True), _t(w, True)
    y = F.conv2d(xt, wtt, stride=s, padding=p)
    dy = rng.normal(size=tuple(y.shape))
    y.backward(_t(dy))
    dx, dw = C.conv2d_backward(x, w, s, p, dy)
    assert np.allclose(dx, xt.grad.numpy(), rtol=1e-11, atol=1e-12)
    assert np.allclose(dw, wtt.grad.numpy(), rtol=1e-11, atol=1e-12)
    wt = rng.normal(size=(3, 5, 4, 4))
    xt, wtt = _t(x, True), _t(wt, True)
    y = F.conv_transpose2d(xt, wtt, stride=s, padding=p)
    dy = rng.normal(size=tuple(y.shape))
    y.backward(_t(dy))
    dx, dw = C.conv_transpose2d_backward(x, wt, s, p, dy)
    assert np.allclose(dx, xt.grad.numpy(), rtol=1e-11, atol=1e-12)
    assert np.allclose(dw, wtt.grad.numpy(), rtol=1e-11, atol=1e-12)


def test_batchnorm_training_mode_matches_torch():
    rng = np.random.default_rng(3)
    x = rng.normal(loc=0.5, scale=2.0, size=(4, 3, 5, 5))
    g, b = rng.normal(size=3), rng.normal(size=3)
    xt, gt, bt = _t(x, True), _t(g, True), _t(b, True)
    y = F.batch_norm(xt, None, None, gt, bt, training=True, eps=C.BN_EPS)
    ours, cache = C.batchnorm(x, g, b)
    assert np.allclose(ours, y.detach().numpy(), rtol=1e-12, atol=1e-12)
    dy = rng.normal(size=x.shape)
    y.backward(_t(dy))
    dx, dg, db = C.batchnorm_backward(dy, g, cache)
    assert np.allclose(dx, xt.grad.numpy(), rtol=1e-10, atol=1e-12)
    assert np.allclose(dg, gt.grad.numpy(), rtol=1e-12) and np.allclose(db, bt.grad.numpy())


def _torch_pair(G, D, x, z, arch):
    """The same pair in torch autograd (float64)."""
    gl, dl = O.g_layout(arch), O.d_layout(arch)
    Gp = {k: _t(v.copy(), True) for k, v in O.unflatten(G, gl).items()}
    Dp = {k: _t(v.copy(), True) for k, v in O.unflatten(D, dl).items()}
    h = _t(z).reshape(z.shape[0], -1, 1, 1)
    for i in range(4):
        s, p = (1, 0) if i == 0 else (2, 1)
        h = F.conv_transpose2d(h, Gp["W%d" % (i + 1)], stride=s, padding=p)
        h = torch.relu(F.batch_norm(h, None, None, Gp["gamma%d" % (i + 1)],
                                    Gp["beta%d" % (i + 1)], training=True, eps=C.BN_EPS))
    fake = torch.tanh(F.conv_transpose2d(h, Gp["W5"], stride=2, padding=1))

    def disc(X):
        a = X
        for i in range(4):
            a = F.leaky_relu(F.conv2d(a, Dp["W%d" % (i + 1)], stride=2, padding=1),
                             arch.leaky_slope)
        return F.conv2d(a, Dp["W5"]).reshape(-1)

    bce = F.binary_cross_entropy_with_logits
    B = x.shape[0]
    real = _t(x).reshape(B, 3, 64, 64)
    one, zero = torch.ones(B, dtype=torch.float64), torch.zeros(B, dtype=torch.float64)
    ld = bce(disc(real), one) + bce(disc(fake.detach()), zero)
    gD = torch.autograd.grad(ld, [Dp[k] for k, _ in dl])
    lg = bce(disc(fake), one)
    gG = torch.autograd.grad(lg, [Gp[k] for k, _ in gl])
    return (np.concatenate([g.numpy().reshape(-1) for g in gG]),
            np.concatenate([g.numpy().reshape(-1) for g in gD]), float(lg.detach()),
            float(ld.detach()))


def _tiny_pair(seed):
    arch = O.Arch(**TINY)
    s = O.create(1, 2, arch, seed)
    rng = np.random.default_rng(seed)
    # larger weights than the initialisation so that every layer matters
    G = s.Gw[0] * 10.0
    D = s.Dw[1] * 10.0
    x = rng.uniform(-1, 1, size=(arch.batch, 12288))
    z = rng.normal(size=(arch.batch, arch.z_dim))
    return arch, G, D, x, z


@pytest.mark.parametrize("seed", [0, 5])
def test_pair_gradients_match_torch_autograd(seed):
    arch, G, D, x, z = _tiny_pair(seed)
    gG, gD, info = O.pair_gradients(G, D, x, z, arch)
    tG, tD, lg, ld = _torch_pair(G, D, x, z, arch)
    assert info["LG"] == pytest.approx(lg, rel=1e-12) and info["LD"] == pytest.approx(ld, rel=1e-12)
    assert np.allclose(gG, tG, rtol=1e-9, atol=1e-12 * np.abs(tG).max())
    assert np.allclose(gD, tD, rtol=1e-9, atol=1e-12 * np.abs(tD).max())


def test_pair_gradients_match_finite_differences():
    arch, G, D, x, z = _tiny_pair(3)
    gG, gD, _ = O.pair_gradients(G, D, x, z, arch)
    rng = np.random.default_rng(1)

    def losses(Gv, Dv):
        fg = O.g_forward(O.unflatten(Gv, O.g_layout(arch)), z, arch)
        lg_ = O.d_forward(O.unflatten(Dv, O.d_layout(arch)), np.vstack([x, fg["F"]]), arch)["logit"]
        return O.pair_losses(lg_[:arch.batch], lg_[arch.batch:])

    h = 1e-6
    for k in rng.choice(len(G), 8, replace=False):
        e = np.zeros_like(G)
        e[k] = h
        num = (losses(G + e, D)[0] - losses(G - e, D)[0]) / (2 * h)
        assert num == pytest.approx(gG[k], rel=1e-5, abs=1e-9)
    for k in rng.choice(len(D), 8, replace=False):
        e = np.zeros_like(D)
        e[k] = h
        # L_D with the fakes held fixed: the generator does not move when D does
        num = (losses(G, D + e)[1] - losses(G, D - e)[1]) / (2 * h)
        assert num == pytest.approx(gD[k], rel=1e-5, abs=1e-9)


def test_undecided_discriminator_gives_ln2():
    arch, G, D, x, z = _tiny_pair(2)
    Dp = O.unflatten(D.copy(), O.d_layout(arch))
    Dp["W5"][:] = 0.0
    D0 = np.concatenate([Dp[k].reshape(-1) for k, _ in O.d_layout(arch)])
    _, _, info = O.pair_gradients(G, D0, x, z, arch)
    assert info["LG"] == pytest.approx(math.log(2), abs=1e-15)
    assert info["LD"] == pytest.approx(2 * math.log(2), abs=1e-15)


def test_initialisation_moments_and_output_range():
    arch = O.Arch(kind="dcgan", z_dim=100, ngf=16, ndf=16, x_dim=12288, batch=4)
    s = O.create(1, 1, arch, 1811)
    Gp = O.unflatten(s.Gw[0], O.g_layout(arch))
    Dp = O.unflatten(s.Dw[0], O.d_layout(arch))
    w = np.concatenate([Gp["W2"].ravel(), Dp["W4"].ravel()])
    assert abs(w.mean()) < 5e-4 and abs(w.std() - 0.02) < 5e-4
    assert abs(Gp["gamma1"].mean() - 1.0) < 0.01 and np.all(Gp["beta1"] == 0.0)
    assert np.array_equal(s.Gw[0], s.Gw[0].astype(np.float32))
    z = np.random.default_rng(0).normal(size=(4, 100))
    F_ = O.g_forward(Gp, z, arch)["F"]
    assert F_.shape == (4, 12288) and np.all(np.abs(F_) <= 1.0)
    # batch normalisation in training mode: each generator layer's output has zero batch mean
    h = O.g_forward(Gp, z, arch)["cache"][1][2]
    assert np.allclose(h.mean(axis=(0, 2, 3)), Gp["beta2"], atol=1e-12)


def test_float32_accumulation_variant_is_the_same_arithmetic():
    """oracle.dcgan.ACC = float32 sums every convolution and batch-norm statistic in float32
    (tests use the spread between it and the float64 oracle to set their tolerances). On a
    small network it must agree with the float64 oracle to float32 rounding, and differ from it
    (the switch takes effect)."""
    from oracle import dcgan as DC
    a = O.Arch(kind="dcgan", precision="fp32", batch=3, z_dim=8, x_dim=12288, ngf=4, ndf=4)
    s = O.create(1, 1, a, 3)
    rng = np.random.default_rng(0)
    x = rng.uniform(-1, 1, size=(3, 12288))
    z = rng.normal(size=(3, 8))
    ref = O.pair_gradients(s.Gw[0], s.Dw[0], x, z, a)
    try:
        DC.ACC = np.float32
        got = O.pair_gradients(s.Gw[0], s.Dw[0], x, z, a)
    finally:
        DC.ACC = np.float64
    for r, g in zip(ref[:2], got[:2]):
        d = np.max(np.abs(g - r)) / np.max(np.abs(r))
        assert 0 < d < 1e-4, d
