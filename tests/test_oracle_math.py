"""Pins for the oracle's losses, gradients, Adam step, bf16 rounding and whole iterations.

Checks come from closed forms (the ln 2 loss of an undecided discriminator, Adam's first step),
central finite differences, and independent library routines (torch autograd, torch's BCE,
torch.optim.Adam and torch's bfloat16 conversion, all on the CPU).
"""

import math

import numpy as np
import pytest

from oracle import lipz_oracle as O

torch = pytest.importorskip("torch")

TINY = dict(z_dim=3, hidden=4, x_dim=5, batch=2)


def _tiny_state(seed=5, rows=1, cols=1, **kw):
    arch = O.Arch(**{**TINY, **kw})
    return O.create(rows, cols, arch, seed)


def test_bce_of_undecided_discriminator_is_ln2():
    """A discriminator whose last layer is zero outputs sigmoid(0) = 1/2 on every input:
    each BCE term is ln 2, so L_G = ln 2 and L_D = 2 ln 2 for every pair and every fitness."""
    arch = O.Arch(z_dim=8, hidden=16, x_dim=12, batch=10)
    s = O.create(2, 3, arch, 11)
    dl = O.d_layout(arch)
    for c in range(s.cells):
        P = O.unflatten(s.Dw[c], dl)
        P["W3"][:] = 0.0
        P["b3"][:] = 0.0
    pool = np.random.default_rng(0).uniform(-1, 1, size=(50, 12))
    ev = O.eval_neighborhoods(s, O.batches(s, pool))
    ln2 = math.log(2.0)
    assert np.all(np.abs(ev["LG"] - ln2) <= 2 * np.finfo(float).eps)
    assert np.all(np.abs(ev["LD"] - 2 * ln2) <= 4 * np.finfo(float).eps)
    assert np.allclose(ev["fG"], ln2, rtol=0, atol=1e-15)
    assert np.allclose(ev["fD"], 2 * ln2, rtol=0, atol=1e-15)


def test_pair_losses_match_torch_bce():
    rng = np.random.default_rng(3)
    lr_, lf = rng.normal(scale=4, size=7), rng.normal(scale=4, size=7)
    lg, ld = O.pair_losses(lr_, lf)
    F = torch.nn.functional.binary_cross_entropy_with_logits
    tr, tf = torch.tensor(lr_), torch.tensor(lf)
    ref_d = F(tr, torch.ones(7, dtype=torch.float64)) + F(tf, torch.zeros(7, dtype=torch.float64))
    ref_g = F(tf, torch.ones(7, dtype=torch.float64))
    assert ld == pytest.approx(float(ref_d), rel=1e-14)
    assert lg == pytest.approx(float(ref_g), rel=1e-14)
    # softplus never overflows and tends to x / 0 at the ends
    assert O.softplus(np.array([1000.0]))[0] == 1000.0
    assert O.softplus(np.array([-1000.0]))[0] == 0.0


def _losses_for(Gflat, Dflat, x, z, arch, detach_fake=None):
    gl, dl = O.g_layout(arch), O.d_layout(arch)
    F = O.g_forward(O.unflatten(Gflat, gl), z, arch)["F"] if detach_fake is None else detach_fake
    logit = O.d_forward(O.unflatten(Dflat, dl), np.vstack([x, F]), arch)["logit"]
    B = x.shape[0]
    return O.pair_losses(logit[:B], logit[B:])


def _tiny_pair(seed):
    arch = O.Arch(**TINY)
    rng = np.random.default_rng(seed)
    G = rng.normal(scale=0.8, size=O.n_params(O.g_layout(arch)))
    D = rng.normal(scale=0.8, size=O.n_params(O.d_layout(arch)))
    x = rng.uniform(-1, 1, size=(arch.batch, arch.x_dim))
    z = rng.normal(size=(arch.batch, arch.z_dim))
    return arch, G, D, x, z


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_gradients_match_central_finite_differences(seed):
    arch, G, D, x, z = _tiny_pair(seed)
    gG, gD, _ = O.pair_gradients(G, D, x, z, arch)
    h = 1e-6
    F = O.g_forward(O.unflatten(G, O.g_layout(arch)), z, arch)["F"]
    # discriminator: L_D with the fake batch held fixed
    for k in range(D.size):
        Dp, Dm = D.copy(), D.copy()
        Dp[k] += h
        Dm[k] -= h
        fd = (_losses_for(G, Dp, x, z, arch, F)[1] - _losses_for(G, Dm, x, z, arch, F)[1]) / (2 * h)
        assert abs(fd - gD[k]) <= 1e-6 * max(1.0, abs(fd)), (k, fd, gD[k])
    # generator: L_G through the discriminator
    for k in range(G.size):
        Gp, Gm = G.copy(), G.copy()
        Gp[k] += h
        Gm[k] -= h
        fd = (_losses_for(Gp, D, x, z, arch)[0] - _losses_for(Gm, D, x, z, arch)[0]) / (2 * h)
        assert abs(fd - gG[k]) <= 1e-6 * max(1.0, abs(fd)), (k, fd, gG[k])


def _torch_grads(G, D, x, z, arch):
    """The same pair through torch autograd in float64 (an independent implementation)."""
    t = lambda a: torch.tensor(a, dtype=torch.float64, requires_grad=True)
    gl, dl = O.g_layout(arch), O.d_layout(arch)
    Gp = {k: t(v.copy()) for k, v in O.unflatten(G, gl).items()}
    Dp = {k: t(v.copy()) for k, v in O.unflatten(D, dl).items()}
    lin = torch.nn.functional.linear
    zt = torch.tensor(z)
    h = torch.relu(lin(zt, Gp["W1"], Gp["b1"]))
    h = torch.relu(lin(h, Gp["W2"], Gp["b2"]))
    fake = torch.tanh(lin(h, Gp["W3"], Gp["b3"]))

    def disc(X):
        g = torch.nn.functional.leaky_relu(lin(X, Dp["W1"], Dp["b1"]), arch.leaky_slope)
        g = torch.nn.functional.leaky_relu(lin(g, Dp["W2"], Dp["b2"]), arch.leaky_slope)
        return lin(g, Dp["W3"], Dp["b3"])[:, 0]

    bce = torch.nn.functional.binary_cross_entropy_with_logits
    B = x.shape[0]
    one, zero = torch.ones(B, dtype=torch.float64), torch.zeros(B, dtype=torch.float64)
    ld = bce(disc(torch.tensor(x)), one) + bce(disc(fake.detach()), zero)
    gD = torch.autograd.grad(ld, [Dp[k] for k, _ in dl])
    lg = bce(disc(fake), one)
    gG = torch.autograd.grad(lg, [Gp[k] for k, _ in gl])
    return (np.concatenate([g.numpy().reshape(-1) for g in gG]),
            np.concatenate([g.numpy().reshape(-1) for g in gD]))


@pytest.mark.parametrize("seed", [0, 4])
def test_gradients_match_torch_autograd(seed):
    arch = O.Arch(z_dim=6, hidden=10, x_dim=9, batch=7)
    rng = np.random.default_rng(seed)
    G = rng.normal(scale=0.5, size=O.n_params(O.g_layout(arch)))
    D = rng.normal(scale=0.5, size=O.n_params(O.d_layout(arch)))
    x = rng.uniform(-1, 1, size=(7, 9))
    z = rng.normal(size=(7, 6))
    gG, gD, _ = O.pair_gradients(G, D, x, z, arch)
    tG, tD = _torch_grads(G, D, x, z, arch)
    assert np.allclose(gG, tG, rtol=1e-12, atol=1e-14)
    assert np.allclose(gD, tD, rtol=1e-12, atol=1e-14)


def test_bf16_mode_tracks_fp32_gradients():
    arch = O.Arch(z_dim=16, hidden=32, x_dim=24, batch=16)
    rng = np.random.default_rng(9)
    G = rng.normal(scale=0.3, size=O.n_params(O.g_layout(arch)))
    D = rng.normal(scale=0.3, size=O.n_params(O.d_layout(arch)))
    x = rng.uniform(-1, 1, size=(16, 24))
    z = rng.normal(size=(16, 16))
    g32 = O.pair_gradients(G, D, x, z, arch)
    b16 = O.pair_gradients(G, D, x, z, O.Arch(**{**arch.__dict__, "precision": "bf16"}))
    for a, b in ((g32[0], b16[0]), (g32[1], b16[1])):
        assert np.max(np.abs(a - b)) <= 0.05 * np.max(np.abs(a))


def test_round_bf16_matches_torch_and_ties_to_even():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.normal(scale=s, size=4000) for s in (1e-30, 1e-3, 1.0, 1e3, 1e30)])
    x = x.astype(np.float32)
    ref = torch.tensor(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(O.round_bf16(x.astype(np.float64)), ref)
    assert O.round_bf16(np.array([1.0 + 2.0 ** -8]))[0] == 1.0            # tie -> even
    assert O.round_bf16(np.array([1.0 + 3 * 2.0 ** -8]))[0] == 1.0 + 2.0 ** -6  # tie -> even
    assert O.round_bf16(np.array([1.0 + 3 * 2.0 ** -9]))[0] == 1.0 + 2.0 ** -7


def test_adam_first_step_closed_form_and_zero_gradient():
    arch = O.Arch(lr=2e-4, beta1=0.5, beta2=0.999, eps=1e-8)
    g = np.array([1e-3, -2.0, 0.0, 5e-9, -1e-12])
    w0 = np.array([0.1, -0.2, 0.3, 0.0, 1.0])
    w1, m1, v1, t1 = O.adam_step(w0, np.zeros(5), np.zeros(5), 0, g, arch.lr, arch)
    # after one step m_hat = g and v_hat = g^2, so the move is lr * g / (|g| + eps)
    assert np.allclose(w1, w0 - arch.lr * g / (np.abs(g) + arch.eps), rtol=1e-13, atol=0)
    assert w1[2] == w0[2] and t1 == 1


def test_adam_matches_torch_optim_over_steps():
    arch = O.Arch(lr=1e-3, beta1=0.5, beta2=0.999, eps=1e-8)
    rng = np.random.default_rng(1)
    w = rng.normal(size=11)
    p = torch.tensor(w.copy(), requires_grad=True)
    opt = torch.optim.Adam([p], lr=arch.lr, betas=(arch.beta1, arch.beta2), eps=arch.eps)
    m, v, step = np.zeros(11), np.zeros(11), 0
    for _ in range(5):
        g = rng.normal(size=11)
        p.grad = torch.tensor(g.copy())
        opt.step()
        w, m, v, step = O.adam_step(w, m, v, step, g, arch.lr, arch)
    assert np.allclose(w, p.detach().numpy(), rtol=1e-12, atol=1e-15)


def test_one_by_one_grid_ties_keep_the_centre():
    s = _tiny_state(rows=1, cols=1)
    pool = np.random.default_rng(0).uniform(-1, 1, size=(20, 5))
    data = O.batches(s, pool)
    ev = O.eval_neighborhoods(s, data)
    # all five slots hold the same individuals, so every pair scores the same
    assert np.all(ev["LG"] == ev["LG"][0, 0, 0]) and np.all(ev["LD"] == ev["LD"][0, 0, 0])
    sel = O.select_replace(s, ev)
    assert sel["sel_g"][0] == 0 and sel["sel_d"][0] == 0


def test_zero_learning_rate_moves_nothing_but_counts_steps():
    s = _tiny_state(rows=2, cols=2, lr=0.0)
    pool = np.random.default_rng(0).uniform(-1, 1, size=(20, 5))
    s1 = O.iterate(s, pool, 1)
    nbr = O.neighbors(2, 2)
    ev = O.eval_neighborhoods(s, O.batches(s, pool))
    sel = O.select_replace(s, ev)
    for c in range(4):
        assert np.array_equal(s1.Gw[c], s.Gw[nbr[c][sel["sel_g"][c]]])
        assert np.array_equal(s1.Dw[c], s.Dw[nbr[c][sel["sel_d"][c]]])
    assert np.all(s1.Gstep == 1) and np.all(s1.Dstep == 1) and s1.t == 1
    assert np.any(s1.Gm != 0.0)


def test_iteration_is_deterministic_and_state_bytes_round_trip():
    s = _tiny_state(rows=2, cols=3, seed=99)
    pool = np.random.default_rng(1).uniform(-1, 1, size=(30, 5))
    a = O.iterate(s, pool, 2)
    b = O.iterate(s, pool, 2)
    for f in ("Gw", "Gm", "Gv", "Dw", "Dm", "Dv", "Gstep", "Dstep", "Glr", "Dlr"):
        assert np.array_equal(getattr(a, f), getattr(b, f))
    buf = O.state_to_bytes(a)
    c = O.state_from_bytes(buf, a.arch)
    assert c.t == 2 and c.seed == 99 and c.rows == 2 and c.cols == 3
    for f in ("Gw", "Dw", "Gm", "Dv"):
        assert np.array_equal(getattr(c, f), getattr(a, f).astype(np.float32))


def test_training_lowers_the_pair_losses():
    """One Adam step along the gradient, at a learning rate small enough for the linear
    approximation, lowers L_D for the discriminator and L_G for the generator."""
    arch, G, D, x, z = _tiny_pair(7)
    gG, gD, losses = O.pair_gradients(G, D, x, z, arch)
    lr = 1e-4
    G1 = O.adam_step(G, 0 * G, 0 * G, 0, gG, lr, arch)[0]
    D1 = O.adam_step(D, 0 * D, 0 * D, 0, gD, lr, arch)[0]
    F = O.g_forward(O.unflatten(G, O.g_layout(arch)), z, arch)["F"]
    assert _losses_for(G, D1, x, z, arch, F)[1] < losses["LD"]
    assert _losses_for(G1, D, x, z, arch)[0] < losses["LG"]


def _torch_adam_step(w, m, v, step, g, lr, arch):
    """One step of torch.optim.Adam resumed from (m, v, step) (an independent implementation)."""
    p = torch.tensor(np.array(w, np.float64), requires_grad=True)
    opt = torch.optim.Adam([p], lr=float(lr), betas=(arch.beta1, arch.beta2), eps=arch.eps)
    opt.state[p] = {"step": torch.tensor(float(step)),
                    "exp_avg": torch.tensor(np.array(m, np.float64)),
                    "exp_avg_sq": torch.tensor(np.array(v, np.float64))}
    p.grad = torch.tensor(np.array(g, np.float64))
    opt.step()
    st = opt.state[p]
    return (p.detach().numpy(), st["exp_avg"].numpy(), st["exp_avg_sq"].numpy(),
            int(st["step"].item()))


@pytest.mark.parametrize("mutation", [False, True])
def test_later_minibatch_steps_continue_adam_on_fresh_batches(mutation):
    """K = 3 minibatch steps per iteration equal the K = 1 iteration followed, in every cell, by
    two steps of torch.optim.Adam (moments, step count and the cell's lr carried over) on torch
    autograd gradients of the cell's own pair, on the minibatch of streams BATCH + 256 k and
    NOISE + 256 k; selection and the lr mutation happen once."""
    kw = dict(lr=1e-3, lr_mutation=mutation, lr_mut_std=1e-4, lr_mut_prob=0.5)
    s = _tiny_state(rows=2, cols=3, seed=3, **kw)
    s3 = _tiny_state(rows=2, cols=3, seed=3, train_steps=3, **kw)
    pool = np.random.default_rng(2).uniform(-1, 1, size=(40, 5))
    one = O.iterate(s, pool, 1)
    three = O.iterate(s3, pool, 1)
    a = s.arch
    for c in range(s.cells):
        G = (one.Gw[c], one.Gm[c], one.Gv[c], int(one.Gstep[c]))
        D = (one.Dw[c], one.Dm[c], one.Dv[c], int(one.Dstep[c]))
        for k in (1, 2):
            idx = O.mulhi(O.draw_words(3, 3 + 256 * k, 0, c, a.batch), pool.shape[0])
            x = pool[idx.astype(np.int64)]
            z = O.draw_normals(3, 4 + 256 * k, 0, c, a.batch * a.z_dim).reshape(a.batch, -1)
            gG, gD = _torch_grads(G[0], D[0], x, z, a)
            G = _torch_adam_step(*G, gG, one.Glr[c], a)
            D = _torch_adam_step(*D, gD, one.Dlr[c], a)
        for got, ref in ((three.Gw[c], G[0]), (three.Gm[c], G[1]), (three.Gv[c], G[2]),
                         (three.Dw[c], D[0]), (three.Dm[c], D[1]), (three.Dv[c], D[2])):
            assert np.allclose(got, ref, rtol=1e-11, atol=1e-15)
        assert three.Gstep[c] == G[3] == 3 and three.Dstep[c] == D[3] == 3
        assert three.Glr[c] == one.Glr[c] and three.Dlr[c] == one.Dlr[c]
    assert three.t == 1


def test_later_minibatch_steps_draw_fresh_batches():
    """Step k's minibatch comes from its own streams: no two steps of a cell share their noise,
    and step 0 is the evaluation minibatch."""
    a = O.Arch(**TINY)
    pool = np.random.default_rng(0).uniform(-1, 1, size=(1000, 5))
    zs = [O.draw_batch(7, 4, 1, pool, a, k)[1] for k in range(3)]
    assert np.array_equal(zs[0], O.draw_batch(7, 4, 1, pool, a)[1])
    assert not np.array_equal(zs[0], zs[1]) and not np.array_equal(zs[1], zs[2])


@pytest.mark.parametrize("layer,row", [("G1", 3), ("G2", 0), ("D1", 2), ("D1", 9), ("D2", 5),
                                       ("D2", 11)])
def test_flipped_derivative_branch_equals_the_other_side_of_the_kink(layer, row):
    """pair_gradients(flip=...) takes the other branch of a ReLU / LeakyReLU derivative at the
    named elements (for comparisons with implementations whose pre-activation lands on the other
    side of 0). Pinned against torch autograd: the bias of the element's unit is set so that
    the element's pre-activation is +1e-9; flipping it must give the gradients that autograd
    computes with the pre-activation at -1e-9 (bias lowered by 2e-9), where the derivative is
    the other branch and every other quantity moves by O(1e-9). D rows 7.. are the fake batch,
    whose derivative serves both losses."""
    arch = O.Arch(z_dim=6, hidden=10, x_dim=9, batch=7)
    rng = np.random.default_rng(11)
    gl, dl = O.g_layout(arch), O.d_layout(arch)
    G = rng.normal(scale=0.5, size=O.n_params(gl))
    D = rng.normal(scale=0.5, size=O.n_params(dl))
    x = rng.uniform(-1, 1, size=(7, 9))
    z = rng.normal(size=(7, 6))
    net, lay = (G, gl) if layer[0] == "G" else (D, dl)
    bname = "b" + layer[1]
    off = 0
    for name, shape in lay:
        if name == bname:
            break
        off += int(np.prod(shape))
    pre = O.pair_gradients(G, D, x, z, arch)[2]["pre"][layer]
    unit = int(np.argmax(np.abs(pre[row])))    # a unit that carries a real delta
    eps = 1e-9
    net[off + unit] += eps - pre[row, unit]    # now pre[row, unit] = +eps
    info = O.pair_gradients(G, D, x, z, arch)[2]
    assert abs(info["pre"][layer][row, unit] - eps) < 1e-12
    others = np.delete(info["pre"][layer][:, unit], row)
    assert np.min(np.abs(others)) > 1e-6       # no other row crosses 0 with the shift
    flip = {layer: np.zeros_like(info["pre"][layer], dtype=bool)}
    flip[layer][row, unit] = True
    fG, fD, _ = O.pair_gradients(G, D, x, z, arch, flip=flip)
    nG, nD, _ = O.pair_gradients(G, D, x, z, arch)
    net[off + unit] -= 2 * eps                 # pre[row, unit] = -eps
    tG, tD = _torch_grads(G, D, x, z, arch)
    assert np.allclose(fG, tG, rtol=1e-6, atol=1e-8) and np.allclose(fD, tD, rtol=1e-6, atol=1e-8)
    # and the flip mattered: the unflipped gradients are the other side's
    assert np.max(np.abs(np.concatenate([nG - tG, nD - tD]))) > 1e-4
