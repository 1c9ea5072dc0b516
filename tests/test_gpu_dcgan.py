"""GPU parity of the DCGAN networks (Table 1, CelebA column) against the oracle: the
initialisation, the evaluation of every (cell, slot) pair and one training step of every
cell's selected pair, at small widths in fp32 and bf16 (1e-4 / 2e-2 max-norm relative), and
sampled outputs of the 3x3, width-64, B = 128 configuration."""

import numpy as np
import pytest

from oracle import lipz_oracle as O

from helpers import max_rel, oracle_arch, per_tensor

pytestmark = pytest.mark.gpu

TOL = {0: 1e-4, 1: 2e-2}


@pytest.fixture(scope="module")
def L():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1811_12843_gb300 import _build
    _build.build()
    import paper_1811_12843_gb300 as lib
    return lib


def _field_pool(seed, n):
    import lipz_synth
    return lipz_synth.field_pool(seed, n=n)


def _grid(L, rows, cols, seed, pool, **kw):
    kw = {**dict(kind=1, x_dim=12288, z_dim=8, ngf=4, ndf=4, batch=4), **kw}
    g = L.Grid(rows, cols, seed=seed, **kw)
    g.set_data(pool)
    return g


def _state(g):
    return O.state_from_bytes(g.export_state(), oracle_arch(g.arch))


def test_dcgan_initialisation_matches_the_oracle(L):
    pool = _field_pool(1, 20)
    g = _grid(L, 2, 2, 7, pool, z_dim=100, ngf=8, ndf=8)
    s = _state(g)
    ref = O.create(2, 2, oracle_arch(g.arch), 7)
    for got, want in ((s.Gw, ref.Gw), (s.Dw, ref.Dw)):
        assert np.max(np.abs(got - want)) <= 1e-6 * np.max(np.abs(want))
    lay = O.unflatten(s.Gw[0], O.g_layout(ref.arch))
    assert np.all(lay["beta2"] == 0.0) and abs(lay["gamma1"].mean() - 1.0) < 0.02


@pytest.mark.parametrize("precision,rows,cols,batch,width", [
    ("fp32", 1, 2, 4, 4),
    ("bf16", 2, 2, 4, 4),
    ("bf16", 1, 1, 8, 8),
    ("fp32", 2, 1, 3, 8),   # odd batch
])
def test_dcgan_eval_parity(L, precision, rows, cols, batch, width):
    pool = _field_pool(2, 40)
    g = _grid(L, rows, cols, 3, pool, precision=precision, batch=batch, ngf=width, ndf=width)
    s = _state(g)
    ref = O.eval_neighborhoods(s, O.batches(s, pool))
    ev = g.eval(pairs=True)
    tol = TOL[g.arch.precision]
    assert max_rel(g.logits(), ref["logits"]) < tol
    for k in ("LG", "LD", "fG", "fD"):
        assert max_rel(ev[k], ref[k]) < tol, k


@pytest.mark.parametrize("rows,cols,batch,ngf", [(1, 1, 4, 8), (1, 2, 3, 8), (1, 1, 4, 64),
                                                 (2, 1, 5, 64)])
def test_dcgan_tensor_core_eval(L, rows, cols, batch, ngf):
    """bf16 with widths that are multiples of 64 runs the evaluation on the tensor-core
    implicit-GEMM kernel (the discriminator's convolutions; with ngf = 64 also the generator's
    transposed convolutions by output parity class and channel-last batch norm): every logit
    and loss against the oracle."""
    pool = _field_pool(5, 30)
    g = _grid(L, rows, cols, 9, pool, precision="bf16", batch=batch, ngf=ngf, ndf=64)
    s = _state(g)
    ref = O.eval_neighborhoods(s, O.batches(s, pool))
    ev = g.eval(pairs=True)
    assert max_rel(g.logits(), ref["logits"]) < 2e-2
    for k in ("LG", "LD", "fG", "fD"):
        assert max_rel(ev[k], ref[k]) < 2e-2, k


@pytest.mark.parametrize("precision,width,rows,cols,batch", [("fp32", 4, 2, 2, 4),
                                                            ("bf16", 4, 2, 2, 4),
                                                            ("bf16", 64, 1, 2, 16),
                                                            ("bf16", (128, 64), 1, 1, 16)])
def test_dcgan_one_iteration_parity(L, precision, width, rows, cols, batch):
    """Selection bit-exact given the engine's fitness; then the last step's gradients and the
    Adam state per cell against the oracle (a cell whose pre-activations came within rounding
    distance of a kink is excused, as in the MLP checks). Width 64 in bf16 runs the training
    forward on the tensor-core kernel with channel-last activations. At that width every cell
    has pre-activations within 1e-8 of a kink, and batch normalisation's backward spreads a
    flipped derivative over the whole channel: the CUDA-core and the tensor-core paths both
    reach 1.4-4.7 % there (B = 16), so that case is held to 7.5 % per cell and 5 % median.
    A generator twice as wide (ngf 128, ndf 64) takes the kernel variants the width-64 case
    does not: the output layer by parity class, and the wide first-layer variant for the
    generator's input gradient. Its single cell lands at 6.9 % with the tensor cores and 6.8 %
    with the CUDA-core kernels (measured side by side on the same inputs; the two differ from
    each other by 7 %), so it is held to the 7.5 % per-cell rule only."""
    pool = _field_pool(3, 40)
    ngf, ndf = width if isinstance(width, tuple) else (width, width)
    width = min(ngf, ndf)
    g = _grid(L, rows, cols, 11, pool, precision=precision, keep_grads=1, ngf=ngf, ndf=ndf,
              batch=batch)
    a = oracle_arch(g.arch)
    tol = TOL[g.arch.precision]
    for it in range(2 if width < 64 else 1):
        s = _state(g)
        data = O.batches(s, pool)
        ev = g.eval()
        sel = g.select()
        ref_sel = O.select_replace(s, {"fG": ev["fG"].astype(np.float64),
                                       "fD": ev["fD"].astype(np.float64)})
        assert np.array_equal(sel["sel_g"], ref_sel["sel_g"])
        assert np.array_equal(sel["sel_d"], ref_sel["sel_d"])
        g.train()
        new, grads = O.train_step(s, ref_sel, data, keep_grads=True)
        got = _state(g)
        assert np.array_equal(got.Gstep, new.Gstep) and np.array_equal(got.Dstep, new.Dstep)
        gg, gd = g.gradients()
        worst = np.zeros(s.cells)
        for pop, gpu, r in (("G", gg, grads["gG"]), ("D", gd, grads["gD"]),
                            ("G", got.Gm, new.Gm), ("D", got.Dm, new.Dm)):
            lay = O.g_layout(a) if pop == "G" else O.d_layout(a)
            for c in range(s.cells):
                worst[c] = max(worst[c], max(per_tensor(gpu[c:c + 1], r[c:c + 1], lay).values()))
        ok = worst < tol
        kinky = grads["kink"] < (1e-5 if precision == "fp32" else 1e-3)
        assert np.all(ok | kinky), (it, worst)
        if precision == "fp32":
            assert np.sum(~ok) <= 1, (it, worst)
        elif width >= 64:
            assert np.all(worst < 0.075), (it, worst)
            if ngf == ndf:
                assert np.median(worst) < 0.05, (it, worst)
        else:
            assert np.all(worst < 5 * tol) and np.median(worst) < 2 * tol, (it, worst)


def test_dcgan_fused_iterate_equals_separate_calls_and_is_deterministic(L):
    pool = _field_pool(4, 30)
    a = _grid(L, 2, 2, 5, pool, precision="bf16")
    b = _grid(L, 2, 2, 5, pool, precision="bf16")
    a.iterate(2)
    for _ in range(2):
        b.eval()
        b.select()
        b.train()
    assert a.export_state() == b.export_state()


def test_dcgan_full_width_3x3_b128_sampled(L):
    """The 3x3 DCGAN configuration (width 64: 512/256/128/64 channels, z = 100, B = 128,
    bf16): one cell's centre generator on its noise (the full batch, for the batch
    statistics) and the logits of sampled rows against the oracle."""
    pool = _field_pool(1811, 600)
    g = _grid(L, 3, 3, 1811, pool, precision="bf16", z_dim=100, ngf=64, ndf=64, batch=128)
    s = _state(g)
    c = 4
    data = O.batches(s, pool, cells=[c])
    g.eval()
    x, z = g.batch()
    a = s.arch
    gl, dl = O.g_layout(a), O.d_layout(a)
    F = O.g_forward(O.unflatten(s.Gw[c], gl), data[c][1], a)["F"]
    logits = g.logits()
    rows = np.r_[0:8, 128:136]  # real rows, then the centre generator's fakes
    X = np.vstack([data[c][0], F])[rows]
    lg = O.d_forward(O.unflatten(s.Dw[c], dl), X, a)["logit"]
    assert max_rel(logits[c, 0, rows], lg) < 2e-2


def test_dcgan_tma_and_gathered_activations_agree_bit_for_bit(L, monkeypatch):
    """The tensor-core convolutions load their channel-last A tiles through activation maps by
    TMA; with LIPZ_CONV_GATHER=1 the gather warps load them instead. Both hand the MMA the same
    bytes, so one iteration (evaluation, selection, training) ends in the same state."""
    pool = _field_pool(6, 40)
    kw = dict(precision="bf16", ngf=64, ndf=64, batch=16, z_dim=100)
    a = _grid(L, 2, 2, 7, pool, **kw)
    a.iterate(1)
    monkeypatch.setenv("LIPZ_CONV_GATHER", "1")
    b = _grid(L, 2, 2, 7, pool, **kw)
    b.iterate(1)
    assert a.export_state() == b.export_state()
