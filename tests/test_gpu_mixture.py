"""GPU parity of the generator-mixture step (Section 3 step 4): the Gaussian-kernel block means
of every cell's evaluation rows against the oracle (1e-4 fp32 / 2e-2 bf16, max-norm relative),
and the ES-(1+1) step given the engine's own block means (the same decision wherever the two
scores differ by more than the fp32 rounding band)."""

import numpy as np
import pytest

from oracle import lipz_oracle as O

from helpers import max_rel, oracle_arch

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


def _pool(seed, n, dim):
    import lipz_synth
    return lipz_synth.blob_pool(seed, n=n, dim=dim)


def _arch(g):
    a = oracle_arch(g.arch)
    a.mixture, a.mix_sigma = bool(g.arch.mixture), float(g.arch.mix_sigma)
    return a


def _check_mixture(g, pool, cells=None):
    """One evaluation: block means against the oracle, then the ES step given the engine's
    block means. Returns the number of accepted mutations among the checked cells."""
    a = _arch(g)
    s = O.state_from_bytes(g.export_state(), a)
    w0 = g.mixture()
    assert np.array_equal(w0.astype(np.float64), s.mix)
    data = O.batches(s, pool, cells=cells)
    g.eval()
    w, S, score = g.mixture(blocks=True)
    ref = O.mixture_update(s, data, cells=cells)
    idx = range(s.cells) if cells is None else cells
    tol = TOL[g.arch.precision]
    accepted = 0
    for c in idx:
        assert max_rel(S[c], ref["S"][c]) < tol, (c, S[c], ref["S"][c])
        assert np.allclose(S[c], S[c].T, rtol=0, atol=1e-6)
        nrm = O.draw_normals(s.seed, O.STREAM_MIX, s.t, c, 5)
        wr, acc, old, new = O.mixture_step(s.mix[c], S[c].astype(np.float64), nrm, a.mix_sigma)
        band = 1e-5 * max(1.0, abs(old))
        if abs(new - old) > band:
            assert np.allclose(w[c], wr, rtol=0, atol=1e-6), (c, w[c], wr)
            assert score[c] == pytest.approx(new if acc else old, rel=1e-4, abs=1e-6)
            accepted += int(acc)
        assert np.isclose(w[c].sum(), 1.0, atol=1e-5) and np.all(w[c] >= 0)
    return accepted


@pytest.mark.parametrize("precision,rows,cols,batch", [
    ("fp32", 2, 2, 100),    # CUDA-core path: stored Gram matrix
    ("bf16", 3, 3, 100),    # tensor-core Gram kernel: 600 rows = 5 row tiles, 3 column blocks
    ("bf16", 2, 3, 129),    # 774 rows: ragged row tile and a 6-column last block
    ("bf16", 1, 1, 37),     # degenerate torus, one column block of 222
    ("bf16", 2, 2, 20),     # batch below 32: the stored-Gram path in bf16
])
def test_mixture_step_against_the_oracle(L, precision, rows, cols, batch):
    pool = _pool(21, 4000, 784)
    g = L.Grid(rows, cols, seed=5, precision=precision, batch=batch, mixture=1, mix_sigma=0.05)
    g.set_data(pool)
    acc = 0
    for it in range(3):
        acc += _check_mixture(g, pool)
        g.select()
        g.train()
    st = O.state_from_bytes(g.export_state(), _arch(g))
    assert np.allclose(st.mix, g.mixture(), rtol=0, atol=0)
    if rows * cols > 1:
        assert acc > 0  # some mutation was kept


def test_mixture_is_deterministic_and_resumes(L):
    pool = _pool(22, 3000, 784)
    kw = dict(precision="bf16", mixture=1, mix_sigma=0.05)
    a = L.Grid(3, 3, seed=8, **kw)
    b = L.Grid(3, 3, seed=8, **kw)
    for g in (a, b):
        g.set_data(pool)
    a.iterate(3)
    b.iterate(2)
    c = L.Grid(3, 3, seed=1, **kw)
    c.set_data(pool)
    c.import_state(b.export_state())
    b.iterate(1)
    c.iterate(1)
    assert a.export_state() == b.export_state() == c.export_state()
    assert not np.allclose(a.mixture(), 0.2)


def test_mixture_off_keeps_uniform_weights_and_refuses_scores(L):
    pool = _pool(23, 2000, 784)
    g = L.Grid(2, 2, seed=3)
    g.set_data(pool)
    g.iterate(2)
    assert np.allclose(g.mixture(), 0.2)
    with pytest.raises(L.LipzError) as e:
        g.mixture(blocks=True)
    assert e.value.code == L.LIPZ_ERR_STATE


def test_mixture_full_size_12x12_sampled_cells(L):
    """The benchmark workload with the mixture step (tensor-core Gram kernel over 144 cells):
    block means and ES steps of sampled cells, including the wrap-around corners."""
    pool = _pool(1811, 60000, 784)
    g = L.Grid(12, 12, seed=1811, precision="bf16", mixture=1, mix_sigma=0.05)
    g.set_data(pool)
    g.iterate(1)
    _check_mixture(g, pool, cells=[0, 11, 77, 143])
