"""Pins for the oracle's generator-mixture step (Section 3 step 4): the Gaussian-kernel MMD
score of a weighted mixture and the ES-(1+1) update.

Checks come from an independent library routine (scipy's pairwise squared distances), from the
definition of the weighted MMD as the MMD of a sample in which each generator's fakes are
repeated in proportion to its weight, from the positive definiteness of the Gaussian kernel, and
from cases with known answers.
"""

import numpy as np
import pytest

from oracle import lipz_oracle as O

cdist = pytest.importorskip("scipy.spatial.distance").cdist


def _blocks_scipy(X, B):
    K = np.exp(-cdist(X, X, "sqeuclidean") / X.shape[1])
    nb = X.shape[0] // B
    return np.array([[K[a * B:(a + 1) * B, b * B:(b + 1) * B].mean() for b in range(nb)]
                     for a in range(nb)])


def _mmd2_samples(P, Q):
    """Biased squared MMD between two unweighted samples, from scipy distances."""
    d = P.shape[1]
    k = lambda U, V: np.exp(-cdist(U, V, "sqeuclidean") / d).mean()
    return k(P, P) + k(Q, Q) - 2.0 * k(P, Q)


def test_blocks_match_scipy_pairwise_distances():
    rng = np.random.default_rng(0)
    X = rng.uniform(-1, 1, size=(6 * 7, 11))
    S = O.mixture_blocks(X, 7)
    assert S.shape == (6, 6)
    assert np.allclose(S, _blocks_scipy(X, 7), rtol=1e-13, atol=0)
    assert np.allclose(S, S.T, rtol=0, atol=1e-15) and np.all((S > 0) & (S <= 1))


def test_weighted_score_is_the_mmd_of_the_replicated_mixture():
    """With rational weights w_i = m_i / M, the weighted score equals the plain biased MMD^2
    between the real rows and the sample holding slot i's fakes m_i times."""
    rng = np.random.default_rng(1)
    B, d = 6, 9
    X = np.vstack([rng.normal(loc=mu, size=(B, d)) for mu in (0.0, 0.2, 0.5, -0.3, 1.0, 0.05)])
    S = O.mixture_blocks(X, B)
    for m in ([1, 1, 1, 1, 1], [3, 0, 1, 0, 2], [0, 0, 0, 0, 1], [5, 1, 0, 2, 0]):
        w = np.array(m, float) / sum(m)
        mix = np.vstack([X[B * (1 + i):B * (2 + i)] for i in range(5) for _ in range(m[i])])
        assert O.mmd2(w, S) == pytest.approx(_mmd2_samples(X[:B], mix), rel=1e-12, abs=1e-15)


def test_score_is_nonnegative_and_zero_for_perfect_fakes():
    rng = np.random.default_rng(2)
    B = 5
    X = rng.uniform(-1, 1, size=(6 * B, 8))
    S = O.mixture_blocks(X, B)
    for _ in range(50):
        w = rng.dirichlet(np.ones(5))
        assert O.mmd2(w, S) >= -1e-15
    x = X[:B]
    S0 = O.mixture_blocks(np.vstack([x] * 6), B)
    assert abs(O.mmd2(rng.dirichlet(np.ones(5)), S0)) < 1e-15


def test_es_step_keeps_only_improvements_and_stays_on_the_simplex():
    """Slot 0's fakes are the real rows, the others are far: moving weight to slot 0 lowers the
    score (accepted), moving it away raises it (rejected); a zero mutation changes nothing."""
    rng = np.random.default_rng(3)
    B = 4
    x = rng.uniform(-1, 1, size=(B, 6))
    far = [x + 3.0 + i for i in range(4)]
    S = O.mixture_blocks(np.vstack([x, x] + far), B)
    w = np.full(5, 0.2)
    up = np.array([3.0, -1.0, -1.0, -1.0, -1.0])
    w1, acc, old, new = O.mixture_step(w, S, up, 0.05)
    assert acc and new < old and np.isclose(w1.sum(), 1.0) and w1[0] > 0.2 and np.all(w1 >= 0)
    w2, acc2, old2, new2 = O.mixture_step(w, S, -up, 0.05)
    assert not acc2 and new2 > old2 and np.array_equal(w2, w)
    w3, acc3, _, _ = O.mixture_step(w, S, up, 0.0)
    assert not acc3 and np.array_equal(w3, w)
    # a mutation that clips every weight to 0 leaves w as it was
    w4, acc4, _, _ = O.mixture_step(w, S, np.full(5, -10.0), 1.0)
    assert np.array_equal(w4, w)
    # clipping: one weight driven below zero becomes exactly 0
    w5, _, _, new5 = O.mixture_step(w, S, np.array([1.0, -5.0, 0.0, 0.0, 0.0]), 0.1)
    cand = np.maximum(w + 0.1 * np.array([1.0, -5.0, 0.0, 0.0, 0.0]), 0)
    assert new5 == pytest.approx(O.mmd2(cand / cand.sum(), S), rel=1e-14)


def test_grid_mixture_update_draws_its_own_stream_and_converges_on_a_perfect_slot():
    """On a 1x1 torus all five slots hold the same generator, so every mixture scores the same;
    the update's mutation normals are the first five of stream MIX at the iteration."""
    arch = O.Arch(z_dim=3, hidden=4, x_dim=5, batch=6, mixture=True, mix_sigma=0.01)
    s = O.create(1, 1, arch, 7)
    pool = np.random.default_rng(0).uniform(-1, 1, size=(50, 5))
    data = O.batches(s, pool)
    mx = O.mixture_update(s, data)
    S = mx["S"][0]
    assert np.allclose(S[1:, 1:], S[1, 1]) and np.allclose(S[1:, 0], S[1, 0])
    nrm = O.draw_normals(7, O.STREAM_MIX, 0, 0, 5)
    cand = np.maximum(0.2 + 0.01 * nrm, 0)
    assert mx["score_new"][0] == pytest.approx(O.mmd2(cand / cand.sum(), S), rel=1e-12)
    assert mx["score"][0] == pytest.approx(O.mmd2(np.full(5, 0.2), S), rel=1e-12)
    s2 = O.iterate(s, pool, 3)
    assert np.isclose(s2.mix.sum(), 1.0) and np.all(s2.mix >= 0)
    buf = O.state_to_bytes(s2)
    assert np.allclose(O.state_from_bytes(buf, arch).mix, s2.mix.astype(np.float32))
