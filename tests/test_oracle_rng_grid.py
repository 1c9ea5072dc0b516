"""Pins for the oracle's random numbers, torus neighbourhoods, initialisation and selection.

Each check is against something other than the oracle itself: published known-answer vectors,
brute force on small grids, closed forms, or exhaustive enumeration.
"""

import math
import os

import numpy as np
import pytest

from oracle import lipz_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _kat_rows():
    rows = []
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                rows.append([int(v, 16) for v in line.split()])
    return rows


def test_philox_known_answer_vectors():
    rows = _kat_rows()
    assert len(rows) == 3
    for r in rows:
        out = O.philox4x32_10(np.array(r[:4], np.uint64), (r[4], r[5]))
        assert [int(v) for v in out] == r[6:10]


def test_draw_words_counter_mapping():
    # word k of a (stream, t, cell) sequence is word k % 4 of block (k // 4, cell, t, stream)
    seed = (7 << 32) | 1234
    w = O.draw_words(seed, 4, 9, 3, 10)
    for k in range(10):
        blk = O.philox4x32_10(np.array([k // 4, 3, 9, 4], np.uint64), (1234, 7))
        assert int(w[k]) == int(blk[k % 4])


def test_uniform_words_statistics():
    w = O.draw_words(1811, O.STREAM_BATCH, 0, 0, 1 << 16).astype(np.float64) / 2 ** 32
    assert abs(w.mean() - 0.5) < 0.005
    assert abs(w.var() - 1.0 / 12) < 0.002


def test_mulhi_exact_buckets():
    # mulhi(w, n) = j exactly on [ceil(j 2^32 / n), ceil((j+1) 2^32 / n))
    for n in (1, 2, 3, 4, 5, 7, 100, 60000):
        for j in sorted({0, 1, n // 2, n - 1}):
            lo = -(-(j << 32) // n)
            hi = -(-((j + 1) << 32) // n) - 1
            assert int(O.mulhi(np.array([lo]), n)[0]) == j
            assert int(O.mulhi(np.array([hi]), n)[0]) == j
            if lo > 0:
                assert int(O.mulhi(np.array([lo - 1]), n)[0]) == j - 1


def test_box_muller_closed_forms_and_moments():
    # u1 = 1 (top bits all ones) gives r = 0; v = 0 gives (r, 0)
    a, b = O.box_muller(np.array([0xFFFFFFFF]), np.array([0]))
    assert a[0] == 0.0 and b[0] == 0.0
    a, b = O.box_muller(np.array([0]), np.array([0]))
    assert a[0] == pytest.approx(math.sqrt(-2 * math.log(2.0 ** -24)), rel=1e-15)
    assert b[0] == 0.0
    z = O.draw_normals(3, O.STREAM_NOISE, 5, 2, 200000)
    assert abs(z.mean()) < 0.01
    assert abs(z.var() - 1.0) < 0.02
    # fourth moment of a standard normal is 3
    assert abs((z ** 4).mean() - 3.0) < 0.1


def _torus_brute(rows, cols):
    """Neighbourhoods by definition: the cell itself plus the cells one step away along the
    row or the column, wrapping around the torus edges."""
    nb = []
    for r in range(rows):
        for q in range(cols):
            nb.append([(r, q), ((r - 1 + rows) % rows, q), ((r + 1) % rows, q),
                       (r, (q - 1 + cols) % cols), (r, (q + 1) % cols)])
    return np.array([[a * cols + b for a, b in cells] for cells in nb])


@pytest.mark.parametrize("rows,cols", [(1, 1), (2, 2), (3, 3), (1, 4), (4, 4), (3, 5), (12, 12)])
def test_neighbourhoods_brute_force_and_invariants(rows, cols):
    nbr = O.neighbors(rows, cols)
    assert np.array_equal(nbr, _torus_brute(rows, cols))
    cells = rows * cols
    # every cell appears exactly 5 times over all slots (each slot map is a bijection)
    counts = np.bincount(nbr.reshape(-1), minlength=cells)
    assert np.all(counts == 5)
    for s in range(5):
        assert sorted(nbr[:, s]) == list(range(cells))
    # symmetry: c' in N(c)  <=>  c in N(c')
    for c in range(cells):
        for cp in nbr[c]:
            assert c in nbr[cp]


def test_neighbourhood_special_grids():
    assert np.all(O.neighbors(1, 1) == 0)
    n2 = O.neighbors(2, 2)
    assert np.array_equal(n2[:, 1], n2[:, 2]) and np.array_equal(n2[:, 3], n2[:, 4])
    n3 = O.neighbors(3, 3)
    for c in range(9):
        assert len(set(n3[c])) == 5
        right = (c // 3) * 3 + (c % 3 + 1) % 3
        # horizontally adjacent 3x3 neighbourhoods share their whole row (3 cells)
        assert len(set(n3[c]) & set(n3[right])) == 3
    n4 = O.neighbors(4, 5)
    for c in range(20):
        right = (c // 5) * 5 + (c % 5 + 1) % 5
        assert len(set(n4[c]) & set(n4[right])) == 2


def test_xavier_init_bounds_and_variance():
    a = O.Arch()
    gl = O.g_layout(a)
    flat = O.init_params(1811, O.STREAM_INIT_G, 3, gl)
    P = O.unflatten(flat, gl)
    for name, (fo, fi) in (("W1", (256, 64)), ("W2", (256, 256)), ("W3", (784, 256))):
        bound = math.sqrt(6.0 / (fi + fo))
        w = P[name]
        assert np.all(np.abs(w) < bound * (1 + 1e-7))
        assert abs(w.var() / (bound ** 2 / 3.0) - 1.0) < 0.05
        assert abs(w.mean()) < 0.05 * bound
        assert np.array_equal(w, w.astype(np.float32))
    for name in ("b1", "b2", "b3"):
        assert np.all(P[name] == 0.0)
    other = O.init_params(1811, O.STREAM_INIT_G, 4, gl)
    assert not np.array_equal(flat, other)
    assert np.array_equal(flat, O.init_params(1811, O.STREAM_INIT_G, 3, gl))


def _word_for_bucket(j, n):
    return ((j << 32) + (1 << 31)) // n


def test_tournament_size2_enumeration():
    rng = np.random.default_rng(0)
    seen = set()
    for trial in range(30):
        f = rng.integers(0, 3, size=5).astype(np.float64)  # many exact ties
        for j0 in range(5):
            for j1 in range(4):
                w = np.array([_word_for_bucket(j0, 5), _word_for_bucket(j1, 4)], np.uint64)
                a = j0
                b = j1 + (1 if j1 >= a else 0)
                seen.add((a, b))
                win = O.tournament(f, w, 2)
                assert win in (a, b)
                other = b if win == a else a
                assert f[win] <= f[other]
                if f[win] == f[other]:
                    assert win < other
    # the 20 word buckets give the 20 ordered pairs of distinct slots, each once
    assert len(seen) == 20 and all(a != b for a, b in seen)


def test_tournament_size5_is_argmin_and_if_better_keeps_best():
    rng = np.random.default_rng(1)
    arch = O.Arch(tournament_size=5)
    for _ in range(200):
        f = rng.normal(size=5)
        w = rng.integers(0, 2 ** 32, size=5, dtype=np.uint64)
        assert O.tournament(f, w, 5) == int(np.argmin(f))
        assert O.select_slot(f, w, arch) == int(np.argmin(f))
    arch2 = O.Arch(tournament_size=2)
    for _ in range(500):
        f = rng.normal(size=5)
        w = rng.integers(0, 2 ** 32, size=2, dtype=np.uint64)
        s = O.select_slot(f, w, arch2)
        assert f[s] <= f[0]            # never replaced by a worse individual
        if np.argmin(f) == 0:
            assert s == 0              # a centre that is the neighbourhood's best is kept
    # an exact tie with the centre keeps the centre
    assert O.select_slot(np.zeros(5), np.array([0, 0], np.uint64), arch2) == 0


def test_best_individual_survives_a_grid_selection():
    """'Selection keeps the best-fitness individual': the global best is its own neighbourhood's
    best, so its cell keeps it; with tournament size 5 every cell adopts its neighbourhood best."""
    rng = np.random.default_rng(2)
    for rows, cols in ((3, 3), (4, 5)):
        nbr = O.neighbors(rows, cols)
        f_cell = rng.normal(size=rows * cols)
        best = int(np.argmin(f_cell))
        for size in (2, 5):
            arch = O.Arch(tournament_size=size)
            for c in range(rows * cols):
                f5 = f_cell[nbr[c]]
                w = rng.integers(0, 2 ** 32, size=size, dtype=np.uint64)
                s = O.select_slot(f5, w, arch)
                if c == best:
                    assert nbr[c][s] == best
                if size == 5:
                    assert nbr[c][s] == nbr[c][int(np.argmin(f5))]


def test_lr_mutation():
    a = O.Arch(lr_mutation=True, lr_mut_prob=0.0)
    assert O.mutate_lr(2e-4, 1, O.STREAM_MUT_G, 0, 0, a) == 2e-4
    a1 = O.Arch(lr_mutation=True, lr_mut_prob=1.0)
    deltas = np.array([O.mutate_lr(2e-4, 1, O.STREAM_MUT_G, t, c, a1) - 2e-4
                       for t in range(20) for c in range(50)])
    assert np.all(deltas != 0.0)
    assert abs(deltas.mean()) < 2e-5 and abs(deltas.std() / 1e-4 - 1.0) < 0.1
    assert O.mutate_lr(0.0, 1, O.STREAM_MUT_G, 0, 0, O.Arch(lr_mut_prob=1.0, lr_mut_std=1.0)) >= 1e-8
    half = O.Arch(lr_mut_prob=0.5)
    changed = np.mean([O.mutate_lr(2e-4, 2, O.STREAM_MUT_D, t, c, half) != 2e-4
                       for t in range(20) for c in range(50)])
    assert abs(changed - 0.5) < 0.05
