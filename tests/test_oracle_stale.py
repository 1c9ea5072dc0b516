"""Pins for the oracle's stale-neighbour schedule (the asynchronous cells of Section 3 emulated
deterministically: a cell sees its own centre as of the iteration and its neighbours one
iteration late). Checked against the plain synchronous evaluation of each snapshot, and
against the selection sources with a zero learning rate (where Adam moves nothing)."""

import numpy as np
import pytest

from oracle import lipz_oracle as O

TINY = dict(z_dim=3, hidden=4, x_dim=5, batch=6)


def _setup(rows=2, cols=3, **kw):
    arch = O.Arch(**{**TINY, **kw})
    s0 = O.create(rows, cols, arch, 11)
    pool = np.random.default_rng(4).uniform(-1, 1, size=(60, 5))
    return arch, s0, pool


def test_first_iteration_equals_the_synchronous_one():
    arch, s0, pool = _setup(stale_neighbors=True)
    sync = O.Arch(**{**TINY})
    a = O.iterate(s0, pool, 1)
    b = O.iterate(O.State(**{**s0.__dict__, "arch": sync}), pool, 1)
    for f in ("Gw", "Dw", "Gm", "Dv", "Gstep", "Dstep"):
        assert np.array_equal(getattr(a, f), getattr(b, f))


def test_stale_evaluation_pairs_come_from_the_right_snapshots():
    """Pair (i, j) of a stale evaluation takes generator i and discriminator j from the current
    snapshot when the slot is the centre, else from the previous one: each such pair's losses
    equal those of the plain evaluation of the snapshot (or mixed pair) it names."""
    arch, s0, pool = _setup()
    s1 = O.iterate(s0, pool, 1)
    data = O.batches(s1, pool)
    ev = O.eval_neighborhoods(s1, data, prev=s0)
    cur = O.eval_neighborhoods(s1, data)
    old = O.eval_neighborhoods(s0, data)
    assert not np.allclose(cur["LG"], old["LG"])
    # generator and discriminator both neighbours: the previous snapshot's pair
    assert np.array_equal(ev["LG"][:, 1:, 1:], old["LG"][:, 1:, 1:])
    assert np.array_equal(ev["LD"][:, 1:, 1:], old["LD"][:, 1:, 1:])
    # both centres: the current pair
    assert np.array_equal(ev["LG"][:, 0, 0], cur["LG"][:, 0, 0])
    # current centre generator against a previous neighbour discriminator: a mixed snapshot
    gl, dl = O.g_layout(arch), O.d_layout(arch)
    nbr = O.neighbors(s1.rows, s1.cols)
    for c in range(s1.cells):
        x, z = data[c]
        F = O.g_forward(O.unflatten(s1.Gw[c], gl), z, arch)["F"]
        for j in range(1, 5):
            lg = O.d_forward(O.unflatten(s0.Dw[nbr[c][j]], dl), np.vstack([x, F]), arch)["logit"]
            lgg, ldd = O.pair_losses(lg[:arch.batch], lg[arch.batch:])
            assert ev["LG"][c, 0, j] == pytest.approx(lgg, rel=1e-12)
            assert ev["LD"][c, 0, j] == pytest.approx(ldd, rel=1e-12)


def test_stale_selection_brings_the_previous_individual():
    """With lr = 0 Adam moves nothing, so a cell whose tournament picked neighbour slot s holds
    exactly the previous snapshot's individual nbr[c][s] afterwards (its step count + 1)."""
    arch, s0, pool = _setup(rows=3, cols=3, lr=0.0, tournament_size=5, replace_mode="always",
                            stale_neighbors=True)
    s1 = O.iterate(s0, pool, 1)
    # perturb s1 so that the two snapshots differ
    s1.Gw = s1.Gw + 0.01
    s1.Dw = s1.Dw - 0.01
    data = O.batches(s1, pool)
    ev = O.eval_neighborhoods(s1, data, prev=s0)
    sel = O.select_replace(s1, ev)
    new = O.train_step(s1, sel, data, pool=pool, prev=s0)
    nbr = O.neighbors(3, 3)
    moved = 0
    for c in range(9):
        for pop, ks in (("G", sel["sel_g"][c]), ("D", sel["sel_d"][c])):
            src = (s1 if ks == 0 else s0)
            k = nbr[c][ks]
            assert np.array_equal(getattr(new, pop + "w")[c], getattr(src, pop + "w")[k])
            assert getattr(new, pop + "step")[c] == getattr(src, pop + "step")[k] + 1
            moved += int(ks != 0)
    assert moved > 0
    # and iterate() carries the previous snapshot itself
    two = O.iterate(s0, pool, 2)
    s1b = O.iterate(s0, pool, 1)
    ref = O.iterate(s1b, pool, 1, prev=s0)
    assert np.array_equal(two.Gw, ref.Gw) and np.array_equal(two.Dstep, ref.Dstep)


def test_stale_neighbours_need_one_step_per_iteration():
    arch, s0, pool = _setup(stale_neighbors=True, train_steps=2)
    with pytest.raises(ValueError):
        O.iterate(s0, pool, 1)
