"""GPU parity of the stale-neighbour schedule (asynchronous cells, Section 3): every evaluation
reads the cell's own centre from the current snapshot and its four neighbours from the other
snapshot (the previous iteration's centres), and a selected neighbour brings that older
individual. Checked in lockstep against the oracle given the engine's previous state."""

import numpy as np
import pytest

from oracle import lipz_oracle as O

from helpers import gradient_parity, max_rel, oracle_arch

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


def _lockstep(g, pool, prev, label):
    """One stale iteration against the oracle started from the engine's current and previous
    states: evaluation within tolerance, selection bit-exact given the engine's fitness, then
    the new state's step counts and lrs exactly, the gradients by the rules of
    helpers.gradient_parity, and the moments and weights as Adam steps of the selected (possibly
    older) individual given the engine's own gradient. Returns the state it started from."""
    a = oracle_arch(g.arch)
    s = O.state_from_bytes(g.export_state(), a)
    tol = TOL[g.arch.precision]
    data = O.batches(s, pool)
    ref = O.eval_neighborhoods(s, data, prev=prev)
    ev = g.eval(pairs=True)
    for k in ("LG", "LD", "fG", "fD"):
        assert max_rel(ev[k], ref[k]) < tol, k
    assert max_rel(g.logits(), ref["logits"]) < tol
    sel = g.select()
    ref_sel = O.select_replace(s, {"fG": ev["fG"].astype(np.float64),
                                   "fD": ev["fD"].astype(np.float64)})
    assert np.array_equal(sel["sel_g"], ref_sel["sel_g"])
    assert np.array_equal(sel["sel_d"], ref_sel["sel_d"])
    g.train()
    new, grads = O.train_step(s, ref_sel, data, keep_grads=True, prev=prev)
    got = O.state_from_bytes(g.export_state(), a)
    assert np.array_equal(got.Gstep, new.Gstep) and np.array_equal(got.Dstep, new.Dstep)
    assert np.allclose(got.Glr, new.Glr, rtol=1e-6) and np.allclose(got.Dlr, new.Dlr, rtol=1e-6)
    gg, gd = g.gradients()
    nbr = O.neighbors(s.rows, s.cols)

    def source(pop, c):
        slot = int(ref_sel["sel_" + pop.lower()][c])
        return O._slot_state(s, prev, slot), int(nbr[c][slot])

    def pair_inputs(c):
        (SG, kg), (SD, kd) = source("G", c), source("D", c)
        return (SG.Gw[kg], SD.Dw[kd]) + tuple(data[c])

    gradient_parity(label, a, gg, gd, grads["gG"], grads["gD"], tol, pair_inputs)
    for pop, gpu_g in (("G", gg), ("D", gd)):
        for c in range(s.cells):
            S, k = source(pop, c)
            w1, m1, v1, _ = O.adam_step(getattr(S, pop + "w")[k], getattr(S, pop + "m")[k],
                                        getattr(S, pop + "v")[k], getattr(S, pop + "step")[k],
                                        gpu_g[c].astype(np.float64),
                                        float(np.float32(getattr(new, pop + "lr")[c])), a)
            for f, r in (("w", w1), ("m", m1), ("v", v1)):
                v = getattr(got, pop + f)[c]
                assert np.max(np.abs(v - r)) <= 1e-6 * np.max(np.abs(r)) + 1e-12, (pop, f, c)
    return s, ref_sel


@pytest.mark.parametrize("precision,rows,cols,batch", [
    ("fp32", 2, 3, 100),   # CUDA-core path
    ("bf16", 3, 3, 100),   # tensor-core path (both snapshots in one index space)
])
def test_stale_neighbours_lockstep(L, precision, rows, cols, batch):
    pool = _pool(31, 4000, 784)
    g = L.Grid(rows, cols, seed=9, precision=precision, batch=batch, keep_grads=1,
               stale_neighbors=1, tournament_size=5, replace_mode="always")
    g.set_data(pool)
    prev, picked = None, 0
    for it in range(4):
        s, sel = _lockstep(g, pool, prev, "stale %s %dx%d it %d" % (precision, rows, cols, it))
        if it > 0:
            picked += int(np.sum(sel["sel_g"] != 0) + np.sum(sel["sel_d"] != 0))
        prev = s
    assert picked > 0  # some stale neighbour was selected


def test_stale_first_iteration_and_import_equal_the_synchronous_schedule(L):
    """No older snapshot exists right after create or import: that iteration is the
    synchronous one, bit for bit; the next one differs."""
    pool = _pool(32, 3000, 784)
    a = L.Grid(3, 3, seed=4, precision="bf16", stale_neighbors=1)
    b = L.Grid(3, 3, seed=4, precision="bf16")
    for g in (a, b):
        g.set_data(pool)
        g.iterate(1)
    assert a.export_state() == b.export_state()
    a.iterate(1)
    b.iterate(1)
    assert a.export_state() != b.export_state()
    st = b.export_state()
    a.import_state(st)
    b.import_state(st)
    a.iterate(1)
    b.iterate(1)
    assert a.export_state() == b.export_state()


def test_stale_fused_adam_equals_stored_gradient_path(L):
    """Selected stale individuals come from the other snapshot through the fused-Adam
    backward's maps as well: bit-identical to the stored-gradient path."""
    pool = _pool(33, 3000, 784)
    kw = dict(precision="bf16", stale_neighbors=1, tournament_size=5, replace_mode="always")
    a = L.Grid(3, 3, seed=6, **kw)
    b = L.Grid(3, 3, seed=6, keep_grads=1, **kw)
    for g in (a, b):
        g.set_data(pool)
    for it in range(4):
        a.iterate(1)
        b.iterate(1)
        assert a.export_state() == b.export_state(), it
