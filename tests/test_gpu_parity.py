"""GPU parity: the CUDA engine (through the C ABI) against the CPU oracle, step by step.

Tolerances (max-norm relative error per tensor, max|gpu - ref| / max|ref|): 1e-4 for the fp32
path and 2e-2 for the bf16-operand / fp32-accumulate path. Integer work (neighbourhoods,
minibatch indices, tournament choices given the same fitness) is compared bit-exactly.
"""

import numpy as np
import pytest

from oracle import lipz_oracle as O

from helpers import (BF16_CEIL, FP32_FLIP_BAND, cell_errors, gradient_parity, max_rel,
                     oracle_arch)

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


def _grid(L, rows, cols, seed, pool, **kw):
    g = L.Grid(rows, cols, seed=seed, **kw)
    g.set_data(pool)
    return g


def _to_oracle(g, arch):
    return O.state_from_bytes(g.export_state(), oracle_arch(arch))


# ------------------------------------------------------------------------------------------
def test_init_is_bit_exact(L):
    g = L.Grid(2, 3, seed=1811)
    s = _to_oracle(g, g.arch)
    ref = O.create(2, 3, oracle_arch(g.arch), 1811)
    assert np.array_equal(s.Gw, ref.Gw) and np.array_equal(s.Dw, ref.Dw)
    assert np.all(s.Gm == 0) and np.all(s.Dv == 0) and np.all(s.Gstep == 0)
    assert np.allclose(s.Glr, np.float32(2e-4))


@pytest.mark.parametrize("precision", ["fp32", "bf16"])
def test_minibatch_draw(L, precision):
    pool = _pool(3, 5000, 784)
    g = _grid(L, 2, 2, 77, pool, precision=precision)
    g.eval()
    x, z = g.batch()
    s = _to_oracle(g, g.arch)
    data = O.batches(s, pool)
    for c in range(4):
        xr, zr = data[c]
        if precision == "fp32":
            assert np.array_equal(x[c], xr.astype(np.float32))        # indices bit-exact
            assert np.max(np.abs(z[c] - zr)) < 2e-6 * max(1.0, np.max(np.abs(zr)))
        else:
            assert np.array_equal(x[c], O.round_bf16(xr))
            assert np.max(np.abs(z[c] - O.round_bf16(zr))) <= 2 ** -7 * np.max(np.abs(zr))


def _check_eval(g, s, ev_ref, tol, cells=None):
    ev = g.eval(pairs=True)
    logits = g.logits()
    sl = slice(None) if cells is None else list(cells)
    assert max_rel(logits[sl], ev_ref["logits"][sl]) < tol
    for k in ("LG", "LD", "fG", "fD"):
        assert max_rel(ev[k][sl], ev_ref[k][sl]) < tol, k
    return ev


@pytest.mark.parametrize("precision,rows,cols,batch", [
    ("fp32", 2, 2, 100),    # 2x2 fp32, B=100 (one-iteration parity config)
    ("fp32", 1, 1, 37),     # degenerate 1x1 torus, ragged batch
    ("fp32", 1, 4, 64),
    ("bf16", 2, 2, 100),
    ("bf16", 3, 3, 129),    # ragged tile tails on the tensor-core path
])
def test_eval_parity(L, precision, rows, cols, batch):
    pool = _pool(5, 3000, 784)
    g = _grid(L, rows, cols, 11, pool, precision=precision, batch=batch)
    s = _to_oracle(g, g.arch)
    ref = O.eval_neighborhoods(s, O.batches(s, pool))
    _check_eval(g, s, ref, TOL[g.arch.precision])


def test_eval_parity_tiny_arch_simt(L):
    """Shapes the tensor-core kernels do not take run on the CUDA-core kernels."""
    pool = _pool(6, 200, 5)
    g = _grid(L, 2, 3, 4, pool, z_dim=3, hidden=4, x_dim=5, batch=7)
    s = _to_oracle(g, g.arch)
    ref = O.eval_neighborhoods(s, O.batches(s, pool))
    _check_eval(g, s, ref, 1e-4)


def _one_iteration_check(L, g, pool, tol, x_host=None, label="", cells=None):
    """Eval, select (bit-exact given the engine's own fitness), train: gradients by the rules of
    helpers.gradient_parity (every cell bounded), the Adam arithmetic of both populations given
    the engine's own gradient, and the updated weights. ``cells`` restricts the comparison to a
    sample (the oracle then runs only those cells). Returns the number of weight elements that
    differed beyond the tolerance with a gradient inside the noise band of zero."""
    a = oracle_arch(g.arch)
    assert not a.lr_mutation  # the weight checks below take the individual's own lr
    s = _to_oracle(g, g.arch)
    sample = list(range(s.cells)) if cells is None else list(cells)
    data = O.batches(s, pool, x_host, cells=None if cells is None else sample)
    ref = O.eval_neighborhoods(s, data, cells=None if cells is None else sample)
    ev = _check_eval(g, s, ref, tol, cells=None if cells is None else sample)
    sel = g.select()
    # the tournament is a pure function of (fitness, Philox words): feed the engine's fitness
    ref_sel = O.select_replace(s, {"fG": ev["fG"].astype(np.float64),
                                   "fD": ev["fD"].astype(np.float64)})
    assert np.array_equal(sel["sel_g"], ref_sel["sel_g"])
    assert np.array_equal(sel["sel_d"], ref_sel["sel_d"])
    g.train()
    gg, gd = g.gradients()
    got = _to_oracle(g, g.arch)
    assert got.t == s.t + 1
    nbr = O.neighbors(s.rows, s.cols)
    src_g = nbr[np.arange(s.cells), ref_sel["sel_g"]]
    src_d = nbr[np.arange(s.cells), ref_sel["sel_d"]]
    assert np.array_equal(got.Gstep, s.Gstep[src_g] + 1)
    assert np.array_equal(got.Dstep, s.Dstep[src_d] + 1)
    # the oracle's gradients of every sampled cell's new centre pair
    refG = np.zeros((len(sample), s.Gw.shape[1]))
    refD = np.zeros((len(sample), s.Dw.shape[1]))
    for i, c in enumerate(sample):
        x, z = data[c]
        refG[i], refD[i], _ = O.pair_gradients(s.Gw[src_g[c]], s.Dw[src_d[c]], x, z, a)

    def pair_inputs(i):
        c = sample[i]
        return (s.Gw[src_g[c]], s.Dw[src_d[c]]) + tuple(data[c])

    refG, refD, _ = gradient_parity(label or "one-iteration", a, gg[sample], gd[sample], refG,
                                    refD, tol, pair_inputs)
    flagged = 0
    for pop, lay, src, gpu_g, ref_g in (("G", O.g_layout(a), src_g, gg, refG),
                                        ("D", O.d_layout(a), src_d, gd, refD)):
        W, M, V, S, LR = (getattr(s, pop + f) for f in ("w", "m", "v", "step", "lr"))
        w_got = getattr(got, pop + "w")
        for i, c in enumerate(sample):
            k = src[c]
            lr = float(np.float32(LR[k]))
            # Adam given the engine's own gradient: fp32 arithmetic against float64
            w1 = O.adam_step(W[k], M[k], V[k], S[k], gpu_g[c].astype(np.float64), lr, a)[0]
            assert np.max(np.abs(w_got[c] - w1)) <= 1e-6 * np.max(np.abs(w1)) + 1e-9, (pop, c)
            # the updated weights against the oracle's Adam step on the oracle's gradient.
            # Adam's early steps move an element by about lr * sign(g): an element whose
            # gradient lies within the comparison's noise band of zero (|g_ref| <= 2 |g_gpu -
            # g_ref| + tol * max|g_ref| of its tensor) may move the other way
            w_ref = O.adam_step(W[k], M[k], V[k], S[k], ref_g[i], lr, a)[0]
            off = 0
            for name, shape in lay:
                n = int(np.prod(shape))
                sl = slice(off, off + n)
                off += n
                d = np.abs(w_got[c, sl] - w_ref[sl])
                bad = d > tol * np.max(np.abs(w_ref[sl]))
                if np.any(bad):
                    gr = ref_g[i, sl][bad]
                    gq = gpu_g[c, sl][bad].astype(np.float64)
                    band = tol * np.max(np.abs(ref_g[i, sl]))
                    assert np.all(np.abs(gr) <= 2 * np.abs(gq - gr) + band + 1e-12), (pop, name, c)
                    flagged += int(bad.sum())
    return flagged


def test_one_iteration_fp32_2x2(L):
    """2x2 torus, fp32, B = 100, one grid iteration."""
    pool = _pool(1811, 60000, 784)
    g = _grid(L, 2, 2, 1811, pool, keep_grads=1)
    flagged = _one_iteration_check(L, g, pool, 1e-4, label="fp32 2x2 B=100")
    assert flagged <= 20


def test_lockstep_fp32_3x3_twenty_iterations(L):
    """3x3 torus, fp32, B = 100: twenty iterations, each checked against the oracle started from
    the engine's previous state."""
    pool = _pool(1811, 60000, 784)
    g = _grid(L, 3, 3, 0, pool, keep_grads=1)
    for it in range(20):
        _one_iteration_check(L, g, pool, 1e-4, label="fp32 3x3 B=100 it %d" % it)
    assert g.t == 20


def test_one_iteration_bf16_5x5_b256(L):
    """5x5 torus, bf16 operands / fp32 accumulation and Adam masters, B = 256."""
    pool = _pool(2, 60000, 784)
    g = _grid(L, 5, 5, 2, pool, precision="bf16", batch=256, keep_grads=1)
    for it in range(2):
        _one_iteration_check(L, g, pool, 2e-2, label="bf16 5x5 B=256 it %d" % it)


def test_one_iteration_bf16_3x3_b100(L):
    """3x3 torus, bf16, B = 100 (the benchmark's batch, 100 valid rows of each 128-row tile in
    the backward's K dimension), lr 2e-4: three iterations, every cell's gradients, Adam and
    weights against the oracle."""
    pool = _pool(1811, 60000, 784)
    g = _grid(L, 3, 3, 1811, pool, precision="bf16", batch=100, keep_grads=1)
    for it in range(3):
        _one_iteration_check(L, g, pool, 2e-2, label="bf16 3x3 B=100 it %d" % it)


@pytest.mark.parametrize("rows,cols,batch", [(3, 3, 100), (2, 3, 129)])
def test_fused_adam_equals_stored_gradient_path(L, rows, cols, batch):
    """Unless the gradients are kept, the tensor-core backward applies Adam to the weight
    matrices inside its epilogue (the gradient never leaves the accumulator). Its state after
    every iteration must equal, bit for bit, the path that stores the gradients and runs the
    separate Adam kernel (the one checked against the oracle above)."""
    pool = _pool(9, 5000, 784)
    a = _grid(L, rows, cols, 31, pool, precision="bf16", batch=batch)
    b = _grid(L, rows, cols, 31, pool, precision="bf16", batch=batch, keep_grads=1)
    for it in range(3):
        a.iterate(1)
        b.iterate(1)
        assert a.export_state() == b.export_state(), it


@pytest.mark.parametrize("precision", ["fp32", "bf16"])
def test_iterate_equals_separate_calls(L, precision):
    """lipz_iterate selects inside the fitness kernel; the result must equal, bit for bit, the
    separate eval / select / train calls (mutation on, so the lr path is covered too)."""
    pool = _pool(12, 3000, 784)
    kw = dict(precision=precision, lr_mutation=1, lr_mut_prob=0.5, lr_mut_std=1e-4)
    a = _grid(L, 3, 4, 5, pool, **kw)
    b = _grid(L, 3, 4, 5, pool, **kw)
    for it in range(2):
        a.iterate(1)
        b.eval()
        b.select()
        b.train()
        assert a.export_state() == b.export_state(), it


def test_selection_modes_and_mutation(L):
    pool = _pool(8, 4000, 784)
    g = _grid(L, 3, 4, 8, pool, keep_grads=1, tournament_size=5, replace_mode="always",
              lr_mutation=1, lr_mut_prob=1.0, lr_mut_std=1e-4)
    for _ in range(2):
        s = _to_oracle(g, g.arch)
        data = O.batches(s, pool)
        ev = g.eval()
        sel = g.select()
        ref_sel = O.select_replace(s, {"fG": ev["fG"].astype(np.float64),
                                       "fD": ev["fD"].astype(np.float64)})
        assert np.array_equal(sel["sel_g"], ref_sel["sel_g"])
        assert np.array_equal(sel["sel_g"], np.argmin(ev["fG"], axis=1))
        g.train()
        new = O.train_step(s, ref_sel, data)
        got = _to_oracle(g, g.arch)
        assert np.allclose(got.Glr, new.Glr, rtol=1e-6, atol=1e-12)
        assert np.allclose(got.Dlr, new.Dlr, rtol=1e-6, atol=1e-12)
        assert not np.allclose(got.Glr, 2e-4)


def test_host_batch_iteration(L):
    import lipz_synth
    g = L.Grid(2, 3, seed=5, keep_grads=1)
    g.set_data(_pool(1, 100, 784))
    x = lipz_synth.host_batch(9, 6, 100)
    s = _to_oracle(g, g.arch)
    fg, fd = np.zeros((6, 5), np.float32), np.zeros((6, 5), np.float32)
    L.lipz_iterate_batch(g.h, x, fg, fd)
    data = O.batches(s, None, x)
    ref = O.eval_neighborhoods(s, data)
    assert max_rel(fg, ref["fG"]) < 1e-4 and max_rel(fd, ref["fD"]) < 1e-4
    sel = O.select_replace(s, {"fG": fg.astype(np.float64), "fD": fd.astype(np.float64)})
    new = O.train_step(s, sel, data)
    got = _to_oracle(g, g.arch)
    assert max_rel(got.Dm, new.Dm) < 1e-4


def test_host_batch_pipelined_equals_one_call_at_a_time(L):
    """lipz_iterate_batch_next uploads the next call's minibatch while the current iteration
    runs; a sequence of calls (cycling two pinned buffers, then a call whose x_host is not the
    announced one, then plain calls mixed in) ends in the same state and fitnesses as the same
    minibatches through lipz_iterate_batch, bit for bit."""
    import torch
    import lipz_synth
    pool = _pool(3, 2000, 784)
    a = _grid(L, 3, 3, 12, pool, precision="bf16")
    b = _grid(L, 3, 3, 12, pool, precision="bf16")
    xs = [torch.from_numpy(lipz_synth.host_batch(40 + i, 9, 100)).pin_memory() for i in range(3)]
    order = [0, 1, 0, 1, 2, 0, 1]
    fa = [np.zeros((9, 5), np.float32) for _ in range(2)]
    fb = [np.zeros((9, 5), np.float32) for _ in range(2)]
    for i, k in enumerate(order):
        # call 4 announces xs[0] but is followed by xs[2]; call 5 is a plain call
        nxt = xs[order[i + 1]] if i + 1 < len(order) else None
        if i == 3:
            nxt = xs[0]
        if i == 5:
            L.lipz_iterate_batch(a.h, xs[k], fa[0], fa[1])
        else:
            L.lipz_iterate_batch_next(a.h, xs[k], nxt, fa[0], fa[1])
        L.lipz_iterate_batch(b.h, xs[k], fb[0], fb[1])
        assert np.array_equal(fa[0], fb[0]) and np.array_equal(fa[1], fb[1]), i
    assert a.export_state() == b.export_state()


def test_host_batch_async_equals_one_call_at_a_time(L):
    """lipz_iterate_batch_async runs one call ahead: it enqueues its iteration and returns once
    the previous call's has completed, with that call's fitnesses in its (alternating, pinned)
    result buffers. A sequence of calls (a minibatch announced and then not used, a synchronous
    call in between, lipz_synchronize to finish) gives the same fitnesses and state as the same
    minibatches through lipz_iterate_batch, bit for bit; uploads into a staging buffer wait for
    the iteration that last read it (a call never waits for its own iteration)."""
    import torch
    import lipz_synth
    pool = _pool(3, 2000, 784)
    a = _grid(L, 3, 3, 12, pool, precision="bf16")
    b = _grid(L, 3, 3, 12, pool, precision="bf16")
    xs = [torch.from_numpy(lipz_synth.host_batch(50 + i, 9, 100)).pin_memory() for i in range(3)]
    order = [0, 1, 2, 0, 1, 2, 0, 1, 0]
    res = [[torch.zeros((9, 5), dtype=torch.float32).pin_memory() for _ in range(2)]
           for _ in range(2)]
    ref = []
    fb = [np.zeros((9, 5), np.float32) for _ in range(2)]
    pending = None  # index of the call whose results the next call completes
    for i, k in enumerate(order):
        nxt = xs[order[i + 1]] if i + 1 < len(order) else None
        if i == 4:
            nxt = xs[0]  # announced, then call 5 uses xs[2]: the early upload is dropped
        L.lipz_iterate_batch(b.h, xs[k], fb[0], fb[1])
        ref.append((fb[0].copy(), fb[1].copy()))
        if i == 6:
            # a synchronous call in between completes the pending one first
            L.lipz_iterate_batch(a.h, xs[k], res[i % 2][0], res[i % 2][1])
        else:
            L.lipz_iterate_batch_async(a.h, xs[k], nxt, res[i % 2][0], res[i % 2][1])
        if pending is not None:
            got = res[pending % 2]
            assert np.array_equal(got[0].numpy(), ref[pending][0]), pending
            assert np.array_equal(got[1].numpy(), ref[pending][1]), pending
        pending = None if i == 6 else i
        if i == 6:
            assert np.array_equal(res[0][0].numpy(), ref[6][0])
    L.lipz_synchronize(a.h)
    last = len(order) - 1
    assert np.array_equal(res[last % 2][0].numpy(), ref[last][0])
    assert np.array_equal(res[last % 2][1].numpy(), ref[last][1])
    assert a.export_state() == b.export_state()
    # a non-finite loss of call n is reported by call n + 1 (or by lipz_synchronize)
    s = _to_oracle(a, a.arch)
    s.Dw[2, 5] = np.nan
    a.import_state(O.state_to_bytes(s))
    L.lipz_iterate_batch_async(a.h, xs[0], xs[1], res[0][0], res[0][1])
    with pytest.raises(L.LipzError) as e:
        L.lipz_iterate_batch_async(a.h, xs[1], None, res[1][0], res[1][1])
    assert e.value.code == L.LIPZ_ERR_NONFINITE
    L.lipz_synchronize(a.h)  # drained: nothing left to report
    s.Dw[2, 5] = 0.0
    a.import_state(O.state_to_bytes(s))
    L.lipz_iterate_batch_async(a.h, xs[0], None, res[0][0], res[0][1])
    L.lipz_synchronize(a.h)


def test_determinism_and_resume(L):
    pool = _pool(4, 2000, 784)
    a = _grid(L, 3, 3, 21, pool, precision="bf16")
    b = _grid(L, 3, 3, 21, pool, precision="bf16")
    a.iterate(3)
    b.iterate(2)
    mid = b.export_state()
    c = _grid(L, 3, 3, 999, pool, precision="bf16")
    c.import_state(mid)                 # resume replaces seed and iteration counter too
    b.iterate(1)
    c.iterate(1)
    sa, sb, sc = a.export_state(), b.export_state(), c.export_state()
    assert sa == sb == sc


def test_call_order_and_nonfinite_detection(L):
    pool = _pool(4, 500, 784)
    g = _grid(L, 2, 2, 3, pool)
    with pytest.raises(L.LipzError) as e:
        g.select()
    assert e.value.code == L.LIPZ_ERR_STATE
    g.eval()
    with pytest.raises(L.LipzError) as e:
        g.train()
    assert e.value.code == L.LIPZ_ERR_STATE
    # plant a NaN in cell 2's discriminator through the state interface (a host-side fault)
    s = _to_oracle(g, g.arch)
    s.Dw[2, 5] = np.nan
    g.import_state(O.state_to_bytes(s))
    with pytest.raises(L.LipzError) as e:
        g.eval()
    assert e.value.code == L.LIPZ_ERR_NONFINITE


def test_full_size_12x12_bf16_sampled_cells(L):
    """The benchmark workload (12x12 torus, bf16, B = 100, tensor-core path): two iterations;
    in each, a sample of cells (corners, an interior cell, wrap-around neighbours) against the
    oracle computed cell by cell: losses, fitness, selection (bit-exact), gradients, Adam and
    the updated weights. The gradients come from the stored-gradient path; the fused-Adam path
    that the benchmark runs must leave the same state, bit for bit, at this size."""
    pool = _pool(1811, 60000, 784)
    g = _grid(L, 12, 12, 1811, pool, precision="bf16", keep_grads=1)
    f = _grid(L, 12, 12, 1811, pool, precision="bf16")
    for it, cells in enumerate(([0, 13, 77, 143], [11, 66, 132, 140])):
        _one_iteration_check(L, g, pool, 2e-2, label="bf16 12x12 B=100 it %d" % it, cells=cells)
        f.iterate(1)
        sg, sf = _to_oracle(g, g.arch), _to_oracle(f, f.arch)
        for k in ("Gw", "Gm", "Gv", "Dw", "Dm", "Dv", "Gstep", "Dstep"):
            assert np.array_equal(getattr(sg, k), getattr(sf, k)), (it, k)
    assert np.all(np.isfinite(sg.Gw)) and np.all(np.isfinite(sg.Dw))


def test_bf16_5x5_b256_fifty_iterations_sampled_lockstep(L):
    """5x5 torus, bf16, B = 256, fifty grid iterations; at every fifth iteration and the last
    the engine's state is handed to the oracle and one full iteration is compared (losses,
    fitness, selection bit-exact given the engine's fitness, every cell's gradients, Adam and
    the updated weights); the iterations between run unchecked, so drift of any kind
    accumulates into the checked ones."""
    pool = _pool(2, 60000, 784)
    g = _grid(L, 5, 5, 50, pool, precision="bf16", batch=256, keep_grads=1)
    checked = set(range(0, 50, 5)) | {49}
    for it in range(50):
        if it in checked:
            _one_iteration_check(L, g, pool, 2e-2, label="bf16 5x5 B=256 it %d" % it)
        else:
            g.iterate(1)
    assert g.t == 50
    s = _to_oracle(g, g.arch)
    assert np.all(np.isfinite(s.Gw)) and np.all(np.isfinite(s.Dw))
    assert np.all(s.Gstep >= 1) and np.all(s.Gstep <= 50)


def test_large_grid_20x20_bf16_sampled(L):
    """A 20x20 torus (400 cells, 10,000 pairs per iteration): sampled cells against the oracle,
    then two iterations with bit-exact selection and bounded weight moves."""
    pool = _pool(3, 60000, 784)
    g = _grid(L, 20, 20, 7, pool, precision="bf16")
    for it in range(2):
        s = _to_oracle(g, g.arch)
        cells = [0, 19, 210, 399]
        data = O.batches(s, pool, cells=cells)
        ref = O.eval_neighborhoods(s, data, cells=cells)
        ev = _check_eval(g, s, ref, 2e-2, cells=cells)
        sel = g.select()
        ref_sel = O.select_replace(s, {"fG": ev["fG"].astype(np.float64),
                                       "fD": ev["fD"].astype(np.float64)})
        assert np.array_equal(sel["sel_g"], ref_sel["sel_g"])
        assert np.array_equal(sel["sel_d"], ref_sel["sel_d"])
        g.train()
        got = _to_oracle(g, g.arch)
        nbr = O.neighbors(20, 20)
        src = nbr[np.arange(400), sel["sel_d"]]
        lr = float(np.max(s.Dlr))
        ulp = 2 * np.spacing(np.float32(np.max(np.abs(s.Dw))))
        # Adam moves an element by lr * |m_hat| / (sqrt(v_hat) + eps): at most lr on the first
        # step, at most lr (1 - beta1) / sqrt(1 - beta2) (about 15.8 lr here) afterwards
        bound = lr if it == 0 else lr * (1 - 0.5) / np.sqrt(1 - 0.999)
        assert np.max(np.abs(got.Dw - s.Dw[src])) <= bound * (1 + 1e-5) + ulp
        assert np.all(got.Dstep == s.Dstep[src] + 1)


def _k_step_iteration_check(L, g, pool, tol, label):
    """One iteration with arch.train_steps = K: the selection bit-exact given the engine's own
    fitness, then the state after the K Adam steps against the oracle's: step counts and lrs
    exactly; the last step's gradients and both moments per cell (the worst of the cell's 36
    tensors):
      fp32: every cell within tol, except a cell whose pre-activations came within
        FP32_FLIP_BAND of 0 in one of its K steps (a derivative branch the engine may take the
        other way; at most a quarter of the cells), which stays within the bf16 ceiling;
      bf16: every cell within 5 tol and the median cell within tol (after K steps the worst of
        36 tensors is taken; an error of the method, such as a wrong minibatch, fake slot, step
        count or moment, is of order one).
    A weight of any cell may miss the tolerance only by less than the K Adam moves (about lr
    each) that a near-zero gradient can turn either way, and only rarely."""
    a = oracle_arch(g.arch)
    K = a.train_steps
    s = _to_oracle(g, g.arch)
    data = O.batches(s, pool)
    ev = g.eval()
    sel = g.select()
    ref_sel = O.select_replace(s, {"fG": ev["fG"].astype(np.float64),
                                   "fD": ev["fD"].astype(np.float64)})
    assert np.array_equal(sel["sel_g"], ref_sel["sel_g"])
    assert np.array_equal(sel["sel_d"], ref_sel["sel_d"])
    g.train()
    new, grads = O.train_step(s, ref_sel, data, keep_grads=True, pool=pool)
    got = _to_oracle(g, g.arch)
    assert got.t == s.t + 1
    nbr = O.neighbors(s.rows, s.cols)
    src_g = nbr[np.arange(s.cells), ref_sel["sel_g"]]
    assert np.array_equal(got.Gstep, s.Gstep[src_g] + K) and np.array_equal(got.Gstep, new.Gstep)
    assert np.array_equal(got.Dstep, new.Dstep)
    assert np.allclose(got.Glr, new.Glr, rtol=1e-6) and np.allclose(got.Dlr, new.Dlr, rtol=1e-6)
    gg, gd = g.gradients()
    worst = np.zeros(s.cells)
    pairs = [("G", gg, grads["gG"]), ("D", gd, grads["gD"])]
    for pop in ("G", "D"):
        pairs += [(pop, getattr(got, pop + f), getattr(new, pop + f)) for f in ("m", "v")]
    for pop, gpu, ref in pairs:
        lay = O.g_layout(a) if pop == "G" else O.d_layout(a)
        worst = np.maximum(worst, cell_errors(gpu, ref, lay).max(axis=1))
    ok = worst < tol
    if a.precision == "fp32":
        near = grads["kink"] < FP32_FLIP_BAND
        assert np.all(ok | near), (label, "mismatch without a kink", np.where(~ok)[0], worst)
        assert np.all(worst <= BF16_CEIL * 2e-2), (label, worst)
        assert np.sum(~ok) <= max(1, s.cells // 4), (label, worst)
    else:
        assert np.all(worst < 5 * tol) and np.median(worst) < tol, (label, worst)
    print("PARITY %s cells=%d worst=%.3e median=%.3e" % (label, s.cells, worst.max(),
                                                         np.median(worst)))
    for pop, lay in (("G", O.g_layout(a)), ("D", O.d_layout(a))):
        w_got, w_ref = getattr(got, pop + "w"), getattr(new, pop + "w")
        off, flagged, total = 0, 0, 0
        for name, shape in lay:
            n = int(np.prod(shape))
            d = np.abs(w_got[:, off:off + n] - w_ref[:, off:off + n])
            bad = d > tol * np.max(np.abs(w_ref[:, off:off + n]))
            assert np.all(d[bad] <= 2.5 * K * a.lr), (pop, name, float(np.max(d)))
            flagged += int(bad.sum())
            total += d.size
            off += n
        assert flagged <= max(20, total // 2000), (pop, flagged)


@pytest.mark.parametrize("precision,rows,cols,batch,K", [
    ("fp32", 2, 2, 100, 3),
    ("bf16", 3, 3, 129, 2),
    ("bf16", 2, 3, 100, 4),
])
def test_k_minibatch_steps_against_the_oracle(L, precision, rows, cols, batch, K):
    """train_steps = K: after the selection every cell's new centre pair takes K Adam steps,
    step k >= 1 on a fresh minibatch of the step-k streams. In bf16 the learning rate is 1e-6:
    at 2e-4 the elements whose gradient is at bf16 noise level take Adam moves of either sign
    (about lr each, the same in the one-step check) and those differences feed the next step's
    gradients, so only the first step would be compared at the tolerance."""
    pool = _pool(14, 6000, 784)
    kw = dict(lr_mutation=1, lr_mut_prob=0.5)
    if precision == "bf16":
        kw.update(lr=1e-6, lr_mut_std=1e-7)
    g = _grid(L, rows, cols, 40 + K, pool, precision=precision, batch=batch, keep_grads=1,
              train_steps=K, **kw)
    tol = TOL[g.arch.precision]
    for it in range(2):
        _k_step_iteration_check(L, g, pool, tol, "K=%d %s %dx%d B=%d it %d"
                                % (K, precision, rows, cols, batch, it))


def test_k_minibatch_steps_fused_adam_bit_exact(L):
    """The in-place later steps through the fused-Adam backward equal the stored-gradient path
    bit for bit; K = 1 leaves the default iteration unchanged."""
    pool = _pool(15, 4000, 784)
    a = _grid(L, 3, 3, 17, pool, precision="bf16", train_steps=3)
    b = _grid(L, 3, 3, 17, pool, precision="bf16", train_steps=3, keep_grads=1)
    c = _grid(L, 3, 3, 17, pool, precision="bf16", train_steps=1)
    d = _grid(L, 3, 3, 17, pool, precision="bf16")
    for it in range(2):
        a.iterate(1)
        b.iterate(1)
        c.iterate(1)
        d.iterate(1)
        assert a.export_state() == b.export_state(), it
        assert c.export_state() == d.export_state(), it
    sa = _to_oracle(a, a.arch)
    assert np.all(sa.Gstep >= 6) and np.all(sa.Gstep % 3 == 0)


def test_k_minibatch_steps_need_the_pool(L):
    """Steps k >= 1 draw from the pool: with caller batches and no pool the training call fails
    with LIPZ_ERR_STATE instead of reading unset memory."""
    import lipz_synth
    g = L.Grid(1, 2, seed=3, train_steps=2)
    x = lipz_synth.host_batch(2, 2, 100)
    fg, fd = np.zeros((2, 5), np.float32), np.zeros((2, 5), np.float32)
    with pytest.raises(L.LipzError) as e:
        L.lipz_iterate_batch(g.h, x, fg, fd)
    assert e.value.code == L.LIPZ_ERR_STATE and "pool" in str(e.value)


@pytest.mark.parametrize("rows,cols,batch,stale", [(3, 3, 100, 0), (2, 2, 129, 0), (1, 1, 37, 0),
                                                   (3, 4, 100, 1), (12, 12, 100, 0)])
def test_pair_kernels_equal_one_cta_kernels(L, monkeypatch, rows, cols, batch, stale):
    """The evaluation runs on CTA pairs (two SMs share each weight chunk, M = 256 per MMA);
    LIPZ_FWD_SINGLE=1 at grid creation keeps the one-CTA kernels (M = 128). Both accumulate
    every output in the same order, so the logits, the fitness and the whole iteration agree
    bit for bit: duplicated neighbours (2x2, 1x1), ragged batches and stale neighbours (an
    individual in one or four problems) included."""
    pool = _pool(21, 4000, 784)
    kw = dict(precision="bf16", batch=batch, stale_neighbors=stale)
    a = _grid(L, rows, cols, 5, pool, **kw)
    monkeypatch.setenv("LIPZ_FWD_SINGLE", "1")
    b = _grid(L, rows, cols, 5, pool, **kw)
    monkeypatch.delenv("LIPZ_FWD_SINGLE")
    for it in range(3):
        ea, eb = a.eval(pairs=True), b.eval(pairs=True)
        assert np.array_equal(a.logits(), b.logits()), it
        for k in ("LG", "LD", "fG", "fD"):
            assert np.array_equal(ea[k], eb[k]), (it, k)
        xa, _ = a.batch()
        assert np.all(np.isfinite(xa))
        a.select()
        b.select()
        a.train()
        b.train()
    assert a.export_state() == b.export_state()
