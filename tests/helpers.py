"""Shared test helpers: engine <-> oracle state conversion and tolerance checks."""

import numpy as np

from oracle import lipz_oracle as O


def oracle_arch(arch) -> O.Arch:
    """The oracle's Arch for an engine lipz_arch."""
    return O.Arch(z_dim=arch.z_dim, hidden=arch.hidden, x_dim=arch.x_dim, batch=arch.batch,
                  precision="bf16" if arch.precision == 1 else "fp32", lr=float(arch.lr),
                  beta1=float(arch.beta1), beta2=float(arch.beta2), eps=float(arch.eps),
                  tournament_size=arch.tournament_size,
                  replace_mode="always" if arch.replace_mode == 1 else "if_better",
                  lr_mutation=bool(arch.lr_mutation), lr_mut_std=float(arch.lr_mut_std),
                  lr_mut_prob=float(arch.lr_mut_prob), leaky_slope=float(arch.leaky_slope),
                  train_steps=int(arch.train_steps), mixture=bool(arch.mixture),
                  mix_sigma=float(arch.mix_sigma),
                  stale_neighbors=bool(arch.stale_neighbors),
                  kind="dcgan" if arch.kind == 1 else "mlp", ngf=int(arch.ngf),
                  ndf=int(arch.ndf))


def max_rel(got, ref) -> float:
    """Max-norm relative error max|got - ref| / max|ref| (0 if both are all zero)."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.max(np.abs(ref)) if ref.size else 0.0
    num = np.max(np.abs(got - ref)) if ref.size else 0.0
    if den == 0.0:
        return float(num)
    return float(num / den)


def per_tensor(flat_got, flat_ref, layout):
    """max_rel per named tensor of flat parameter vectors ([cells, P])."""
    out = {}
    off = 0
    for name, shape in layout:
        n = int(np.prod(shape))
        out[name] = max_rel(flat_got[..., off:off + n], flat_ref[..., off:off + n])
        off += n
    return out


# ---- gradient parity ----------------------------------------------------------------------
# ReLU / LeakyReLU derivatives jump at 0. An engine that rounds a pre-activation differently
# from the float64 oracle takes the other branch wherever that pre-activation lies within its
# rounding distance of 0, and the difference in that one derivative moves every gradient fed
# by the element's batch row (by up to a few 1e-2 of the tensor's largest value).
#
# fp32: the engine's pre-activations differ from the oracle's by fp32 accumulation error
# (below 1e-6 at these sizes), so only elements within FP32_FLIP_BAND of 0 can flip (a few
# tenths of an element per cell). A cell that misses the tolerance is compared again with the
# oracle's gradients for every choice of branches at those elements (pair_gradients(flip=)),
# and must meet the tolerance under one of them.
#
# bf16: the operands of every product are rounded to bf16, and a value that lands on the other
# side of a rounding boundary moves the next pre-activations by up to ~1e-3, so hundreds of
# elements per cell can flip and no enumeration is possible. The oracle itself, with float32
# instead of float64 products and otherwise the same code, differs from the float64 oracle by
# up to 2e-2 in a few cells (median 1e-3). The rule is an error budget: every cell within
# BF16_CEIL x tol, at most a quarter of the cells (at least two) above tol, and the median cell
# within
# BF16_MEDIAN x tol (the engine's medians lie at 1e-3 to 5e-3). A method error (a wrong row,
# cell, slot or tile tail) is of order one.
FP32_FLIP_BAND = 2e-6
MAX_FLIPS = 8
BF16_CEIL = 2.5
BF16_MEDIAN = 0.35


def cell_errors(gpu, ref, layout):
    """[cells, tensors] max-norm relative error of each cell's named tensors."""
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    out, off = [], 0
    for _, shape in layout:
        n = int(np.prod(shape))
        d = np.max(np.abs(gpu[:, off:off + n] - ref[:, off:off + n]), axis=1)
        den = np.max(np.abs(ref[:, off:off + n]), axis=1)
        out.append(np.where(den > 0, d / np.where(den > 0, den, 1.0), d))
        off += n
    return np.stack(out, axis=1)


def _flip_variants(a, Gf, Df, x, z):
    """The oracle's gradients for every choice of derivative branch at the pre-activations
    within FP32_FLIP_BAND of 0 (none flipped first)."""
    import itertools
    pre = O.pair_gradients(Gf, Df, x, z, a)[2]["pre"]
    near = [(k, idx) for k, p in pre.items() for idx in zip(*np.nonzero(np.abs(p) < FP32_FLIP_BAND))]
    assert len(near) <= MAX_FLIPS, ("too many pre-activations at a kink", len(near))
    for n in range(1, len(near) + 1):
        for sub in itertools.combinations(near, n):
            flip = {k: np.zeros(p.shape, bool) for k, p in pre.items()}
            for k, idx in sub:
                flip[k][idx] = True
            gG, gD, _ = O.pair_gradients(Gf, Df, x, z, a, flip=flip)
            yield gG, gD


def gradient_parity(label, a, gg, gd, refG, refD, tol, pair_inputs):
    """Checks the engine's gradients gg, gd [cells, P] against the oracle's refG, refD by the
    rules above; pair_inputs(c) -> (G params, D params, x, z) of the cell's selected pair.
    Returns the accepted reference gradients (a flipped variant where fp32 needed one) and the
    per-cell worst errors."""
    gl, dl = O.g_layout(a), O.d_layout(a)
    refG, refD = np.array(refG, np.float64), np.array(refD, np.float64)
    err = np.concatenate([cell_errors(gg, refG, gl), cell_errors(gd, refD, dl)], axis=1)
    worst = err.max(axis=1)
    names = ["G" + n for n, _ in gl] + ["D" + n for n, _ in dl]
    if a.precision == "fp32":
        for c in np.nonzero(worst >= tol)[0]:
            Gf, Df, x, z = pair_inputs(int(c))
            for vG, vD in _flip_variants(a, Gf, Df, x, z):
                e = np.concatenate([cell_errors(gg[c:c + 1], vG[None], gl),
                                    cell_errors(gd[c:c + 1], vD[None], dl)], axis=1)[0]
                if e.max() < tol:
                    refG[c], refD[c], worst[c], err[c] = vG, vD, e.max(), e
                    break
            else:
                raise AssertionError((label, "cell", int(c), "misses the tolerance under every "
                                      "branch choice", dict(zip(names, err[c]))))
    else:
        assert np.all(worst <= BF16_CEIL * tol), (label, "ceiling", worst)
        assert np.sum(worst > tol) <= max(2, len(worst) // 4), (label, "count", worst)
        assert np.median(worst) <= BF16_MEDIAN * tol, (label, "median", worst)
    print("PARITY %s cells=%d worst=%.3e median=%.3e per-tensor-max {%s}" % (
        label, len(worst), worst.max(), np.median(worst),
        ", ".join("%s: %.1e" % (n, v) for n, v in zip(names, err.max(axis=0)))))
    return refG, refD, worst
