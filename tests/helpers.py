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
