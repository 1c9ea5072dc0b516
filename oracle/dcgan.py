"""CPU oracle for the DCGAN networks of Lipizzaner's CelebA setting (Table 1, DCGAN column).

TEST INFRASTRUCTURE, like ``oracle.lipz_oracle`` (which dispatches here for ``Arch.kind ==
"dcgan"``): only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU arms use it.

The paper gives the DCGAN column of Table 1 only as sizes (input 100, four hidden layers,
64 x 64 x 3 outputs, tanh, batch 128, lr 5e-5); the networks follow the DCGAN architecture of
Radford, Metz and Chintala (ICLR 2016), the one its settings describe:

  G: z (100) -> ConvT 4x4 /1 -> 8g x 4 x 4 -> BN, ReLU -> ConvT 4x4 /2 -> 4g x 8 x 8 -> BN, ReLU
     -> 2g x 16 x 16 -> BN, ReLU -> g x 32 x 32 -> BN, ReLU -> ConvT 4x4 /2 -> 3 x 64 x 64, tanh
  D: 3 x 64 x 64 -> Conv 4x4 /2 -> d x 32 x 32, LeakyReLU(0.2) -> 2d x 16 x 16 -> 4d x 8 x 8
     -> 8d x 4 x 4 (each LeakyReLU) -> Conv 4x4 /1 -> 1 logit

with g = ngf, d = ndf (64 in the 512/256/128/64 configuration), stride-2 layers padded by 1,
no convolution biases, batch normalisation only in the generator, in training mode (the
statistics of the batch it is applied to: one generator slot's B samples), eps 1e-5.
Weights start N(0, 0.02^2), batch-norm scales 1 + N(0, 0.02^2) and shifts 0 (the DCGAN paper's
initialisation). Images are stored channel-major per sample (C, H, W), 12,288 values.

bf16 mode rounds at the same kind of points as the MLP: every operand of a convolution
(weights, input activations, back-propagated deltas) is rounded to bfloat16 and products
accumulate exactly (here: float64); batch normalisation works on the unrounded convolution
output; batch-norm parameters, gradients and optimiser state stay unrounded.

Every convolution is written out from its definition, one kernel tap at a time (a numpy einsum
per (ky, kx)); nothing is blocked or reordered beyond that.
"""

from __future__ import annotations

import math
from typing import Dict, List, Tuple

import numpy as np

BN_EPS = 1e-5
INIT_STD = 0.02

# Accumulation type of every sum (convolutions, batch-norm statistics and their gradients).
# float64 is the oracle. float32 is the same arithmetic summed in another order and precision:
# the spread between the two shows how far an implementation that accumulates in fp32 may land
# from the oracle without any error of method (tests use it to justify their tolerances).
ACC = np.float64


def _a(x):
    return np.asarray(x).astype(ACC, copy=False)


# --------------------------------------------------------------------------------------------
# Parameter layouts (PyTorch conventions: ConvTranspose2d weight [in][out][kh][kw], Conv2d
# weight [out][in][kh][kw]).
# --------------------------------------------------------------------------------------------
def g_layout(a) -> List[Tuple[str, Tuple[int, ...]]]:
    g = a.ngf
    ch = [a.z_dim, 8 * g, 4 * g, 2 * g, g]
    out = []
    for i in range(4):
        out += [("W%d" % (i + 1), (ch[i], ch[i + 1], 4, 4)), ("gamma%d" % (i + 1), (ch[i + 1],)),
                ("beta%d" % (i + 1), (ch[i + 1],))]
    out.append(("W5", (g, 3, 4, 4)))
    return out


def d_layout(a) -> List[Tuple[str, Tuple[int, ...]]]:
    d = a.ndf
    ch = [3, d, 2 * d, 4 * d, 8 * d]
    out = [("W%d" % (i + 1), (ch[i + 1], ch[i], 4, 4)) for i in range(4)]
    out.append(("W5", (1, 8 * d, 4, 4)))
    return out


def init_params(normals: np.ndarray, layout) -> np.ndarray:
    """Flat initial parameters from the flat vector's normals (element k takes normal k):
    weights 0.02 n, batch-norm scales 1 + 0.02 n, shifts 0; stored as float32."""
    flat = np.zeros(len(normals), dtype=np.float64)
    off = 0
    for name, shape in layout:
        n = int(np.prod(shape))
        v = normals[off:off + n]
        if name.startswith("W"):
            flat[off:off + n] = (INIT_STD * v).astype(np.float32)
        elif name.startswith("gamma"):
            flat[off:off + n] = (1.0 + INIT_STD * v).astype(np.float32)
        off += n
    return flat


# --------------------------------------------------------------------------------------------
# Convolutions from their definitions.
# --------------------------------------------------------------------------------------------
def conv2d(x: np.ndarray, w: np.ndarray, s: int, p: int) -> np.ndarray:
    """y[n, o, i, j] = sum_{c, ky, kx} x[n, c, s i - p + ky, s j - p + kx] w[o, c, ky, kx]
    (x read as 0 outside the image)."""
    N, C, H, W = x.shape
    O, _, k, _ = w.shape
    Ho, Wo = (H + 2 * p - k) // s + 1, (W + 2 * p - k) // s + 1
    xp = _a(np.pad(x, ((0, 0), (0, 0), (p, p), (p, p))))
    w = _a(w)
    y = np.zeros((N, O, Ho, Wo), ACC)
    for ky in range(k):
        for kx in range(k):
            win = xp[:, :, ky:ky + s * (Ho - 1) + 1:s, kx:kx + s * (Wo - 1) + 1:s]
            y += np.einsum("nchw,oc->nohw", win, w[:, :, ky, kx], optimize=True)
    return y.astype(np.float64)


def conv2d_backward(x, w, s, p, dy) -> Tuple[np.ndarray, np.ndarray]:
    """Gradients of conv2d with respect to x and w given dL/dy."""
    N, C, H, W = x.shape
    O, _, k, _ = w.shape
    Ho, Wo = dy.shape[2], dy.shape[3]
    xp = _a(np.pad(x, ((0, 0), (0, 0), (p, p), (p, p))))
    w, dy = _a(w), _a(dy)
    dxp = np.zeros_like(xp)
    dw = np.zeros(w.shape, ACC)
    for ky in range(k):
        for kx in range(k):
            sl = (slice(None), slice(None), slice(ky, ky + s * (Ho - 1) + 1, s),
                  slice(kx, kx + s * (Wo - 1) + 1, s))
            dw[:, :, ky, kx] = np.einsum("nohw,nchw->oc", dy, xp[sl], optimize=True)
            dxp[sl] += np.einsum("nohw,oc->nchw", dy, w[:, :, ky, kx], optimize=True)
    return dxp[:, :, p:p + H, p:p + W].astype(np.float64), dw.astype(np.float64)


def conv_transpose2d(x: np.ndarray, w: np.ndarray, s: int, p: int) -> np.ndarray:
    """y[n, o, s i - p + ky, s j - p + kx] += x[n, c, i, j] w[c, o, ky, kx] for every input
    pixel and tap (outputs cropped by p on each side): the adjoint of conv2d."""
    N, C, H, W = x.shape
    _, O, k, _ = w.shape
    Hf, Wf = s * (H - 1) + k, s * (W - 1) + k
    x, w = _a(x), _a(w)
    full = np.zeros((N, O, Hf, Wf), ACC)
    for ky in range(k):
        for kx in range(k):
            full[:, :, ky:ky + s * (H - 1) + 1:s, kx:kx + s * (W - 1) + 1:s] += np.einsum(
                "nchw,co->nohw", x, w[:, :, ky, kx], optimize=True)
    return full[:, :, p:Hf - p, p:Wf - p].astype(np.float64)


def conv_transpose2d_backward(x, w, s, p, dy) -> Tuple[np.ndarray, np.ndarray]:
    """Gradients of conv_transpose2d with respect to x and w given dL/dy."""
    N, C, H, W = x.shape
    _, O, k, _ = w.shape
    Hf, Wf = s * (H - 1) + k, s * (W - 1) + k
    x, w = _a(x), _a(w)
    dfull = np.zeros((N, O, Hf, Wf), ACC)
    dfull[:, :, p:Hf - p, p:Wf - p] = dy
    dx = np.zeros(x.shape, ACC)
    dw = np.zeros(w.shape, ACC)
    for ky in range(k):
        for kx in range(k):
            d = dfull[:, :, ky:ky + s * (H - 1) + 1:s, kx:kx + s * (W - 1) + 1:s]
            dx += np.einsum("nohw,co->nchw", d, w[:, :, ky, kx], optimize=True)
            dw[:, :, ky, kx] = np.einsum("nchw,nohw->co", x, d, optimize=True)
    return dx.astype(np.float64), dw.astype(np.float64)


# --------------------------------------------------------------------------------------------
# Batch normalisation in training mode (Ioffe & Szegedy 2015), per channel over (N, H, W).
# --------------------------------------------------------------------------------------------
def batchnorm(x, gamma, beta):
    mu = _a(x).mean(axis=(0, 2, 3)).astype(np.float64)
    var = _a((x - mu[None, :, None, None]) ** 2).mean(axis=(0, 2, 3)).astype(np.float64)
    inv = 1.0 / np.sqrt(var + BN_EPS)
    xhat = (x - mu[None, :, None, None]) * inv[None, :, None, None]
    return gamma[None, :, None, None] * xhat + beta[None, :, None, None], (xhat, inv)


def batchnorm_backward(dy, gamma, cache):
    xhat, inv = cache
    m = dy.shape[0] * dy.shape[2] * dy.shape[3]
    dbeta = _a(dy).sum(axis=(0, 2, 3)).astype(np.float64)
    dgamma = _a(dy * xhat).sum(axis=(0, 2, 3)).astype(np.float64)
    dx = (gamma * inv)[None, :, None, None] * (
        dy - dbeta[None, :, None, None] / m - xhat * (dgamma / m)[None, :, None, None])
    return dx, dgamma, dbeta


# --------------------------------------------------------------------------------------------
# Networks.
# --------------------------------------------------------------------------------------------
def _lrelu(x, slope):
    return np.where(x > 0.0, x, slope * x)


def g_forward(P: Dict[str, np.ndarray], z: np.ndarray, arch, rb) -> Dict[str, object]:
    """Generator on z [B, z_dim]: fakes F [B, 3 * 64 * 64] (rounded as stored in bf16 mode)
    and what the backward needs."""
    h = z.reshape(z.shape[0], -1, 1, 1)
    cache = []
    for i in range(4):
        s, p = (1, 0) if i == 0 else (2, 1)
        hin = rb(h)
        c = conv_transpose2d(hin, rb(P["W%d" % (i + 1)]), s, p)
        y, bn = batchnorm(c, P["gamma%d" % (i + 1)], P["beta%d" % (i + 1)])
        h = np.maximum(y, 0.0)
        cache.append((hin, c, y, bn))
    hin = rb(h)
    F = rb(np.tanh(conv_transpose2d(hin, rb(P["W5"]), 2, 1)))
    return {"F": F.reshape(F.shape[0], -1), "cache": cache, "h4": hin}


def d_forward(P: Dict[str, np.ndarray], X: np.ndarray, arch, rb) -> Dict[str, object]:
    """Discriminator on X [N, 3 * 64 * 64] (rows as stored): logits [N] and the layer inputs."""
    a = X.reshape(X.shape[0], 3, 64, 64)
    ins, pre = [], []
    for i in range(4):
        ain = rb(a)
        c = conv2d(ain, rb(P["W%d" % (i + 1)]), 2, 1)
        ins.append(ain)
        pre.append(c)
        a = _lrelu(c, arch.leaky_slope)
    ain = rb(a)
    ins.append(ain)
    logit = conv2d(ain, rb(P["W5"]), 1, 0).reshape(-1)
    return {"logit": logit, "ins": ins, "pre": pre}


def d_backward(P, fd, dlogit, arch, rb, need_dx: bool):
    """Back-propagation of dL/dlogit [N] through the discriminator: weight gradients and, with
    need_dx, dL/dX [N, 3, 64, 64]. Deltas enter each convolution rounded (bf16 mode)."""
    N = dlogit.shape[0]
    grads = {}
    d = rb(dlogit.reshape(N, 1, 1, 1))
    dx, grads["W5"] = conv2d_backward(fd["ins"][4], rb(P["W5"]), 1, 0, d)
    for i in range(3, -1, -1):
        d = rb(dx * np.where(fd["pre"][i] > 0.0, 1.0, arch.leaky_slope))
        if i == 0 and not need_dx:
            _, grads["W1"] = conv2d_backward(fd["ins"][0], rb(P["W1"]), 2, 1, d)
            dx = None
        else:
            dx, grads["W%d" % (i + 1)] = conv2d_backward(fd["ins"][i], rb(P["W%d" % (i + 1)]),
                                                         2, 1, d)
    return grads, dx


def pair_gradients(Gflat, Dflat, x, z, arch, rb, unflatten, pair_losses, sigmoid):
    """dL_D/dv (fake batch detached) and dL_G/du through D at its pre-update parameters, for one
    generator-discriminator pair on one minibatch (real rows x [B, 12288], noise z [B, z_dim])."""
    gl, dl = g_layout(arch), d_layout(arch)
    G, D = unflatten(Gflat, gl), unflatten(Dflat, dl)
    B = x.shape[0]
    fg = g_forward(G, z, arch, rb)
    X = rb(np.vstack([x, fg["F"]]))
    fd = d_forward(D, X, arch, rb)
    logit = fd["logit"]
    sg = sigmoid(logit)
    dl_d = np.concatenate([(sg[:B] - 1.0) / B, sg[B:] / B])
    dl_g = (sg[B:] - 1.0) / B
    gD, _ = d_backward(D, fd, dl_d, arch, rb, need_dx=False)
    # the generator's loss through D's fake rows
    fd_fake = {"ins": [a[B:] for a in fd["ins"]], "pre": [c[B:] for c in fd["pre"]]}
    _, dF = d_backward(D, fd_fake, dl_g, arch, rb, need_dx=True)
    F = fg["F"].reshape(B, 3, 64, 64)
    d = rb(dF * (1.0 - F * F))
    gG = {}
    dh, gG["W5"] = conv_transpose2d_backward(fg["h4"], rb(G["W5"]), 2, 1, d)
    kink = math.inf
    for i in range(3, -1, -1):
        hin, c, y, bn = fg["cache"][i]
        dy = dh * (y > 0.0)
        dc, gG["gamma%d" % (i + 1)], gG["beta%d" % (i + 1)] = batchnorm_backward(
            dy, G["gamma%d" % (i + 1)], bn)
        s, p = (1, 0) if i == 0 else (2, 1)
        dh, gG["W%d" % (i + 1)] = conv_transpose2d_backward(hin, rb(G["W%d" % (i + 1)]), s, p,
                                                            rb(dc))
        kink = min(kink, float(np.min(np.abs(y))))
    for c in fd["pre"]:
        kink = min(kink, float(np.min(np.abs(c))))
    lg, ld = pair_losses(logit[:B], logit[B:])
    flatG = np.concatenate([gG[n].reshape(-1) for n, _ in gl])
    flatD = np.concatenate([gD[n].reshape(-1) for n, _ in dl])
    return flatG, flatD, {"LG": lg, "LD": ld, "kink": kink}
