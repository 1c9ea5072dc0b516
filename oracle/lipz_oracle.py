"""CPU oracle for one grid iteration of Lipizzaner's coevolutionary GAN training.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU
baseline / reference arm may import or run this module. The product path (the CUDA library
and its Python binding) never calls it, and this module never imports the product.

What it computes follows the method section of arXiv 1811.12843 (Section 3, "Coevolutionary GAN
Training", steps 1-3 and 5) and its settings table (Table 1), written as plain numpy in float64:

  1. every cell of an R x C toroidal grid holds one generator (params u_i, learning rate delta_i)
     and one discriminator (v_j, gamma_j), randomly initialised (step 1);
  2. each generator is evaluated against each discriminator of its cell's 5-cell von Neumann
     neighbourhood (centre, N, S, W, E; Section 2 "Scaling Evolutionary Computing for ML"),
     L(u_i, v_j) on one minibatch; a discriminator's fitness averages its interactions, a
     generator's averages its own (step 2);
  3. size-2 tournament selection in each neighbourhood, then one gradient (Adam) update of the
     selected pair, with optional Gaussian mutation of the learning rate (step 3, Table 1).

Readings where the paper is silent (each with its reason in the design notes):
  * fitness is a loss for both populations, lower is better: f_G = mean_j L_G, f_D = mean_i L_D;
  * L_D is the SUM of the real-batch and fake-batch BCE means; L_G is the non-saturating loss;
  * iterations run on a synchronous snapshot of all centres; with ``stale_neighbors`` (the
    asynchronous schedule of Section 3 emulated deterministically) a cell sees its own centre
    as of the iteration and its four neighbours as they were one iteration earlier (at the
    first iteration: as they are), both for the evaluation and as selection sources;
  * tournament entrants are distinct slots; a tie goes to the lower slot; the centre is replaced
    by the winner only if the winner's fitness is strictly lower (``if_better``) -- or always;
  * the pair is trained on the same minibatch that was used for its evaluation, with the fake
    batch detached for the discriminator gradient and both gradients taken at the pre-update
    parameters; one Adam step (Kingma & Ba 2015, Algorithm 1) per iteration by default;
  * with ``train_steps`` K > 1 (an iteration read as an epoch of K minibatch steps, Section 4's
    footnote equating iteration, generation and epoch), steps k = 1..K-1 train the cell's new
    centre pair again, each on a fresh minibatch drawn from the step-k streams (stream id +
    256 k); selection and lr mutation happen once, before step 0;
  * random draws come from Philox4x32-10 (Salmon et al., SC'11) keyed by the seed, with the
    counter (block index, cell, iteration, stream);
  * mixture weights (step 4): one ES-(1+1) step per iteration on each cell's weights w over its
    five neighbourhood generators, scored, in place of FID (no Inception network here), by the
    squared maximum mean discrepancy (Gretton et al., JMLR 2012) with the Gaussian kernel
    exp(-||a - b||^2 / x_dim) between the w-weighted fakes of the evaluation and the real
    minibatch (the same rows the discriminators saw in step 2); a mutation adds sigma N(0, 1)
    to every weight, clips at 0 and renormalises, and is kept only if it lowers the score;
  * in bf16 mode every operand of a matrix product (weights, activations, back-propagated
    deltas) is rounded to bfloat16 (round to nearest even), products accumulate exactly (here:
    float64), biases, logits, losses, gradients and optimiser state stay unrounded.

Parity of the whole iteration against the paper is pinned only through its pieces (Philox
known-answer vectors, torus invariants, the ln 2 BCE case, finite-difference gradients, Adam's
closed-form first step, torch cross-checks, exhaustive tournament checks); see tests/.
"""

from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Tuple

import numpy as np

# --------------------------------------------------------------------------------------------
# Counter-based random numbers: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random
# numbers: as easy as 1, 2, 3", SC'11). Multipliers and Weyl key increments are the ones that
# paper publishes for the 4x32 variant.
# --------------------------------------------------------------------------------------------
_PHILOX_M0 = np.uint64(0xD2511F53)
_PHILOX_M1 = np.uint64(0xCD9E8D57)
_PHILOX_W0 = 0x9E3779B9
_PHILOX_W1 = 0xBB67AE85
_MASK32 = np.uint64(0xFFFFFFFF)

# Stream ids (the fourth counter word); part of the library's documented contract.
STREAM_INIT_G = 1
STREAM_INIT_D = 2
STREAM_BATCH = 3
STREAM_NOISE = 4
STREAM_TOUR_G = 5
STREAM_TOUR_D = 6
STREAM_MUT_G = 7
STREAM_MUT_D = 8
STREAM_MIX = 9
# Minibatch step k of an iteration draws from stream id + STEP_STREAM_STRIDE * k.
STEP_STREAM_STRIDE = 256


def philox4x32_10(ctr: np.ndarray, key: Tuple[int, int]) -> np.ndarray:
    """Ten Philox rounds on counters ``ctr`` ([..., 4] of 32-bit values) with key (k0, k1).

    One round: the products M0*c0 and M1*c2 are split into high/low halves; the new counter is
    (hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0). The key is bumped by the Weyl constants between
    rounds.
    """
    ctr = np.asarray(ctr, dtype=np.uint64)
    c0, c1, c2, c3 = (ctr[..., i].copy() for i in range(4))
    k0, k1 = int(key[0]) & 0xFFFFFFFF, int(key[1]) & 0xFFFFFFFF
    for rnd in range(10):
        if rnd:
            k0 = (k0 + _PHILOX_W0) & 0xFFFFFFFF
            k1 = (k1 + _PHILOX_W1) & 0xFFFFFFFF
        p0 = _PHILOX_M0 * c0
        p1 = _PHILOX_M1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        c0, c1, c2, c3 = hi1 ^ c1 ^ np.uint64(k0), lo1, hi0 ^ c3 ^ np.uint64(k1), lo0
    return np.stack([c0, c1, c2, c3], axis=-1)


def draw_words(seed: int, stream: int, t: int, cell: int, n: int) -> np.ndarray:
    """The first ``n`` 32-bit words of the (stream, t, cell) sequence: word k is output word
    k % 4 of the Philox block with counter (k // 4, cell, t, stream), key = (seed lo, seed hi)."""
    nb = (n + 3) // 4
    ctr = np.zeros((nb, 4), dtype=np.uint64)
    ctr[:, 0] = np.arange(nb, dtype=np.uint64)
    ctr[:, 1] = cell
    ctr[:, 2] = t
    ctr[:, 3] = stream
    out = philox4x32_10(ctr, (seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF))
    return out.reshape(-1)[:n]


def mulhi(w: np.ndarray, n: int) -> np.ndarray:
    """floor(w * n / 2^32): maps a uniform 32-bit word onto {0, .., n-1} without floats."""
    return (np.asarray(w, dtype=np.uint64) * np.uint64(n)) >> np.uint64(32)


def box_muller(wa: np.ndarray, wb: np.ndarray) -> Tuple[np.ndarray, np.ndarray]:
    """Two standard normals from two words (Box & Muller 1958): u1 = (top 24 bits + 1) / 2^24 in
    (0, 1], v = (top 24 bits) / 2^24 in [0, 1); r = sqrt(-2 ln u1); (r cos 2 pi v, r sin 2 pi v)."""
    u1 = ((np.asarray(wa, dtype=np.uint64) >> np.uint64(8)).astype(np.float64) + 1.0) * 2.0 ** -24
    v = (np.asarray(wb, dtype=np.uint64) >> np.uint64(8)).astype(np.float64) * 2.0 ** -24
    r = np.sqrt(-2.0 * np.log(u1))
    return r * np.cos(2.0 * math.pi * v), r * np.sin(2.0 * math.pi * v)


def draw_normals(seed: int, stream: int, t: int, cell: int, n: int) -> np.ndarray:
    """``n`` normals: block i's words (w0, w1, w2, w3) give normals 4i..4i+3 as
    box_muller(w0, w1) followed by box_muller(w2, w3)."""
    nb = (n + 3) // 4
    w = draw_words(seed, stream, t, cell, 4 * nb).reshape(nb, 4)
    out = np.empty((nb, 4), dtype=np.float64)
    out[:, 0], out[:, 1] = box_muller(w[:, 0], w[:, 1])
    out[:, 2], out[:, 3] = box_muller(w[:, 2], w[:, 3])
    return out.reshape(-1)[:n]


# --------------------------------------------------------------------------------------------
# Configuration (Table 1 for the MLP/MNIST column) and parameter layout.
# --------------------------------------------------------------------------------------------
@dataclasses.dataclass
class Arch:
    z_dim: int = 64          # input neurons (Table 1)
    hidden: int = 256        # neurons per hidden layer, 2 hidden layers (Table 1)
    x_dim: int = 784         # output neurons (Table 1)
    batch: int = 100         # batch size (Table 1)
    precision: str = "fp32"  # "fp32" or "bf16"
    lr: float = 2e-4         # initial learning rate (Table 1)
    beta1: float = 0.5
    beta2: float = 0.999
    eps: float = 1e-8
    tournament_size: int = 2  # Table 1
    replace_mode: str = "if_better"  # or "always"
    lr_mutation: bool = False
    lr_mut_std: float = 1e-4  # mutation rate (Table 1)
    lr_mut_prob: float = 0.5  # mutation probability (Table 1)
    leaky_slope: float = 0.2
    train_steps: int = 1      # Adam steps of the new centre pair per iteration
    mixture: bool = False     # evolve each neighbourhood's generator-mixture weights
    stale_neighbors: bool = False  # neighbours seen one iteration late (asynchronous cells)
    mix_sigma: float = 0.01   # mixture mutation scale (Table 1)
    kind: str = "mlp"         # "mlp" (Table 1, MNIST column) or "dcgan" (CelebA column)
    ngf: int = 64             # DCGAN generator width (channels 8g, 4g, 2g, g)
    ndf: int = 64             # DCGAN discriminator width (channels d, 2d, 4d, 8d)


def g_layout(a: Arch) -> List[Tuple[str, Tuple[int, ...]]]:
    """Generator tensors in storage order; weights are [out][in] row-major."""
    if a.kind == "dcgan":
        return _dcgan().g_layout(a)
    return [("W1", (a.hidden, a.z_dim)), ("b1", (a.hidden,)),
            ("W2", (a.hidden, a.hidden)), ("b2", (a.hidden,)),
            ("W3", (a.x_dim, a.hidden)), ("b3", (a.x_dim,))]


def d_layout(a: Arch) -> List[Tuple[str, Tuple[int, ...]]]:
    """Discriminator tensors in storage order; weights are [out][in] row-major."""
    if a.kind == "dcgan":
        return _dcgan().d_layout(a)
    return [("W1", (a.hidden, a.x_dim)), ("b1", (a.hidden,)),
            ("W2", (a.hidden, a.hidden)), ("b2", (a.hidden,)),
            ("W3", (1, a.hidden)), ("b3", (1,))]


def _dcgan():
    from oracle import dcgan
    return dcgan


def n_params(layout) -> int:
    return sum(int(np.prod(s)) for _, s in layout)


def unflatten(flat: np.ndarray, layout) -> Dict[str, np.ndarray]:
    """Views of the named tensors inside one flat parameter vector."""
    out, off = {}, 0
    for name, shape in layout:
        n = int(np.prod(shape))
        out[name] = flat[off:off + n].reshape(shape)
        off += n
    return out


def neighbors(rows: int, cols: int) -> np.ndarray:
    """nbr[c] = (centre, north, south, west, east) on the torus, cells numbered r * cols + col.
    Duplicates are kept (a 1x1 grid has the centre in all five slots)."""
    nbr = np.empty((rows * cols, 5), dtype=np.int64)
    for r in range(rows):
        for q in range(cols):
            nbr[r * cols + q] = [r * cols + q,
                                 ((r - 1) % rows) * cols + q,
                                 ((r + 1) % rows) * cols + q,
                                 r * cols + (q - 1) % cols,
                                 r * cols + (q + 1) % cols]
    return nbr


def xavier_bound(fan_in: int, fan_out: int) -> np.float32:
    """Glorot & Bengio (2010) uniform bound sqrt(6 / (fan_in + fan_out)), stored as float32."""
    return np.float32(math.sqrt(6.0 / (fan_in + fan_out)))


def init_params(seed: int, stream: int, cell: int, layout) -> np.ndarray:
    """Step 1: random weights. Element k of a weight tensor takes word k of the flat vector's
    sequence: s = word >> 8, q = (2 s + 1 - 2^24) / 2^24 in (-1, 1), w = float32(a * q) with a the
    tensor's Xavier bound. Biases start at zero."""
    total = n_params(layout)
    words = draw_words(seed, stream, 0, cell, total)
    flat = np.zeros(total, dtype=np.float64)
    off = 0
    for name, shape in layout:
        n = int(np.prod(shape))
        if name.startswith("W"):
            s = (words[off:off + n] >> np.uint64(8)).astype(np.float64)
            q = (2.0 * s + 1.0 - 2.0 ** 24) * 2.0 ** -24
            a = float(xavier_bound(shape[1], shape[0]))
            flat[off:off + n] = (a * q).astype(np.float32)
        off += n
    return flat


# --------------------------------------------------------------------------------------------
# Arithmetic helpers.
# --------------------------------------------------------------------------------------------
def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bfloat16 value (8 significant bits), ties to even."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)
    return np.ldexp(np.round(m * 256.0), e - 8)


def softplus(x: np.ndarray) -> np.ndarray:
    """log(1 + e^x), written max(x, 0) + log1p(e^-|x|) so that it never overflows."""
    return np.maximum(x, 0.0) + np.log1p(np.exp(-np.abs(x)))


def sigmoid(x: np.ndarray) -> np.ndarray:
    return 0.5 * (1.0 + np.tanh(0.5 * x))


class _Rounder:
    def __init__(self, arch: Arch):
        if arch.precision not in ("fp32", "bf16"):
            raise ValueError("precision must be fp32 or bf16")
        self.bf16 = arch.precision == "bf16"

    def __call__(self, x):
        return round_bf16(x) if self.bf16 else np.asarray(x, dtype=np.float64)


def g_forward(P: Dict[str, np.ndarray], z: np.ndarray, arch: Arch) -> Dict[str, np.ndarray]:
    """Generator MLP: z -> ReLU(256) -> ReLU(256) -> tanh(784). Returns every activation."""
    rb = _Rounder(arch)
    if arch.kind == "dcgan":
        return _dcgan().g_forward(P, z, arch, rb)
    zq = rb(z)
    h1 = rb(np.maximum(zq @ rb(P["W1"]).T + P["b1"], 0.0))
    h2 = rb(np.maximum(h1 @ rb(P["W2"]).T + P["b2"], 0.0))
    F = rb(np.tanh(h2 @ rb(P["W3"]).T + P["b3"]))
    return {"z": zq, "h1": h1, "h2": h2, "F": F}


def _lrelu(x, slope):
    return np.where(x > 0.0, x, slope * x)


def d_forward(P: Dict[str, np.ndarray], X: np.ndarray, arch: Arch) -> Dict[str, np.ndarray]:
    """Discriminator MLP: x -> LeakyReLU(256) -> LeakyReLU(256) -> logit (sigmoid in the loss)."""
    rb = _Rounder(arch)
    if arch.kind == "dcgan":
        return _dcgan().d_forward(P, X, arch, rb)
    Xq = rb(X)
    g1 = rb(_lrelu(Xq @ rb(P["W1"]).T + P["b1"], arch.leaky_slope))
    g2 = rb(_lrelu(g1 @ rb(P["W2"]).T + P["b2"], arch.leaky_slope))
    logit = g2 @ rb(P["W3"])[0] + P["b3"][0]
    return {"X": Xq, "g1": g1, "g2": g2, "logit": logit}


def pair_losses(logit_real: np.ndarray, logit_fake: np.ndarray) -> Tuple[float, float]:
    """L_D = mean BCE(D(x), 1) + mean BCE(D(G(z)), 0);  L_G = mean BCE(D(G(z)), 1).
    With sigmoid outputs, BCE(l, 1) = softplus(-l) and BCE(l, 0) = softplus(l)."""
    ld = float(np.mean(softplus(-logit_real)) + np.mean(softplus(logit_fake)))
    lg = float(np.mean(softplus(-logit_fake)))
    return lg, ld


# --------------------------------------------------------------------------------------------
# Grid state.
# --------------------------------------------------------------------------------------------
@dataclasses.dataclass
class State:
    rows: int
    cols: int
    arch: Arch
    seed: int
    t: int
    Gw: np.ndarray   # [cells, PG] parameters (float64 holding float32 values after init)
    Gm: np.ndarray
    Gv: np.ndarray
    Gstep: np.ndarray  # [cells] int64
    Glr: np.ndarray    # [cells]
    Dw: np.ndarray
    Dm: np.ndarray
    Dv: np.ndarray
    Dstep: np.ndarray
    Dlr: np.ndarray
    mix: np.ndarray = None  # [cells, 5] generator-mixture weights of each neighbourhood

    @property
    def cells(self) -> int:
        return self.rows * self.cols

    def copy(self) -> "State":
        return dataclasses.replace(self, **{f: getattr(self, f).copy() for f in
                                            ("Gw", "Gm", "Gv", "Gstep", "Glr",
                                             "Dw", "Dm", "Dv", "Dstep", "Dlr", "mix")})


def create(rows: int, cols: int, arch: Arch, seed: int) -> State:
    """Step 1 for every cell: Xavier weights, zero biases and moments, lr = arch.lr, step 0."""
    if rows < 1 or cols < 1:
        raise ValueError("grid needs rows, cols >= 1")
    gl, dl = g_layout(arch), d_layout(arch)
    cells = rows * cols
    if arch.kind == "dcgan":
        # weights N(0, 0.02^2) and batch-norm scales 1 + N(0, 0.02^2) from the normals of the
        # cell's init stream (normal k for flat element k)
        init = lambda stream, c, lay: _dcgan().init_params(
            draw_normals(seed, stream, 0, c, n_params(lay)), lay)
    else:
        init = lambda stream, c, lay: init_params(seed, stream, c, lay)
    Gw = np.stack([init(STREAM_INIT_G, c, gl) for c in range(cells)])
    Dw = np.stack([init(STREAM_INIT_D, c, dl) for c in range(cells)])
    lr = float(np.float32(arch.lr))
    return State(rows, cols, arch, seed, 0,
                 Gw, np.zeros_like(Gw), np.zeros_like(Gw), np.zeros(cells, np.int64),
                 np.full(cells, lr), Dw, np.zeros_like(Dw), np.zeros_like(Dw),
                 np.zeros(cells, np.int64), np.full(cells, lr), np.full((cells, 5), 0.2))


def draw_batch(seed: int, t: int, cell: int, pool: np.ndarray, arch: Arch, step: int = 0
               ) -> Tuple[np.ndarray, np.ndarray]:
    """Cell ``cell``'s minibatch at iteration ``t``, minibatch step ``step``: B pool rows at
    indices mulhi(word_b, n) (stream BATCH + 256 step) and z = B x z_dim normals (stream
    NOISE + 256 step), row-major."""
    off = STEP_STREAM_STRIDE * step
    w = draw_words(seed, STREAM_BATCH + off, t, cell, arch.batch)
    idx = mulhi(w, pool.shape[0]).astype(np.int64)
    x = pool[idx].astype(np.float64)
    z = draw_normals(seed, STREAM_NOISE + off, t, cell, arch.batch * arch.z_dim)
    return x, z.reshape(arch.batch, arch.z_dim)


def batches(state: State, pool: Optional[np.ndarray], x_host: Optional[np.ndarray] = None,
            cells=None):
    """Per-cell (x, z) for the state's current iteration. ``x_host`` ([cells, B, x_dim]) replaces
    the pool draw when the caller supplies the real minibatches itself. With ``cells``, only
    those cells' batches are drawn (the others are None)."""
    a = state.arch
    out = []
    for c in range(state.cells):
        if cells is not None and c not in cells:
            out.append(None)
        elif x_host is not None:
            z = draw_normals(state.seed, STREAM_NOISE, state.t, c, a.batch * a.z_dim)
            out.append((np.asarray(x_host[c], np.float64), z.reshape(a.batch, a.z_dim)))
        else:
            out.append(draw_batch(state.seed, state.t, c, pool, a))
    return out


# --------------------------------------------------------------------------------------------
# Step 2: all-pairs evaluation and fitness.
# --------------------------------------------------------------------------------------------
def _slot_state(state: State, prev: Optional[State], s: int) -> State:
    """The snapshot slot ``s`` of a neighbourhood is read from: the cell's own centre (s = 0)
    from ``state``; the neighbours from ``prev`` when given (stale neighbours), else ``state``."""
    return state if (s == 0 or prev is None) else prev


def eval_neighborhoods(state: State, data, cells=None, prev: Optional[State] = None
                       ) -> Dict[str, np.ndarray]:
    """For each cell c and slots (i, j): generator nbr[c][i] against discriminator nbr[c][j] on
    cell c's minibatch. Returns L_G, L_D [cells, 5(i), 5(j)], fitness f_G = mean_j L_G[c, i, :],
    f_D = mean_i L_D[c, :, j], and the logits [cells, 5(j), 6B] (real rows, then the fakes of
    generator slots 0..4). With ``cells``, only those cells are evaluated (others stay 0). With
    ``prev``, the neighbour slots 1..4 hold ``prev``'s individuals (stale neighbours)."""
    a = state.arch
    gl, dl = g_layout(a), d_layout(a)
    nbr = neighbors(state.rows, state.cols)
    only = cells
    cells, B = state.cells, a.batch
    LG = np.zeros((cells, 5, 5))
    LD = np.zeros((cells, 5, 5))
    logits = np.zeros((cells, 5, 6 * B))
    for c in (range(cells) if only is None else only):
        x, z = data[c]
        fakes = [g_forward(unflatten(_slot_state(state, prev, i).Gw[nbr[c][i]], gl), z, a)["F"]
                 for i in range(5)]
        X = np.vstack([x] + fakes)
        for j in range(5):
            lg = d_forward(unflatten(_slot_state(state, prev, j).Dw[nbr[c][j]], dl), X,
                           a)["logit"]
            logits[c, j] = lg
            for i in range(5):
                LG[c, i, j], LD[c, i, j] = pair_losses(lg[:B], lg[B * (i + 1):B * (i + 2)])
    return {"LG": LG, "LD": LD, "fG": LG.mean(axis=2), "fD": LD.mean(axis=1), "logits": logits}


# --------------------------------------------------------------------------------------------
# Step 4: generator-mixture weights, ES-(1+1).
# --------------------------------------------------------------------------------------------
def mixture_blocks(X: np.ndarray, B: int) -> np.ndarray:
    """S[a][b] = mean of the Gaussian kernel exp(-||X_r - X_s||^2 / dim) over the rows r of block
    a and s of block b, blocks of B rows (block 0 the real rows, block 1 + i the fakes of
    generator slot i)."""
    X = np.asarray(X, np.float64)
    n, dim = X.shape
    K = np.empty((n, n))
    for r in range(n):
        K[r] = np.exp(-((X - X[r]) ** 2).sum(axis=1) / dim)
    nb = n // B
    S = np.empty((nb, nb))
    for a in range(nb):
        for b in range(nb):
            S[a, b] = K[a * B:(a + 1) * B, b * B:(b + 1) * B].mean()
    return S


def mmd2(w: np.ndarray, S: np.ndarray) -> float:
    """Squared MMD between the mixture sum_i w_i (fakes of slot i) and the real rows, from the
    block means: sum_ij w_i w_j S[1+i][1+j] - 2 sum_i w_i S[1+i][0] + S[0][0]."""
    w = np.asarray(w, np.float64)
    return float(w @ S[1:, 1:] @ w - 2.0 * (w @ S[1:, 0]) + S[0, 0])


def mixture_step(w: np.ndarray, S: np.ndarray, normals: np.ndarray, sigma: float):
    """ES-(1+1): w' = max(w + sigma n, 0) / sum (w kept if that sum is 0); w' replaces w iff
    mmd2(w') < mmd2(w). Returns (new w, accepted, mmd2(w), mmd2(w'))."""
    w = np.asarray(w, np.float64)
    cand = np.maximum(w + sigma * np.asarray(normals, np.float64), 0.0)
    tot = cand.sum()
    cand = cand / tot if tot > 0.0 else w.copy()
    old, new = mmd2(w, S), mmd2(cand, S)
    acc = new < old
    return (cand if acc else w.copy()), bool(acc), old, new


def mixture_update(state: State, data, cells=None, prev: Optional[State] = None
                   ) -> Dict[str, np.ndarray]:
    """Every cell's ES-(1+1) step on its mixture weights, scored on the evaluation's rows: the
    real minibatch and the fakes of the five neighbourhood generators on the cell's noise (as
    the discriminators received them, i.e. rounded to bf16 in bf16 mode). The mutation's five
    normals are the first five of the cell's stream MIX at the iteration."""
    a = state.arch
    rb = _Rounder(a)
    gl = g_layout(a)
    nbr = neighbors(state.rows, state.cols)
    n = state.cells
    out = {"S": np.zeros((n, 6, 6)), "mix": state.mix.copy(), "accept": np.zeros(n, bool),
           "score": np.zeros(n), "score_new": np.zeros(n)}
    for c in (range(n) if cells is None else cells):
        x, z = data[c]
        fakes = [g_forward(unflatten(_slot_state(state, prev, i).Gw[nbr[c][i]], gl), z, a)["F"]
                 for i in range(5)]
        S = mixture_blocks(rb(np.vstack([x] + fakes)), a.batch)
        nrm = draw_normals(state.seed, STREAM_MIX, state.t, c, 5)
        w, acc, old, new = mixture_step(state.mix[c], S, nrm, a.mix_sigma)
        out["S"][c], out["mix"][c], out["accept"][c] = S, w, acc
        out["score"][c], out["score_new"][c] = old, new
    return out


# --------------------------------------------------------------------------------------------
# Step 3a: tournament selection, replacement, learning-rate mutation.
# --------------------------------------------------------------------------------------------
def tournament(f5: np.ndarray, words: np.ndarray, size: int) -> int:
    """Draw ``size`` distinct slots (entrant m is the mulhi(word_m, 5 - m)-th slot not yet drawn,
    in ascending order) and return the entrant with the lowest fitness, the lower slot on a tie."""
    if not 1 <= size <= 5:
        raise ValueError("tournament size must be in 1..5")
    remaining = [0, 1, 2, 3, 4]
    entrants = [remaining.pop(int(mulhi(words[m], 5 - m))) for m in range(size)]
    best = entrants[0]
    for e in entrants[1:]:
        if f5[e] < f5[best] or (f5[e] == f5[best] and e < best):
            best = e
    return best


def select_slot(f5: np.ndarray, words: np.ndarray, arch: Arch) -> int:
    """The slot whose individual becomes the new centre: the tournament winner if it is strictly
    fitter than the centre (``if_better``) or unconditionally (``always``); else the centre."""
    win = tournament(f5, words, arch.tournament_size)
    if arch.replace_mode == "always":
        return win
    if arch.replace_mode != "if_better":
        raise ValueError("replace_mode must be if_better or always")
    return win if f5[win] < f5[0] else 0


def mutate_lr(lr: float, seed: int, stream: int, t: int, cell: int, arch: Arch) -> float:
    """Gaussian hyper-parameter update (step 3; Table 1 rate and probability): with probability
    p (word0 < floor(p * 2^32)) add std * N(0, 1) (Box-Muller on word1, word2, cosine branch);
    the result is kept >= 1e-8."""
    w = draw_words(seed, stream, t, cell, 4)
    thr = min(int(math.floor(arch.lr_mut_prob * 4294967296.0)), 4294967296)
    if int(w[0]) >= thr:
        return lr
    n, _ = box_muller(w[1:2], w[2:3])
    return max(lr + arch.lr_mut_std * float(n[0]), 1e-8)


def select_replace(state: State, ev) -> Dict[str, np.ndarray]:
    """Slots chosen for every cell's new centre generator and discriminator."""
    a = state.arch
    sel_g = np.zeros(state.cells, np.int64)
    sel_d = np.zeros(state.cells, np.int64)
    for c in range(state.cells):
        sel_g[c] = select_slot(ev["fG"][c], draw_words(state.seed, STREAM_TOUR_G, state.t, c,
                                                       a.tournament_size), a)
        sel_d[c] = select_slot(ev["fD"][c], draw_words(state.seed, STREAM_TOUR_D, state.t, c,
                                                       a.tournament_size), a)
    return {"sel_g": sel_g, "sel_d": sel_d}


# --------------------------------------------------------------------------------------------
# Step 3b: gradients of the selected pair and the Adam update.
# --------------------------------------------------------------------------------------------
def pair_gradients(Gflat: np.ndarray, Dflat: np.ndarray, x: np.ndarray, z: np.ndarray,
                   arch: Arch, flip: Optional[Dict[str, np.ndarray]] = None
                   ) -> Tuple[np.ndarray, np.ndarray, Dict[str, float]]:
    """dL_D/dv (fake batch detached) and dL_G/du (through D at its pre-update parameters), by
    the chain rule, layer by layer. Returns flat gradients in the parameter layouts.

    The derivative of ReLU / LeakyReLU jumps at 0, so an implementation whose pre-activation
    lands on the other side of 0 (another rounding of the same sum) takes the other branch
    there. ``flip`` (MLP only) names such elements: {"G1", "G2", "D1", "D2"} -> boolean arrays
    shaped like the pre-activations that ``info["pre"]`` returns (G: [B, h]; D: [2B, h], real
    rows then fake rows); a True element takes the other branch of the derivative. The values
    of the activations are unchanged (they are continuous at 0)."""
    a = arch
    rb = _Rounder(a)
    if a.kind == "dcgan":
        if flip:
            raise ValueError("flip is defined for the MLP networks")
        return _dcgan().pair_gradients(Gflat, Dflat, x, z, a, rb, unflatten, pair_losses, sigmoid)
    gl, dl = g_layout(a), d_layout(a)
    G, D = unflatten(Gflat, gl), unflatten(Dflat, dl)
    B = x.shape[0]
    fg = g_forward(G, z, a)
    fd = d_forward(D, np.vstack([x, fg["F"]]), a)
    logit = fd["logit"]
    s = sigmoid(logit)
    dl_d = np.concatenate([(s[:B] - 1.0) / B, s[B:] / B])   # dL_D / d logit, real then fake rows
    dl_g = (s[B:] - 1.0) / B                                 # dL_G / d logit of fake rows
    slope = a.leaky_slope

    gD = {name: np.zeros(shape) for name, shape in dl}
    gG = {name: np.zeros(shape) for name, shape in gl}
    g1, g2, X = fd["g1"], fd["g2"], fd["X"]
    # Rows of the discriminator chain: [real, fake (D loss), fake (G loss)].
    dl3 = np.concatenate([dl_d, dl_g])
    g2_3 = np.vstack([g2, g2[B:]])
    g1_3 = np.vstack([g1, g1[B:]])
    fl = flip or {}

    def side(y, name, rows3=False):
        # which side of 0 each pre-activation lies on (the activation has its sign), with the
        # elements named in ``flip`` on the other side; D's fake rows serve both losses
        pos = y > 0.0
        f = fl.get(name)
        if f is not None:
            pos = pos ^ (np.vstack([f, f[B:]]) if rows3 else f)
        return pos

    w3 = rb(D["W3"])[0]
    gD["W3"][0] = dl_d @ g2
    gD["b3"][0] = dl_d.sum()
    d2 = rb(dl3[:, None] * w3[None, :] * np.where(side(g2_3, "D2", True), 1.0, slope))
    gD["W2"][:] = d2[:2 * B].T @ g1
    gD["b2"][:] = d2[:2 * B].sum(axis=0)
    d1 = rb((d2 @ rb(D["W2"])) * np.where(side(g1_3, "D1", True), 1.0, slope))
    gD["W1"][:] = d1[:2 * B].T @ X
    gD["b1"][:] = d1[:2 * B].sum(axis=0)
    # Generator chain: through D's first layer into the fakes, then back through G.
    dF = d1[2 * B:] @ rb(D["W1"])
    F, h2, h1, zq = fg["F"], fg["h2"], fg["h1"], fg["z"]
    a3 = rb(dF * (1.0 - F * F))
    gG["W3"][:] = a3.T @ h2
    gG["b3"][:] = a3.sum(axis=0)
    a2 = rb((a3 @ rb(G["W3"])) * side(h2, "G2"))
    gG["W2"][:] = a2.T @ h1
    gG["b2"][:] = a2.sum(axis=0)
    a1 = rb((a2 @ rb(G["W2"])) * side(h1, "G1"))
    gG["W1"][:] = a1.T @ zq
    gG["b1"][:] = a1.sum(axis=0)
    lg, ld = pair_losses(logit[:B], logit[B:])
    flatG = np.concatenate([gG[n].reshape(-1) for n, _ in gl])
    flatD = np.concatenate([gD[n].reshape(-1) for n, _ in dl])
    # Distance of the closest pre-activation to a kink of ReLU / LeakyReLU (where the derivative
    # jumps): a diagnostic for comparisons with implementations that round differently.
    pre = {"G1": zq @ rb(G["W1"]).T + G["b1"], "G2": h1 @ rb(G["W2"]).T + G["b2"],
           "D1": X @ rb(D["W1"]).T + D["b1"], "D2": g1 @ rb(D["W2"]).T + D["b2"]}
    kink = min(float(np.min(np.abs(p))) for p in pre.values())
    return flatG, flatD, {"LG": lg, "LD": ld, "kink": kink, "pre": pre}


def adam_step(w, m, v, step, g, lr, arch: Arch):
    """One Adam update (Kingma & Ba 2015, Algorithm 1) with the individual's own step count."""
    t1 = step + 1
    m1 = arch.beta1 * m + (1.0 - arch.beta1) * g
    v1 = arch.beta2 * v + (1.0 - arch.beta2) * g * g
    mhat = m1 / (1.0 - arch.beta1 ** t1)
    vhat = v1 / (1.0 - arch.beta2 ** t1)
    return w - lr * mhat / (np.sqrt(vhat) + arch.eps), m1, v1, t1


def train_step(state: State, sel, data, keep_grads: bool = False,
               pool: Optional[np.ndarray] = None, prev: Optional[State] = None):
    """Every cell's new centre pair (the selected slots' individuals with their optimiser state)
    takes one Adam step on the cell's minibatch, reading only the snapshot ``state``; with
    ``arch.train_steps`` K > 1 it then takes K-1 more steps, step k on the cell's fresh step-k
    minibatch from ``pool``, each at the parameters the previous step left (no selection and no
    lr mutation in between). The kept gradients are the last step's; ``kink`` is the closest
    approach of any step's pre-activations to 0. With ``prev`` (stale neighbours), a selected
    neighbour slot brings ``prev``'s individual."""
    a = state.arch
    nbr = neighbors(state.rows, state.cols)
    new = state.copy()
    grads = {"gG": np.zeros_like(state.Gw), "gD": np.zeros_like(state.Dw),
             "kink": np.zeros(state.cells)}
    for c in range(state.cells):
        sg = int(nbr[c][sel["sel_g"][c]])
        sd = int(nbr[c][sel["sel_d"][c]])
        SG = _slot_state(state, prev, int(sel["sel_g"][c]))
        SD = _slot_state(state, prev, int(sel["sel_d"][c]))
        lr_g, lr_d = float(SG.Glr[sg]), float(SD.Dlr[sd])
        if a.lr_mutation:
            lr_g = mutate_lr(lr_g, state.seed, STREAM_MUT_G, state.t, c, a)
            lr_d = mutate_lr(lr_d, state.seed, STREAM_MUT_D, state.t, c, a)
        x, z = data[c]
        gG, gD, info = pair_gradients(SG.Gw[sg], SD.Dw[sd], x, z, a)
        grads["kink"][c] = info["kink"]
        new.Gw[c], new.Gm[c], new.Gv[c], new.Gstep[c] = adam_step(
            SG.Gw[sg], SG.Gm[sg], SG.Gv[sg], SG.Gstep[sg], gG, lr_g, a)
        new.Dw[c], new.Dm[c], new.Dv[c], new.Dstep[c] = adam_step(
            SD.Dw[sd], SD.Dm[sd], SD.Dv[sd], SD.Dstep[sd], gD, lr_d, a)
        new.Glr[c], new.Dlr[c] = lr_g, lr_d
        grads["gG"][c], grads["gD"][c] = gG, gD
    if a.stale_neighbors and a.train_steps > 1:
        raise ValueError("stale neighbours are defined for one training step per iteration")
    if a.train_steps > 1 and pool is None:
        raise ValueError("train_steps > 1 draws its later minibatches from the pool")
    for k in range(1, a.train_steps):
        for c in range(state.cells):
            x, z = draw_batch(state.seed, state.t, c, pool, a, k)
            gG, gD, info = pair_gradients(new.Gw[c], new.Dw[c], x, z, a)
            grads["kink"][c] = min(grads["kink"][c], info["kink"])
            new.Gw[c], new.Gm[c], new.Gv[c], new.Gstep[c] = adam_step(
                new.Gw[c], new.Gm[c], new.Gv[c], new.Gstep[c], gG, new.Glr[c], a)
            new.Dw[c], new.Dm[c], new.Dv[c], new.Dstep[c] = adam_step(
                new.Dw[c], new.Dm[c], new.Dv[c], new.Dstep[c], gD, new.Dlr[c], a)
            grads["gG"][c], grads["gD"][c] = gG, gD
    new.t = state.t + 1
    return (new, grads) if keep_grads else new


def iterate(state: State, pool: Optional[np.ndarray], n_iters: int = 1,
            x_host: Optional[np.ndarray] = None, record: bool = False,
            prev: Optional[State] = None):
    """Steps 2, 3 (and 4 with ``arch.mixture``) and 5: ``n_iters`` synchronous grid
    iterations. Returns the new state (and, with ``record``, the per-iteration evaluations and
    selections). With
    ``arch.stale_neighbors`` each iteration's neighbours come from the state one iteration
    older (``prev`` for the first iteration; when None, the first iteration uses ``state``)."""
    log = []
    for _ in range(n_iters):
        data = batches(state, pool, x_host)
        ev = eval_neighborhoods(state, data, prev=prev)
        mx = mixture_update(state, data, prev=prev) if state.arch.mixture else None
        sel = select_replace(state, ev)
        new = train_step(state, sel, data, pool=pool, prev=prev)
        if mx is not None:
            new.mix = mx["mix"]
        if state.arch.stale_neighbors:
            prev = state
        state = new
        if record:
            log.append({"eval": ev, "sel": sel, "mix": mx})
    return (state, log) if record else state


# --------------------------------------------------------------------------------------------
# State bytes: the engine's documented export layout (little-endian), so that a state can move
# between the engine and the oracle.
#   header (64 bytes): u32 magic 0x5A50494C ("LIPZ"), u32 version 2, i32 rows, i32 cols,
#     i32 z_dim, i32 hidden, i32 x_dim, i32 batch, i32 precision (0 fp32, 1 bf16), i32 0,
#     i64 t, u64 seed, 8 zero bytes
#   then f32 Gw[cells][PG], Gm, Gv, Dw[cells][PD], Dm, Dv, i32 Gstep[cells], Dstep[cells],
#     f32 Glr[cells], Dlr[cells], f32 mix[cells][5].
# --------------------------------------------------------------------------------------------
_MAGIC = 0x5A50494C


def state_to_bytes(s: State) -> bytes:
    a = s.arch
    hdr = np.zeros(16, dtype=np.uint32)
    hdr[0], hdr[1] = _MAGIC, 2
    hdr[2:10] = [s.rows, s.cols, a.z_dim, a.hidden, a.x_dim, a.batch,
                 1 if a.precision == "bf16" else 0, 0]
    h = hdr.tobytes()
    h = h[:40] + np.array([s.t], np.int64).tobytes() + np.array([s.seed], np.uint64).tobytes() \
        + bytes(8)
    parts = [h] + [getattr(s, f).astype(np.float32).tobytes()
                   for f in ("Gw", "Gm", "Gv", "Dw", "Dm", "Dv")]
    parts += [s.Gstep.astype(np.int32).tobytes(), s.Dstep.astype(np.int32).tobytes(),
              s.Glr.astype(np.float32).tobytes(), s.Dlr.astype(np.float32).tobytes(),
              s.mix.astype(np.float32).tobytes()]
    return b"".join(parts)


def state_from_bytes(buf: bytes, arch: Arch) -> State:
    hdr = np.frombuffer(buf[:40], dtype=np.int32)
    if int(np.frombuffer(buf[:4], np.uint32)[0]) != _MAGIC or int(hdr[1]) != 2:
        raise ValueError("not a version-2 grid state")
    rows, cols = int(hdr[2]), int(hdr[3])
    if (int(hdr[4]), int(hdr[5]), int(hdr[6]), int(hdr[7])) != (arch.z_dim, arch.hidden,
                                                              arch.x_dim, arch.batch):
        raise ValueError("state does not match the architecture")
    t = int(np.frombuffer(buf[40:48], np.int64)[0])
    seed = int(np.frombuffer(buf[48:56], np.uint64)[0])
    cells = rows * cols
    PG, PD = n_params(g_layout(arch)), n_params(d_layout(arch))
    off = 64
    arrs = {}
    for f, p in (("Gw", PG), ("Gm", PG), ("Gv", PG), ("Dw", PD), ("Dm", PD), ("Dv", PD)):
        n = cells * p
        arrs[f] = np.frombuffer(buf[off:off + 4 * n], np.float32).astype(np.float64).reshape(cells, p)
        off += 4 * n
    for f, dt in (("Gstep", np.int32), ("Dstep", np.int32), ("Glr", np.float32),
                  ("Dlr", np.float32)):
        v = np.frombuffer(buf[off:off + 4 * cells], dt)
        arrs[f] = v.astype(np.int64 if dt == np.int32 else np.float64)
        off += 4 * cells
    arrs["mix"] = np.frombuffer(buf[off:off + 20 * cells], np.float32).astype(
        np.float64).reshape(cells, 5)
    off += 20 * cells
    if off != len(buf):
        raise ValueError("state size mismatch")
    return State(rows, cols, arch, seed, t, **arrs)
