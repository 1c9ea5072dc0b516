"""Python binding of the GB300 grid-iteration engine (liblipz.so, C ABI in include/lipz.h).

The functions below carry the C names and only marshal arguments: every step of a grid
iteration runs in the library's CUDA kernels. Output arrays are numpy float32/int32 arrays
(or anything exposing ``data_ptr()``, e.g. a pinned torch tensor) that the caller owns.
If the library has not been built, importing works but the first call raises
``LipzError``; there is no fallback implementation.
"""

import ctypes
import os

import numpy as np

__all__ = [
    "LipzError", "lipz_arch", "arch_default", "library_path", "load",
    "lipz_arch_default", "lipz_grid_create", "lipz_grid_destroy", "lipz_set_stream",
    "lipz_synchronize", "lipz_set_data", "lipz_eval_neighborhoods", "lipz_select_replace",
    "lipz_train_step", "lipz_iterate", "lipz_iterate_batch", "lipz_iterate_batch_next",
    "lipz_iterate_batch_async",
    "lipz_state_bytes",
    "lipz_export_state", "lipz_import_state", "lipz_get_iteration", "lipz_get_batch",
    "lipz_get_logits", "lipz_get_gradients", "lipz_get_mixture", "lipz_profile_enable",
    "lipz_profile_read",
    "lipz_fitness_from_logits_noalloc", "lipz_last_error", "lipz_status_string", "PHASES",
    "EXPORTED", "Grid", "param_counts",
]

LIPZ_OK, LIPZ_ERR_INVALID, LIPZ_ERR_CUDA, LIPZ_ERR_OOM = 0, 1, 2, 3
LIPZ_ERR_NONFINITE, LIPZ_ERR_TIMEOUT, LIPZ_ERR_STATE = 4, 5, 6
LIPZ_MLP, LIPZ_DCGAN64 = 0, 1
LIPZ_FP32, LIPZ_BF16 = 0, 1
LIPZ_REPLACE_IF_BETTER, LIPZ_REPLACE_ALWAYS = 0, 1
LIPZ_NOALLOC_MAX_CELLS = 4096


def library_path() -> str:
    return os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib", "liblipz.so")


class LipzError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__("lipz error %d: %s" % (code, msg))
        self.code = code


class lipz_arch(ctypes.Structure):
    _fields_ = [
        ("struct_size", ctypes.c_uint32), ("kind", ctypes.c_int32),
        ("precision", ctypes.c_int32), ("z_dim", ctypes.c_int32), ("hidden", ctypes.c_int32),
        ("x_dim", ctypes.c_int32), ("batch", ctypes.c_int32), ("lr", ctypes.c_float),
        ("beta1", ctypes.c_float), ("beta2", ctypes.c_float), ("eps", ctypes.c_float),
        ("tournament_size", ctypes.c_int32), ("replace_mode", ctypes.c_int32),
        ("lr_mutation", ctypes.c_int32), ("lr_mut_std", ctypes.c_float),
        ("lr_mut_prob", ctypes.c_float), ("leaky_slope", ctypes.c_float),
        ("keep_grads", ctypes.c_int32), ("force_simt", ctypes.c_int32),
        ("train_steps", ctypes.c_int32), ("mixture", ctypes.c_int32),
        ("mix_sigma", ctypes.c_float), ("stale_neighbors", ctypes.c_int32),
        ("ngf", ctypes.c_int32), ("ndf", ctypes.c_int32),
    ]


_P = ctypes.c_void_p
_I = ctypes.c_int
# name -> (restype, argtypes)
_SIGS = {
    "lipz_arch_default": (_I, [ctypes.POINTER(lipz_arch)]),
    "lipz_grid_create": (_I, [_I, _I, ctypes.POINTER(lipz_arch), ctypes.c_uint64,
                              ctypes.POINTER(_P)]),
    "lipz_grid_destroy": (_I, [_P]),
    "lipz_set_stream": (_I, [_P, _P]),
    "lipz_synchronize": (_I, [_P]),
    "lipz_set_data": (_I, [_P, _P, ctypes.c_int64, ctypes.c_int32]),
    "lipz_eval_neighborhoods": (_I, [_P, _P, _P, _P, _P]),
    "lipz_select_replace": (_I, [_P, _P, _P]),
    "lipz_train_step": (_I, [_P]),
    "lipz_iterate": (_I, [_P, _I]),
    "lipz_iterate_batch": (_I, [_P, _P, _P, _P]),
    "lipz_iterate_batch_next": (_I, [_P, _P, _P, _P, _P]),
    "lipz_iterate_batch_async": (_I, [_P, _P, _P, _P, _P]),
    "lipz_state_bytes": (_I, [_P, ctypes.POINTER(ctypes.c_size_t)]),
    "lipz_export_state": (_I, [_P, _P, ctypes.c_size_t]),
    "lipz_import_state": (_I, [_P, _P, ctypes.c_size_t]),
    "lipz_get_iteration": (_I, [_P, ctypes.POINTER(ctypes.c_int64)]),
    "lipz_get_batch": (_I, [_P, _P, _P]),
    "lipz_get_logits": (_I, [_P, _P]),
    "lipz_get_gradients": (_I, [_P, _P, _P]),
    "lipz_get_mixture": (_I, [_P, _P, _P, _P]),
    "lipz_profile_enable": (_I, [_P, _I]),
    "lipz_profile_read": (_I, [_P, _P, _P, _P, _I]),
    "lipz_fitness_from_logits_noalloc": (_I, [_P, ctypes.c_int32, ctypes.c_int32, _P, _P, _P]),
    "lipz_last_error": (ctypes.c_char_p, [_P]),
    "lipz_status_string": (ctypes.c_char_p, [_I]),
}
EXPORTED = tuple(_SIGS)

_lib = None


def load():
    """Load liblipz.so (built in-tree by ``_build.build()``); raise if it is missing."""
    global _lib
    if _lib is None:
        path = library_path()
        if not os.path.exists(path):
            raise LipzError(LIPZ_ERR_INVALID, "liblipz.so is not built (%s); run "
                            "python -m paper_1811_12843_gb300._build" % path)
        lib = ctypes.CDLL(path)
        for name, (res, args) in _SIGS.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def _ptr(a):
    if a is None:
        return None
    if hasattr(a, "data_ptr"):
        return ctypes.c_void_p(a.data_ptr())
    if isinstance(a, np.ndarray):
        if not a.flags["C_CONTIGUOUS"]:
            raise ValueError("arrays passed to the engine must be C-contiguous")
        return ctypes.c_void_p(a.ctypes.data)
    if isinstance(a, (bytearray, memoryview)):
        return ctypes.c_void_p(ctypes.addressof(ctypes.c_char.from_buffer(a)))
    raise TypeError("unsupported buffer type %r" % type(a))


def _check(g, rc):
    if rc != LIPZ_OK:
        raise LipzError(rc, lipz_last_error(g))
    return rc


# ---- C-named wrappers -------------------------------------------------------------------
def lipz_arch_default() -> lipz_arch:
    a = lipz_arch()
    _check(None, load().lipz_arch_default(ctypes.byref(a)))
    return a


def lipz_grid_create(rows, cols, arch, seed):
    h = _P()
    _check(None, load().lipz_grid_create(int(rows), int(cols), ctypes.byref(arch),
                                         ctypes.c_uint64(int(seed)), ctypes.byref(h)))
    return h


def lipz_grid_destroy(g):
    return _check(g, load().lipz_grid_destroy(g))


def lipz_set_stream(g, stream):
    s = stream if isinstance(stream, int) else getattr(stream, "cuda_stream", stream)
    return _check(g, load().lipz_set_stream(g, _P(int(s or 0))))


def lipz_synchronize(g):
    return _check(g, load().lipz_synchronize(g))


def lipz_set_data(g, pool):
    pool = np.ascontiguousarray(pool, dtype=np.float32)
    return _check(g, load().lipz_set_data(g, _ptr(pool), pool.shape[0], pool.shape[1]))


def lipz_eval_neighborhoods(g, fit_g=None, fit_d=None, pair_lg=None, pair_ld=None):
    return _check(g, load().lipz_eval_neighborhoods(g, _ptr(fit_g), _ptr(fit_d), _ptr(pair_lg),
                                                    _ptr(pair_ld)))


def lipz_select_replace(g, sel_g=None, sel_d=None):
    return _check(g, load().lipz_select_replace(g, _ptr(sel_g), _ptr(sel_d)))


def lipz_train_step(g):
    return _check(g, load().lipz_train_step(g))


def lipz_iterate(g, n_iters):
    return _check(g, load().lipz_iterate(g, int(n_iters)))


def lipz_iterate_batch(g, x_host, fit_g=None, fit_d=None):
    return _check(g, load().lipz_iterate_batch(g, _ptr(x_host), _ptr(fit_g), _ptr(fit_d)))


def lipz_iterate_batch_next(g, x_host, x_next=None, fit_g=None, fit_d=None):
    """lipz_iterate_batch that uploads the next call's minibatch (x_next) while this one runs."""
    return _check(g, load().lipz_iterate_batch_next(g, _ptr(x_host), _ptr(x_next), _ptr(fit_g),
                                                    _ptr(fit_d)))


def lipz_iterate_batch_async(g, x_host, x_next=None, fit_g=None, fit_d=None):
    """lipz_iterate_batch_next one call ahead: enqueues this iteration, returns once the previous
    call's has completed (its fitness buffers filled, its device status returned)."""
    return _check(g, load().lipz_iterate_batch_async(g, _ptr(x_host), _ptr(x_next), _ptr(fit_g),
                                                     _ptr(fit_d)))


def lipz_state_bytes(g) -> int:
    n = ctypes.c_size_t()
    _check(g, load().lipz_state_bytes(g, ctypes.byref(n)))
    return n.value


def lipz_export_state(g) -> bytes:
    buf = bytearray(lipz_state_bytes(g))
    _check(g, load().lipz_export_state(g, _ptr(buf), len(buf)))
    return bytes(buf)


def lipz_import_state(g, data: bytes):
    buf = bytearray(data)
    return _check(g, load().lipz_import_state(g, _ptr(buf), len(buf)))


def lipz_get_iteration(g) -> int:
    t = ctypes.c_int64()
    _check(g, load().lipz_get_iteration(g, ctypes.byref(t)))
    return t.value


def lipz_get_batch(g, x=None, z=None):
    return _check(g, load().lipz_get_batch(g, _ptr(x), _ptr(z)))


def lipz_get_logits(g, logits):
    return _check(g, load().lipz_get_logits(g, _ptr(logits)))


def lipz_get_gradients(g, grad_g=None, grad_d=None):
    return _check(g, load().lipz_get_gradients(g, _ptr(grad_g), _ptr(grad_d)))


def lipz_get_mixture(g, weights=None, blocks=None, score=None):
    return _check(g, load().lipz_get_mixture(g, _ptr(weights), _ptr(blocks), _ptr(score)))


PHASES = ("batch", "g_fwd", "d_fwd", "fitness", "select", "train_fwd", "train_bwd", "adam",
          "mixture")


def lipz_profile_enable(g, enable=True):
    return _check(g, load().lipz_profile_enable(g, 1 if enable else 0))


def lipz_profile_read(g):
    """{phase: (device ms, executions, kernel launches)} since the last read."""
    n = len(PHASES)
    ms = np.zeros(n, np.float64)
    cnt = np.zeros(n, np.int64)
    la = np.zeros(n, np.int64)
    _check(g, load().lipz_profile_read(g, _ptr(ms), _ptr(cnt), _ptr(la), n))
    return {p: (float(ms[i]), int(cnt[i]), int(la[i])) for i, p in enumerate(PHASES)}


def _device_f32(t, need, what):
    """Refuse anything but a contiguous float32 CUDA tensor of at least `need` elements: the
    library launches a kernel on these addresses and cannot check them itself."""
    ok = (hasattr(t, "is_cuda") and t.is_cuda and str(getattr(t, "dtype", "")) == "torch.float32"
          and t.is_contiguous())
    if not ok:
        raise LipzError(LIPZ_ERR_INVALID, "lipz_fitness_from_logits_noalloc: %s must be a "
                        "contiguous float32 CUDA tensor" % what)
    if t.numel() < need:
        raise LipzError(LIPZ_ERR_INVALID, "lipz_fitness_from_logits_noalloc: %s holds %d "
                        "elements, %d needed" % (what, t.numel(), need))


def lipz_fitness_from_logits_noalloc(logits, cells, batch, fit_g, fit_d, stream=0):
    """Fitness from device logits with no device allocation (all buffers are device tensors
    the caller owns). Raises LipzError with the status code on failure; buffers that are not
    contiguous float32 CUDA tensors of the needed sizes are refused before the library is
    called."""
    cells, batch = int(cells), int(batch)
    # sizes outside the library's limits go through unchecked: the library refuses them itself,
    # launching nothing
    if 1 <= cells <= LIPZ_NOALLOC_MAX_CELLS and batch >= 1:
        _device_f32(logits, cells * 30 * batch, "logits")
        _device_f32(fit_g, cells * 5, "fit_g")
        _device_f32(fit_d, cells * 5, "fit_d")
    s = stream if isinstance(stream, int) else getattr(stream, "cuda_stream", stream)
    rc = load().lipz_fitness_from_logits_noalloc(_ptr(logits), int(cells), int(batch),
                                                 _ptr(fit_g), _ptr(fit_d), _P(int(s or 0)))
    if rc != LIPZ_OK:
        msg = lipz_status_string(rc)
        if rc == LIPZ_ERR_INVALID:
            msg += " (cells must be in 1..%d, batch >= 1)" % LIPZ_NOALLOC_MAX_CELLS
        raise LipzError(rc, "lipz_fitness_from_logits_noalloc: " + msg)
    return rc


def lipz_last_error(g) -> str:
    s = load().lipz_last_error(g)
    return s.decode() if s else ""


def lipz_status_string(code) -> str:
    return load().lipz_status_string(int(code)).decode()


# ---- convenience --------------------------------------------------------------------------
def arch_default(**overrides) -> lipz_arch:
    """Table 1 MLP defaults with field overrides; precision may be given as "fp32"/"bf16"."""
    a = lipz_arch_default()
    for k, v in overrides.items():
        if k == "precision" and isinstance(v, str):
            v = {"fp32": LIPZ_FP32, "bf16": LIPZ_BF16}[v]
        if k == "replace_mode" and isinstance(v, str):
            v = {"if_better": LIPZ_REPLACE_IF_BETTER, "always": LIPZ_REPLACE_ALWAYS}[v]
        setattr(a, k, v)
    return a


def param_counts(z_dim, hidden, x_dim, kind=LIPZ_MLP, ngf=64, ndf=64):
    """(PG, PD): parameters of one generator and one discriminator."""
    if kind == LIPZ_DCGAN64:
        ch = [z_dim, 8 * ngf, 4 * ngf, 2 * ngf, ngf]
        pg = sum(ch[i] * ch[i + 1] * 16 + 2 * ch[i + 1] for i in range(4)) + ngf * 3 * 16
        dh = [3, ndf, 2 * ndf, 4 * ndf, 8 * ndf]
        pd = sum(dh[i] * dh[i + 1] * 16 for i in range(4)) + 8 * ndf * 16
        return pg, pd
    pg = hidden * z_dim + hidden + hidden * hidden + hidden + x_dim * hidden + x_dim
    pd = hidden * x_dim + hidden + hidden * hidden + hidden + hidden + 1
    return pg, pd


class Grid:
    """Owning handle of one grid with numpy-returning helpers."""

    def __init__(self, rows, cols, arch=None, seed=0, **overrides):
        self.arch = arch if arch is not None else arch_default(**overrides)
        self.rows, self.cols, self.cells = rows, cols, rows * cols
        self.h = lipz_grid_create(rows, cols, self.arch, seed)
        a = self.arch
        self.PG, self.PD = param_counts(a.z_dim, a.hidden, a.x_dim, a.kind, a.ngf, a.ndf)

    def close(self):
        if self.h:
            lipz_grid_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_stream(self, stream):
        lipz_set_stream(self.h, stream)

    def set_data(self, pool):
        lipz_set_data(self.h, pool)

    def eval(self, pairs=False):
        C = self.cells
        fg, fd = np.zeros((C, 5), np.float32), np.zeros((C, 5), np.float32)
        lg = np.zeros((C, 5, 5), np.float32) if pairs else None
        ld = np.zeros((C, 5, 5), np.float32) if pairs else None
        lipz_eval_neighborhoods(self.h, fg, fd, lg, ld)
        out = {"fG": fg, "fD": fd}
        if pairs:
            out.update(LG=lg, LD=ld)
        return out

    def select(self):
        sg, sd = np.zeros(self.cells, np.int32), np.zeros(self.cells, np.int32)
        lipz_select_replace(self.h, sg, sd)
        return {"sel_g": sg, "sel_d": sd}

    def train(self):
        lipz_train_step(self.h)

    def iterate(self, n=1):
        lipz_iterate(self.h, n)

    def synchronize(self):
        lipz_synchronize(self.h)

    def export_state(self) -> bytes:
        return lipz_export_state(self.h)

    def import_state(self, data: bytes):
        lipz_import_state(self.h, data)

    @property
    def t(self) -> int:
        return lipz_get_iteration(self.h)

    def batch(self):
        a = self.arch
        x = np.zeros((self.cells, a.batch, a.x_dim), np.float32)
        z = np.zeros((self.cells, a.batch, a.z_dim), np.float32)
        lipz_get_batch(self.h, x, z)
        return x, z

    def logits(self):
        out = np.zeros((self.cells, 5, 6 * self.arch.batch), np.float32)
        lipz_get_logits(self.h, out)
        return out

    def mixture(self, blocks=False):
        """Mixture weights [cells, 5]; with ``blocks`` also the last evaluation's kernel block
        means [cells, 6, 6] and squared-MMD scores [cells] (needs arch.mixture)."""
        w = np.zeros((self.cells, 5), np.float32)
        if not blocks:
            lipz_get_mixture(self.h, w)
            return w
        S = np.zeros((self.cells, 6, 6), np.float32)
        sc = np.zeros(self.cells, np.float32)
        lipz_get_mixture(self.h, w, S, sc)
        return w, S, sc

    def gradients(self):
        gg = np.zeros((self.cells, self.PG), np.float32)
        gd = np.zeros((self.cells, self.PD), np.float32)
        lipz_get_gradients(self.h, gg, gd)
        return gg, gd
