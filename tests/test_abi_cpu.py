"""The C-ABI library without a GPU: it builds, loads, exports every declared entry point, and
rejects bad arguments before touching the device."""

import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    with open(os.path.join(ROOT, "include", "lipz.h")) as f:
        src = f.read()
    return sorted(set(re.findall(r"LIPZ_API\s+[\w\s\*]+?\b(lipz_\w+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_1811_12843_gb300 import _build
    _build.build()
    import paper_1811_12843_gb300 as L
    return L.load()


def test_header_declares_the_boundary():
    names = _declared()
    for must in ("lipz_grid_create", "lipz_eval_neighborhoods", "lipz_select_replace",
                 "lipz_train_step", "lipz_iterate", "lipz_export_state", "lipz_import_state"):
        assert must in names


def test_library_exports_every_declared_symbol(lib):
    import paper_1811_12843_gb300 as L
    names = _declared()
    out = subprocess.run(["nm", "-D", "--defined-only", L.library_path()], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (lipz_\w+)", out))
    assert set(names) <= exported, set(names) - exported
    # and the Python binding wraps exactly the declared calls
    assert sorted(L.EXPORTED) == names
    for n in names:
        assert hasattr(lib, n)


def test_arch_struct_layout_matches(lib):
    import paper_1811_12843_gb300 as L
    a = L.lipz_arch_default()
    assert a.struct_size == ctypes.sizeof(L.lipz_arch)
    assert (a.z_dim, a.hidden, a.x_dim, a.batch, a.tournament_size) == (64, 256, 784, 100, 2)
    assert abs(a.lr - 2e-4) < 1e-9 and abs(a.beta1 - 0.5) < 1e-9 and abs(a.leaky_slope - 0.2) < 1e-7


def test_create_rejects_bad_arguments_without_a_device(lib):
    import paper_1811_12843_gb300 as L
    a = L.lipz_arch_default()
    with pytest.raises(L.LipzError) as e:
        L.lipz_grid_create(0, 3, a, 1)
    assert e.value.code == L.LIPZ_ERR_INVALID and "rows" in str(e.value)
    bad = L.lipz_arch_default()
    bad.tournament_size = 6
    with pytest.raises(L.LipzError) as e:
        L.lipz_grid_create(2, 2, bad, 1)
    assert e.value.code == L.LIPZ_ERR_INVALID
    assert a.train_steps == 1
    for k in (0, -1, 65537):
        bad = L.lipz_arch_default()
        bad.train_steps = k
        with pytest.raises(L.LipzError) as e:
            L.lipz_grid_create(2, 2, bad, 1)
        assert e.value.code == L.LIPZ_ERR_INVALID and "train_steps" in str(e.value)
    bad = L.lipz_arch_default()
    bad.struct_size = 4
    with pytest.raises(L.LipzError):
        L.lipz_grid_create(2, 2, bad, 1)
    assert L.lipz_status_string(L.LIPZ_ERR_STATE) == "call out of order"


def test_param_counts_match_the_paper_sizes():
    import paper_1811_12843_gb300 as L
    assert L.param_counts(64, 256, 784) == (283920, 267009)


def test_noalloc_wrapper_refuses_bad_buffers_before_the_library(lib):
    """The allocation-free fitness call launches a kernel on the addresses it is given, and the
    library cannot check them: the wrapper refuses host arrays, wrong dtypes, non-contiguous
    and short tensors with LIPZ_ERR_INVALID. No device exists here, so a refusal that reached
    the library would fail differently."""
    import numpy as np
    import torch
    import paper_1811_12843_gb300 as L
    cells, batch = 2, 3
    host = np.zeros(cells * 30 * batch, np.float32)
    out = np.zeros(cells * 5, np.float32)
    cases = [
        (host, out, out, "logits"),                                      # numpy, not a device tensor
        (torch.zeros(cells * 30 * batch), out, out, "logits"),           # CPU tensor
    ]
    for logits, fg, fd, what in cases:
        with pytest.raises(L.LipzError) as e:
            L.lipz_fitness_from_logits_noalloc(logits, cells, batch, fg, fd)
        assert e.value.code == L.LIPZ_ERR_INVALID and what in str(e.value)

    class FakeCuda:
        """Stands in for a CUDA tensor (no device here): only the attributes the check reads."""

        def __init__(self, n, dtype="torch.float32", contiguous=True):
            self.is_cuda, self.dtype, self._n, self._c = True, dtype, n, contiguous

        def is_contiguous(self):
            return self._c

        def numel(self):
            return self._n

        def data_ptr(self):
            raise AssertionError("the wrapper passed a refused buffer on")

    ok_l, ok_o = FakeCuda(cells * 30 * batch), FakeCuda(cells * 5)
    bad = [
        (FakeCuda(cells * 30 * batch - 1), ok_o, ok_o, "logits"),        # one logit short
        (ok_l, FakeCuda(cells * 5 - 1), ok_o, "fit_g"),                  # short output
        (ok_l, ok_o, FakeCuda(cells * 5, dtype="torch.float64"), "fit_d"),
        (FakeCuda(cells * 30 * batch, contiguous=False), ok_o, ok_o, "logits"),
    ]
    for logits, fg, fd, what in bad:
        with pytest.raises(L.LipzError) as e:
            L.lipz_fitness_from_logits_noalloc(logits, cells, batch, fg, fd)
        assert e.value.code == L.LIPZ_ERR_INVALID and what in str(e.value)
