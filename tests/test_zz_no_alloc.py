"""The allocation-free fitness entry point, for callers that cannot call cudaMalloc (a serving
loop whose device memory another allocator has fully reserved, or a latency-critical path that
cannot take the implicit synchronisation of cudaMalloc / cudaFree).

Its output must match the fitness that lipz_eval_neighborhoods returns for the same logits,
on two calls in a row of different sizes (the shared scratch array keeps the previous call's
contents, which must not leak into the next result). This file is collected last.
"""

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1811_12843_gb300 import _build
    _build.build()
    import lipz_synth
    import paper_1811_12843_gb300 as L
    return torch, L, lipz_synth


def _reference(L, lipz_synth, rows, cols, precision, batch, seed):
    g = L.Grid(rows, cols, seed=seed, precision=precision, batch=batch)
    g.set_data(lipz_synth.blob_pool(seed, n=1000, dim=784))
    ev = g.eval()
    logits = g.logits()
    g.close()
    return logits, ev["fG"], ev["fD"]


def test_noalloc_fitness_matches_eval_on_two_calls(env):
    torch, L, lipz_synth = env
    cases = [(3, 4, "bf16", 100, 7), (2, 2, "fp32", 37, 8)]
    refs = [_reference(L, lipz_synth, *c) for c in cases]
    stream = torch.cuda.current_stream()
    for (rows, cols, _, batch, _), (logits, fg_ref, fd_ref) in zip(cases, refs):
        cells = rows * cols
        dl = torch.from_numpy(logits).cuda()
        fg = torch.full((cells, 5), float("nan"), device="cuda")
        fd = torch.full((cells, 5), float("nan"), device="cuda")
        L.lipz_fitness_from_logits_noalloc(dl, cells, batch, fg, fd, stream)
        torch.cuda.synchronize()
        for got, ref in ((fg.cpu().numpy(), fg_ref), (fd.cpu().numpy(), fd_ref)):
            assert np.max(np.abs(got - ref)) <= 1e-4 * np.max(np.abs(ref))


def test_noalloc_rejects_sizes_beyond_the_limit(env):
    torch, L, _ = env
    dl = torch.zeros(30, device="cuda")
    out = torch.zeros(5, device="cuda")
    with pytest.raises(L.LipzError) as e:
        L.lipz_fitness_from_logits_noalloc(dl, 4097, 1, out, out)
    assert e.value.code == L.LIPZ_ERR_INVALID
    with pytest.raises(L.LipzError) as e:
        L.lipz_fitness_from_logits_noalloc(dl, 0, 1, out, out)
    assert e.value.code == L.LIPZ_ERR_INVALID
