"""dc_drift_sums_noalloc: the drift sums for callers that cannot allocate
device memory while running (fixed start-up memory budgets, hosts that may
not call cudaMalloc after initialisation).  Checked through the C ABI
against dc_drift_sums on the same inputs and against the sums written out in
fp64, over calls in a row that share the library's fixed scratch array, on
the default stream and on a stream of the caller's.  This file is collected
last."""

import numpy as np
import pytest

from synth import WORKLOADS, gen

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dc():
    from paper_2608_16354_gb300 import _build, binding
    _build.build()
    binding.lib()
    return binding


def _fp64_sums(w, xn, xr):
    """sum ||(x_now - x_ref) W_e^T||^2 and sum ||x_now W_e^T + b_e + pos||^2
    per scene, in fp64."""
    We = w["w_embed"].astype(np.float64)
    out = []
    for s in range(xn.shape[0]):
        du = (xn[s].astype(np.float64) - xr[s]) @ We.T
        u = xn[s].astype(np.float64) @ We.T + w["b_embed"] + w["pos"]
        out += [np.sum(du * du), np.sum(u * u)]
    return np.array(out)


def _check(dc, model, w, xn, xr, stream=None):
    B = xn.shape[0]
    tn = torch.tensor(xn, device="cuda", dtype=torch.float32)
    tr = torch.tensor(xr, device="cuda", dtype=torch.float32)
    ref = torch.zeros(2 * B, device="cuda", dtype=torch.float32)
    got = torch.full((2 * B,), float("nan"), device="cuda", dtype=torch.float32)
    if stream is not None:
        stream.wait_stream(torch.cuda.current_stream())
    dc.drift_sums(model, tn, tr, ref, stream=stream)
    dc.drift_sums_noalloc(model, tn, tr, got, stream=stream)
    torch.cuda.synchronize()
    g, r = got.cpu().numpy().astype(np.float64), ref.cpu().numpy().astype(np.float64)
    exact = _fp64_sums(w, xn, xr)
    assert np.all(np.isfinite(g))
    assert np.all(np.abs(g - r) <= 1e-5 * np.abs(r)), (g, r)
    assert np.all(np.abs(g - exact) <= 1e-5 * np.abs(exact)), (g, exact)


def test_noalloc_drift_sums_match_allocating_entry(dc):
    wl = WORKLOADS["c2"].with_(n_blocks=1, frames=2, rows=9, cols=17, batch=6, steps=2)
    w = gen.weights(wl)
    model = dc.Model(wl, gen.flat_blob(wl, w))
    rng = np.random.default_rng(11)
    for call, B in enumerate((6, 3)):  # two calls in a row, different inputs and sizes
        xn = rng.standard_normal((B, wl.n_tokens, wl.channels)).astype(np.float32)
        xr = (xn + 0.05 * (call + 1) * rng.standard_normal(xn.shape)).astype(np.float32)
        _check(dc, model, w, xn, xr)
    # one scene on a stream of the caller's, twice in a row
    side = torch.cuda.Stream()
    for call in range(2):
        xn = rng.standard_normal((1, wl.n_tokens, wl.channels)).astype(np.float32)
        xr = (xn + 0.1 * rng.standard_normal(xn.shape)).astype(np.float32)
        _check(dc, model, w, xn, xr, stream=side)
    # more scenes than the model (and the fixed scratch) holds is refused
    big = torch.zeros((7, wl.n_tokens, wl.channels), device="cuda", dtype=torch.float32)
    with pytest.raises(dc.DCError):
        dc.drift_sums_noalloc(model, big, big, torch.zeros(14, device="cuda", dtype=torch.float32))
    model.close()
