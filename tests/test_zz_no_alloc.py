"""dc_drift_sums_noalloc: the drift sums for callers that cannot allocate
device memory while running (fixed start-up memory budgets, hosts that may
not call cudaMalloc after initialisation).  Checked through the C ABI
against dc_drift_sums on the same inputs, over two calls in a row that share
the library's fixed scratch array.  This file is collected last."""

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


def test_noalloc_drift_sums_match_allocating_entry(dc):
    wl = WORKLOADS["c2"].with_(n_blocks=1, frames=2, rows=9, cols=17, batch=6, steps=2)
    model = dc.Model(wl, gen.flat_blob(wl, gen.weights(wl)))
    rng = np.random.default_rng(11)
    for call, B in enumerate((6, 3)):  # two calls in a row, different inputs and sizes
        xn = rng.standard_normal((B, wl.n_tokens, wl.channels)).astype(np.float32)
        xr = (xn + 0.05 * (call + 1) * rng.standard_normal(xn.shape)).astype(np.float32)
        tn = torch.tensor(xn, device="cuda", dtype=torch.float32)
        tr = torch.tensor(xr, device="cuda", dtype=torch.float32)
        ref = torch.zeros(2 * B, device="cuda", dtype=torch.float32)
        got = torch.full((2 * B,), float("nan"), device="cuda", dtype=torch.float32)
        dc.drift_sums(model, tn, tr, ref)
        dc.drift_sums_noalloc(model, tn, tr, got)
        torch.cuda.synchronize()
        g, r = got.cpu().numpy(), ref.cpu().numpy()
        assert np.all(np.isfinite(g))
        assert np.all(np.abs(g - r) <= 1e-5 * np.abs(r)), (call, g, r)
    # more scenes than the model (and the fixed scratch) holds is refused
    big = torch.zeros((7, wl.n_tokens, wl.channels), device="cuda", dtype=torch.float32)
    with pytest.raises(dc.DCError):
        dc.drift_sums_noalloc(model, big, big, torch.zeros(14, device="cuda", dtype=torch.float32))
    model.close()
