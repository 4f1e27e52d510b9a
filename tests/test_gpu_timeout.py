"""Failure detection of the device kernels, made to fire on purpose.

Every wait of the tensor-core kernels (GEMM, attention, adaLN table) is
bounded: when one gives up, the kernel records a code in the model's error
word, drains the copies and MMAs it has issued, frees its tensor memory and
returns; later tensor-core launches of the call skip their work, and the
host returns DC_ERR_DEVICE_TIMEOUT and clears the word.  Here the wait limit
is cut to 1 ns (dc_set_wait_limit), so every wait that is not satisfied at
once gives up: the call must come back with DC_ERR_DEVICE_TIMEOUT (not hang,
not fault), the stream must complete, and with the limit restored the next
call on the same model must give exactly the result of a call made before,
which the oracle confirms (Eq. 1 interface and Euler update, bf16 bound)."""

import numpy as np
import pytest

from oracle import controller as Ctl
from oracle import planner as P
from synth import WORKLOADS, gen

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

DC_ERR_DEVICE_TIMEOUT = 4


@pytest.fixture(scope="module")
def dc():
    from paper_2608_16354_gb300 import _build, binding
    _build.build()
    binding.lib()
    return binding


def rel(a, b):
    return float(np.linalg.norm(np.asarray(a, np.float64) - b) / max(np.linalg.norm(b), 1e-30))


@pytest.mark.timeout(300)
def test_bounded_waits_run_out_and_the_model_recovers(dc):
    # d 3072 / dh 128, 2025 tokens, one block: the GEMMs run K loops of up to
    # 12288 (tens of microseconds per tile), so their epilogue waits, and the
    # attention's, outlast any wait limit of a few microseconds (an mbarrier
    # try_wait itself may block for a while before it reports "not yet");
    # one compute and one reuse step
    wl = WORKLOADS["c5"].with_(n_blocks=1, frames=1, rows=45, cols=45, batch=1, steps=2)
    w = gen.weights(wl)
    K = wl.steps
    sig = gen.sigmas(K)
    x1 = gen.latents(wl)
    trajs = list(gen.scene_trajectories(wl))
    forced = np.array([[0, P.COMPUTE, P.REUSE]] * wl.batch, np.uint8)
    model = dc.Model(wl, gen.flat_blob(wl, w), max_batch=wl.batch, max_steps=K)
    na = dc.AnchorArgs(K, wl.h_max, dict(L0=0, T0=0, L1=0, T1=0, valid=0), dict(q0=None, q1=None))
    sched = dc.SchedArgs(K, sig, na, 0.0, forced=forced)

    def run():
        lat = torch.tensor(x1, device="cuda")
        dc.denoise(model, lat, trajs, sched)
        torch.cuda.synchronize()
        return lat.cpu().numpy()

    before = run()
    dc.set_wait_limit(model, 1)
    lat = torch.tensor(x1, device="cuda")
    with pytest.raises(dc.DCError) as ei:
        dc.denoise(model, lat, trajs, sched)
    assert ei.value.status == DC_ERR_DEVICE_TIMEOUT, str(ei.value)
    torch.cuda.synchronize()  # every launch of the failed call has returned
    dc.set_wait_limit(model, 0)
    after = run()
    assert np.array_equal(after, before)
    model.close()
    # and the recovered result is the oracle's (forced schedule replay)
    om = Ctl.build(wl, w)
    ref = Ctl.denoise(om, x1, trajs, sig, dict(valid=0), None, 0.0, K, wl.h_max,
                      forced=forced.tolist())
    assert rel(after, ref["x"]) <= 2e-2
    assert rel(after - x1, ref["x"] - x1) <= 2e-2
