"""Replica harness on the GPU: scenes split across replicas (emulated in one
process, one model instance per replica) and across batches give every
scene exactly the latents and the record of a single call over all scenes --
scenes share no state (Sec. 3.2), and every kernel treats rows, slots and
scenes independently."""

import numpy as np
import pytest

from oracle import controller as Ctl
from synth import WORKLOADS, gen

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dc():
    from paper_2608_16354_gb300 import _build, binding
    _build.build()
    binding.lib()
    return binding


@pytest.mark.parametrize("world,batch", [(2, None), (3, 1), (2, 2)])
def test_sharded_serving_equals_one_call(dc, world, batch):
    from paper_2608_16354_gb300 import replicas
    wl = WORKLOADS["c2"].with_(n_blocks=2, frames=3, rows=10, cols=13, batch=5, steps=10,
                               rho_tar=0.4)
    w = gen.weights(wl)
    om = Ctl.build(wl, w)
    K, H = wl.steps, wl.h_max
    sig = gen.sigmas(K)
    q0, q1 = gen.synthetic_q_tables(K, H)
    anc, tabs, tau, _ = Ctl.calibrate(om, wl, gen.calibration_trajectories(wl),
                                      gen.anchor_noise(wl), sig, q0, q1, wl.target())
    sched = dc.SchedArgs(K, sig, dc.AnchorArgs(K, H, anc, tabs), tau)
    x1 = np.asarray(gen.latents(wl), np.float32)
    trajs = list(gen.scene_trajectories(wl))
    one = dc.Model(wl, gen.flat_blob(wl, w), max_batch=wl.batch)
    x_ref = x1.copy()
    rec = dc.denoise_host(one, x_ref, trajs, sched)
    one.close()
    assert rec["n_reuse"].sum() >= 1
    merged = {}
    for r in range(world):
        m = dc.Model(wl, gen.flat_blob(wl, w), max_batch=3)
        merged.update(replicas.serve_shard(m, x1, trajs, sched, r, world, batch))
        m.close()
    assert sorted(merged) == list(range(wl.batch))
    for s in range(wl.batch):
        x, st = merged[s]
        assert np.array_equal(x, x_ref[s]), s
        for key, v in st.items():
            assert np.array_equal(np.asarray(v), np.asarray(rec[key][s]), equal_nan=True), (s, key)
