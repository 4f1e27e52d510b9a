"""Sampler-state snapshots through the C ABI (dc_denoise_steps).

A call stopped after any step and resumed from its snapshot -- on the same
model instance or on another one -- ends with the latents and the record of
the uninterrupted call bit for bit, through drift checks, refusals, replans
and guidance; the resumed result therefore still matches the oracle's
controller (Sec. 3.2) as the uninterrupted call does.  Invalid resumes fail
before any launch."""

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


def _calibrated(wl):
    w = gen.weights(wl)
    om = Ctl.build(wl, w)
    K, H = wl.steps, wl.h_max
    sig = gen.sigmas(K)
    q0, q1 = gen.synthetic_q_tables(K, H)
    anc, tabs, tau, _ = Ctl.calibrate(om, wl, gen.calibration_trajectories(wl),
                                      gen.anchor_noise(wl), sig, q0, q1, wl.target())
    return w, om, sig, anc, tabs, tau


def _same_record(a, b):
    for key in a:
        if key == "launches":
            continue
        x, y = np.asarray(a[key]), np.asarray(b[key])
        if x.dtype.kind == "f":
            assert np.array_equal(x, y, equal_nan=True), key
        else:
            assert np.array_equal(x, y), key


def _straight(dc, model, x1, trajs, sched):
    lat = torch.tensor(np.asarray(x1, np.float32), device="cuda")
    st = dc.denoise(model, lat, list(trajs), sched)
    torch.cuda.synchronize()
    return lat.cpu().numpy(), st


def _resumed(dc, models, x1, trajs, sched, stops):
    """Run through each k in stops, saving and resuming between calls; the
    i-th call runs on models[i % len(models)] with fresh latent storage."""
    snap = None
    for i, k in enumerate(stops):
        m = models[i % len(models)]
        lat = torch.tensor(np.asarray(x1, np.float32), device="cuda")
        if snap is not None:
            lat.fill_(np.nan)  # the snapshot supplies x_{k0+1}
        last = i == len(stops) - 1
        st, out = dc.denoise_steps(m, lat, list(trajs), sched, k, resume=snap, save=not last)
        torch.cuda.synchronize()
        if not last:
            info = dc.snapshot_info(out)
            assert info["k_done"] == k and info["B"] == len(trajs)
            snap = out
    return lat.cpu().numpy(), st


def test_fp32_controller_resume_after_every_step(dc):
    wl = WORKLOADS["c1"]
    w, om, sig, anc, tabs, tau = _calibrated(wl)
    K, H = wl.steps, wl.h_max
    x1 = gen.latents(wl)
    trajs = gen.scene_trajectories(wl)
    model = dc.Model(wl, gen.flat_blob(wl, w))
    sched = dc.SchedArgs(K, sig, dc.AnchorArgs(K, H, anc, tabs), tau)
    ref_x, ref_st = _straight(dc, model, x1, trajs, sched)
    assert ref_st["n_reuse"][0] >= 1
    for k in range(1, K):
        got, st = _resumed(dc, [model], x1, trajs, sched, [k, K])
        assert np.array_equal(got, ref_x), k
        _same_record(st, ref_st)
    model.close()
    # and the resumed call is the oracle's controller run
    ref = Ctl.denoise(om, x1, trajs, sig, anc, tabs, tau, K, H)
    assert st["executed"][0].tolist()[1:] == ref["executed"][0][1:]
    assert np.linalg.norm(got - ref["x"]) <= 1e-4 * np.linalg.norm(ref["x"])


def test_fp32_refusals_and_replans_across_a_snapshot(dc):
    """Zero drift thresholds: every planned reuse is refused and the suffix
    replanned; the replanned plan travels in the snapshot."""
    wl = WORKLOADS["c1"]
    w = gen.weights(wl)
    K, H = wl.steps, wl.h_max
    sig = gen.sigmas(K)
    q0, q1 = gen.synthetic_q_tables(K, H)
    z = np.zeros((K, H + 1))
    anc = dict(L0=0.0, T0=0.0, L1=10.0, T1=1.0, valid=1)
    tabs = dict(q0=q0, q1=q1, d0=z, d1=z)
    x1 = gen.latents(wl)
    trajs = gen.scene_trajectories(wl)
    a, b = dc.Model(wl, gen.flat_blob(wl, w)), dc.Model(wl, gen.flat_blob(wl, w))
    sched = dc.SchedArgs(K, sig, dc.AnchorArgs(K, H, anc, tabs), 0.2)
    ref_x, ref_st = _straight(dc, a, x1, trajs, sched)
    assert ref_st["n_veto"][0] >= 1 and ref_st["n_replan"][0] >= 1
    for stops in ([3, K], [2, 5, K], list(range(1, K + 1))):
        got, st = _resumed(dc, [a, b], x1, trajs, sched, stops)
        assert np.array_equal(got, ref_x), stops
        _same_record(st, ref_st)
    a.close()
    b.close()


@pytest.mark.parametrize("forced", [False, True])
def test_bf16_guidance_migrates_between_instances(dc, forced):
    """bf16 model with guidance (two branch caches per scene), under the
    calibrated controller or a forced schedule with reuses; the call hops
    between two model instances."""
    base = WORKLOADS["c2"].with_(n_blocks=2, frames=3, rows=10, cols=13, batch=3, steps=10,
                                 rho_tar=0.4)
    w, om, sig, anc, tabs, tau = _calibrated(base)
    wl = base.with_(batch=2)
    K, H = wl.steps, wl.h_max
    x1 = gen.latents(wl)
    trajs = gen.scene_trajectories(base)[:2]
    a = dc.Model(wl, gen.flat_blob(wl, w), max_batch=4)
    b = dc.Model(wl, gen.flat_blob(wl, w), max_batch=4)
    acts = None
    if forced:
        acts = np.array([[0, 1, 2, 2, 1, 2, 2, 2, 1, 2, 1],
                         [0, 1, 1, 2, 2, 1, 2, 1, 2, 2, 2]], np.uint8)
    sched = dc.SchedArgs(K, sig, dc.AnchorArgs(K, H, anc, tabs), tau, cfg_scale=3.0,
                         forced=acts)
    ref_x, ref_st = _straight(dc, a, x1, trajs, sched)
    if forced:
        assert ref_st["n_reuse"].sum() == 12
    got, st = _resumed(dc, [b, a, b], x1, trajs, sched, [3, 6, K])
    assert np.array_equal(got, ref_x)
    _same_record(st, ref_st)
    a.close()
    b.close()


def test_invalid_resumes_fail_before_launch(dc):
    wl = WORKLOADS["c1"]
    w, om, sig, anc, tabs, tau = _calibrated(wl)
    K, H = wl.steps, wl.h_max
    x1 = gen.latents(wl)
    trajs = gen.scene_trajectories(wl)
    model = dc.Model(wl, gen.flat_blob(wl, w))
    sched = dc.SchedArgs(K, sig, dc.AnchorArgs(K, H, anc, tabs), tau)
    lat = torch.tensor(x1, device="cuda")
    _, snap = dc.denoise_steps(model, lat, list(trajs), sched, 4, save=True)
    before = lat.clone()
    bad = []
    other_tau = dc.SchedArgs(K, sig, dc.AnchorArgs(K, H, anc, tabs), tau * 0.5)
    bad.append(lambda: dc.denoise_steps(model, lat, list(trajs), other_tau, K, resume=snap))
    moved = [t.copy() for t in trajs]
    moved[0][-1, 0] += 1.0
    bad.append(lambda: dc.denoise_steps(model, lat, moved, sched, K, resume=snap))
    bad.append(lambda: dc.denoise_steps(model, lat, list(trajs), sched, 4, resume=snap))
    bad.append(lambda: dc.denoise_steps(model, lat, list(trajs), sched, K + 1, resume=snap))
    cut = snap[:-1]
    bad.append(lambda: dc.denoise_steps(model, lat, list(trajs), sched, K, resume=cut))
    magic = snap.copy()
    magic[0] ^= 1
    bad.append(lambda: dc.denoise_steps(model, lat, list(trajs), sched, K, resume=magic))
    for f in bad:
        with pytest.raises(dc.DCError):
            f()
    torch.cuda.synchronize()
    assert torch.equal(lat, before)
    # a bf16 model (of another width) rejects the fp32 snapshot
    bwl = wl.with_(dtype="bf16", d_model=192, n_heads=3)
    bw = gen.weights(bwl)
    other = dc.Model(bwl, gen.flat_blob(bwl, bw))
    with pytest.raises(dc.DCError):
        dc.denoise_steps(other, lat, list(trajs), sched, K, resume=snap)
    other.close()
    model.close()
