"""Pins for separate guidance branches (Sec. 3.2) in the oracle's sampler:
scale 1 reduces to the single-branch run, an all-compute run equals Euler on
v_u + g (v_c - v_u) evaluated by direct model calls, and a reuse step of
each branch reads that branch's own cache."""

import numpy as np

import synth
from oracle import controller as Ctl
from oracle import dit as O
from oracle import planner as P
from synth import gen


def _setup():
    wl = synth.WORKLOADS["c1"]
    w = gen.weights(wl)
    for k in list(w):
        if k.startswith("blk"):
            w[k] = np.asarray(w[k]) * 4
    m = Ctl.build(wl, w)
    K, H = wl.steps, wl.h_max
    sig = gen.sigmas(K)
    q0, q1 = gen.synthetic_q_tables(K, H)
    z = [[0.0] * (H + 1) for _ in range(K)]
    tabs = dict(q0=q0, q1=q1, d0=z, d1=z)
    anc = dict(L0=0.0, T0=0.0, L1=5.0, T1=1.0, valid=1)
    return wl, m, K, H, sig, tabs, anc


def test_scale_one_is_the_conditional_branch():
    wl, m, K, H, sig, tabs, anc = _setup()
    x1 = gen.latents(wl)
    tr = gen.scene_trajectories(wl)
    a = Ctl.denoise(m, x1, tr, sig, anc, tabs, 10.0, K, H, veto=False)
    b = Ctl.denoise(m, x1, tr, sig, anc, tabs, 10.0, K, H, veto=False, cfg_scale=1.0)
    assert a["executed"] == b["executed"]
    assert np.abs(a["x"] - b["x"]).max() < 1e-12


def test_all_compute_guidance_equals_direct_evaluation():
    wl, m, K, H, sig, tabs, anc = _setup()
    x1 = gen.latents(wl)
    tr = gen.scene_trajectories(wl)
    g = 2.5
    out = Ctl.denoise(m, x1, tr, sig, anc, tabs, 0.0, K, H, cfg_scale=g,
                      forced=[[0] + [P.COMPUTE] * K])
    x = np.asarray(x1[0], np.float64).copy()
    null = np.zeros((wl.n_poses, 3))
    for k in range(1, K + 1):
        v_c = m.full_step(x, sig[k - 1], tr[0])[0]
        v_u = m.full_step(x, sig[k - 1], null)[0]
        x = O.euler(x, v_u + g * (v_c - v_u), sig[k - 1], sig[k])
    assert np.abs(out["x"][0] - x).max() < 1e-13


def test_reuse_reads_each_branch_cache():
    """A forced schedule with one reuse at step 3 after a refresh at step 2:
    the guided velocity at step 3 uses r_c(2) with the trajectory and r_u(2)
    with the null trajectory."""
    wl, m, K, H, sig, tabs, anc = _setup()
    x1 = gen.latents(wl)
    tr = gen.scene_trajectories(wl)
    g = 1.7
    forced = [[0, P.COMPUTE, P.COMPUTE, P.REUSE] + [P.COMPUTE] * (K - 3)]
    out = Ctl.denoise(m, x1, tr, sig, anc, tabs, 0.0, K, H, cfg_scale=g, forced=forced, keep_trace=True)
    null = np.zeros((wl.n_poses, 3))
    x2, x3 = out["trace"][1][0], out["trace"][2][0]
    r_c = m.full_step(x2, sig[1], tr[0])[2]
    r_u = m.full_step(x2, sig[1], null)[2]
    v_c = m.reuse_step(x3, r_c, sig[2], tr[0])[0]
    v_u = m.reuse_step(x3, r_u, sig[2], null)[0]
    x4 = O.euler(x3, v_u + g * (v_c - v_u), sig[2], sig[3])
    assert np.abs(out["trace"][3][0] - x4).max() < 1e-13
