"""Pins for the oracle's anchor drift tables (Eq. 5) and the drift it logs at
each pre-reuse check (Eq. 12), on a backbone whose trace has a closed form.

With every block gate at zero the block stack is the identity, and with the
output head's weight at zero and its bias at a vector c the velocity is c at
every token and step.  The Euler sampler then gives x_k = x_1 + (sigma_k - 1) c
(sigma_1 = 1), the backbone input is u_k = x_k W_e^T + b_e + pos, and

    u_{k'} - u_k = (sigma_{k'} - sigma_k) 1 (W_e c)^T      (the same row at every token)

so the numerator of Eq. 5 / Eq. 12 is |sigma_{k'} - sigma_k| sqrt(N) ||W_e c||
without running the sampler, and the denominator is the norm of the LATER
input.  A table built from the wrong pair of steps, or normalised by the
earlier input, misses these values."""

import math

import numpy as np

import synth
from oracle import controller as Ctl
from oracle import dit as O
from oracle import planner as P
from synth import gen

C_VEL = np.array([1.5, -2.0, 0.75, 3.0])  # the constant velocity (c1 has C = 4)


def _constant_velocity_model(wl):
    w = gen.weights(wl)
    d, L = wl.d_model, wl.n_blocks
    w_ada = np.array(w["w_ada"], np.float64)
    b_ada = np.array(w["b_ada"], np.float64)
    for l in range(L):
        for g in (2, 5):  # gate1, gate2 rows of block l
            rows = slice((6 * l + g) * d, (6 * l + g + 1) * d)
            w_ada[rows] = 0.0
            b_ada[rows] = 0.0
    w = dict(w, w_ada=w_ada, b_ada=b_ada, w_final=np.zeros_like(w["w_final"]),
             b_final=C_VEL.copy())
    return O.Model(wl, w), w


def _u_closed(w, x1, sig_k):
    """u at the step whose sigma is sig_k, from x_k = x_1 + (sig_k - 1) c."""
    x = np.asarray(x1, np.float64) + (sig_k - 1.0) * C_VEL
    return x @ np.asarray(w["w_embed"], np.float64).T + w["b_embed"] + w["pos"]


def _d_closed(w, x1, sig, k_ref, k_now, n_tok, eps=P.EPS):
    """Eq. 5 / Eq. 12 between steps k_ref < k_now (1-based) in closed form."""
    row = np.asarray(w["w_embed"], np.float64) @ C_VEL  # W_e c, one row of u_{k'} - u_k
    num = abs(sig[k_now - 1] - sig[k_ref - 1]) * math.sqrt(n_tok) * float(np.linalg.norm(row))
    u_now = _u_closed(w, x1, sig[k_now - 1])
    return num / (math.sqrt(float(np.sum(u_now * u_now))) + eps)


def test_constant_velocity_trace_closed_form():
    wl = synth.WORKLOADS["c1"]
    m, w = _constant_velocity_model(wl)
    K, H = wl.steps, wl.h_max
    sig = gen.sigmas(K)
    x1 = gen.anchor_noise(wl)
    _, us = Ctl.anchor_trace_drift(m, x1, gen.calibration_trajectories(wl)[0], sig, K, H)
    for k in range(1, K + 1):
        assert np.abs(us[k] - _u_closed(w, x1, sig[k - 1])).max() < 1e-12, k


def test_anchor_drift_table_closed_form():
    """Every entry d_{j,l} of the Eq. 5 table, j = 1..K-1, l = 1..min(H, K-j)."""
    wl = synth.WORKLOADS["c1"]
    m, w = _constant_velocity_model(wl)
    K, H = wl.steps, wl.h_max
    sig = gen.sigmas(K)
    x1 = gen.anchor_noise(wl)
    d, _ = Ctl.anchor_trace_drift(m, x1, gen.calibration_trajectories(wl)[5], sig, K, H)
    n_checked = 0
    for j in range(1, K):
        for l in range(1, H + 1):
            if j + l > K:
                assert d[j][l] == 0.0
                continue
            want = _d_closed(w, x1, sig, j, j + l, wl.n_tokens)
            assert abs(d[j][l] - want) <= 1e-12 * want, (j, l, d[j][l], want)
            n_checked += 1
    assert n_checked == sum(min(H, K - j) for j in range(1, K))
    # the drift grows with the lag at every refresh step (|sigma| steps add up)
    for j in range(1, K - 1):
        assert d[j][1] < d[j][2]


def test_controller_logged_drift_closed_form():
    """A scripted call: thresholds so loose that every check accepts, so the
    plan runs as made and each logged d_obs compares the step's input with
    the input of its refresh step (Eq. 12)."""
    wl = synth.WORKLOADS["c1"]
    m, w = _constant_velocity_model(wl)
    K, H = wl.steps, wl.h_max
    sig = gen.sigmas(K)
    q0, q1 = gen.synthetic_q_tables(K, H)
    big = [[1e9] * (H + 1) for _ in range(K)]
    tabs = dict(q0=q0, q1=q1, d0=big, d1=big)
    anc = dict(L0=0.0, T0=0.0, L1=10.0, T1=1.0, valid=1)
    tr = gen.scene_trajectories(wl)
    x1 = gen.latents(wl)
    out = Ctl.denoise(m, x1, tr, sig, anc, tabs, 1e9, K, H)
    log = out["log"][0]
    assert len(log) >= 3 and all(e["accept"] for e in log)
    ages = {e["h"] for e in log}
    assert max(ages) >= 2  # some checks reach back more than one step
    for e in log:
        k, j = e["k"], e["j"]
        assert j == k - e["h"]
        want = _d_closed(w, x1[0], sig, j, k, wl.n_tokens)
        assert abs(e["d_obs"] - want) <= 1e-12 * want, (e, want)
    # the sampler's output is the closed-form latent after the last step
    assert np.abs(out["x"][0] - (x1[0] + (sig[K] - 1.0) * C_VEL)).max() < 1e-12
