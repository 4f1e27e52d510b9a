"""Pins for the oracle's backbone, interface and sampler (Eq. 1 split of the
synthetic DiT).  Library routines (torch fp64 modules) and closed forms pin
each op; special cases pin the reuse/compute equivalence."""

import math

import numpy as np
import pytest
import torch

import synth
from oracle import dit as O
from oracle import controller as Ctl
from oracle import planner as P
from synth import gen

def _t(a):
    return torch.tensor(np.asarray(a, np.float64), dtype=torch.float64)


def test_layer_norm_vs_torch():
    x = np.random.default_rng(0).standard_normal((37, 72)) * 3 + 1
    ref = torch.nn.functional.layer_norm(_t(x), (72,), eps=1e-6).numpy()
    assert np.abs(O.layer_norm(x) - ref).max() < 1e-12


def test_gelu_silu_vs_torch():
    x = np.linspace(-8, 8, 1001)
    assert np.abs(O.gelu_tanh(x) - torch.nn.functional.gelu(_t(x), approximate="tanh").numpy()).max() < 1e-13
    assert np.abs(O.silu(x) - torch.nn.functional.silu(_t(x)).numpy()).max() < 1e-13


def test_softmax_closed_form():
    p = O.softmax(np.array([[0.0, math.log(3.0)]]))
    assert np.allclose(p, [[0.25, 0.75]], atol=1e-15, rtol=0)


@pytest.mark.parametrize("n,d,heads", [(50, 64, 4), (33, 72, 6)])
def test_attention_vs_torch_multihead(n, d, heads):
    """MHSA + out-projection against torch.nn.MultiheadAttention with the
    same packed [q|k|v] in-projection: pins the split order, the head layout
    and the 1/sqrt(dh) scale."""
    rng = np.random.default_rng(1)
    a = rng.standard_normal((n, d))
    w_qkv = rng.standard_normal((3 * d, d)) * 0.2
    b_qkv = rng.standard_normal(3 * d) * 0.1
    w_o = rng.standard_normal((d, d)) * 0.2
    b_o = rng.standard_normal(d) * 0.1
    ours = O.linear(O.attention(a, w_qkv, b_qkv, heads), w_o, b_o)
    mha = torch.nn.MultiheadAttention(d, heads, bias=True, batch_first=True, dtype=torch.float64)
    with torch.no_grad():
        mha.in_proj_weight.copy_(_t(w_qkv))
        mha.in_proj_bias.copy_(_t(b_qkv))
        mha.out_proj.weight.copy_(_t(w_o))
        mha.out_proj.bias.copy_(_t(b_o))
        ref, _ = mha(_t(a)[None], _t(a)[None], _t(a)[None], need_weights=False)
    assert np.abs(ours - ref[0].numpy()).max() < 1e-12


def _torch_block(wb, h, mod, heads):
    """The block written with torch modules (LayerNorm without affine,
    MultiheadAttention, Linear, GELU(tanh))."""
    d = h.shape[1]
    f64 = dict(dtype=torch.float64)
    ln = torch.nn.LayerNorm(d, eps=1e-6, elementwise_affine=False, **f64)
    mha = torch.nn.MultiheadAttention(d, heads, bias=True, batch_first=True, **f64)
    fc1 = torch.nn.Linear(d, wb["w_1"].shape[0], **f64)
    fc2 = torch.nn.Linear(wb["w_1"].shape[0], d, **f64)
    with torch.no_grad():
        mha.in_proj_weight.copy_(_t(wb["w_qkv"]))
        mha.in_proj_bias.copy_(_t(wb["b_qkv"]))
        mha.out_proj.weight.copy_(_t(wb["w_o"]))
        mha.out_proj.bias.copy_(_t(wb["b_o"]))
        fc1.weight.copy_(_t(wb["w_1"]))
        fc1.bias.copy_(_t(wb["b_1"]))
        fc2.weight.copy_(_t(wb["w_2"]))
        fc2.bias.copy_(_t(wb["b_2"]))
        x = _t(h)
        m = {k: _t(v) for k, v in mod.items()}
        a = ln(x) * (1 + m["scale1"]) + m["shift1"]
        o, _ = mha(a[None], a[None], a[None], need_weights=False)
        x = x + m["gate1"] * o[0]
        a = ln(x) * (1 + m["scale2"]) + m["shift2"]
        x = x + m["gate2"] * fc2(torch.nn.functional.gelu(fc1(a), approximate="tanh"))
    return x.numpy()


def test_block_vs_torch_modules():
    wl = synth.WORKLOADS["c1"]
    w = gen.weights(wl)
    rng = np.random.default_rng(3)
    h = rng.standard_normal((wl.n_tokens, wl.d_model))
    mod = {k: rng.standard_normal(wl.d_model) * 0.3
           for k in ("shift1", "scale1", "gate1", "shift2", "scale2", "gate2")}
    wb = {k: np.asarray(v, np.float64) * 10 for k, v in O.block_weights(w, 1).items()}
    ours = O.block(wb, h, mod, wl.n_heads)
    ref = _torch_block(wb, h, mod, wl.n_heads)
    assert np.abs(ours - ref).max() < 1e-11


def test_block_zero_gates_is_identity():
    wl = synth.WORKLOADS["c1"]
    w = gen.weights(wl)
    h = np.random.default_rng(4).standard_normal((wl.n_tokens, wl.d_model))
    mod = {k: np.full(wl.d_model, 0.7) for k in ("shift1", "scale1", "shift2", "scale2")}
    mod["gate1"] = np.zeros(wl.d_model)
    mod["gate2"] = np.zeros(wl.d_model)
    assert np.array_equal(O.block(O.block_weights(w, 0), h, mod, wl.n_heads), h)


def test_timestep_features_closed_form():
    f = O.timestep_features(0.0)
    assert np.array_equal(f, np.concatenate([np.ones(128), np.zeros(128)]))
    f = O.timestep_features(0.001)  # t = 1: i = 0 has frequency 1
    assert abs(f[0] - math.cos(1.0)) < 1e-15 and abs(f[128] - math.sin(1.0)) < 1e-15
    assert abs(f[64] - math.cos(0.01)) < 1e-15  # f_64 = 10000^(-1/2)


def test_pose_features():
    poses = [(1.0, 2.0, 3.0), (11.0, 2.0, -3.0), (1.0, -18.0, 3.0)]
    f = O.pose_features(poses)
    assert np.allclose(f, [0, 0, 0, 1.0, 0.0, 2 * math.pi - 6.0, 0.0, -2.0, 0.0], atol=1e-15)


def test_modulation_layout():
    """With b_ada = e_i and W_ada = 0, the i-th element of the stacked
    modulation lands in the documented chunk."""
    wl = synth.WORKLOADS["c1"]
    d, L = wl.d_model, wl.n_blocks
    w = {"w_ada": np.zeros(((6 * L + 2) * d, d)), "b_ada": np.zeros((6 * L + 2) * d)}
    w["b_ada"][6 * d + 2 * d + 5] = 1.0  # block 1, gate1, channel 5
    w["b_ada"][6 * L * d + d + 7] = 2.0  # final scale, channel 7
    blocks, fin = O.modulation(w, np.zeros(d), L, d)
    assert blocks[1]["gate1"][5] == 1.0 and blocks[1]["gate1"].sum() == 1.0
    assert fin["scale"][7] == 2.0 and fin["shift"].sum() == 0.0


def test_constant_velocity_sampler_closed_form():
    """With W_f = 0 and b_f = c the head returns c everywhere, so K Euler
    steps from sigma = 1 to 0 give x_K = x_1 - c exactly (dyadic values)."""
    wl = synth.WORKLOADS["c1"]
    w = gen.weights(wl)
    w["w_final"] = np.zeros_like(w["w_final"])
    w["b_final"] = np.array([0.5, -0.25, 1.0, 0.125])
    m = O.Model(wl, w)
    x = np.random.default_rng(5).standard_normal((wl.n_tokens, wl.channels))
    K = 8
    sig = gen.sigmas(K)
    xk = x.copy()
    for k in range(K):
        v, _, _ = m.full_step(xk, sig[k], gen.unicycle(5, 0, 8))
        xk = O.euler(xk, v, sig[k], sig[k + 1])
    assert np.abs(xk - (x - w["b_final"])).max() < 1e-14


def test_reuse_equals_compute_when_blocks_are_identity():
    """Zero gates make r = 0 and h_L = u, so a reuse step reproduces the full
    step exactly (Eq. 1: H(x, r_j) with r_j = r_k)."""
    wl = synth.WORKLOADS["c1"]
    w = gen.weights(wl)
    d, L = wl.d_model, wl.n_blocks
    for l in range(L):  # zero the gate rows of the ada table
        w["w_ada"][6 * l * d + 2 * d:6 * l * d + 3 * d] = 0
        w["w_ada"][6 * l * d + 5 * d:6 * l * d + 6 * d] = 0
    m = O.Model(wl, w)
    x = np.random.default_rng(6).standard_normal((wl.n_tokens, wl.channels))
    traj = gen.unicycle(5, 0, 8)
    v, u, r = m.full_step(x, 0.7, traj)
    assert np.abs(r).max() == 0.0
    v2, _ = m.reuse_step(x, r, 0.7, traj)
    assert np.array_equal(v, v2)


def test_controller_invariants_tiny():
    """Sec. 3.2 invariants on the tiny workload: first step full, charge never
    above tau, a zero budget gives no reuse, and an all-compute forced
    schedule equals full inference."""
    wl = synth.WORKLOADS["c1"]
    w = gen.weights(wl)
    m = Ctl.build(wl, w)
    K, H = wl.steps, wl.h_max
    sig = gen.sigmas(K)
    q0, q1 = gen.synthetic_q_tables(K, H)
    anc, tabs, tau, reached = Ctl.calibrate(m, wl, gen.calibration_trajectories(wl),
                                            gen.anchor_noise(wl), sig, q0, q1, wl.target())
    assert anc["valid"] and reached
    x1 = gen.latents(wl)
    tr = gen.scene_trajectories(wl)
    out = Ctl.denoise(m, x1, tr, sig, anc, tabs, tau, K, H)
    assert out["executed"][0][1] == P.COMPUTE
    assert out["stats"][0]["charge"] <= tau
    assert out["stats"][0]["n_reuse"] == wl.target_reuses
    zero = Ctl.denoise(m, x1, tr, sig, anc, tabs, 0.0, K, H)
    assert zero["stats"][0]["n_reuse"] == 0
    allc = Ctl.denoise(m, x1, tr, sig, anc, tabs, tau, K, H,
                       forced=[[0] + [P.COMPUTE] * K])
    assert np.array_equal(allc["x"], zero["x"])


def test_controller_veto_refresh_and_replan():
    """With zero drift thresholds every planned reuse is vetoed: each veto
    evaluates the backbone, keeps the charge, and replans only the suffix."""
    wl = synth.WORKLOADS["c1"]
    m = Ctl.build(wl, gen.weights(wl))
    K, H = wl.steps, wl.h_max
    sig = gen.sigmas(K)
    q0, q1 = gen.synthetic_q_tables(K, H)
    zero = [[0.0] * (H + 1) for _ in range(K)]
    tabs = dict(q0=q0, q1=q1, d0=zero, d1=zero)
    anc = dict(L0=0.0, T0=0.0, L1=10.0, T1=1.0, valid=1)
    tr = gen.scene_trajectories(wl)
    out = Ctl.denoise(m, gen.latents(wl), tr, sig, anc, tabs, 0.2, K, H)
    st = out["stats"][0]
    assert st["n_reuse"] == 0 and st["n_veto"] >= 1 and st["charge"] == 0.0
    assert all(e["accept"] is False for e in out["log"][0])
    # each veto happened at a step the (re)plan had marked as a reuse
    plan = out["plans"][0]["actions"]
    assert out["log"][0][0]["k"] == min(k for k in range(1, K + 1) if plan[k] == P.REUSE)
