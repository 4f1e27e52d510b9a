"""Pins for the oracle's joint run responses (Eq. 6-7): every tangent is
checked against central finite differences of the primal in fp64, one DiT
block against torch.func.jvp (forward-mode AD) of the block written with torch
modules, the propagated perturbation P_t e against differencing the
nonlinear sampler itself, and the table against a closed form (last row)
and an exact zero (identity blocks)."""

import math

import numpy as np
import pytest
import torch

import synth
from oracle import dit as O
from oracle import response as R
from synth import gen


def _fd(f, x, dx, h=1e-6):
    return (f(x + h * dx) - f(x - h * dx)) / (2 * h)


def _rel(a, b):
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def test_layer_norm_and_gelu_tangents_vs_finite_differences():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((7, 40)) * 2 + 0.5
    dx = rng.standard_normal((7, 40))
    assert _rel(R.layer_norm_jvp(x, dx), _fd(O.layer_norm, x, dx)) < 1e-8
    z = np.linspace(-6, 6, 301)
    assert _rel(R.gelu_tanh_grad(z) * 1.0, _fd(O.gelu_tanh, z, np.ones_like(z))) < 1e-8
    t = torch.tensor(z, dtype=torch.float64, requires_grad=True)
    torch.nn.functional.gelu(t, approximate="tanh").sum().backward()
    assert np.abs(R.gelu_tanh_grad(z) - t.grad.numpy()).max() < 1e-14


def test_attention_tangent_vs_finite_differences():
    rng = np.random.default_rng(1)
    q, k, v = (rng.standard_normal((3, 20, 8)) * s for s in (2.0, 1.0, 1.0))
    dq, dk, dv = (rng.standard_normal((3, 20, 8)) for _ in range(3))
    _, do = R.attention_jvp(q, k, v, dq, dk, dv)
    fd = (O.attention_core(q + 1e-6 * dq, k + 1e-6 * dk, v + 1e-6 * dv)
          - O.attention_core(q - 1e-6 * dq, k - 1e-6 * dk, v - 1e-6 * dv)) / 2e-6
    assert _rel(do, fd) < 1e-8


def test_block_tangent_vs_torch_jvp():
    """torch.func.jvp (forward-mode AD) of the block written with torch modules
    (LayerNorm, MultiheadAttention, Linear, GELU(tanh)) in fp64."""
    wl = synth.WORKLOADS["c1"]
    w = gen.weights(wl)
    rng = np.random.default_rng(2)
    n, d = 24, wl.d_model
    h = rng.standard_normal((n, d))
    dh = rng.standard_normal((n, d))
    mod = {k: rng.standard_normal(d) * 0.3 for k in ("shift1", "scale1", "gate1", "shift2", "scale2", "gate2")}
    wb = {k: np.asarray(v, np.float64) * 10 for k, v in O.block_weights(w, 1).items()}
    f64 = dict(dtype=torch.float64)
    ln = torch.nn.LayerNorm(d, eps=1e-6, elementwise_affine=False, **f64)
    mha = torch.nn.MultiheadAttention(d, wl.n_heads, bias=True, batch_first=True, **f64)
    fc1 = torch.nn.Linear(d, wb["w_1"].shape[0], **f64)
    fc2 = torch.nn.Linear(wb["w_1"].shape[0], d, **f64)
    T = lambda a: torch.tensor(np.asarray(a, np.float64))
    with torch.no_grad():
        mha.in_proj_weight.copy_(T(wb["w_qkv"])); mha.in_proj_bias.copy_(T(wb["b_qkv"]))
        mha.out_proj.weight.copy_(T(wb["w_o"])); mha.out_proj.bias.copy_(T(wb["b_o"]))
        fc1.weight.copy_(T(wb["w_1"])); fc1.bias.copy_(T(wb["b_1"]))
        fc2.weight.copy_(T(wb["w_2"])); fc2.bias.copy_(T(wb["b_2"]))
    m = {k: T(v) for k, v in mod.items()}

    def blk(x):
        a = ln(x) * (1 + m["scale1"]) + m["shift1"]
        o, _ = mha(a[None], a[None], a[None], need_weights=False)
        x = x + m["gate1"] * o[0]
        a = ln(x) * (1 + m["scale2"]) + m["shift2"]
        return x + m["gate2"] * fc2(torch.nn.functional.gelu(fc1(a), approximate="tanh"))

    from torch.nn.attention import SDPBackend, sdpa_kernel
    with sdpa_kernel(SDPBackend.MATH):  # the reference kernel, which has forward-mode AD
        _, ref = torch.func.jvp(blk, (T(h),), (T(dh),))
    _, got = R.block_jvp(wb, h, dh, mod, wl.n_heads)
    assert _rel(got, ref.detach().numpy()) < 1e-11


def _tiny():
    wl = synth.WORKLOADS["c1"]
    w = gen.weights(wl)
    for k in list(w):  # stronger blocks so the Jacobian is far from the identity
        if k.startswith("blk"):
            w[k] = np.asarray(w[k]) * 8
    return wl, O.Model(wl, w)


def test_velocity_tangent_vs_finite_differences():
    wl, m = _tiny()
    rng = np.random.default_rng(3)
    x = rng.standard_normal((wl.n_tokens, wl.channels))
    dx = rng.standard_normal(x.shape)
    poses = gen.unicycle(4.0, 0.2, wl.n_poses)
    f = lambda y: m.full_step(y, 0.6, poses)[0]
    assert _rel(R.velocity_jvp(m, x, dx, 0.6, poses), _fd(f, x, dx, 1e-5)) < 1e-7


def test_propagated_perturbation_vs_nonlinear_sampler():
    """P_t e against re-running the sampler with v_t + h e (and every later
    velocity recomputed by the model), differenced centrally."""
    wl, m = _tiny()
    K = 6
    sig = gen.sigmas(K)
    poses = gen.unicycle(4.0, 0.2, wl.n_poses)
    x1 = gen.latents(wl)[0]
    xs, _ = R.frozen_trace(m, x1, poses, sig, K)
    e = np.random.default_rng(4).standard_normal(x1.shape)
    t = 2

    def final(hh):
        x = xs[t].copy()
        v = m.full_step(x, sig[t - 1], poses)[0] + hh * e
        x = O.euler(x, v, sig[t - 1], sig[t])
        for k in range(t + 1, K + 1):
            x = O.euler(x, m.full_step(x, sig[k - 1], poses)[0], sig[k - 1], sig[k])
        return x

    fd = (final(1e-5) - final(-1e-5)) / 2e-5
    got = R.propagate(m, xs, poses, sig, K, t, e)
    assert _rel(got, fd) < 1e-7
    # the Jacobians matter: the frozen-sampler-only product dsig_t e is far off
    assert _rel((sig[t] - sig[t - 1]) * e, fd) > 1e-3


def test_response_table_closed_forms():
    wl, m = _tiny()
    K, H = 5, 3
    sig = gen.sigmas(K)
    poses = gen.unicycle(4.0, 0.2, wl.n_poses)
    x1 = gen.latents(wl)[0]
    q, xs, rs = R.response_table(m, x1, poses, sig, K, H)
    # last row: only l = 1 exists and nothing follows step K: G = dsig_K e
    e = m.reuse_step(xs[K], rs[K - 1], sig[K - 1], poses)[0] - m.reuse_step(xs[K], rs[K], sig[K - 1], poses)[0]
    want = abs(sig[K] - sig[K - 1]) * np.linalg.norm(e) / (np.linalg.norm(xs[K + 1]) + 1e-6)
    assert abs(q[K - 1][1] - want) <= 1e-13 * want
    assert all(q[j][h] == 0.0 for j in range(1, K) for h in range(min(H, K - j) + 1, H + 1))
    assert all(q[j][h] > 0.0 for j in range(1, K) for h in range(1, min(H, K - j) + 1))


def test_identity_blocks_give_zero_response():
    """Zero gates: every r is 0, so every e (Eq. 6) and every q vanish."""
    wl = synth.WORKLOADS["c1"]
    w = gen.weights(wl)
    d, L = wl.d_model, wl.n_blocks
    for l in range(L):
        w["w_ada"][6 * l * d + 2 * d:6 * l * d + 3 * d] = 0
        w["w_ada"][6 * l * d + 5 * d:6 * l * d + 6 * d] = 0
    m = O.Model(wl, w)
    K, H = 4, 2
    q, _, _ = R.response_table(m, gen.latents(wl)[0], gen.unicycle(3.0, 0.1, wl.n_poses), gen.sigmas(K), K, H)
    assert all(v == 0.0 for row in q for v in row)
