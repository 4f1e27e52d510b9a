"""Oracle: joint run responses q^(i)_{j,h} (Eq. 6-7) of one anchor trace, with
forward-mode Jacobian-vector products of the synthetic DiT, in fp64.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import this
module; only tests, the package's smoke check and the benchmark's CPU
baseline leg use it.  It shares no code with the C++/CUDA library.

Sections followed:
  Eq. 6  e_{j,l} = H_{j+l}(x_{j+l}, r_j) - H_{j+l}(x_{j+l}, r_{j+l}) along one
         full denoising trace (the anchor's trajectory and noise)
  Eq. 7  G_{j,h} = sum_{l<=h} P_{j+l} e_{j,l},  q_{j,h} = ||G_{j,h}|| / (||x_K|| + eps)

READINGS:
  * the terminal latent x_K of the paper is the latent after the last step
    (x_{K+1} here: x_1 is the input of step 1);
  * the denoiser output eps_t is the velocity v_t of step t;
  * P_t, the Jacobian of the terminal latent with respect to eps_t along the
    frozen trace, carries a perturbation through every later model
    evaluation: dx_{t+1} = dsig_t e, dx_{m+1} = dx_m + dsig_m J_m dx_m for
    m = t+1..K, J_m = dv_m/dx_m at the trace point x_m (the sampler's
    coefficients and the conditioning stay frozen).  This is what makes the
    paper's count of O(K^3) unbatched JVPs; P_t = dsig_t I would need none;
  * H_t(x, r) is the reuse interface: u_t(x) + r through the final
    modulated LayerNorm and head (both terms of Eq. 6 use cached r).
"""

import math

import numpy as np

from .dit import (LN_EPS, attention_core, block_weights, embed, euler, f64, gelu_tanh,
                  layer_norm, linear)


# ---------------------------------------------------- op tangents (d f[x] dx)

def layer_norm_jvp(x, dx, eps=LN_EPS):
    """y = (x - mu) / sigma over the last axis; dy = (dx - mean(dx) - y mean(y dx)) / sigma."""
    x, dx = f64(x), f64(dx)
    mu = x.mean(axis=-1, keepdims=True)
    sig = np.sqrt(((x - mu) ** 2).mean(axis=-1, keepdims=True) + eps)
    y = (x - mu) / sig
    return (dx - dx.mean(axis=-1, keepdims=True) - y * (y * dx).mean(axis=-1, keepdims=True)) / sig


def gelu_tanh_grad(x):
    """d/dx of 0.5 x (1 + tanh(k (x + c x^3)))."""
    x = f64(x)
    k, c = math.sqrt(2.0 / math.pi), 0.044715
    t = np.tanh(k * (x + c * x ** 3))
    return 0.5 * (1.0 + t) + 0.5 * x * (1.0 - t * t) * k * (1.0 + 3.0 * c * x * x)


def attention_jvp(q, k, v, dq, dk, dv):
    """o = softmax(q k^T / sqrt dh) v per head and its tangent:
    dS = (dq k^T + q dk^T) / sqrt dh, dP = P (dS - rowsum(P dS)), do = dP v + P dv."""
    q, k, v, dq, dk, dv = (f64(a) for a in (q, k, v, dq, dk, dv))
    dh = q.shape[-1]
    o = np.empty_like(q)
    do = np.empty_like(q)
    for hd in range(q.shape[0]):
        s = q[hd] @ k[hd].T / math.sqrt(dh)
        p = np.exp(s - s.max(axis=1, keepdims=True))
        p /= p.sum(axis=1, keepdims=True)
        ds = (dq[hd] @ k[hd].T + q[hd] @ dk[hd].T) / math.sqrt(dh)
        dp = p * (ds - (p * ds).sum(axis=1, keepdims=True))
        o[hd] = p @ v[hd]
        do[hd] = dp @ v[hd] + p @ dv[hd]
    return o, do


def _split_heads(t, n, heads, dh):
    return t.reshape(n, heads, dh).transpose(1, 0, 2)


def block_jvp(wb, h, dh_, mod, n_heads):
    """One DiT block and its tangent (modulation is constant in x)."""
    n, d = h.shape
    hd = d // n_heads
    a = layer_norm(h) * (1.0 + mod["scale1"]) + mod["shift1"]
    da = layer_norm_jvp(h, dh_) * (1.0 + mod["scale1"])
    qkv = linear(a, wb["w_qkv"], wb["b_qkv"])
    dqkv = f64(da) @ f64(wb["w_qkv"]).T
    q, k, v = (_split_heads(qkv[:, i * d:(i + 1) * d], n, n_heads, hd) for i in range(3))
    dq, dk, dv = (_split_heads(dqkv[:, i * d:(i + 1) * d], n, n_heads, hd) for i in range(3))
    o, do = attention_jvp(q, k, v, dq, dk, dv)
    o = o.transpose(1, 0, 2).reshape(n, d)
    do = do.transpose(1, 0, 2).reshape(n, d)
    h1 = h + mod["gate1"] * linear(o, wb["w_o"], wb["b_o"])
    dh1 = dh_ + mod["gate1"] * (do @ f64(wb["w_o"]).T)
    a2 = layer_norm(h1) * (1.0 + mod["scale2"]) + mod["shift2"]
    da2 = layer_norm_jvp(h1, dh1) * (1.0 + mod["scale2"])
    z = linear(a2, wb["w_1"], wb["b_1"])
    dz = da2 @ f64(wb["w_1"]).T
    m = gelu_tanh(z)
    dm = gelu_tanh_grad(z) * dz
    h2 = h1 + mod["gate2"] * linear(m, wb["w_2"], wb["b_2"])
    dh2 = dh1 + mod["gate2"] * (dm @ f64(wb["w_2"]).T)
    return h2, dh2


def velocity_jvp(model, x, dx, sigma, poses):
    """J dx for the full evaluation v(x) = H(F(u(x))) at one step (Eq. 1)."""
    blocks, fmod = model.mods(sigma, poses)
    h = embed(model.w, x)
    dh_ = f64(dx) @ f64(model.w["w_embed"]).T
    for l, mod in enumerate(blocks):
        h, dh_ = block_jvp(block_weights(model.w, l), h, dh_, mod, model.heads)
    da = layer_norm_jvp(h, dh_) * (1.0 + fmod["scale"])
    return da @ f64(model.w["w_final"]).T


# ---------------------------------------------------------------- Eq. 6 and 7

def frozen_trace(model, noise, poses, sig, K):
    """Full evaluations at every step: x_1..x_{K+1} and the cached r_1..r_K."""
    xs = [None, f64(noise).copy()]
    rs = [None]
    for k in range(1, K + 1):
        v, _, r = model.full_step(xs[k], sig[k - 1], poses)
        rs.append(r)
        xs.append(euler(xs[k], v, sig[k - 1], sig[k]))
    return xs, rs


def propagate(model, xs, poses, sig, K, t, e):
    """P_t e: inject dsig_t e after step t and carry it through steps t+1..K."""
    dx = (float(sig[t]) - float(sig[t - 1])) * f64(e)
    for m in range(t + 1, K + 1):
        dx = dx + (float(sig[m]) - float(sig[m - 1])) * velocity_jvp(model, xs[m], dx, sig[m - 1], poses)
    return dx


def response_table(model, noise, poses, sig, K, H, eps=1e-6):
    """q_{j,h} (Eq. 7) for j = 1..K-1, h = 1..min(H, K-j); [K][H+1], other
    entries 0.  Also returns the trace."""
    xs, rs = frozen_trace(model, noise, poses, sig, K)
    den = float(np.linalg.norm(xs[K + 1])) + eps
    q = [[0.0] * (H + 1) for _ in range(K)]
    for j in range(1, K):
        G = np.zeros_like(xs[1])
        for l in range(1, min(H, K - j) + 1):
            t = j + l
            e = model.reuse_step(xs[t], rs[j], sig[t - 1], poses)[0] - \
                model.reuse_step(xs[t], rs[t], sig[t - 1], poses)[0]      # Eq. 6
            G = G + propagate(model, xs, poses, sig, K, t, e)              # Eq. 7
            q[j][l] = float(np.linalg.norm(G)) / den
    return q, xs, rs
