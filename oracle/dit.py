"""Oracle: the synthetic spatiotemporal DiT backbone, its interface and the
Euler sampler, in plain fp64 NumPy.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import this
module; only tests, the package's smoke check and the benchmark's CPU
baseline leg use it.  It shares no code with the C++/CUDA library.

The paper's generators are not available; the backbone is a random-init
adaLN DiT whose split follows Eq. 1: the backbone input u_k is the embedded
latent, the reusable backbone output is r_k = h_L - u_k (the block stack's
residual), and the interface H_k is the final modulated LayerNorm + linear
head that produces the velocity; the Euler update is the sampler.

Definitions (READING, fixed for this build; the paper is silent):
  u        = x W_e^T + b_e + pos                      (tokens x d)
  c_{k,s}  = W_t2 silu(W_t1 tfeat(1000 sigma_k) + b_t1) + b_t2
             + W_traj pfeat(poses_s) + b_traj
  mod      = W_ada silu(c) + b_ada  -> per block (shift1, scale1, gate1,
             shift2, scale2, gate2), then final (shift, scale)
  block    : a = LN(h)(1 + scale1) + shift1;  h += gate1 * (MHSA(a) W_o^T + b_o)
             a = LN(h)(1 + scale2) + shift2;  h += gate2 * (gelu_tanh(a W_1^T + b_1) W_2^T + b_2)
  LN       : no affine, eps 1e-6, population variance over d
  MHSA     : qkv = a W_qkv^T + b_qkv, split [q | k | v], heads contiguous in d,
             softmax(q k^T / sqrt(dh)) v over all tokens of the scene
  head     : v = (LN(h_L)(1 + scale) + shift) W_f^T + b_f
  Euler    : x_{k+1} = x_k + (sigma_{k+1} - sigma_k) v_k
"""

import math

import numpy as np

LN_EPS = 1e-6
TEMB_DIM = 256


def f64(a):
    return np.asarray(a, dtype=np.float64)


def layer_norm(x, eps=LN_EPS):
    x = f64(x)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def silu(x):
    x = f64(x)
    return x / (1.0 + np.exp(-x))


def gelu_tanh(x):
    x = f64(x)
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def softmax(s, axis=-1):
    s = f64(s)
    m = s.max(axis=axis, keepdims=True)
    e = np.exp(s - m)
    return e / e.sum(axis=axis, keepdims=True)


def linear(x, w, b):
    """y = x W^T + b with W stored [out][in]."""
    return f64(x) @ f64(w).T + f64(b)


def timestep_features(sigma):
    """Sinusoidal features of t = 1000 sigma: [cos(t f_i), sin(t f_i)],
    f_i = exp(-ln(10000) i / 128), i = 0..127."""
    t = 1000.0 * float(sigma)
    half = TEMB_DIM // 2
    f = np.exp(-math.log(10000.0) * np.arange(half, dtype=np.float64) / half)
    return np.concatenate([np.cos(t * f), np.sin(t * f)])


def _wrap(a):
    r = math.remainder(a, 2.0 * math.pi)
    return math.pi if r == -math.pi else r


def pose_features(poses):
    """Planned poses relative to the first: (dx / 10, dy / 10, wrap(dpsi)) per
    pose, flattened (3 P values)."""
    p = f64(poses)
    out = np.zeros((p.shape[0], 3))
    for t in range(p.shape[0]):
        out[t, 0] = (p[t, 0] - p[0, 0]) / 10.0
        out[t, 1] = (p[t, 1] - p[0, 1]) / 10.0
        out[t, 2] = _wrap(p[t, 2] - p[0, 2])
    return out.reshape(-1)


def conditioning(w, sigma, poses):
    temb = linear(silu(linear(timestep_features(sigma), w["w_t1"], w["b_t1"])), w["w_t2"], w["b_t2"])
    traj = linear(pose_features(poses), w["w_traj"], w["b_traj"])
    return temb + traj


def modulation(w, c, n_blocks, d):
    """All adaLN vectors for one (step, scene): list of per-block dicts and
    the final (shift, scale)."""
    m = linear(silu(c), w["w_ada"], w["b_ada"])
    blocks = []
    for l in range(n_blocks):
        v = m[6 * l * d:6 * (l + 1) * d].reshape(6, d)
        blocks.append(dict(shift1=v[0], scale1=v[1], gate1=v[2],
                           shift2=v[3], scale2=v[4], gate2=v[5]))
    f = m[6 * n_blocks * d:].reshape(2, d)
    return blocks, dict(shift=f[0], scale=f[1])


def embed(w, x):
    """Backbone input u = x W_e^T + b_e + pos."""
    return linear(x, w["w_embed"], w["b_embed"]) + f64(w["pos"])


def attention_core(q, k, v):
    """softmax(q k^T / sqrt(dh)) v per head; q, k, v: [heads][n][dh]."""
    q, k, v = f64(q), f64(k), f64(v)
    dh = q.shape[-1]
    o = np.empty_like(q)
    for hd in range(q.shape[0]):
        p = softmax(q[hd] @ k[hd].T / math.sqrt(dh))
        o[hd] = p @ v[hd]
    return o


def attention(a, w_qkv, b_qkv, n_heads):
    n, d = a.shape
    dh = d // n_heads
    qkv = linear(a, w_qkv, b_qkv)
    q = qkv[:, :d].reshape(n, n_heads, dh).transpose(1, 0, 2)
    k = qkv[:, d:2 * d].reshape(n, n_heads, dh).transpose(1, 0, 2)
    v = qkv[:, 2 * d:].reshape(n, n_heads, dh).transpose(1, 0, 2)
    return attention_core(q, k, v).transpose(1, 0, 2).reshape(n, d)


def block(wb, h, mod, n_heads):
    a = layer_norm(h) * (1.0 + mod["scale1"]) + mod["shift1"]
    o = attention(a, wb["w_qkv"], wb["b_qkv"], n_heads)
    h = h + mod["gate1"] * linear(o, wb["w_o"], wb["b_o"])
    a = layer_norm(h) * (1.0 + mod["scale2"]) + mod["shift2"]
    m = gelu_tanh(linear(a, wb["w_1"], wb["b_1"]))
    h = h + mod["gate2"] * linear(m, wb["w_2"], wb["b_2"])
    return h


def block_weights(w, l):
    return {k: w[f"blk{l}.{k}"] for k in ("w_qkv", "b_qkv", "w_o", "b_o", "w_1", "b_1", "w_2", "b_2")}


def backbone(w, u, mods, n_heads):
    """F_k of Eq. 1: returns h_L (r_k = h_L - u_k)."""
    h = f64(u)
    for l, mod in enumerate(mods):
        h = block(block_weights(w, l), h, mod, n_heads)
    return h


def head(w, h, fmod):
    """H_k of Eq. 1 on the block-stack output: the velocity."""
    a = layer_norm(h) * (1.0 + fmod["scale"]) + fmod["shift"]
    return linear(a, w["w_final"], w["b_final"])


def euler(x, v, sigma_k, sigma_next):
    return f64(x) + (float(sigma_next) - float(sigma_k)) * f64(v)


class Model:
    """Weights + shape of the synthetic DiT (fp64 evaluation)."""

    def __init__(self, wl, weights):
        self.wl = wl
        self.w = {k: f64(v) for k, v in weights.items()}
        self.L = wl.n_blocks
        self.d = wl.d_model
        self.heads = wl.n_heads

    def mods(self, sigma, poses):
        return modulation(self.w, conditioning(self.w, sigma, poses), self.L, self.d)

    def full_step(self, x, sigma, poses):
        """One full evaluation: returns (v, u, r) with r = h_L - u."""
        blocks, fmod = self.mods(sigma, poses)
        u = embed(self.w, x)
        hL = backbone(self.w, u, blocks, self.heads)
        v = head(self.w, hL, fmod)
        return v, u, hL - u

    def reuse_step(self, x, r_cached, sigma, poses):
        """One reuse evaluation: h = u_k + r_j, then the interface."""
        _, fmod = self.mods(sigma, poses)
        u = embed(self.w, x)
        v = head(self.w, u + f64(r_cached), fmod)
        return v, u
