"""Seeded synthetic inputs shared by the oracle and the CUDA path.

Everything here is an INPUT: random-init weights, noise latents, planned ego
trajectories, the sampler's sigma schedule and the stand-in anchor response
curves.  None of the method's arithmetic (motion statistics, interpolation,
DP, drift, backbone) is computed here, so the oracle and the product can both
draw their inputs from this module without sharing any method code.

Recipe (also stated in the design notes):
  * weights: every matrix N(0, 0.02), every bias 0, positional table N(0, 0.02);
    one independent stream per tensor (SeedSequence([seed, tensor_id])), so a
    model with fewer blocks has exactly the first blocks of the larger one;
    for bf16 workloads the values are rounded to the nearest bf16 (ties to
    even) here, so both sides see the same exactly-representable weights.
  * latents: N(0, 1) fp32, one stream per scene.
  * trajectories: unicycle at 10 Hz from the origin, initial heading U(-pi, pi],
    headings reported in (-pi, pi] (so yaw differences cross the +-pi seam).
  * anchor q tables (stand-in for the JVP calibration of Eq. 7):
    q^(i)_{j,h} = a_i (1 + 2 (1 - (j-1)/(K-1))^2) h^1.2, a_0 = 0.01, a_1 = 0.03.
"""

import math

import numpy as np

from .configs import Workload

# ---------------------------------------------------------------- rng helpers


def _rng(*key) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(k) for k in key])))


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 (ties to even), returned as fp32."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    u = (u + 0x7FFF + lsb) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).reshape(a.shape)


# ------------------------------------------------------------------- weights

TEMB_DIM = 256  # sinusoidal timestep feature width


def weight_specs(wl: Workload):
    """(name, shape, kind) for every tensor of the synthetic DiT, in the order
    of the flat host blob that the model constructor takes.  Matrices are
    stored [out][in] (y = x W^T + b)."""
    d, c, L = wl.d_model, wl.channels, wl.n_blocks
    dm = wl.mlp_ratio * d
    specs = [
        ("w_embed", (d, c), "w"), ("b_embed", (d,), "b"), ("pos", (wl.n_tokens, d), "w"),
        ("w_t1", (d, TEMB_DIM), "w"), ("b_t1", (d,), "b"),
        ("w_t2", (d, d), "w"), ("b_t2", (d,), "b"),
        ("w_traj", (d, wl.cond_dim), "w"), ("b_traj", (d,), "b"),
        ("w_ada", ((6 * L + 2) * d, d), "w"), ("b_ada", ((6 * L + 2) * d,), "b"),
    ]
    for l in range(L):
        specs += [
            (f"blk{l}.w_qkv", (3 * d, d), "w"), (f"blk{l}.b_qkv", (3 * d,), "b"),
            (f"blk{l}.w_o", (d, d), "w"), (f"blk{l}.b_o", (d,), "b"),
            (f"blk{l}.w_1", (dm, d), "w"), (f"blk{l}.b_1", (dm,), "b"),
            (f"blk{l}.w_2", (d, dm), "w"), (f"blk{l}.b_2", (d,), "b"),
        ]
    specs += [("w_final", (c, d), "w"), ("b_final", (c,), "b")]
    return specs


def _tensor_id(name: str) -> int:
    h = 0
    for ch in name.encode():
        h = (h * 131 + ch) % 2_147_483_647
    return h


class _Weights(dict):
    """Weight dict whose tensors are views, in weight_specs order, into one
    flat fp32 array (`blob`), so that flat_blob need not copy them."""
    blob = None
    views = ()


def _draw(seed, key, shape, std, bf16, out):
    a = (_rng(seed, _tensor_id(key)).standard_normal(shape) * std).astype(np.float32)
    if bf16:
        a = round_to_bf16(a)
    out[...] = a


def weights(wl: Workload, seed: int = None, std: float = 0.02) -> dict:
    """Random-init weights: matrices N(0, std), biases zero.  Every matrix
    (and every block's slice of the ada table) has its own stream, so the
    tensors are drawn in parallel threads with the same values as drawn one
    after another."""
    import os
    from concurrent.futures import ThreadPoolExecutor
    seed = wl.seed if seed is None else seed
    specs = weight_specs(wl)
    total = sum(int(np.prod(shape)) for _, shape, _ in specs)
    blob = np.empty(total, np.float32)
    out = _Weights()
    out.blob = blob
    bf16 = wl.dtype == "bf16"
    jobs, o = [], 0
    for name, shape, kind in specs:
        n = int(np.prod(shape))
        view = blob[o:o + n].reshape(shape)
        o += n
        out[name] = view
        if kind == "b":
            view[...] = 0.0
        elif name == "w_ada":
            # the ada table is drawn row-block by row-block so that it does not
            # depend on L for the blocks that two workloads share
            d = wl.d_model
            for l in range(wl.n_blocks):
                jobs.append((f"w_ada.blk{l}", (6 * d, d), view[6 * d * l:6 * d * (l + 1)]))
            jobs.append(("w_ada.final", (2 * d, d), view[6 * d * wl.n_blocks:]))
        else:
            jobs.append((name, shape, view))
    out.views = tuple(out[n] for n, _, _ in specs)
    big = sum(int(np.prod(sh)) for _, sh, _ in jobs) > (1 << 22)
    workers = min(32, os.cpu_count() or 1) if big else 1
    with ThreadPoolExecutor(workers) as ex:
        for f in [ex.submit(_draw, seed, k, sh, std, bf16, v) for k, sh, v in jobs]:
            f.result()
    return out


def flat_blob(wl: Workload, w: dict) -> np.ndarray:
    """The tensors in weight_specs order as one fp32 array (no copy when w
    is weights()'s own, unmodified dict)."""
    names = [n for n, _, _ in weight_specs(wl)]
    if isinstance(w, _Weights) and w.blob is not None and len(w.views) == len(names) and \
            all(w[n] is v for n, v in zip(names, w.views)):
        return w.blob
    return np.concatenate([np.ascontiguousarray(w[n], np.float32).ravel() for n in names])


# ------------------------------------------------------------------- latents


def latents(wl: Workload, batch: int = None, seed: int = None) -> np.ndarray:
    """Initial noise x_1 for each scene, [B, N, C] fp32, N(0, 1)."""
    seed = wl.seed if seed is None else seed
    batch = wl.batch if batch is None else batch
    return np.stack([_rng(seed, 1000 + s).standard_normal((wl.n_tokens, wl.channels))
                     .astype(np.float32) for s in range(batch)])


def anchor_noise(wl: Workload) -> np.ndarray:
    """Noise used for both anchor traces, [N, C] fp32."""
    return _rng(wl.anchor_noise_seed, 77).standard_normal((wl.n_tokens, wl.channels)).astype(np.float32)


def sigmas(K: int) -> np.ndarray:
    """Flow-matching Euler schedule: sigma_k = 1 - (k-1)/K for k = 1..K and
    sigma_{K+1} = 0, stored 0-based as [K+1]."""
    return np.array([1.0 - k / K for k in range(K)] + [0.0], dtype=np.float64)


# -------------------------------------------------------------- trajectories


def unicycle(v: float, omega: float, n_poses: int, dt: float = 0.1,
             psi0: float = 0.0, p0=(0.0, 0.0)) -> np.ndarray:
    """Planned poses [P, 3] = (x, y, psi): constant speed v (m/s) and yaw rate
    omega (rad/s) at spacing dt; heading reported in (-pi, pi]."""
    out = np.zeros((n_poses, 3), np.float64)
    x, y, psi = float(p0[0]), float(p0[1]), float(psi0)
    for t in range(n_poses):
        out[t] = (x, y, math.atan2(math.sin(psi), math.cos(psi)))
        x += v * dt * math.cos(psi)
        y += v * dt * math.sin(psi)
        psi += omega * dt
    return out


def scene_motions(wl: Workload, batch: int = None, seed: int = None):
    """(v, omega, psi0) per scene following the workload's scene mix."""
    seed = wl.seed if seed is None else seed
    batch = wl.batch if batch is None else batch
    r = _rng(seed, 2000)
    out = []
    for s in range(batch):
        psi0 = float(r.uniform(-math.pi, math.pi))
        mix = wl.scene_mix
        if mix == "straight5":
            v, om, psi0 = 5.0, 0.0, 0.0
        elif mix == "thirds":
            kind = s % 3
            v = 0.0 if kind == 0 else float(r.uniform(2.0, 20.0))
            om = float(r.uniform(0.2, 0.5)) if kind == 2 else 0.0
        elif mix == "straight_turn":
            v = float(r.uniform(2.0, 20.0))
            om = 0.0 if s % 2 == 0 else float(r.uniform(0.2, 0.5))
        elif mix == "turning_pm":
            v = float(r.uniform(0.0, 15.0))
            om = float(r.uniform(-0.5, 0.5))
        elif mix == "sharp":
            v, om = 15.0, 0.5
        else:
            raise ValueError(mix)
        out.append((v, om, psi0))
    return out


def scene_trajectories(wl: Workload, batch: int = None, seed: int = None) -> np.ndarray:
    """[B, P, 3] planned poses of the evaluated scenes."""
    return np.stack([unicycle(v, om, wl.n_poses, wl.dt, psi0)
                     for v, om, psi0 in scene_motions(wl, batch, seed)])


def calibration_trajectories(wl: Workload, seed: int = None) -> np.ndarray:
    """[n_calib, P, 3] calibration clips: a quarter stationary, a quarter
    straight, a quarter turning and a quarter unconstrained."""
    seed = wl.seed if seed is None else seed
    r = _rng(seed, 3000)
    clips = []
    for i in range(wl.n_calib):
        kind = i % 4
        psi0 = float(r.uniform(-math.pi, math.pi))
        if kind == 0:
            v, om = 0.0, 0.0
        elif kind == 1:
            v, om = float(r.uniform(2.0, 22.0)), 0.0
        elif kind == 2:
            v = float(r.uniform(2.0, 22.0))
            om = float(r.uniform(0.2, 0.6)) * (1.0 if r.uniform() < 0.5 else -1.0)
        else:
            v, om = float(r.uniform(0.0, 22.0)), float(r.uniform(-0.6, 0.6))
        clips.append(unicycle(v, om, wl.n_poses, wl.dt, psi0))
    return np.stack(clips)


# ------------------------------------------------------- anchor response curves


def synthetic_q_tables(K: int, h_max: int, a0: float = 0.01, a1: float = 0.03):
    """Stand-in joint run responses q^(0), q^(1), each [K][h_max+1] with rows
    j = 1..K-1 and columns h = 1..h_max (row 0 / column 0 unused, zero)."""
    q = []
    for a in (a0, a1):
        t = np.zeros((K, h_max + 1), np.float64)
        for j in range(1, K):
            w = 1.0 + 2.0 * (1.0 - (j - 1) / max(K - 1, 1)) ** 2
            for h in range(1, h_max + 1):
                t[j, h] = a * w * h ** 1.2
        q.append(t)
    return q[0], q[1]


def synthetic_d_tables(K: int, h_max: int, b0: float = 0.02, b1: float = 0.05):
    """Stand-in anchor drift thresholds for planner-only tests (the product
    measures the real ones from anchor traces)."""
    d = []
    for b in (b0, b1):
        t = np.zeros((K, h_max + 1), np.float64)
        for j in range(1, K):
            for h in range(1, h_max + 1):
                t[j, h] = b * h * (1.0 + 0.5 * j / K)
        d.append(t)
    return d[0], d[1]
