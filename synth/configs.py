"""Workload shapes for the synthetic driving world model.

These are sizes only: no part of the method's arithmetic lives here.  The
backbone is a random-init adaLN DiT standing in for the paper's generators
(Wan2.2 5B / A14B and Epona, Sec. 4.1), with latents shaped like a driving
video (views x frames x rows x cols tokens, patch 1) and an ego trajectory of
planned poses at 10 Hz (Sec. 3.1).
"""

from dataclasses import dataclass, field, replace


@dataclass(frozen=True)
class Workload:
    name: str
    dtype: str            # "f32" or "bf16": arithmetic type of the backbone path
    n_blocks: int         # L
    d_model: int          # d
    n_heads: int          # h
    mlp_ratio: int        # MLP hidden = mlp_ratio * d
    channels: int         # C latent channels per token
    views: int
    frames: int
    rows: int
    cols: int
    steps: int            # K denoising steps
    batch: int            # B scenes
    n_poses: int          # P planned poses per scene
    rho_tar: float        # target reuse fraction (Sec. 3.2); None -> target_reuses used
    target_reuses: int = 0
    h_max: int = 4        # maximum cache age
    n_calib: int = 32     # calibration clips (Sec. 4.1 uses 32)
    scene_mix: str = "mixed"
    dt: float = 0.1       # pose spacing (10 Hz)
    seed: int = 0
    anchor_noise_seed: int = 7

    @property
    def n_tokens(self) -> int:
        return self.views * self.frames * self.rows * self.cols

    @property
    def head_dim(self) -> int:
        return self.d_model // self.n_heads

    @property
    def cond_dim(self) -> int:
        # pose features: (dx/10, dy/10, wrapped dpsi) for every planned pose
        return 3 * self.n_poses

    def target(self) -> int:
        """Number of reuses the budget calibration aims for: ceil(rho (K-1))."""
        if self.target_reuses:
            return self.target_reuses
        import math
        return int(math.ceil(self.rho_tar * (self.steps - 1) - 1e-12))

    def flops_per_scene_step(self) -> float:
        """Algorithmic flops of one full backbone pass on one scene:
        L * N * (24 d^2 + 4 N d)  (QKV, out-proj, 4x MLP; QK^T and PV)."""
        n, d = self.n_tokens, self.d_model
        return float(self.n_blocks) * n * (24.0 * d * d + 4.0 * n * d)

    def reuse_bytes_per_scene_step(self) -> float:
        """Algorithmic bytes of one reuse step on one scene: the cached
        feature r_j (N d elements) plus x_k read, x_{k+1} written and the
        refresh latent x_j read for the drift (3 N C fp32)."""
        elt = 4 if self.dtype == "f32" else 2
        return float(self.n_tokens) * (self.d_model * elt + 3 * self.channels * 4)

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


def _poses(frames: int) -> int:
    return 4 * (frames - 1) + 1


# c1: tiny fp32 parity workload
TINY_F32 = Workload(name="tiny-f32-dit-2x64", dtype="f32", n_blocks=2, d_model=64,
                    n_heads=4, mlp_ratio=4, channels=4, views=1, frames=2, rows=8,
                    cols=8, steps=10, batch=1, n_poses=8, rho_tar=0.0,
                    target_reuses=4, scene_mix="straight5")

# c2: the throughput workload (fits one GPU; the bench line is quoted on it)
DIT_S = Workload(name="dit-12x384-n3584-b16-k25", dtype="bf16", n_blocks=12, d_model=384,
                 n_heads=6, mlp_ratio=4, channels=16, views=1, frames=8, rows=16, cols=28,
                 steps=25, batch=16, n_poses=_poses(8), rho_tar=0.4, scene_mix="thirds")

# c3
DIT_XL = Workload(name="dit-28x1152-n14336-b2-k50", dtype="bf16", n_blocks=28, d_model=1152,
                  n_heads=16, mlp_ratio=4, channels=16, views=1, frames=8, rows=32, cols=56,
                  steps=50, batch=2, n_poses=_poses(8), rho_tar=0.5, scene_mix="straight_turn")

# c4
DIT_XL_MV = Workload(name="dit-28x1152-6cam-n10752-b4-k30", dtype="bf16", n_blocks=28,
                     d_model=1152, n_heads=16, mlp_ratio=4, channels=16, views=6, frames=4,
                     rows=16, cols=28, steps=30, batch=4, n_poses=_poses(4), rho_tar=0.5,
                     scene_mix="turning_pm")

# c5
DIT_L = Workload(name="dit-40x3072-n17550-b1-k50", dtype="bf16", n_blocks=40, d_model=3072,
                 n_heads=24, mlp_ratio=4, channels=16, views=1, frames=13, rows=30, cols=45,
                 steps=50, batch=1, n_poses=_poses(13), rho_tar=0.5, scene_mix="sharp")

WORKLOADS = {"c1": TINY_F32, "c2": DIT_S, "c3": DIT_XL, "c4": DIT_XL_MV, "c5": DIT_L}
