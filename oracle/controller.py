"""Oracle: anchor calibration and the causal cache controller around the
synthetic DiT, in fp64.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import this
module; only tests, the package's smoke check and the benchmark's CPU
baseline leg use it.  It shares no code with the C++/CUDA library.

Follows, in order:
  Sec. 3.1  anchor selection over calibration clips
  Eq. 5     anchor input-drift tables from one full trace per anchor
  Sec. 3.2  budget calibration tau(rho_tar)
  Eq. 1     full evaluation (backbone + interface) or reuse of the last r
  Eq. 12 / Sec. 3.2  pre-reuse acceptance test, forced refresh, suffix replan
"""

import numpy as np

from . import planner as P
from .dit import Model, embed, euler, f64


def anchor_trace_drift(model, noise, poses, sig, K, H, eps=P.EPS):
    """Eq. 5 along one full denoising trace: d_{j,l} = ||u_{j+l} - u_j|| /
    (||u_{j+l}|| + eps) for j = 1..K-1, l = 1..min(H, K-j).  Returns the
    [K][H+1] table and the list of u_k."""
    x = f64(noise).copy()
    us = [None]
    for k in range(1, K + 1):
        v, u, _ = model.full_step(x, sig[k - 1], poses)
        us.append(u)
        x = euler(x, v, sig[k - 1], sig[k])
    d = [[0.0] * (H + 1) for _ in range(K)]
    for j in range(1, K):
        for l in range(1, H + 1):
            if j + l <= K:
                d[j][l] = P.drift(us[j + l], us[j], eps)
    return d, us


def calibrate(model, wl, calib_poses, noise, sig, q0, q1, target, eps=P.EPS):
    """Anchors (Sec. 3.1) -> anchor drift tables (Eq. 5) -> tau (Sec. 3.2)."""
    K, H = wl.steps, wl.h_max
    stats = [P.motion_stats(p) for p in calib_poses]
    anc = P.select_anchors([s[0] for s in stats], [s[1] for s in stats])
    tables = dict(q0=q0, q1=q1, d0=None, d1=None)
    if not anc["valid"]:
        z = [[0.0] * (H + 1) for _ in range(K)]
        tables.update(d0=z, d1=z)
        return anc, tables, 0.0, 0
    tables["d0"], _ = anchor_trace_drift(model, noise, calib_poses[anc["i0"]], sig, K, H, eps)
    tables["d1"], _ = anchor_trace_drift(model, noise, calib_poses[anc["i1"]], sig, K, H, eps)
    tau, reached = P.calibrate_budget(calib_poses, anc, tables, target, K, H, eps)
    return anc, tables, tau, reached


def denoise(model, x1, trajs, sig, anc, tables, tau, K, H, veto=True, forced=None,
            eps=P.EPS, keep_trace=False, variant=P.DRIVECACHE, legal=None, cfg_scale=0.0):
    """Run the sampler over B scenes with the causal controller.

    forced: optional [B][K+1] actions to replay verbatim (no planning, no
    checks).  variant: a planner variant of oracle.planner (Table 3
    ablations, fixed-interval baseline); SHUFFLED plans scene s from the
    trajectory of scene (s+1) mod B, FIXED_INTERVAL runs its schedule with no
    charge and no checks, and refusals under FIXED_PLACEMENT keep the fixed
    pattern (no replan).  legal: optional L(k, h) callable for planning and
    replanning.  cfg_scale != 0: separate guidance branches (Sec. 3.2) --
    each scene also runs the unconditional branch (READING: the null
    trajectory, every pose at the origin), each branch keeps its own cached
    r, both compute or reuse together, and v = v_u + g (v_c - v_u).
    Returns dict(x, plans, executed, log, stats, trace)."""
    B = len(trajs)
    plan_traj = [trajs[(s + 1) % B] if variant == P.SHUFFLED else trajs[s] for s in range(B)]
    plans = [P.plan_scene_variant(plan_traj[s], anc, tables, tau, K, H, variant, eps, legal)
             for s in range(B)]
    fixed = variant == P.FIXED_INTERVAL
    acts = [list(p["actions"]) for p in plans]
    if forced is not None:
        acts = [[0] + [int(forced[s][k]) for k in range(1, K + 1)] for s in range(B)]
        for s in range(B):
            acts[s][1] = P.COMPUTE
    x = f64(x1).copy()
    st = [dict(C=0.0, j=0, age=0, r=None, r_u=None, u_ref=None) for _ in range(B)]
    null = [np.zeros_like(np.asarray(trajs[s], np.float64)) for s in range(B)]

    def guided(v_c, v_u):
        return v_u + cfg_scale * (v_c - v_u)
    executed = [[0] * (K + 1) for _ in range(B)]
    log = [[] for _ in range(B)]
    stats = [dict(n_compute=0, n_reuse=0, n_veto=0, n_replan=0) for _ in range(B)]
    trace = [x.copy()] if keep_trace else None
    for k in range(1, K + 1):
        xn = np.empty_like(x)
        for s in range(B):
            S = st[s]
            reuse = False
            if k > 1 and acts[s][k] == P.REUSE:
                if forced is not None or not veto or fixed:
                    reuse = True
                    if forced is None and not fixed:
                        tabs = plans[s]["tabs"]
                        S["C"] = S["C"] + tabs["c"][S["j"]][S["age"] + 1]
                else:
                    h = S["age"] + 1
                    j = S["j"]
                    tabs = plans[s]["tabs"]
                    u_k = embed(model.w, x[s])
                    d_obs = P.drift(u_k, S["u_ref"], eps)
                    dbar = tabs["dbar"][j][h]
                    c_inc = tabs["c"][j][h]
                    ok = P.accept_reuse(d_obs, dbar, c_inc, S["C"], tau, eps)
                    log[s].append(dict(k=k, j=j, h=h, d_obs=d_obs, dbar=dbar, c=c_inc,
                                       C=S["C"], accept=ok))
                    if ok:
                        reuse = True
                        S["C"] = S["C"] + c_inc
                    else:
                        stats[s]["n_veto"] += 1
                        if variant != P.FIXED_PLACEMENT:
                            stats[s]["n_replan"] += 1
                            a, _, _ = P.plan_suffix(tabs["c"], K, H, k, tau - S["C"], legal)
                            for kk in range(k, K + 1):
                                acts[s][kk] = a[kk]
            if reuse:
                v, _ = model.reuse_step(x[s], S["r"], sig[k - 1], trajs[s])
                if cfg_scale != 0.0:
                    v = guided(v, model.reuse_step(x[s], S["r_u"], sig[k - 1], null[s])[0])
                S["age"] += 1
                executed[s][k] = P.REUSE
                stats[s]["n_reuse"] += 1
            else:
                v, u, r = model.full_step(x[s], sig[k - 1], trajs[s])
                if cfg_scale != 0.0:
                    v_u, _, S["r_u"] = model.full_step(x[s], sig[k - 1], null[s])
                    v = guided(v, v_u)
                S["j"], S["age"], S["r"], S["u_ref"] = k, 0, r, u
                executed[s][k] = P.COMPUTE
                stats[s]["n_compute"] += 1
            xn[s] = euler(x[s], v, sig[k - 1], sig[k])
        x = xn
        if keep_trace:
            trace.append(x.copy())
    for s in range(B):
        stats[s]["charge"] = st[s]["C"]
    return dict(x=x, plans=plans, executed=executed, log=log, stats=stats, trace=trace)


def build(wl, weights):
    return Model(wl, weights)
