"""Oracle: the cache controller of DriveCache in plain fp64 Python.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import this
module; only tests, the package's smoke check and the benchmark's CPU
baseline leg use it.  It shares no code with the C++/CUDA library.

Every quantity is a Python float (IEEE binary64), summed left to right in
step order, so that a reader can check each function against the paper line
by line.  Readings of points the paper leaves open are marked READING.

Sections followed:
  Eq. 2   motion statistics L_s, Theta_s
  Sec. 3.1 anchor selection (z-scores, low-motion / moving-turn anchors)
  Eq. 3   normalisation against the anchor pair, support gate
  Eq. 4   motion intensity D_s
  Eq. 8   one-sided interpolation of q (and of the drift threshold d)
  Eq. 9   monotone envelope Q and increments c_hat
  Eq. 10  DP transitions, Eq. 11 maximal reuse count, backtracking (Sec. 3.2)
  Sec. 3.2 budget calibration tau(rho_tar)
  Eq. 12 / Sec. 3.2 causal acceptance test and suffix replanning
  Table 3 ablations (no motion prior, shuffled trajectory, translation only,
          rotation only, fixed placement) and the fixed-interval baseline of
          Table 1, as planner variants
  Sec. 3.2 model-specific legality: expert boundaries, segment-local caches
          and no-cache steps as masks L(k, h)
"""

import math

INF = math.inf
COMPUTE = 1
REUSE = 2
EPS = 1e-6  # READING: one epsilon (1e-6) for Eq. 3, 5, 7, 12 and the veto slack


# ------------------------------------------------------------------ Eq. 2

def wrap(a: float) -> float:
    """Angle difference wrapped into (-pi, pi].  READING: IEEE remainder by
    2 pi (exact), with -pi mapped to +pi."""
    r = math.remainder(a, 2.0 * math.pi)
    if r == -math.pi:
        r = math.pi
    return r


def motion_stats(poses):
    """Eq. 2: L = sum_t ||p_t - p_{t-1}||_2, Theta = sum_t |wrap(psi_t - psi_{t-1})|,
    over consecutive planned poses (x, y, psi)."""
    L = 0.0
    T = 0.0
    for t in range(1, len(poses)):
        dx = float(poses[t][0]) - float(poses[t - 1][0])
        dy = float(poses[t][1]) - float(poses[t - 1][1])
        L = L + math.sqrt(dx * dx + dy * dy)
        T = T + abs(wrap(float(poses[t][2]) - float(poses[t - 1][2])))
    return L, T


# ---------------------------------------------------------- Sec. 3.1 anchors

def _mean_std(v):
    n = len(v)
    s = 0.0
    for a in v:
        s = s + a
    mean = s / n
    ss = 0.0
    for a in v:
        ss = ss + (a - mean) * (a - mean)
    return mean, math.sqrt(ss / n)  # READING: population standard deviation


def _zscores(v):
    mean, std = _mean_std(v)
    if std == 0.0:
        return [0.0 for _ in v]  # READING: constant dimension -> z = 0
    return [(a - mean) / std for a in v]


def _median(v):
    s = sorted(v)
    n = len(s)
    if n % 2 == 1:
        return s[n // 2]
    return (s[n // 2 - 1] + s[n // 2]) / 2.0


def select_anchors(Ls, Ts):
    """Sec. 3.1: z-score L and Theta over the calibration clips; the
    low-motion anchor minimises zL + zTheta; among clips with Theta above the
    calibration median (strict), L > L0 and Theta > Theta0, the moving-turn
    anchor maximises zL * zTheta.  Ties go to the lowest clip index.  An empty
    candidate set makes the anchor pair invalid (full-inference fallback).

    Returns dict(L0, T0, L1, T1, valid, i0, i1)."""
    n = len(Ls)
    zL = _zscores(Ls)
    zT = _zscores(Ts)
    i0 = 0
    best = zL[0] + zT[0]
    for i in range(1, n):
        s = zL[i] + zT[i]
        if s < best:
            best, i0 = s, i
    L0, T0 = Ls[i0], Ts[i0]
    med = _median(Ts)
    i1 = -1
    bestp = -INF
    for i in range(n):
        if Ts[i] > med and Ls[i] > L0 and Ts[i] > T0:
            p = zL[i] * zT[i]
            if i1 < 0 or p > bestp:
                bestp, i1 = p, i
    if i1 < 0:
        return dict(L0=L0, T0=T0, L1=0.0, T1=0.0, valid=0, i0=i0, i1=-1)
    return dict(L0=L0, T0=T0, L1=Ls[i1], T1=Ts[i1], valid=1, i0=i0, i1=i1)


# ------------------------------------------------------------- Eq. 3 and 4

def normalize(L, T, anc, eps=EPS):
    """Eq. 3: z^L = (L - L0) / max(L1 - L0, eps), likewise for Theta."""
    zL = (L - anc["L0"]) / max(anc["L1"] - anc["L0"], eps)
    zT = (T - anc["T0"]) / max(anc["T1"] - anc["T0"], eps)
    return zL, zT


def is_supported(zL, zT):
    """Sec. 3.1: supported only when (zL, zT) lies in [0, 1]^2."""
    return 0.0 <= zL <= 1.0 and 0.0 <= zT <= 1.0


def intensity(zL, zT):
    """Eq. 4: D = (1/sqrt 2) sqrt(zL^2 + zT^2), evaluated as
    sqrt(zL^2 + zT^2) / sqrt(2)."""
    return math.sqrt(zL * zL + zT * zT) / math.sqrt(2.0)


# -------------------------------------------------------------- Eq. 8 and 9

def interpolate(t0, t1, D, K, H):
    """Eq. 8: t~_{j,h} = t0_{j,h} + D max(t1_{j,h} - t0_{j,h}, 0), for
    j = 1..K-1 and h = 1..H (tables indexed [j][h], row/col 0 unused)."""
    out = [[0.0] * (H + 1) for _ in range(K)]
    for j in range(1, K):
        for h in range(1, H + 1):
            a = float(t0[j][h])
            b = float(t1[j][h])
            out[j][h] = a + D * max(b - a, 0.0)
    return out


def envelope(qt, K, H):
    """Eq. 9: Q_{j,h} = max_{l<=h} q~_{j,l}, c_hat_{j,h} = Q_{j,h} - Q_{j,h-1},
    Q_{j,0} = 0.  Returns (Q, c_hat)."""
    Q = [[0.0] * (H + 1) for _ in range(K)]
    c = [[0.0] * (H + 1) for _ in range(K)]
    for j in range(1, K):
        run = -INF
        for h in range(1, H + 1):
            run = max(run, qt[j][h])
            Q[j][h] = run
        for h in range(1, H + 1):
            c[j][h] = Q[j][h] - Q[j][h - 1]
    return Q, c


def scene_tables(tables, D, K, H):
    """Per-scene c_hat (Eq. 8-9 on q) and drift threshold d_bar (Eq. 8 on d)."""
    qt = interpolate(tables["q0"], tables["q1"], D, K, H)
    Q, c = envelope(qt, K, H)
    dbar = interpolate(tables["d0"], tables["d1"], D, K, H)
    return dict(qt=qt, Q=Q, c=c, dbar=dbar)


# ---------------------------------------------------------- Eq. 10 and 11

def default_legal(k, h, H):
    """READING of L(k, h): reuse at step k with cache age h is legal iff
    1 <= h <= H_max; step 1 is always a full evaluation."""
    return 1 <= h <= H and k >= 2


def dp_tables(c, K, H, k0=1, legal=None):
    """Eq. 10 from J_{k0}(0,0) = 0 over steps k0..K.

    J[k][n][h] is the minimum cumulative response after step k with n reuses
    since step k0 and cache age h.  For a refresh state (h = 0) the argmin
    over the previous step's ages is stored (smallest h on ties), which is all
    backtracking needs (Sec. 3.2).  legal(k, h) says whether reusing at step k
    with age h is allowed."""
    if legal is None:
        def legal(k, h):
            return default_legal(k, h, H)
    nmax = K - k0
    J = {k0: [[INF] * (H + 1) for _ in range(nmax + 1)]}
    arg = {}
    J[k0][0][0] = 0.0
    for k in range(k0, K):
        cur = J[k]
        nxt = [[INF] * (H + 1) for _ in range(nmax + 1)]
        argk = [-1] * (nmax + 1)
        for n in range(nmax + 1):
            # J_{k+1}(n, 0) = min_h J_k(n, h)
            best, bh = INF, -1
            for h in range(H + 1):
                if cur[n][h] < best:
                    best, bh = cur[n][h], h
            nxt[n][0] = best
            argk[n] = bh
        for n in range(nmax):
            for h in range(H):
                if cur[n][h] == INF:
                    continue
                if not legal(k + 1, h + 1):
                    continue
                cand = cur[n][h] + c[k - h][h + 1]
                if cand < nxt[n + 1][h + 1]:
                    nxt[n + 1][h + 1] = cand
        J[k + 1] = nxt
        arg[k + 1] = argk
    return J, arg


def cost_curve(J, K, H):
    """m(n) = min_h J_K(n, h) for every n (INF where infeasible)."""
    out = []
    for row in J[K]:
        m = INF
        for v in row:
            if v < m:
                m = v
        out.append(m)
    return out


def best_count(m, tau):
    """Eq. 11: B* = max{n : min_h J_K(n, h) <= tau} (0 when none)."""
    b = 0
    for n, v in enumerate(m):
        if v < INF and v <= tau:  # infeasible counts (J = +inf) never qualify
            b = n
    return b


def backtrack(J, arg, K, H, k0, nstar):
    """Recover the minimum-response schedule with nstar reuses: final age =
    smallest argmin of J_K(nstar, .); a reuse state steps back to (n-1, h-1);
    a refresh state steps back to the stored argmin.  Returns actions for
    steps k0..K as a dict k -> COMPUTE/REUSE."""
    row = J[K][nstar]
    h, best = -1, INF
    for hh in range(H + 1):
        if row[hh] < best:
            best, h = row[hh], hh
    acts = {}
    n, k = nstar, K
    while k > k0:
        if h > 0:
            acts[k] = REUSE
            n, h = n - 1, h - 1
        else:
            acts[k] = COMPUTE
            h = arg[k][n]
        k -= 1
    acts[k0] = COMPUTE
    return acts, best


def plan_suffix(c, K, H, k0, budget, legal=None):
    """Exact DP placement on steps k0..K starting from a full evaluation at
    k0 under `budget`; returns (actions dict, n_reuse, cost)."""
    J, arg = dp_tables(c, K, H, k0, legal)
    m = cost_curve(J, K, H)
    nstar = best_count(m, budget)
    acts, cost = backtrack(J, arg, K, H, k0, nstar)
    return acts, nstar, cost


def plan_scene(poses, anc, tables, tau, K, H, eps=EPS, legal=None):
    """dc_plan: Eq. 2 -> Eq. 3 gate -> Eq. 4 -> Eq. 8/9 -> Eq. 10/11.

    Returns dict(actions[list of K+1, index 0 unused], n_reuse, cost,
    supported, D, L, T, tabs)."""
    L, T = motion_stats(poses)
    acts = [0] + [COMPUTE] * K
    res = dict(actions=acts, n_reuse=0, cost=0.0, supported=0, D=0.0, L=L, T=T, tabs=None)
    if not anc["valid"]:
        return res
    zL, zT = normalize(L, T, anc, eps)
    if not is_supported(zL, zT):
        return res
    D = intensity(zL, zT)
    tabs = scene_tables(tables, D, K, H)
    a, n, cost = plan_suffix(tabs["c"], K, H, 1, tau, legal)
    for k in range(1, K + 1):
        acts[k] = a[k]
    res.update(n_reuse=n, cost=cost, supported=1, D=D, tabs=tabs)
    return res


# ------------------------------------------------------ Sec. 3.2 budget tau

def calibrate_budget(clip_poses, anc, tables, target, K, H, eps=EPS, legal=None):
    """Smallest table-cost threshold tau whose median B* over the calibration
    clips reaches `target` reuses.  READING: candidates are the finite values
    min_h J_K(n, h) of every supported clip; unsupported clips count as 0
    reuses; the median of an even count is the mean of the two middle values.
    Returns (tau, reached)."""
    curves = []
    cands = set()
    for poses in clip_poses:
        L, T = motion_stats(poses)
        if not anc["valid"]:
            curves.append(None)
            continue
        zL, zT = normalize(L, T, anc, eps)
        if not is_supported(zL, zT):
            curves.append(None)
            continue
        D = intensity(zL, zT)
        tabs = scene_tables(tables, D, K, H)
        J, _ = dp_tables(tabs["c"], K, H, 1, legal)
        m = cost_curve(J, K, H)
        curves.append(m)
        for v in m:
            if v < INF:
                cands.add(v)
    if not cands:
        return 0.0, 0
    ordered = sorted(cands)
    for tau in ordered:
        counts = [0 if m is None else best_count(m, tau) for m in curves]
        if _median([float(x) for x in counts]) >= target:
            return tau, 1
    return ordered[-1], 0


# ------------------------------------------------- Eq. 12 causal acceptance

def drift(u_now, u_ref, eps=EPS):
    """Eq. 5 / Eq. 12: ||u_now - u_ref||_2 / (||u_now||_2 + eps) over the whole
    per-scene backbone input (READING of the norm axes: all tokens and
    channels)."""
    import numpy as np
    a = np.asarray(u_now, np.float64)
    b = np.asarray(u_ref, np.float64)
    num = math.sqrt(float(np.sum((a - b) * (a - b))))
    den = math.sqrt(float(np.sum(a * a)))
    return num / (den + eps)


def accept_reuse(d_obs, dbar, c_inc, charge, tau, eps=EPS):
    """Sec. 3.2: accept the h-th reuse of the run from j only when
    d_obs <= d_bar_{j,h} + eps and C_k + c_hat_{j,h} <= tau."""
    return d_obs <= dbar + eps and charge + c_inc <= tau


# ------------------------------------- Table 3 ablations, Table 1 baseline
#
# The paper names these variants without defining them; the READINGS below
# are the ones the library implements (variant ids match include/drivecache.h).

DRIVECACHE = 0         # the method as published
NO_MOTION_PRIOR = 1    # READING: every scene is planned at D = 1/2, no support gate
SHUFFLED = 2           # READING: scene s is planned from the trajectory of scene (s+1) mod B
TRANSLATION_ONLY = 3   # READING: D = z^L, supported iff 0 <= z^L <= 1
ROTATION_ONLY = 4      # READING: D = z^Theta, supported iff 0 <= z^Theta <= 1
FIXED_PLACEMENT = 5    # READING: B* of the method, spread evenly (no DP placement), no replan
FIXED_INTERVAL = 6     # READING: `budget` reuses spread evenly for every scene; no charge, no veto


def variant_intensity(L, T, anc, variant, eps=EPS):
    """(supported, D) of a scene under a planner variant (Eq. 3-4 for the
    method itself)."""
    if not anc["valid"]:
        return 0, 0.0
    if variant == NO_MOTION_PRIOR:
        return 1, 0.5
    zL, zT = normalize(L, T, anc, eps)
    if variant == TRANSLATION_ONLY:
        return (1, zL) if 0.0 <= zL <= 1.0 else (0, 0.0)
    if variant == ROTATION_ONLY:
        return (1, zT) if 0.0 <= zT <= 1.0 else (0, 0.0)
    if not is_supported(zL, zT):
        return 0, 0.0
    return 1, intensity(zL, zT)


def even_schedule(n, K, H, legal=None):
    """READING of fixed placement and of the fixed-interval baseline: n reuses
    spread evenly over steps 2..K -- step k is a reuse iff
    floor((k-1) n / (K-1)) > floor((k-2) n / (K-1)) -- except that a reuse
    whose cache age would be illegal (L(k, h), default 1 <= h <= H_max) is a
    full evaluation instead.  Returns the action list (index 0 unused)."""
    leg = legal or (lambda k, h: default_legal(k, h, H))
    acts = [0] * (K + 1)
    acts[1] = COMPUTE
    age = 0
    for k in range(2, K + 1):
        want = K > 1 and (k - 1) * n // (K - 1) > (k - 2) * n // (K - 1)
        if want and leg(k, age + 1):
            acts[k] = REUSE
            age += 1
        else:
            acts[k] = COMPUTE
            age = 0
    return acts


def schedule_cost(acts, c, K):
    """Sum of c_hat_{j,h} over the reuses of a schedule (j = last full
    evaluation, h = age), in step order."""
    total = 0.0
    j, age = 1, 0
    for k in range(2, K + 1):
        if acts[k] == REUSE:
            age += 1
            total = total + c[j][age]
        else:
            j, age = k, 0
    return total


def plan_scene_variant(poses, anc, tables, budget, K, H, variant, eps=EPS, legal=None):
    """dc_plan under a planner variant.  `budget` is tau, except for
    FIXED_INTERVAL where it is the number of reuses."""
    if variant == FIXED_INTERVAL:
        L, T = motion_stats(poses)
        acts = even_schedule(int(budget), K, H, legal)
        n = sum(1 for k in range(2, K + 1) if acts[k] == REUSE)
        return dict(actions=acts, n_reuse=n, cost=0.0, supported=1, D=0.0, L=L, T=T, tabs=None)
    if variant in (DRIVECACHE, SHUFFLED, FIXED_PLACEMENT):
        res = plan_scene(poses, anc, tables, budget, K, H, eps, legal)
        if variant == FIXED_PLACEMENT and res["supported"]:
            acts = even_schedule(res["n_reuse"], K, H, legal)
            res["actions"] = acts
            res["n_reuse"] = sum(1 for k in range(2, K + 1) if acts[k] == REUSE)
            res["cost"] = schedule_cost(acts, res["tabs"]["c"], K)
        return res
    L, T = motion_stats(poses)
    acts = [0] + [COMPUTE] * K
    res = dict(actions=acts, n_reuse=0, cost=0.0, supported=0, D=0.0, L=L, T=T, tabs=None)
    sup, D = variant_intensity(L, T, anc, variant, eps)
    if not sup:
        return res
    tabs = scene_tables(tables, D, K, H)
    a, n, cost = plan_suffix(tabs["c"], K, H, 1, budget, legal)
    for k in range(1, K + 1):
        acts[k] = a[k]
    res.update(n_reuse=n, cost=cost, supported=1, D=D, tabs=tabs)
    return res


def calibrate_budget_variant(clip_poses, anc, tables, target, K, H, variant, eps=EPS, legal=None):
    """Sec. 3.2 calibration under a planner variant: the motion variants use
    their own intensity; FIXED_PLACEMENT keeps the method's tau (it changes
    placement, not count); FIXED_INTERVAL returns the reuse count itself
    (reached iff the even schedule holds `target` reuses)."""
    if variant == FIXED_INTERVAL:
        acts = even_schedule(target, K, H, legal)
        n = sum(1 for k in range(2, K + 1) if acts[k] == REUSE)
        return float(target), 1 if n >= target else 0
    if variant in (DRIVECACHE, SHUFFLED, FIXED_PLACEMENT):
        return calibrate_budget(clip_poses, anc, tables, target, K, H, eps, legal)
    curves = []
    cands = set()
    for poses in clip_poses:
        L, T = motion_stats(poses)
        sup, D = variant_intensity(L, T, anc, variant, eps)
        if not sup:
            curves.append(None)
            continue
        tabs = scene_tables(tables, D, K, H)
        J, _ = dp_tables(tabs["c"], K, H, 1, legal)
        m = cost_curve(J, K, H)
        curves.append(m)
        for v in m:
            if v < INF:
                cands.add(v)
    if not cands:
        return 0.0, 0
    ordered = sorted(cands)
    for tau in ordered:
        counts = [0 if m is None else best_count(m, tau) for m in curves]
        if _median([float(x) for x in counts]) >= target:
            return tau, 1
    return ordered[-1], 0


# ------------------------------------------ Sec. 3.2 model-specific legality

def legal_mask(K, H, expert_boundary=0, segment_len=0, no_cache_until=0):
    """L(k, h) of Eq. 10 for the model-specific rules of Sec. 3.2, as a
    [K+1][H+1] 0/1 list (index [k][h]).  A reuse at step k with cache age h
    refreshes at j = k - h.  READINGS:
      * always: 1 <= h <= H_max and k >= 2 (the first step is computed);
      * expert_boundary b > 0 (two experts, steps 1..b and b+1..K): j and k
        lie in the same expert -- no run crosses the boundary;
      * segment_len T > 0 (autoregressive segments of T steps, caches local
        to one denoising call): floor((j-1)/T) == floor((k-1)/T), so the
        first step of every segment is computed;
      * no_cache_until p > 0 (native no-cache steps 1..p): k > p."""
    m = [[0] * (H + 1) for _ in range(K + 1)]
    for k in range(2, K + 1):
        for h in range(1, H + 1):
            j = k - h
            if j < 1:
                continue
            if expert_boundary > 0 and (j <= expert_boundary) != (k <= expert_boundary):
                continue
            if segment_len > 0 and (j - 1) // segment_len != (k - 1) // segment_len:
                continue
            if no_cache_until > 0 and k <= no_cache_until:
                continue
            m[k][h] = 1
    return m


def legal_fn(mask):
    """The callable form plan_suffix and dp_tables take."""
    return lambda k, h: 1 <= h < len(mask[0]) and k >= 2 and mask[k][h] != 0
