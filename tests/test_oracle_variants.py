"""Pins for the oracle's planner variants: the Table 3 ablations (no motion
prior, shuffled trajectory, translation only, rotation only, fixed
placement) and the fixed-interval baseline of Table 1.  The paper names
them without formulas; the readings are in oracle.planner.  Pins: schedules
worked by hand (tests/golden/even_schedule_hand.json), the DP's own optimal
cost, closed forms of the one-coordinate intensities, and invariants."""

import json
import math
import os
import random

import numpy as np
import pytest

from oracle import planner as P
from synth import gen

HERE = os.path.dirname(os.path.abspath(__file__))
CH = {"C": P.COMPUTE, "R": P.REUSE}


def _acts(s):
    return [0] + [CH[c] for c in s]


@pytest.mark.parametrize("case", json.load(open(os.path.join(HERE, "golden", "even_schedule_hand.json")))["cases"])
def test_even_schedule_hand_cases(case):
    assert P.even_schedule(case["n"], case["K"], case["H"]) == _acts(case["actions"])


@pytest.mark.parametrize("seed", range(20))
def test_even_schedule_properties(seed):
    """Evenness: with no age limit in the way, exactly n reuses whose gaps
    differ by at most one; with H, no run longer than H."""
    rng = random.Random(seed)
    K = rng.randint(2, 60)
    n = rng.randint(0, K - 1)
    a = P.even_schedule(n, K, K)
    pos = [k for k in range(2, K + 1) if a[k] == P.REUSE]
    assert len(pos) == n and a[1] == P.COMPUTE
    if n >= 2:
        gaps = np.diff(pos)
        assert gaps.max() - gaps.min() <= 1
    H = rng.randint(1, 4)
    b = P.even_schedule(n, K, H)
    run = 0
    for k in range(2, K + 1):
        run = run + 1 if b[k] == P.REUSE else 0
        assert run <= H
        if b[k] == P.REUSE:
            assert a[k] == P.REUSE  # the age limit only removes reuses


@pytest.mark.parametrize("seed", range(10))
def test_schedule_cost_equals_dp_cost(seed):
    """The cost of the DP's own optimal schedule, re-added along the schedule,
    is the DP's min_h J_K(B*, h) (dyadic costs: exact)."""
    rng = random.Random(100 + seed)
    K, H = rng.randint(3, 30), rng.randint(1, 5)
    c = [[0.0] * (H + 1) for _ in range(K)]
    for j in range(1, K):
        for h in range(1, H + 1):
            c[j][h] = rng.randint(0, 64) / 1024.0
    budget = rng.choice([0.0, 0.1, 0.5, 5.0])
    acts, n, cost = P.plan_suffix(c, K, H, 1, budget)
    a = [0] + [acts[k] for k in range(1, K + 1)]
    assert P.schedule_cost(a, c, K) == cost


def _tables(K, H):
    q0, q1 = gen.synthetic_q_tables(K, H)
    d0, d1 = gen.synthetic_d_tables(K, H)
    return dict(q0=q0, q1=q1, d0=d0, d1=d1)


ANC = dict(L0=0.0, T0=0.0, L1=40.0, T1=1.5, valid=1)


def test_no_motion_prior_is_one_plan_for_all_scenes():
    K, H = 25, 4
    tabs = _tables(K, H)
    c = P.scene_tables(tabs, 0.5, K, H)["c"]
    ref, n, cost = P.plan_suffix(c, K, H, 1, 0.3)
    trajs = [gen.unicycle(0.0, 0.0, 29), gen.unicycle(12.0, 0.0, 29), gen.unicycle(8.0, 0.4, 29),
             gen.unicycle(30.0, 0.9, 29)]  # the last is outside the support
    for t in trajs:
        r = P.plan_scene_variant(t, ANC, tabs, 0.3, K, H, P.NO_MOTION_PRIOR)
        assert r["supported"] == 1 and r["D"] == 0.5
        assert r["actions"][1:] == [ref[k] for k in range(1, K + 1)] and r["cost"] == cost
    assert P.plan_scene(trajs[3], ANC, tabs, 0.3, K, H)["supported"] == 0


def test_translation_only_and_rotation_only_closed_forms():
    """A straight scene has z^Theta = 0, so the method's Eq. 4 gives
    D = z^L / sqrt 2 while translation-only gives z^L (ratio sqrt 2);
    likewise a turn in place for rotation-only.  One-coordinate variants
    ignore the other coordinate's support."""
    K, H = 25, 4
    tabs = _tables(K, H)
    straight = gen.unicycle(10.0, 0.0, 29)          # L = 28 m, Theta = 0
    L, T = P.motion_stats(straight)
    m = P.plan_scene_variant(straight, ANC, tabs, 0.3, K, H, P.DRIVECACHE)
    t = P.plan_scene_variant(straight, ANC, tabs, 0.3, K, H, P.TRANSLATION_ONLY)
    assert abs(t["D"] - L / 40.0) < 1e-15
    assert abs(t["D"] / m["D"] - math.sqrt(2.0)) < 1e-14
    turn = gen.unicycle(0.0, 0.25, 29)              # L = 0, Theta = 0.7
    L, T = P.motion_stats(turn)
    m = P.plan_scene_variant(turn, ANC, tabs, 0.3, K, H, P.DRIVECACHE)
    r = P.plan_scene_variant(turn, ANC, tabs, 0.3, K, H, P.ROTATION_ONLY)
    assert abs(r["D"] - T / 1.5) < 1e-15
    assert abs(r["D"] / m["D"] - math.sqrt(2.0)) < 1e-14
    # z^Theta > 1: out of the method's support, inside translation-only's
    sharp = gen.unicycle(10.0, 1.0, 29)
    assert P.plan_scene_variant(sharp, ANC, tabs, 0.3, K, H, P.DRIVECACHE)["supported"] == 0
    assert P.plan_scene_variant(sharp, ANC, tabs, 0.3, K, H, P.TRANSLATION_ONLY)["supported"] == 1
    assert P.plan_scene_variant(sharp, ANC, tabs, 0.3, K, H, P.ROTATION_ONLY)["supported"] == 0


@pytest.mark.parametrize("tau", [0.05, 0.2, 0.5])
def test_fixed_placement_keeps_count_and_spreads_it(tau):
    K, H = 25, 4
    tabs = _tables(K, H)
    for t in (gen.unicycle(6.0, 0.0, 29), gen.unicycle(10.0, 0.3, 29)):
        m = P.plan_scene_variant(t, ANC, tabs, tau, K, H, P.DRIVECACHE)
        f = P.plan_scene_variant(t, ANC, tabs, tau, K, H, P.FIXED_PLACEMENT)
        assert f["actions"] == P.even_schedule(m["n_reuse"], K, H)
        assert f["n_reuse"] == m["n_reuse"]  # count <= K/2 here, never cut by H
        assert f["cost"] == P.schedule_cost(f["actions"], m["tabs"]["c"], K)
        assert f["cost"] >= m["cost"]         # the DP placement is optimal for its count


def test_fixed_interval_ignores_motion_and_budget():
    K, H = 25, 4
    tabs = _tables(K, H)
    want = P.even_schedule(10, K, H)
    for t in (gen.unicycle(0.0, 0.0, 29), gen.unicycle(30.0, 0.9, 29)):
        r = P.plan_scene_variant(t, dict(ANC, valid=0), tabs, 10, K, H, P.FIXED_INTERVAL)
        assert r["actions"] == want and r["n_reuse"] == 10
    assert P.calibrate_budget_variant([], ANC, tabs, 10, K, H, P.FIXED_INTERVAL) == (10.0, 1)


def test_variant_calibration_matches_method_for_placement_and_shuffle():
    from synth import WORKLOADS
    wl = WORKLOADS["c2"]
    K, H = wl.steps, wl.h_max
    clips = gen.calibration_trajectories(wl)
    stats = [P.motion_stats(c) for c in clips]
    anc = P.select_anchors([s[0] for s in stats], [s[1] for s in stats])
    tabs = _tables(K, H)
    ref = P.calibrate_budget(list(clips), anc, tabs, wl.target(), K, H)
    for v in (P.DRIVECACHE, P.SHUFFLED, P.FIXED_PLACEMENT):
        assert P.calibrate_budget_variant(list(clips), anc, tabs, wl.target(), K, H, v) == ref
    # a motion variant calibrates on its own intensities and still reaches the target
    tau, reached = P.calibrate_budget_variant(list(clips), anc, tabs, wl.target(), K, H, P.NO_MOTION_PRIOR)
    assert reached == 1
    n = P.plan_scene_variant(clips[0], anc, tabs, tau, K, H, P.NO_MOTION_PRIOR)["n_reuse"]
    assert n >= wl.target()  # every clip has the same plan, so the median is this count


def test_controller_variants_tiny():
    """Controller invariants per variant on the tiny workload: the shuffled
    run plans each scene from its neighbour's trajectory; fixed interval runs
    its schedule unchecked; fixed placement refuses without replanning."""
    import synth
    from oracle import controller as Ctl
    wl = synth.WORKLOADS["c1"].with_(batch=3)
    m = Ctl.build(wl, gen.weights(wl))
    K, H = wl.steps, wl.h_max
    sig = gen.sigmas(K)
    q0, q1 = gen.synthetic_q_tables(K, H)
    trajs = [gen.unicycle(2.0, 0.0, 8), gen.unicycle(5.0, 0.1, 8), gen.unicycle(0.5, 0.3, 8)]
    zero = [[0.0] * (H + 1) for _ in range(K)]
    tabs = dict(q0=q0, q1=q1, d0=zero, d1=zero)
    anc = dict(L0=0.0, T0=0.0, L1=5.0, T1=1.0, valid=1)
    x1 = np.stack([gen.latents(wl.with_(batch=1), seed=s)[0] for s in range(3)])
    sh = Ctl.denoise(m, x1, trajs, sig, anc, tabs, 10.0, K, H, variant=P.SHUFFLED)
    for s in range(3):
        ref = P.plan_scene(trajs[(s + 1) % 3], anc, tabs, 10.0, K, H)
        assert sh["plans"][s]["actions"][1:] == ref["actions"][1:]
    fi = Ctl.denoise(m, x1, trajs, sig, anc, tabs, 4, K, H, variant=P.FIXED_INTERVAL)
    for s in range(3):
        assert fi["executed"][s][1:] == P.even_schedule(4, K, H)[1:] and fi["log"][s] == []
    fp = Ctl.denoise(m, x1, trajs, sig, anc, tabs, 10.0, K, H, variant=P.FIXED_PLACEMENT)
    for s in range(3):
        st = fp["stats"][s]
        assert st["n_replan"] == 0 and st["n_veto"] == len(fp["log"][s])
        assert all(e["accept"] is False for e in fp["log"][s])  # zero thresholds refuse everything
        assert st["n_reuse"] == 0
