"""The C-ABI library on the CPU: it loads, exports every symbol that
include/drivecache.h declares, and its host planner (Eq. 2-11, Sec. 3.1-3.2)
agrees bit for bit with the oracle on schedules, counts, costs and tau."""

import math
import os
import random
import re

import numpy as np
import pytest

from oracle import planner as P
from synth import WORKLOADS, gen

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def dc():
    from paper_2608_16354_gb300 import _build, binding
    _build.build()
    binding.lib()
    return binding


def _declared_symbols():
    names = set()
    inc = os.path.join(ROOT, "include")
    for f in os.listdir(inc):
        if f.endswith(".h"):
            src = open(os.path.join(inc, f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(dc_[a-z_0-9]+)\s*\(", src))
    return sorted(names)


def test_library_exports_every_declared_symbol(dc):
    lib = dc.lib()
    syms = _declared_symbols()
    assert len(syms) >= 14
    for s in syms:
        assert hasattr(lib, s), s


def _rand_tables(rng, K, H, dyadic=False):
    def t(scale):
        a = np.zeros((K, H + 1))
        for j in range(1, K):
            for h in range(1, H + 1):
                a[j, h] = rng.randint(0, 64) / 1024.0 if dyadic else rng.uniform(0, scale)
        return a
    return dict(q0=t(0.05), q1=t(0.08), d0=t(0.03), d1=t(0.05))


def test_motion_stats_bit_exact(dc):
    rng = random.Random(1)
    for _ in range(50):
        poses = gen.unicycle(rng.uniform(0, 25), rng.uniform(-0.7, 0.7), rng.randint(1, 60), 0.1,
                             rng.uniform(-math.pi, math.pi), (rng.uniform(-50, 50), rng.uniform(-50, 50)))
        assert dc.motion_stats(poses) == P.motion_stats(poses)


def test_select_anchors_bit_exact(dc):
    rng = random.Random(2)
    for trial in range(200):
        n = rng.randint(1, 40)
        Ls = [rng.choice([0.0, 3.0, rng.uniform(0, 80)]) for _ in range(n)]
        Ts = [rng.choice([0.0, 1.0, rng.uniform(0, 3)]) for _ in range(n)]
        a = dc.select_anchors(Ls, Ts)
        b = P.select_anchors(Ls, Ts)
        assert a == b


@pytest.mark.parametrize("seed", range(30))
def test_plan_bit_exact_random(dc, seed):
    rng = random.Random(1000 + seed)
    K = rng.randint(1, 50)
    H = rng.randint(1, 6)
    tabs = _rand_tables(rng, K, H, dyadic=seed % 2 == 0)
    anc = dict(L0=rng.uniform(0, 5), T0=rng.uniform(0, 0.3), L1=rng.uniform(20, 100),
               T1=rng.uniform(1, 3), valid=1)
    legal = None
    if seed % 3 == 0:
        legal = np.ones((K + 1, H + 1), np.uint8)
        for k in range(K + 1):
            for h in range(H + 1):
                legal[k, h] = rng.random() < 0.85
    A = dc.AnchorArgs(K, H, anc, tabs, legal=legal)
    leg = None if legal is None else (lambda k, h: 1 <= h <= H and k >= 2 and legal[k, h] != 0)
    for _ in range(8):
        poses = gen.unicycle(rng.uniform(0, 30), rng.uniform(-0.6, 0.6), 29, 0.1,
                             rng.uniform(-3, 3))
        tau = rng.choice([0.0, rng.uniform(0, 0.5), rng.uniform(0, 3), math.inf])
        got = dc.plan(poses, A, tau, K)
        ref = P.plan_scene(poses, anc, tabs, tau, K, H)
        if ref["supported"] and leg is not None:
            acts, n, cost = P.plan_suffix(ref["tabs"]["c"], K, H, 1, tau, leg)
            ref["actions"] = [0] + [acts[k] for k in range(1, K + 1)]
            ref["n_reuse"], ref["cost"] = n, cost
        assert got["supported"] == ref["supported"]
        assert got["actions"][1:] == ref["actions"][1:]
        assert got["n_reuse"] == ref["n_reuse"]
        assert got["cost"] == ref["cost"]
        assert got["D"] == ref["D"] and got["L"] == ref["L"] and got["T"] == ref["T"]


def test_replan_bit_exact(dc):
    rng = random.Random(7)
    for trial in range(40):
        K = rng.randint(3, 40)
        H = rng.randint(1, 5)
        tabs = _rand_tables(rng, K, H)
        anc = dict(L0=0.0, T0=0.0, L1=50.0, T1=2.0, valid=1)
        A = dc.AnchorArgs(K, H, anc, tabs)
        D = rng.uniform(0, 1)
        k0 = rng.randint(1, K)
        rem = rng.uniform(0, 1)
        prefix = [0] + [rng.choice([1, 2]) for _ in range(K)]
        got = dc.replan(A, D, k0, rem, prefix)
        st = P.scene_tables(tabs, D, K, H)
        acts, n, cost = P.plan_suffix(st["c"], K, H, k0, rem)
        exp = prefix[:k0] + [acts[k] for k in range(k0, K + 1)]
        assert got["actions"] == exp
        assert got["cost"] == cost
        assert got["n_reuse"] == sum(1 for a in exp[1:] if a == 2)


@pytest.mark.parametrize("key", ["c1", "c2", "c3", "c4", "c5"])
def test_calibrate_budget_bit_exact(dc, key):
    wl = WORKLOADS[key]
    K, H = wl.steps, wl.h_max
    clips = gen.calibration_trajectories(wl)
    stats = [P.motion_stats(c) for c in clips]
    anc = P.select_anchors([s[0] for s in stats], [s[1] for s in stats])
    assert anc["valid"] == 1
    q0, q1 = gen.synthetic_q_tables(K, H)
    d0, d1 = gen.synthetic_d_tables(K, H)
    tabs = dict(q0=q0, q1=q1, d0=d0, d1=d1)
    A = dc.AnchorArgs(K, H, anc, tabs)
    tau, reached = dc.calibrate_budget(list(clips), A, wl.target(), K)
    tau_ref, reached_ref = P.calibrate_budget(list(clips), anc, tabs, wl.target(), K, H)
    assert (tau, reached) == (tau_ref, reached_ref)
    assert reached == 1
    # every evaluated scene of the workload is planned identically
    for poses in gen.scene_trajectories(wl):
        got = dc.plan(poses, A, tau, K)
        ref = P.plan_scene(poses, anc, tabs, tau, K, H)
        assert got["actions"][1:] == ref["actions"][1:] and got["cost"] == ref["cost"]


def test_invalid_arguments_are_rejected(dc):
    K, H = 6, 2
    good = dict(q0=np.full((K, H + 1), 0.1), q1=np.full((K, H + 1), 0.2),
                d0=np.full((K, H + 1), 0.1), d1=np.full((K, H + 1), 0.1))
    anc = dict(L0=0.0, T0=0.0, L1=5.0, T1=1.0, valid=1)
    poses = gen.unicycle(3.0, 0.1, 8)
    bad = dict(good)
    bad["q1"] = good["q1"].copy()
    bad["q1"][2, 1] = float("nan")
    with pytest.raises(dc.DCError) as e:
        dc.plan(poses, dc.AnchorArgs(K, H, anc, bad), 1.0, K)
    assert e.value.status == 1 and "finite" in str(e.value)
    neg = dict(good)
    neg["d0"] = good["d0"].copy()
    neg["d0"][1, 2] = -1.0
    with pytest.raises(dc.DCError):
        dc.plan(poses, dc.AnchorArgs(K, H, anc, neg), 1.0, K)
    with pytest.raises(dc.DCError):  # T must equal anchors.K
        dc.plan(poses, dc.AnchorArgs(K, H, anc, good), 1.0, K + 1)
    with pytest.raises(dc.DCError):
        dc.plan(np.array([[0.0, 0.0, float("inf")]]), dc.AnchorArgs(K, H, anc, good), 1.0, K)
    with pytest.raises(dc.DCError):
        dc.replan(dc.AnchorArgs(K, H, anc, good), 1.5, 2, 0.1, [0] + [1] * K)
    with pytest.raises(dc.DCError):
        dc.select_anchors([], [])


def test_invalid_anchor_set_is_full_inference(dc):
    K, H = 8, 3
    tabs = dict(q0=np.zeros((K, H + 1)), q1=np.zeros((K, H + 1)), d0=None, d1=None)
    A = dc.AnchorArgs(K, H, dict(L0=0, T0=0, L1=0, T1=0, valid=0), tabs)
    r = dc.plan(gen.unicycle(5, 0, 8), A, 10.0, K)
    assert r["supported"] == 0 and r["n_reuse"] == 0 and r["actions"][1:] == [1] * K


# ------------------------------------------- planner variants (Table 1, 3)

VARIANTS = range(7)


@pytest.mark.parametrize("variant", VARIANTS)
def test_plan_variants_bit_exact(dc, variant):
    rng = random.Random(500 + variant)
    for trial in range(12):
        K = rng.randint(2, 40)
        H = rng.randint(1, 5)
        tabs = _rand_tables(rng, K, H, dyadic=trial % 2 == 0)
        anc = dict(L0=rng.uniform(0, 5), T0=rng.uniform(0, 0.3), L1=rng.uniform(20, 100),
                   T1=rng.uniform(1, 3), valid=int(trial % 5 != 4))
        A = dc.AnchorArgs(K, H, anc, tabs, variant=variant)
        for _ in range(6):
            poses = gen.unicycle(rng.uniform(0, 30), rng.uniform(-0.6, 0.6), 29, 0.1,
                                 rng.uniform(-3, 3))
            if variant == P.FIXED_INTERVAL:
                budget = rng.randint(0, K - 1)
            else:
                budget = rng.choice([0.0, rng.uniform(0, 0.5), rng.uniform(0, 3), math.inf])
            got = dc.plan(poses, A, budget, K)
            ref = P.plan_scene_variant(poses, anc, tabs, budget, K, H, variant)
            assert got["supported"] == ref["supported"]
            assert got["actions"][1:] == ref["actions"][1:]
            assert got["n_reuse"] == ref["n_reuse"]
            assert got["cost"] == ref["cost"]
            assert got["D"] == ref["D"]


@pytest.mark.parametrize("variant", VARIANTS)
def test_calibrate_variants_bit_exact(dc, variant):
    wl = WORKLOADS["c2"]
    K, H = wl.steps, wl.h_max
    clips = gen.calibration_trajectories(wl)
    stats = [P.motion_stats(c) for c in clips]
    anc = P.select_anchors([s[0] for s in stats], [s[1] for s in stats])
    q0, q1 = gen.synthetic_q_tables(K, H)
    d0, d1 = gen.synthetic_d_tables(K, H)
    tabs = dict(q0=q0, q1=q1, d0=d0, d1=d1)
    A = dc.AnchorArgs(K, H, anc, tabs, variant=variant)
    got = dc.calibrate_budget(list(clips), A, wl.target(), K)
    ref = P.calibrate_budget_variant(list(clips), anc, tabs, wl.target(), K, H, variant)
    assert got == ref
    assert got[1] == 1


def test_fixed_variants_do_not_replan(dc):
    K, H = 12, 3
    tabs = dict(q0=np.full((K, H + 1), 0.1), q1=np.full((K, H + 1), 0.2),
                d0=np.full((K, H + 1), 0.1), d1=np.full((K, H + 1), 0.1))
    anc = dict(L0=0.0, T0=0.0, L1=5.0, T1=1.0, valid=1)
    prefix = [0] + [1, 2, 1, 2, 2, 1, 2, 1, 2, 1, 2, 2]
    for v in (P.FIXED_PLACEMENT, P.FIXED_INTERVAL):
        got = dc.replan(dc.AnchorArgs(K, H, anc, tabs, variant=v), 0.5, 4, 0.1, prefix)
        assert got["actions"] == prefix and got["cost"] == 0.0


def test_variant_arguments_are_checked(dc):
    K, H = 6, 2
    tabs = dict(q0=np.full((K, H + 1), 0.1), q1=np.full((K, H + 1), 0.2),
                d0=np.full((K, H + 1), 0.1), d1=np.full((K, H + 1), 0.1))
    anc = dict(L0=0.0, T0=0.0, L1=5.0, T1=1.0, valid=1)
    poses = gen.unicycle(3.0, 0.1, 8)
    with pytest.raises(dc.DCError):
        dc.plan(poses, dc.AnchorArgs(K, H, anc, tabs, variant=7), 1.0, K)
    fi = dc.AnchorArgs(K, H, anc, tabs, variant=P.FIXED_INTERVAL)
    for bad in (2.5, -1.0, float(K), math.inf):
        with pytest.raises(dc.DCError):
            dc.plan(poses, fi, bad, K)
    assert dc.plan(poses, fi, 2.0, K)["n_reuse"] == 2


# ---------------------------------- model-specific legality (Sec. 3.2)

@pytest.mark.parametrize("rules", [(0, 0, 0), (7, 0, 0), (0, 5, 0), (0, 0, 4), (9, 6, 2)])
def test_legal_mask_bit_exact_and_planning(dc, rules):
    K, H = 25, 4
    m = dc.legal_mask(K, H, *rules)
    assert m.tolist() == P.legal_mask(K, H, *rules)
    rng = random.Random(sum(rules))
    tabs = _rand_tables(rng, K, H, dyadic=True)
    anc = dict(L0=0.0, T0=0.0, L1=40.0, T1=1.5, valid=1)
    A = dc.AnchorArgs(K, H, anc, tabs, legal=m)
    for v in (6.0, 12.0):
        poses = gen.unicycle(v, 0.2, 29)
        got = dc.plan(poses, A, math.inf, K)
        ref = P.plan_scene(poses, anc, tabs, math.inf, K, H, legal=P.legal_fn(P.legal_mask(K, H, *rules)))
        assert got["actions"][1:] == ref["actions"][1:] and got["cost"] == ref["cost"]


def test_legal_mask_arguments(dc):
    with pytest.raises(dc.DCError):
        dc.legal_mask(0, 4)
    with pytest.raises(dc.DCError):
        dc.legal_mask(10, 4, expert_boundary=-1)


@pytest.mark.parametrize("seed", range(24))
def test_plan_and_replan_ties_bit_exact(dc, seed):
    """Coarse costs (0, 1/8, 1/4; all zero for every fourth seed) leave many
    schedules with equal count and cost: the library's tie-break (smallest
    terminal age, smallest age at every refresh) must pick the oracle's
    schedule, which the oracle's pins tie to brute force."""
    rng = random.Random(3000 + seed)
    K = rng.randint(2, 30)
    H = rng.randint(1, 5)
    t = np.zeros((K, H + 1))
    for j in range(1, K):
        for h in range(1, H + 1):
            t[j, h] = 0.0 if seed % 4 == 0 else rng.choice((0.0, 0.125, 0.25))
    tabs = dict(q0=t, q1=t, d0=t, d1=t)
    anc = dict(L0=0.0, T0=0.0, L1=50.0, T1=2.0, valid=1)
    A = dc.AnchorArgs(K, H, anc, tabs)
    st = P.scene_tables(tabs, 0.5, K, H)
    for k0 in sorted({1, rng.randint(1, K), K}):
        for rem in (0.0, 0.125, 0.5, math.inf):
            prefix = [0] + [P.COMPUTE] * K
            got = dc.replan(A, 0.5, k0, rem, prefix)
            acts, n, cost = P.plan_suffix(st["c"], K, H, k0, rem)
            exp = prefix[:k0] + [acts[k] for k in range(k0, K + 1)]
            assert got["actions"] == exp and got["cost"] == cost
            assert got["n_reuse"] == sum(1 for a in exp[1:] if a == P.REUSE)
    poses = gen.unicycle(10.0, 0.2, 29, 0.1)
    for tau in (0.0, 0.25, math.inf):
        got = dc.plan(poses, A, tau, K)
        ref = P.plan_scene(poses, anc, tabs, tau, K, H)
        assert (got["actions"][1:], got["n_reuse"], got["cost"]) == \
            (ref["actions"][1:], ref["n_reuse"], ref["cost"])
