"""Pins for the model-specific legality masks of Sec. 3.2 (expert
boundaries, segment-local caches, native no-cache steps): a mask listed by
hand, brute force over every schedule of small runs with the rules checked
run by run (independently of the mask builder), and invariants of the
planned schedules."""

import itertools
import random

import pytest

from oracle import planner as P


def test_expert_boundary_mask_by_hand():
    """K = 6, H = 2, experts 1..3 | 4..6: a reuse may not refresh across step 3/4."""
    m = P.legal_mask(6, 2, expert_boundary=3)
    legal = {(k, h) for k in range(7) for h in range(3) if m[k][h]}
    assert legal == {(2, 1), (3, 1), (3, 2), (5, 1), (6, 1), (6, 2)}


def test_segment_and_no_cache_masks_by_hand():
    m = P.legal_mask(7, 3, segment_len=3)      # segments 1-3, 4-6, 7
    legal = {(k, h) for k in range(8) for h in range(4) if m[k][h]}
    assert legal == {(2, 1), (3, 1), (3, 2), (5, 1), (6, 1), (6, 2)}
    m = P.legal_mask(5, 2, no_cache_until=3)
    legal = {(k, h) for k in range(6) for h in range(3) if m[k][h]}
    assert legal == {(4, 1), (4, 2), (5, 1), (5, 2)}


def _run_ok(acts, K, H, b, T, p):
    """Every reuse checked against the rules directly: find its refresh."""
    for k in range(2, K + 1):
        if acts[k] != P.REUSE:
            continue
        j = k
        while acts[j] == P.REUSE:
            j -= 1
        if k - j > H:
            return False
        if b and (j <= b) != (k <= b):
            return False
        if T and (j - 1) // T != (k - 1) // T:
            return False
        if p and k <= p:
            return False
    return True


@pytest.mark.parametrize("seed", range(24))
def test_dp_under_masks_matches_brute_force(seed):
    rng = random.Random(77 + seed)
    K = rng.randint(3, 11)
    H = rng.randint(1, 4)
    b = rng.choice([0, rng.randint(1, K - 1)])
    T = rng.choice([0, rng.randint(2, K)])
    p = rng.choice([0, rng.randint(1, K - 1)])
    c = [[0.0] * (H + 1) for _ in range(K)]
    for j in range(1, K):
        for h in range(1, H + 1):
            c[j][h] = rng.randint(0, 32) / 256.0
    budget = rng.choice([0.0, 0.1, 0.3, 10.0])
    best_n, best_cost = 0, 0.0
    for bits in itertools.product((P.COMPUTE, P.REUSE), repeat=K - 1):
        acts = [0, P.COMPUTE] + list(bits)
        if not _run_ok(acts, K, H, b, T, p):
            continue
        n = sum(1 for a in bits if a == P.REUSE)
        cost = P.schedule_cost(acts, c, K)
        if cost <= budget and (n > best_n or (n == best_n and cost < best_cost)):
            best_n, best_cost = n, cost
    mask = P.legal_mask(K, H, b, T, p)
    acts, n, cost = P.plan_suffix(c, K, H, 1, budget, P.legal_fn(mask))
    assert (n, cost) == (best_n, best_cost)
    assert _run_ok([0] + [acts[k] for k in range(1, K + 1)], K, H, b, T, p)


def test_planned_schedules_respect_structure():
    K, H = 40, 4
    rng = random.Random(5)
    c = [[0.0] * (H + 1) for _ in range(K)]
    for j in range(1, K):
        for h in range(1, H + 1):
            c[j][h] = rng.uniform(0.0, 0.01)
    acts, n, _ = P.plan_suffix(c, K, H, 1, 1e9, P.legal_fn(P.legal_mask(K, H, segment_len=10)))
    assert n > 0 and all(acts[k] == P.COMPUTE for k in (1, 11, 21, 31))
    acts, n, _ = P.plan_suffix(c, K, H, 1, 1e9, P.legal_fn(P.legal_mask(K, H, expert_boundary=15)))
    assert acts[16] == P.COMPUTE  # the first low-noise step refreshes
