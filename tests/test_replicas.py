"""Replica harness on the CPU: scene sharding, distributed budget calibration
(Sec. 3.2) over world-size-2 gloo process groups, hand-off of a sampler
snapshot between replicas, and a replica that dies before reporting."""

import math
import multiprocessing as mp
import os
import random
import struct
import traceback

import numpy as np
import pytest

from oracle import planner as P
from synth import WORKLOADS, gen


@pytest.fixture(scope="module")
def dc():
    from paper_2608_16354_gb300 import _build, binding
    _build.build()
    binding.lib()
    return binding


def _anchors(dc, wl, variant=0):
    K, H = wl.steps, wl.h_max
    clips = gen.calibration_trajectories(wl)
    stats = [P.motion_stats(c) for c in clips]
    anc = P.select_anchors([s[0] for s in stats], [s[1] for s in stats])
    q0, q1 = gen.synthetic_q_tables(K, H)
    d0, d1 = gen.synthetic_d_tables(K, H)
    tabs = dict(q0=q0, q1=q1, d0=d0, d1=d1)
    return clips, anc, tabs, dc.AnchorArgs(K, H, anc, tabs, variant=variant)


def test_shard_partitions_contiguously():
    from paper_2608_16354_gb300.replicas import shard
    for n in range(0, 40):
        for world in range(1, 9):
            parts = [shard(n, world, r) for r in range(world)]
            assert [i for p in parts for i in p] == list(range(n))
            sizes = [len(p) for p in parts]
            assert max(sizes) - min(sizes) <= 1 and sizes == sorted(sizes, reverse=True)
    with pytest.raises(ValueError):
        shard(4, 2, 2)


@pytest.mark.parametrize("key", ["c1", "c2"])
def test_cost_curves_match_oracle_dp(dc, key):
    wl = WORKLOADS[key]
    K, H = wl.steps, wl.h_max
    clips, anc, tabs, A = _anchors(dc, wl)
    n_sup = 0
    for poses in clips:
        got, sup = dc.cost_curve(poses, A, K)
        L, T = P.motion_stats(poses)
        zL, zT = P.normalize(L, T, anc)
        assert sup == int(P.is_supported(zL, zT))
        if not sup:
            assert np.all(np.isinf(got))
            continue
        n_sup += 1
        t = P.scene_tables(tabs, P.intensity(zL, zT), K, H)
        J, _ = P.dp_tables(t["c"], K, H, 1)
        ref = P.cost_curve(J, K, H)
        m = min(len(ref), K)
        assert got[:m].tolist() == ref[:m]
        assert np.all(np.isinf(got[m:]))
        assert got[0] == 0.0
    assert n_sup >= 4


@pytest.mark.parametrize("variant", [0, 1, 3, 4])
def test_budget_from_curves_equals_one_host_calibration(dc, variant):
    wl = WORKLOADS["c2"]
    K = wl.steps
    clips, anc, tabs, A = _anchors(dc, wl, variant)
    curves = np.stack([dc.cost_curve(c, A, K)[0] for c in clips])
    rng = random.Random(5)
    for target in range(0, K, 3):
        ref = dc.calibrate_budget(list(clips), A, target, K)
        assert dc.budget_from_curves(curves, target) == ref
        order = list(range(len(clips)))
        rng.shuffle(order)
        assert dc.budget_from_curves(curves[order], target) == ref


def test_budget_from_curves_rejects_bad_input(dc):
    with pytest.raises(dc.DCError):
        dc.budget_from_curves(np.array([[0.0, -1.0]]), 1)
    with pytest.raises(dc.DCError):
        dc.budget_from_curves(np.array([[0.0, math.nan]]), 1)
    assert dc.budget_from_curves(np.full((3, 4), math.inf), 1) == (0.0, 0)


def test_fixed_interval_has_no_cost_curve(dc):
    wl = WORKLOADS["c1"]
    clips, anc, tabs, A = _anchors(dc, wl, variant=6)
    with pytest.raises(dc.DCError):
        dc.cost_curve(clips[0], A, wl.steps)


# ------------------------------------------------ world-size-2 gloo groups

def _snapshot_blob():
    """A well-formed snapshot as include/drivecache.h documents it."""
    B, K, cfg, k_done, dtype, N, d, C, elt = 2, 6, 0, 3, 0, 16, 16, 4, 4
    up = lambda x, a: (x + a - 1) // a * a
    host = 128 + 48 * B + 4 * up(B * (K + 1), 8) + 2 * 8 * B * (K + 1)
    total = up(up(host, 256) + 2 * 4 * B * N * C, 256) + B * N * d * elt
    h = b"DCSNAP01" + struct.pack("<I8iIQQq", 3, B, K, cfg, k_done, dtype, N, d, C, elt, 99,
                                  total, 5)
    body = np.random.default_rng(3).integers(0, 256, total - 128, dtype=np.uint8)
    return np.concatenate([np.frombuffer(h + bytes(128 - len(h)), np.uint8), body])


def _worker(rank, world, port, mode, q):
    try:
        import datetime
        import torch.distributed as dist
        from paper_2608_16354_gb300 import binding, replicas
        os.environ["MASTER_ADDR"] = "127.0.0.1"
        os.environ["MASTER_PORT"] = str(port)
        dist.init_process_group("gloo", rank=rank, world_size=world,
                                timeout=datetime.timedelta(seconds=20))
        if mode == "calibrate":
            wl = WORKLOADS["c2"]
            K = wl.steps
            clips, anc, tabs, A = _anchors(binding, wl)
            got = replicas.calibrate(list(clips), A, wl.target(), K)
            q.put((rank, "ok", got))
        elif mode == "snapshot":
            snap = _snapshot_blob()
            if rank == 0:
                replicas.send_snapshot(snap, 1)
                q.put((rank, "ok", None))
            else:
                r = replicas.recv_snapshot(0)
                q.put((rank, "ok", bool(np.array_equal(r, snap))))
        elif mode == "dies":
            if rank == 1:
                q.put((rank, "ok", "left"))
                q.close()
                q.join_thread()  # the message is out before the process goes
                os._exit(0)  # leaves before the gather, between steps
            parts = [None] * world
            try:
                dist.all_gather_object(parts, {"rank": rank})
                q.put((rank, "ok", "gathered"))
            except Exception as e:  # the survivor learns of it on the host
                q.put((rank, "ok", "error: " + type(e).__name__))
        dist.destroy_process_group()
    except Exception:
        q.put((rank, "fail", traceback.format_exc()))


def _run_group(mode, world=2, timeout=120):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29500 + random.Random(os.getpid() * 7 + len(mode)).randrange(2000)
    ps = [ctx.Process(target=_worker, args=(r, world, port, mode, q)) for r in range(world)]
    for p in ps:
        p.start()
    out = {}
    try:
        for _ in range(world):
            rank, status, val = q.get(timeout=timeout)
            assert status == "ok", val
            out[rank] = val
    finally:
        for p in ps:
            p.join(timeout=30)
            if p.is_alive():
                p.kill()
    return out


def test_distributed_calibration_two_ranks(dc):
    wl = WORKLOADS["c2"]
    clips, anc, tabs, A = _anchors(dc, wl)
    ref = dc.calibrate_budget(list(clips), A, wl.target(), wl.steps)
    out = _run_group("calibrate")
    assert out[0] == ref and out[1] == ref


def test_snapshot_handoff_between_replicas(dc):
    out = _run_group("snapshot")
    assert out[1] is True


def test_replica_that_leaves_is_detected(dc):
    out = _run_group("dies")
    assert out[1] == "left"
    assert out[0].startswith("error")
