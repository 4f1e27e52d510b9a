"""Replica harness for multi-scene serving across GPUs and boxes.

Scenes are independent under DriveCache (each has its own plan, cache, drift
check and charge, Sec. 3.2), so the path shards by scene with no exchange
during denoising: one replica per GPU runs its own contiguous share of the
scenes.  The host side carries only
  - the budget calibration: every replica computes the cost curves of its
    share of the calibration clips (dc_cost_curve), the curves are gathered
    and every replica applies the tau rule to all of them
    (dc_budget_from_curves), so all replicas hold the tau of a one-host
    calibration;
  - the results, gathered to rank 0;
  - preempted calls: a replica that must stop hands the sampler snapshot of
    its running call (dc_denoise_steps) to another replica, which resumes it.
torch.distributed (gloo for host objects) is the transport; every step of the
path runs in libdrivecache.  The shuffled-trajectory ablation (DC_VAR_SHUFFLED)
pairs scenes within one call, so under sharding it pairs them within each
batch.
"""

import numpy as np

from . import binding


def _world(group=None):
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        return dist.get_rank(group), dist.get_world_size(group)
    return 0, 1


def shard(n, world, rank):
    """Contiguous share of n items for `rank` of `world`: sizes differ by at
    most one, lower ranks take the extra items."""
    if world < 1 or not 0 <= rank < world or n < 0:
        raise ValueError("need world >= 1, 0 <= rank < world and n >= 0")
    base, extra = divmod(n, world)
    start = rank * base + min(rank, extra)
    return range(start, start + base + (1 if rank < extra else 0))


def calibrate(clips, anchors, target, T, group=None):
    """Distributed Sec. 3.2 calibration: (tau, reached) on every rank, equal
    to dc_calibrate_budget over all clips."""
    import torch.distributed as dist
    rank, world = _world(group)
    mine = [binding.cost_curve(clips[i], anchors, T)[0] for i in shard(len(clips), world, rank)]
    if world > 1:
        parts = [None] * world
        dist.all_gather_object(parts, mine, group=group)
    else:
        parts = [mine]
    curves = np.array([c for p in parts for c in p], np.float64).reshape(len(clips), T)
    return binding.budget_from_curves(curves, target)


def serve_shard(model, latents, trajs, sched, rank, world, batch=None):
    """Denoise this replica's share of the scenes on its GPU.  latents: host
    fp32 [S, N, C] (all scenes; only the share is read); trajs: S pose
    arrays.  Returns {scene index: (x_out, record)}."""
    S = len(trajs)
    cfg = sched.s.cfg_scale != 0.0
    cap = model.desc.max_batch // (2 if cfg else 1)
    batch = min(batch or cap, cap)
    if batch < 1:
        raise ValueError("max_batch too small for one scene")
    ids = list(shard(S, world, rank))
    out = {}
    for i in range(0, len(ids), batch):
        part = ids[i:i + batch]
        x = np.ascontiguousarray(np.asarray(latents, np.float32)[part])
        rec = binding.denoise_host(model, x, [trajs[s] for s in part], sched)
        for j, s in enumerate(part):
            out[s] = (x[j], {k: (v[j] if isinstance(v, np.ndarray) else v) for k, v in rec.items()
                             if k not in ("backbone_calls", "launches")})
    return out


def serve(model, latents, trajs, sched, group=None, batch=None):
    """All replicas call this with the same scene list; rank 0 returns
    (x [S, N, C], records in scene order), the other ranks None."""
    import torch.distributed as dist
    rank, world = _world(group)
    mine = serve_shard(model, latents, trajs, sched, rank, world, batch)
    if world > 1:
        parts = [None] * world if rank == 0 else None
        dist.gather_object(mine, parts, dst=0, group=group)
    else:
        parts = [mine]
    if rank != 0:
        return None
    merged = {}
    for p in parts:
        merged.update(p)
    if sorted(merged) != list(range(len(trajs))):
        raise RuntimeError("a replica did not report all of its scenes")
    x = np.stack([merged[s][0] for s in range(len(trajs))])
    return x, [merged[s][1] for s in range(len(trajs))]


def send_snapshot(snap, dst, group=None):
    """Hand a sampler snapshot (host uint8 array) to replica `dst`."""
    import torch
    import torch.distributed as dist
    buf = torch.from_numpy(np.ascontiguousarray(snap, np.uint8))
    dist.send(torch.tensor([buf.numel()], dtype=torch.int64), dst, group=group)
    dist.send(buf, dst, group=group)


def recv_snapshot(src, group=None):
    """Receive a snapshot sent by send_snapshot from replica `src`; its header
    is validated (dc_snapshot_info) before it is returned."""
    import torch
    import torch.distributed as dist
    n = torch.zeros(1, dtype=torch.int64)
    dist.recv(n, src, group=group)
    buf = torch.empty(int(n.item()), dtype=torch.uint8)
    dist.recv(buf, src, group=group)
    snap = buf.numpy()
    binding.snapshot_info(snap)
    return snap
