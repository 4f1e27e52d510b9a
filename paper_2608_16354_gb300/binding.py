"""Thin ctypes binding of libdrivecache.so (include/drivecache.h).

Argument marshalling only: every step of the hot path runs in the library.
Device buffers are passed as torch CUDA tensors (data_ptr) and streams as
torch streams; host arrays as NumPy.  There is no fallback: if the library
is missing or was built without a kernel, the call raises.
"""

import ctypes as C
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libdrivecache.so")

COMPUTE, REUSE = 1, 2
# planner variants (DC_VAR_* in include/drivecache.h)
(VAR_DRIVECACHE, VAR_NO_MOTION_PRIOR, VAR_SHUFFLED, VAR_TRANSLATION_ONLY, VAR_ROTATION_ONLY,
 VAR_FIXED_PLACEMENT, VAR_FIXED_INTERVAL) = range(7)
DTYPE_F32, DTYPE_BF16 = 0, 1

STATUS = {0: "DC_OK", 1: "DC_ERR_INVALID_ARG", 2: "DC_ERR_NOMEM", 3: "DC_ERR_CUDA",
          4: "DC_ERR_DEVICE_TIMEOUT", 5: "DC_ERR_NONFINITE", 6: "DC_ERR_UNSUPPORTED"}


class DCError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


class Pose(C.Structure):
    _fields_ = [("x", C.c_double), ("y", C.c_double), ("psi", C.c_double)]


class Trajectory(C.Structure):
    _fields_ = [("poses", C.POINTER(Pose)), ("n_poses", C.c_int)]


class AnchorResponses(C.Structure):
    _fields_ = [("K", C.c_int), ("H_max", C.c_int),
                ("L0", C.c_double), ("T0", C.c_double), ("L1", C.c_double), ("T1", C.c_double),
                ("valid", C.c_int),
                ("q0", C.POINTER(C.c_double)), ("q1", C.POINTER(C.c_double)),
                ("d0", C.POINTER(C.c_double)), ("d1", C.POINTER(C.c_double)),
                ("legal", C.POINTER(C.c_ubyte)), ("eps", C.c_double), ("variant", C.c_int)]


class Schedule(C.Structure):
    _fields_ = [("T", C.c_int), ("action", C.POINTER(C.c_ubyte)), ("n_reuse", C.c_int),
                ("cost", C.c_double), ("supported", C.c_int), ("D", C.c_double),
                ("L", C.c_double), ("Theta", C.c_double)]


class ModelDesc(C.Structure):
    _fields_ = [("dtype", C.c_int), ("n_blocks", C.c_int), ("d_model", C.c_int),
                ("n_heads", C.c_int), ("mlp_ratio", C.c_int), ("channels", C.c_int),
                ("n_tokens", C.c_int), ("n_poses", C.c_int), ("max_batch", C.c_int),
                ("max_steps", C.c_int)]


class Cond(C.Structure):
    _fields_ = [("B", C.c_int), ("traj", C.POINTER(Trajectory))]


class Sched(C.Structure):
    _fields_ = [("K", C.c_int), ("sigmas", C.POINTER(C.c_double)),
                ("anchors", C.POINTER(AnchorResponses)), ("tau", C.c_double),
                ("veto", C.c_int), ("forced", C.POINTER(C.c_ubyte)), ("cfg_scale", C.c_double)]


class RunStats(C.Structure):
    _fields_ = [("planned", C.POINTER(C.c_ubyte)), ("executed", C.POINTER(C.c_ubyte)),
                ("d_obs", C.POINTER(C.c_double)), ("d_bar", C.POINTER(C.c_double)),
                ("checked", C.POINTER(C.c_ubyte)),
                ("n_compute", C.POINTER(C.c_int)), ("n_reuse", C.POINTER(C.c_int)),
                ("n_veto", C.POINTER(C.c_int)), ("n_replan", C.POINTER(C.c_int)),
                ("charge", C.POINTER(C.c_double)), ("supported", C.POINTER(C.c_int)),
                ("D", C.POINTER(C.c_double)),
                ("backbone_calls", C.c_longlong), ("launches", C.c_longlong)]


class SnapshotDesc(C.Structure):
    _fields_ = [("B", C.c_int), ("K", C.c_int), ("cfg", C.c_int), ("k_done", C.c_int),
                ("dtype", C.c_int), ("n_tokens", C.c_int), ("d_model", C.c_int),
                ("channels", C.c_int), ("digest", C.c_ulonglong), ("backbone_calls", C.c_longlong)]


_lib = None


def lib():
    """Load libdrivecache.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: run __graft_entry__.build() first")
    L = C.CDLL(LIB_PATH)
    st = C.c_int
    P = C.POINTER
    sig = {
        "dc_motion_stats": (st, [P(Trajectory), P(C.c_double), P(C.c_double)]),
        "dc_select_anchors": (st, [P(C.c_double), P(C.c_double), C.c_int, P(C.c_double),
                                   P(C.c_int), P(C.c_int)]),
        "dc_plan": (st, [P(Trajectory), P(AnchorResponses), C.c_double, C.c_int, P(Schedule)]),
        "dc_replan": (st, [P(AnchorResponses), C.c_double, C.c_int, C.c_double, P(Schedule)]),
        "dc_calibrate_budget": (st, [P(Trajectory), C.c_int, P(AnchorResponses), C.c_int,
                                     C.c_int, P(C.c_double), P(C.c_int)]),
        "dc_cost_curve": (st, [P(Trajectory), P(AnchorResponses), C.c_int, P(C.c_double),
                               P(C.c_int)]),
        "dc_budget_from_curves": (st, [P(C.c_double), C.c_int, C.c_int, C.c_int,
                                       P(C.c_double), P(C.c_int)]),
        "dc_model_weight_count": (C.c_size_t, [P(ModelDesc)]),
        "dc_model_create": (st, [P(ModelDesc), P(C.c_float), C.c_size_t, C.c_int,
                                 P(C.c_void_p)]),
        "dc_model_destroy": (None, [C.c_void_p]),
        "dc_denoise": (st, [C.c_void_p, C.c_void_p, P(Cond), P(Sched), C.c_void_p, P(RunStats)]),
        "dc_denoise_host": (st, [C.c_void_p, P(C.c_float), P(Cond), P(Sched), C.c_void_p,
                                 P(RunStats)]),
        "dc_denoise_steps": (st, [C.c_void_p, C.c_void_p, P(Cond), P(Sched), C.c_int, C.c_void_p,
                                  C.c_size_t, C.c_void_p, C.c_size_t, C.c_void_p, P(RunStats)]),
        "dc_snapshot_bytes": (C.c_size_t, [P(ModelDesc), C.c_int, C.c_int, C.c_int]),
        "dc_snapshot_info": (st, [C.c_void_p, C.c_size_t, P(SnapshotDesc)]),
        "dc_legal_mask": (st, [C.c_int, C.c_int, C.c_int, C.c_int, C.c_int, P(C.c_ubyte)]),
        "dc_anchor_drift": (st, [C.c_void_p, C.c_void_p, P(Trajectory), C.c_int, P(C.c_double),
                                 C.c_int, C.c_double, P(C.c_double), C.c_void_p]),
        "dc_anchor_response": (st, [C.c_void_p, C.c_void_p, P(Trajectory), C.c_int,
                                    P(C.c_double), C.c_int, C.c_double, P(C.c_double),
                                    C.c_void_p]),
        "dc_drift_sums": (st, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_void_p,
                               C.c_void_p]),
        "dc_drift_sums_noalloc": (st, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_int, C.c_void_p,
                                       C.c_void_p]),
        "dc_cache_copy": (st, [C.c_void_p, C.c_int, C.c_void_p, C.c_size_t, C.c_void_p]),
        "dc_attention": (st, [C.c_int, C.c_void_p, C.c_int, C.c_int, C.c_int, C.c_int, C.c_void_p,
                              C.c_void_p]),
        "dc_profile": (st, [C.c_void_p, C.c_int]),
        "dc_set_wait_limit": (st, [C.c_void_p, C.c_uint]),
        "dc_profile_read": (st, [C.c_void_p, P(C.c_double), P(C.c_longlong), P(C.c_double),
                                 P(C.c_double)]),
        "dc_status_string": (C.c_char_p, [C.c_int]),
        "dc_last_error": (C.c_char_p, []),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    _lib = L
    return L


def _check(status):
    if status != 0:
        raise DCError(status, lib().dc_last_error().decode())


def _dptr(a):
    return a.ctypes.data_as(C.POINTER(C.c_double))


def _bptr(a):
    return a.ctypes.data_as(C.POINTER(C.c_ubyte))


# --------------------------------------------------------------- host side

class TrajectoryArgs:
    """Keeps pose buffers alive while a call uses them."""

    def __init__(self, poses_list):
        self.bufs = [np.ascontiguousarray(np.asarray(p, np.float64).reshape(-1, 3))
                     for p in poses_list]
        self.arr = (Trajectory * len(self.bufs))()
        for i, b in enumerate(self.bufs):
            self.arr[i].poses = b.ctypes.data_as(C.POINTER(Pose))
            self.arr[i].n_poses = b.shape[0]

    def ptr(self, i=0):
        return C.pointer(self.arr[i])


class AnchorArgs:
    """dc_anchor_responses built from Python tables ([K][H+1] nested lists or
    arrays) and anchor statistics."""

    def __init__(self, K, H, anc, tables, legal=None, eps=1e-6, variant=VAR_DRIVECACHE):
        def tab(t):
            if t is None:
                return np.zeros((K, H + 1), np.float64)
            return np.ascontiguousarray(np.asarray(t, np.float64).reshape(K, H + 1))
        self.q0, self.q1 = tab(tables["q0"]), tab(tables["q1"])
        self.d0, self.d1 = tab(tables.get("d0")), tab(tables.get("d1"))
        self.legal = None if legal is None else np.ascontiguousarray(
            np.asarray(legal, np.uint8).reshape(K + 1, H + 1))
        s = AnchorResponses()
        s.K, s.H_max = K, H
        s.L0, s.T0, s.L1, s.T1 = (float(anc["L0"]), float(anc["T0"]),
                                  float(anc["L1"]), float(anc["T1"]))
        s.valid = int(anc["valid"])
        s.q0, s.q1, s.d0, s.d1 = _dptr(self.q0), _dptr(self.q1), _dptr(self.d0), _dptr(self.d1)
        s.legal = _bptr(self.legal) if self.legal is not None else None
        s.eps = eps
        s.variant = int(variant)
        self.s = s

    def ptr(self):
        return C.pointer(self.s)


def legal_mask(K, H, expert_boundary=0, segment_len=0, no_cache_until=0):
    """dc_legal_mask: the L(k, h) mask [K+1][H+1] (uint8) of the model-specific
    rules (expert boundary, segment-local caches, no-cache steps)."""
    out = np.zeros((K + 1, H + 1), np.uint8)
    _check(lib().dc_legal_mask(int(K), int(H), int(expert_boundary), int(segment_len),
                               int(no_cache_until), out.ctypes.data_as(C.POINTER(C.c_ubyte))))
    return out


def motion_stats(poses):
    t = TrajectoryArgs([poses])
    L, T = C.c_double(), C.c_double()
    _check(lib().dc_motion_stats(t.ptr(), C.byref(L), C.byref(T)))
    return L.value, T.value


def select_anchors(Ls, Ts):
    Ls = np.ascontiguousarray(Ls, np.float64)
    Ts = np.ascontiguousarray(Ts, np.float64)
    out = (C.c_double * 4)()
    valid = C.c_int()
    idx = (C.c_int * 2)()
    _check(lib().dc_select_anchors(_dptr(Ls), _dptr(Ts), len(Ls), out, C.byref(valid), idx))
    return dict(L0=out[0], T0=out[1], L1=out[2], T1=out[3], valid=valid.value,
                i0=idx[0], i1=idx[1])


def plan(poses, anchors: AnchorArgs, budget, T):
    t = TrajectoryArgs([poses])
    acts = np.zeros(T + 1, np.uint8)
    s = Schedule()
    s.T, s.action = T, _bptr(acts)
    _check(lib().dc_plan(t.ptr(), anchors.ptr(), float(budget), T, C.byref(s)))
    return dict(actions=acts.tolist(), n_reuse=s.n_reuse, cost=s.cost, supported=s.supported,
                D=s.D, L=s.L, T=s.Theta)


def replan(anchors: AnchorArgs, D, k_refresh, remaining, actions):
    acts = np.ascontiguousarray(actions, np.uint8).copy()
    s = Schedule()
    s.T, s.action = len(acts) - 1, _bptr(acts)
    _check(lib().dc_replan(anchors.ptr(), float(D), int(k_refresh), float(remaining), C.byref(s)))
    return dict(actions=acts.tolist(), n_reuse=s.n_reuse, cost=s.cost)


def calibrate_budget(clip_poses, anchors: AnchorArgs, target, T):
    t = TrajectoryArgs(clip_poses)
    tau = C.c_double()
    reached = C.c_int()
    _check(lib().dc_calibrate_budget(t.arr, len(t.bufs), anchors.ptr(), int(target), int(T),
                                     C.byref(tau), C.byref(reached)))
    return tau.value, reached.value


def cost_curve(poses, anchors: AnchorArgs, T):
    """dc_cost_curve: (curve [T] with inf where infeasible, supported)."""
    t = TrajectoryArgs([poses])
    out = np.empty(int(T), np.float64)
    sup = C.c_int()
    _check(lib().dc_cost_curve(t.ptr(), anchors.ptr(), int(T), _dptr(out), C.byref(sup)))
    return out, sup.value


def budget_from_curves(curves, target):
    """dc_budget_from_curves on a [n, T] array: (tau, reached)."""
    c = np.ascontiguousarray(curves, np.float64)
    tau = C.c_double()
    reached = C.c_int()
    _check(lib().dc_budget_from_curves(_dptr(c), c.shape[0], c.shape[1], int(target),
                                       C.byref(tau), C.byref(reached)))
    return tau.value, reached.value


# -------------------------------------------------------------- device side

def _stream_handle(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return C.c_void_p(stream.cuda_stream)


class Model:
    """A synthetic DiT resident on the current CUDA device."""

    def __init__(self, wl, weights_blob, max_batch=None, max_steps=None, device=-1):
        d = ModelDesc()
        d.dtype = DTYPE_BF16 if wl.dtype == "bf16" else DTYPE_F32
        d.n_blocks, d.d_model, d.n_heads, d.mlp_ratio = wl.n_blocks, wl.d_model, wl.n_heads, wl.mlp_ratio
        d.channels, d.n_tokens, d.n_poses = wl.channels, wl.n_tokens, wl.n_poses
        d.max_batch = max_batch or wl.batch
        d.max_steps = max_steps or wl.steps
        self.desc = d
        self.wl = wl
        blob = np.ascontiguousarray(weights_blob, np.float32)
        n = lib().dc_model_weight_count(C.byref(d))
        if n and n != blob.size:  # n == 0: dc_model_create reports the invalid shape
            raise ValueError(f"weight blob has {blob.size} floats, model expects {n}")
        h = C.c_void_p()
        _check(lib().dc_model_create(C.byref(d), blob.ctypes.data_as(C.POINTER(C.c_float)),
                                     blob.size, int(device), C.byref(h)))
        self.h = h

    def close(self):
        if self.h:
            lib().dc_model_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class StatsArgs:
    def __init__(self, B, K):
        self.planned = np.zeros((B, K + 1), np.uint8)
        self.executed = np.zeros((B, K + 1), np.uint8)
        self.d_obs = np.full((B, K + 1), np.nan)
        self.d_bar = np.full((B, K + 1), np.nan)
        self.checked = np.zeros((B, K + 1), np.uint8)
        self.n_compute = np.zeros(B, np.int32)
        self.n_reuse = np.zeros(B, np.int32)
        self.n_veto = np.zeros(B, np.int32)
        self.n_replan = np.zeros(B, np.int32)
        self.charge = np.zeros(B, np.float64)
        self.supported = np.zeros(B, np.int32)
        self.D = np.zeros(B, np.float64)
        s = RunStats()
        s.planned, s.executed = _bptr(self.planned), _bptr(self.executed)
        s.d_obs, s.d_bar, s.checked = _dptr(self.d_obs), _dptr(self.d_bar), _bptr(self.checked)
        ip = C.POINTER(C.c_int)
        s.n_compute = self.n_compute.ctypes.data_as(ip)
        s.n_reuse = self.n_reuse.ctypes.data_as(ip)
        s.n_veto = self.n_veto.ctypes.data_as(ip)
        s.n_replan = self.n_replan.ctypes.data_as(ip)
        s.charge = _dptr(self.charge)
        s.supported = self.supported.ctypes.data_as(ip)
        s.D = _dptr(self.D)
        self.s = s

    def as_dict(self):
        return dict(planned=self.planned, executed=self.executed, d_obs=self.d_obs,
                    d_bar=self.d_bar, checked=self.checked, n_compute=self.n_compute,
                    n_reuse=self.n_reuse, n_veto=self.n_veto, n_replan=self.n_replan,
                    charge=self.charge, supported=self.supported, D=self.D,
                    backbone_calls=self.s.backbone_calls, launches=self.s.launches)


class SchedArgs:
    def __init__(self, K, sigmas, anchors: AnchorArgs, tau, veto=True, forced=None, cfg_scale=0.0):
        self.sig = np.ascontiguousarray(sigmas, np.float64)
        assert self.sig.size == K + 1
        self.forced = None if forced is None else np.ascontiguousarray(forced, np.uint8)
        s = Sched()
        s.K, s.sigmas = K, _dptr(self.sig)
        s.anchors = anchors.ptr()
        s.tau, s.veto = float(tau), int(veto)
        s.forced = _bptr(self.forced) if self.forced is not None else None
        s.cfg_scale = float(cfg_scale)
        self.anchors = anchors
        self.s = s


def denoise(model: Model, latents, trajs, sched: SchedArgs, stream=None, stats=True):
    """dc_denoise on a CUDA fp32 tensor [B, N, C] (updated in place)."""
    B = latents.shape[0]
    ta = TrajectoryArgs(trajs)
    cond = Cond(B, ta.arr)
    st = StatsArgs(B, sched.s.K) if stats else None
    _check(lib().dc_denoise(model.h, C.c_void_p(latents.data_ptr()), C.byref(cond),
                            C.byref(sched.s), _stream_handle(stream),
                            C.byref(st.s) if st else None))
    return st.as_dict() if st else None


def snapshot_bytes(desc: ModelDesc, B, K, cfg=False):
    """dc_snapshot_bytes (host only); 0 for an invalid argument."""
    return lib().dc_snapshot_bytes(C.byref(desc), int(B), int(K), int(bool(cfg)))


def snapshot_info(snap):
    """dc_snapshot_info on a host uint8 array: the validated header fields."""
    buf = np.ascontiguousarray(snap, np.uint8)
    out = SnapshotDesc()
    _check(lib().dc_snapshot_info(C.c_void_p(buf.ctypes.data), buf.size, C.byref(out)))
    return {f: getattr(out, f) for f, _ in SnapshotDesc._fields_}


def denoise_steps(model: Model, latents, trajs, sched: SchedArgs, k_stop, resume=None,
                  save=False, stream=None, stats=True):
    """dc_denoise_steps on a CUDA fp32 tensor [B, N, C] (updated in place).
    resume: a snapshot (host uint8 array) or None; save: return the state
    after step k_stop as a new host uint8 array.  Returns (stats, snapshot)."""
    B = latents.shape[0]
    ta = TrajectoryArgs(trajs)
    cond = Cond(B, ta.arr)
    st = StatsArgs(B, sched.s.K) if stats else None
    rin = None if resume is None else np.ascontiguousarray(resume, np.uint8)
    out = None
    if save:
        n = snapshot_bytes(model.desc, B, sched.s.K, sched.s.cfg_scale != 0.0)
        out = np.empty(n, np.uint8)
    _check(lib().dc_denoise_steps(
        model.h, C.c_void_p(latents.data_ptr()), C.byref(cond), C.byref(sched.s), int(k_stop),
        C.c_void_p(rin.ctypes.data) if rin is not None else None, rin.size if rin is not None else 0,
        C.c_void_p(out.ctypes.data) if out is not None else None, out.size if out is not None else 0,
        _stream_handle(stream), C.byref(st.s) if st else None))
    return (st.as_dict() if st else None), out


def denoise_host(model: Model, host_latents, trajs, sched: SchedArgs, stream=None, stats=True):
    """dc_denoise_host on a host fp32 array/tensor [B, N, C] (updated in place)."""
    B = host_latents.shape[0]
    ta = TrajectoryArgs(trajs)
    cond = Cond(B, ta.arr)
    st = StatsArgs(B, sched.s.K) if stats else None
    if hasattr(host_latents, "data_ptr"):
        ptr = C.cast(C.c_void_p(host_latents.data_ptr()), C.POINTER(C.c_float))
    else:
        ptr = host_latents.ctypes.data_as(C.POINTER(C.c_float))
    _check(lib().dc_denoise_host(model.h, ptr, C.byref(cond), C.byref(sched.s),
                                 _stream_handle(stream), C.byref(st.s) if st else None))
    return st.as_dict() if st else None


def anchor_drift(model: Model, noise, poses, K, sigmas, H, eps=1e-6, stream=None):
    """dc_anchor_drift: noise is a CUDA fp32 tensor [N, C]; returns [K][H+1]."""
    ta = TrajectoryArgs([poses])
    sig = np.ascontiguousarray(sigmas, np.float64)
    out = np.zeros((K, H + 1), np.float64)
    _check(lib().dc_anchor_drift(model.h, C.c_void_p(noise.data_ptr()), ta.ptr(), int(K),
                                 _dptr(sig), int(H), float(eps), _dptr(out),
                                 _stream_handle(stream)))
    return out



def anchor_response(model: Model, noise, poses, K, sigmas, H, eps=1e-6, stream=None):
    """dc_anchor_response (Eq. 6-7): noise is a CUDA fp32 tensor [N, C];
    returns the joint run responses q [K][H+1]."""
    ta = TrajectoryArgs([poses])
    sig = np.ascontiguousarray(sigmas, np.float64)
    out = np.zeros((K, H + 1), np.float64)
    _check(lib().dc_anchor_response(model.h, C.c_void_p(noise.data_ptr()), ta.ptr(), int(K),
                                    _dptr(sig), int(H), float(eps), _dptr(out),
                                    _stream_handle(stream)))
    return out

def drift_sums(model: Model, x_now, x_ref, out, stream=None):
    """dc_drift_sums on CUDA fp32 tensors x_now/x_ref [B, N, C], out [2B]."""
    _check(lib().dc_drift_sums(model.h, C.c_void_p(x_now.data_ptr()), C.c_void_p(x_ref.data_ptr()),
                               int(x_now.shape[0]), C.c_void_p(out.data_ptr()),
                               _stream_handle(stream)))


def cache_copy(model: Model, scene, dst, stream=None):
    """dc_cache_copy into a CUDA tensor dst of the model dtype, shape [N, d]."""
    _check(lib().dc_cache_copy(model.h, int(scene), C.c_void_p(dst.data_ptr()),
                               dst.numel() * dst.element_size(), _stream_handle(stream)))


def attention(qkv, slots, heads, n_tokens, head_dim, out, stream=None):
    """dc_attention on CUDA tensors (bf16 or fp32, see include/drivecache.h)."""
    import torch
    dtype = DTYPE_BF16 if qkv.dtype == torch.bfloat16 else DTYPE_F32
    _check(lib().dc_attention(dtype, C.c_void_p(qkv.data_ptr()), int(slots), int(heads),
                              int(n_tokens), int(head_dim), C.c_void_p(out.data_ptr()),
                              _stream_handle(stream)))


PROF_NAMES = ["condition", "embed", "ln_mod", "gemm_qkv", "attention", "gemm_out", "gemm_mlp1",
              "gemm_mlp2", "final_compute", "reuse", "drift", "jvp_attention", "jvp_gemm",
              "jvp_other", "cond_mlp"]


def set_wait_limit(model: Model, ns):
    """dc_set_wait_limit: the limit (ns) of the device waits on work in
    progress; 0 restores the default."""
    _check(lib().dc_set_wait_limit(model.h, int(ns)))


def profile(model: Model, enable):
    _check(lib().dc_profile(model.h, int(bool(enable))))


def profile_read(model: Model):
    n = len(PROF_NAMES)
    ms, cnt = (C.c_double * n)(), (C.c_longlong * n)()
    fl, by = (C.c_double * n)(), (C.c_double * n)()
    _check(lib().dc_profile_read(model.h, ms, cnt, fl, by))
    return {PROF_NAMES[i]: dict(ms=ms[i], launches=cnt[i], flops=fl[i], bytes=by[i])
            for i in range(n)}


def drift_sums_noalloc(model: Model, x_now, x_ref, out, stream=None):
    """dc_drift_sums_noalloc: same as drift_sums, with no device allocation
    (fixed scratch inside the library, at most 64 scenes per call)."""
    _check(lib().dc_drift_sums_noalloc(model.h, C.c_void_p(x_now.data_ptr()),
                                       C.c_void_p(x_ref.data_ptr()), int(x_now.shape[0]),
                                       C.c_void_p(out.data_ptr()), _stream_handle(stream)))
