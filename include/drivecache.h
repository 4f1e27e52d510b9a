/*
 * drivecache.h -- C ABI of the GB300 DriveCache hot path.
 *
 * DriveCache (action-aware caching for driving world-model inference) lets a
 * diffusion sampler skip the expensive backbone F_k on some denoising steps
 * by substituting the most recently computed backbone output r_j (Eq. 1).
 * The host planner places those reuses from the planned ego motion with an
 * exact DP under a response budget (Eq. 2-11); at run time a causal drift
 * check (Eq. 12) may refuse a planned reuse, refresh the cache and replan the
 * remaining steps (Sec. 3.2).  The backbone here is a synthetic adaLN DiT.
 *
 * Conventions for every call:
 *  - Steps are 1-based: k = 1..K.  Arrays "[K+1]" leave index 0 unused.
 *  - Response / drift tables are row-major [K][H_max+1] doubles indexed
 *    [j][h]: j = 1..K-1 is the step of the last full evaluation, h = 1..H_max
 *    the cache age; row 0 and column 0 are ignored.
 *  - Actions: DC_ACT_COMPUTE (full backbone evaluation) or DC_ACT_REUSE.
 *  - The caller owns every pointer it passes; the library never keeps one
 *    after the call returns, except the model's own device memory.
 *  - Errors: calls return a dc_status and never abort.  Arguments are
 *    validated before any device work; dc_last_error() gives a thread-local
 *    message for the last failure on the calling thread.
 *  - Host planner calls (dc_motion_stats .. dc_calibrate_budget) are pure
 *    fp64 host code with no device dependency and are thread-safe.
 *  - A dc_model serves one call at a time: its workspace (activations,
 *    caches, profile counters) is shared by every call that takes the model,
 *    so such calls must not overlap, from several threads or on several
 *    streams.  Distinct models (on one device or several) are independent.
 *  - Calls whose results are device arrays (dc_drift_sums,
 *    dc_drift_sums_noalloc, dc_cache_copy, and dc_attention outside its
 *    tensor-core head dims) are asynchronous on their stream; calls that
 *    return host results, or that check a device error word, synchronise
 *    their stream before they return.
 */
#ifndef DRIVECACHE_H
#define DRIVECACHE_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  DC_OK = 0,
  DC_ERR_INVALID_ARG = 1,
  DC_ERR_NOMEM = 2,
  DC_ERR_CUDA = 3,
  DC_ERR_DEVICE_TIMEOUT = 4, /* a bounded device wait gave up */
  DC_ERR_NONFINITE = 5,      /* a latent or drift statistic became NaN/Inf */
  DC_ERR_UNSUPPORTED = 6     /* shape/dtype this build has no kernel for */
} dc_status;

enum { DC_ACT_COMPUTE = 1, DC_ACT_REUSE = 2 };
enum { DC_DTYPE_F32 = 0, DC_DTYPE_BF16 = 1 };

/* One planned ego pose: position in metres, heading in radians. */
typedef struct { double x, y, psi; } dc_pose;

/* A planned trajectory: n_poses consecutive poses (host memory). */
typedef struct { const dc_pose* poses; int n_poses; } dc_trajectory;

/* Planner variants: the method itself, the ablations of Table 3 and the
 * fixed-interval baseline of Table 1 (Sec. 4).  The paper names them without
 * formulas; the readings implemented are:
 *  DC_VAR_DRIVECACHE        the method as published (Sec. 3.1-3.2);
 *  DC_VAR_NO_MOTION_PRIOR   every scene planned at D = 1/2, no support gate;
 *  DC_VAR_SHUFFLED          dc_denoise plans scene s from the trajectory of
 *                           scene (s+1) mod B (the backbone still sees its
 *                           own); dc_plan plans the trajectory it is given;
 *  DC_VAR_TRANSLATION_ONLY  D = z^L, supported iff 0 <= z^L <= 1;
 *  DC_VAR_ROTATION_ONLY     D = z^Theta, supported iff 0 <= z^Theta <= 1;
 *  DC_VAR_FIXED_PLACEMENT   the method's B* reuses spread evenly over steps
 *                           2..T (below) instead of the DP placement; a
 *                           refused reuse is computed and the pattern kept;
 *  DC_VAR_FIXED_INTERVAL    `budget` (an integer) reuses spread evenly for
 *                           every scene, whatever its motion or support; no
 *                           charge and no drift check.
 * Even spreading: step k (2 <= k <= T) is a reuse iff
 * floor((k-1) n / (T-1)) > floor((k-2) n / (T-1)), except that a reuse whose
 * cache age would be illegal (the mask below, or h > H_max) is a full
 * evaluation instead. */
enum {
  DC_VAR_DRIVECACHE = 0,
  DC_VAR_NO_MOTION_PRIOR = 1,
  DC_VAR_SHUFFLED = 2,
  DC_VAR_TRANSLATION_ONLY = 3,
  DC_VAR_ROTATION_ONLY = 4,
  DC_VAR_FIXED_PLACEMENT = 5,
  DC_VAR_FIXED_INTERVAL = 6
};

/* Calibrated anchor responses (Sec. 3.1-3.2).
 *  (L0,T0), (L1,T1): low-motion and moving-turn anchor statistics (Eq. 2);
 *  valid = 0 means no moving-turn anchor exists -> every scene runs full
 *  inference.  q0/q1: joint run responses q^(i)_{j,h} (Eq. 7) of the two
 *  anchors; d0/d1: anchor input drifts d^(i)_{j,h} (Eq. 5).  All four are
 *  [K][H_max+1] (see conventions), finite and >= 0.
 *  legal: optional [K+1][H_max+1] bytes, legal[k][h] != 0 iff reusing at
 *  step k with cache age h is allowed (the L(k,h) mask of Eq. 10); NULL means
 *  every age 1..H_max at every step k >= 2.  eps: the epsilon of Eq. 3 and of
 *  the veto slack (1e-6 by default).  variant: a DC_VAR_* planner variant
 *  (0 = the method). */
typedef struct {
  int K, H_max;
  double L0, T0, L1, T1;
  int valid;
  const double *q0, *q1, *d0, *d1;
  const unsigned char* legal;
  double eps;
  int variant;
} dc_anchor_responses;

/* A per-scene schedule.  action: caller-owned [T+1] bytes (index 0 unused). */
typedef struct {
  int T;
  unsigned char* action;
  int n_reuse;      /* number of REUSE steps */
  double cost;      /* min_h J_T(n_reuse, h) of the plan (Eq. 10-11) */
  int supported;    /* 1 iff (z^L, z^Theta) in [0,1]^2 and anchors valid */
  double D;         /* motion intensity (Eq. 4); 0 when unsupported */
  double L, Theta;  /* motion statistics (Eq. 2) */
} dc_schedule;

/* Eq. 2: total translation L = sum ||p_t - p_{t-1}|| and accumulated
 * absolute wrapped yaw Theta = sum |wrap(psi_t - psi_{t-1})|, wrap into
 * (-pi, pi].  Needs n_poses >= 1 and finite poses. */
dc_status dc_motion_stats(const dc_trajectory* traj, double* L, double* Theta);

/* Sec. 3.1 anchor selection over n >= 1 calibration clips' (L, Theta):
 * population z-scores; low-motion anchor = argmin zL + zTheta; moving-turn
 * anchor = argmax zL * zTheta among clips with Theta > median(Theta),
 * L > L0 and Theta > Theta0; ties to the lowest index.  Writes
 * anchors_out = {L0, T0, L1, T1}, *valid (0 = empty candidate set) and,
 * if index_out != NULL, index_out = {i0, i1} (i1 = -1 when invalid). */
dc_status dc_select_anchors(const double* L, const double* Theta, int n,
                            double anchors_out[4], int* valid, int* index_out);

/* Sec. 3.1-3.2: plan one scene.  Eq. 2 -> Eq. 3 support gate -> Eq. 4 ->
 * Eq. 8/9 scene tables -> Eq. 10 DP from J_1(0,0) = 0 -> Eq. 11 B* under
 * `budget` (tau) -> backtracking (ties: smallest final age, then smallest
 * age before each refresh).  T must equal anc->K; out->action must hold T+1
 * bytes.  An unsupported scene gets an all-COMPUTE schedule.  Under
 * anc->variant the intensity and placement follow the variant (see DC_VAR_*);
 * for DC_VAR_FIXED_INTERVAL `budget` is the reuse count, an integer in
 * [0, T-1], and cost is 0. */
dc_status dc_plan(const dc_trajectory* traj, const dc_anchor_responses* anc, double budget,
                  int T, dc_schedule* out);

/* Sec. 3.2 suffix replanning after a forced full evaluation at step
 * k_refresh: DP from J_{k_refresh}(0,0) = 0 over steps k_refresh..T under
 * `remaining` (= tau - C_k) with the scene tables of intensity D.  Overwrites
 * inout->action[k_refresh..T] (action[k_refresh] = COMPUTE) and leaves the
 * prefix untouched; sets inout->n_reuse to the REUSE count of the whole
 * action array and inout->cost to the suffix plan's cost.  The fixed
 * variants (DC_VAR_FIXED_PLACEMENT, DC_VAR_FIXED_INTERVAL) never replan: the
 * actions are left as they are and cost is set to 0. */
dc_status dc_replan(const dc_anchor_responses* anc, double D, int k_refresh, double remaining,
                    dc_schedule* inout);

/* Sec. 3.2 budget calibration: the smallest table-cost threshold tau whose
 * median B* over the n calibration clips reaches `target` reuses (callers
 * pass target = ceil(rho_tar (T-1))).  Candidates are the finite
 * min_h J_T(n, h) of every supported clip; unsupported clips count as zero
 * reuses.  *reached = 0 if no candidate reaches the target, in which case
 * *tau is the largest candidate.  The motion variants calibrate on their own
 * intensities; DC_VAR_SHUFFLED and DC_VAR_FIXED_PLACEMENT give the method's
 * tau (they change which trajectory or which steps, not the count);
 * DC_VAR_FIXED_INTERVAL returns *tau = target (its reuse count), reached iff
 * the even schedule holds `target` reuses. */
dc_status dc_calibrate_budget(const dc_trajectory* clips, int n, const dc_anchor_responses* anc,
                              int target, int T, double* tau, int* reached);

/* Distributed budget calibration (Sec. 3.2): the tau rule above split into
 * a per-clip part, which any host can run on its share of the calibration
 * clips, and a combining part over the gathered curves.
 * dc_cost_curve writes m_out[n] = min_h J_T(n, h) for n = 0..T-1 (+infinity
 * where n reuses are infeasible) from the clip's own tables; an unsupported
 * clip gets an all-infinite curve and *supported = 0 (supported may be NULL).
 * DC_VAR_FIXED_INTERVAL has no curve (DC_ERR_INVALID_ARG: its budget is the
 * reuse count).  dc_budget_from_curves applies the tau rule to n curves
 * (row-major [n][T]): for the same clips, in any order, it returns exactly
 * what dc_calibrate_budget returns. */
dc_status dc_cost_curve(const dc_trajectory* clip, const dc_anchor_responses* anc, int T,
                        double* m_out, int* supported);
dc_status dc_budget_from_curves(const double* curves, int n, int T, int target, double* tau,
                                int* reached);

/* Sec. 3.2 model-specific legality as the L(k, h) mask of Eq. 10: writes
 * out[k*(H_max+1)+h] = 1 iff reusing at step k with cache age h (refresh at
 * j = k - h) is allowed, for k = 0..K, h = 0..H_max (caller-owned
 * [K+1][H_max+1] bytes).  Always 1 <= h <= H_max and k >= 2; in addition
 *  expert_boundary b > 0: two experts (steps 1..b, b+1..K) and no run
 *    crosses from one to the other (j and k in the same expert);
 *  segment_len T > 0: autoregressive segments of T steps with caches local
 *    to one segment ((j-1)/T == (k-1)/T), so every segment starts computed;
 *  no_cache_until p > 0: steps 1..p are native no-cache steps (k > p).
 * 0 disables a rule.  Pass the result as dc_anchor_responses.legal. */
dc_status dc_legal_mask(int K, int H_max, int expert_boundary, int segment_len,
                        int no_cache_until, unsigned char* out);

/* ------------------------------------------------------------------ model */

/* Shape of the synthetic DiT.  n_tokens = views x frames x rows x cols
 * (patch 1); channels 4 or 16; d_model <= 3072 and head_dim = d_model /
 * n_heads.  bf16: d_model and mlp_ratio * d_model multiples of 192 and
 * head_dim 64, 72 or 128; f32: d_model % 8 == 0 and head_dim 8, 16, 32 or
 * 64.  max_batch (internal scenes per call, two per scene with guidance,
 * <= 64) and max_steps bound the per-call workspace allocated by
 * dc_model_create.  Index bounds: n_blocks <= 4096, mlp_ratio <= 16,
 * n_tokens <= 2^22, max_batch * n_tokens <= 2^25, n_poses <= 65536,
 * max_steps <= 100000. */
typedef struct {
  int dtype;       /* DC_DTYPE_F32 or DC_DTYPE_BF16 */
  int n_blocks, d_model, n_heads, mlp_ratio, channels, n_tokens, n_poses;
  int max_batch, max_steps;
} dc_model_desc;

typedef struct dc_model dc_model;

/* Number of floats dc_model_create expects in host_weights; 0 when desc is
 * NULL or describes a shape dc_model_create rejects.  Host only. */
size_t dc_model_weight_count(const dc_model_desc* desc);

/* Create a model on `device` (the caller's current CUDA device when < 0).
 * host_weights: fp32, all tensors concatenated in this order, matrices
 * [out][in] row-major:
 *   w_embed[d][C] b_embed[d] pos[N][d] w_t1[d][256] b_t1[d] w_t2[d][d] b_t2[d]
 *   w_traj[d][3P] b_traj[d] w_ada[(6L+2)d][d] b_ada[(6L+2)d]
 *   per block l: w_qkv[3d][d] b_qkv[3d] w_o[d][d] b_o[d] w_1[md][d] b_1[md]
 *                w_2[d][md] b_2[d]            (md = mlp_ratio d)
 *   w_final[C][d] b_final[C]
 * For bf16 models the values are converted to bf16 (round to nearest even).
 * The model owns its weights and a workspace for max_batch scenes. */
dc_status dc_model_create(const dc_model_desc* desc, const float* host_weights, size_t n_floats,
                          int device, dc_model** out);
void dc_model_destroy(dc_model* m);

/* Per-scene conditioning: planned poses of each of the B scenes (host). */
typedef struct { int B; const dc_trajectory* traj; } dc_cond;

/* Sampler + controller settings for one dc_denoise call.
 *  sigmas: [K+1] host doubles, sigma_1 .. sigma_{K+1} stored 0-based.
 *  anchors: calibrated responses (anchors->K must equal K); tau: budget.
 *  veto: 1 = check drift and charge before every planned reuse (Eq. 12);
 *        0 = execute the plan as made (the no-veto ablation of Table 3).
 *  The planner variant is anchors->variant (DC_VAR_*).  The reduced-steps
 *  baseline of Table 2 is a plain call with fewer steps (K and sigmas of the
 *  shorter schedule) and a forced all-COMPUTE schedule.
 *  cfg_scale: 0 = one branch; otherwise classifier-free guidance with
 *        separate guidance branches (Sec. 3.2): every scene also runs an
 *        unconditional branch (the null trajectory: all poses at the origin,
 *        so its trajectory features vanish), each branch with its own cache
 *        of r, and v = v_u + cfg_scale (v_c - v_u) drives the Euler step.  The
 *        plan, the drift check (on x) and the charge stay per scene; both
 *        branches compute or reuse together.  Needs 2 B <= max_batch.
 *  forced: NULL, or [B][K+1] actions replayed verbatim (no planning, no
 *        checks; step 1 is always computed). */
typedef struct {
  int K;
  const double* sigmas;
  const dc_anchor_responses* anchors;
  double tau;
  int veto;
  const unsigned char* forced;
  double cfg_scale;
} dc_sched;

/* Optional per-call record (every pointer may be NULL; arrays caller-owned).
 * [B][K+1] arrays are indexed [s*(K+1) + k]. */
typedef struct {
  unsigned char* planned;   /* [B][K+1] initial plan */
  unsigned char* executed;  /* [B][K+1] executed actions */
  double* d_obs;            /* [B][K+1] observed drift at checked steps, NaN elsewhere */
  double* d_bar;            /* [B][K+1] threshold d_bar_{j,h} at checked steps */
  unsigned char* checked;   /* [B][K+1] 0 unchecked, 1 accepted, 2 refused */
  int* n_compute;           /* [B] */
  int* n_reuse;             /* [B] */
  int* n_veto;              /* [B] refused planned reuses */
  int* n_replan;            /* [B] */
  double* charge;           /* [B] final accumulated charge C */
  int* supported;           /* [B] */
  double* D;                /* [B] */
  long long backbone_calls; /* out: scene-steps that ran the block stack */
  long long launches;       /* out: kernels launched by the call */
} dc_run_stats;

/* Run the K-step Euler sampler on B <= max_batch scenes with the cache
 * controller (Eq. 1, Sec. 3.2).  latents: DEVICE fp32 [B][N][C], x_1 in,
 * x_{K+1} out.  stream: a cudaStream_t (NULL = legacy default stream).
 * Device work is enqueued on `stream`; the call synchronises the stream once
 * per step that has a planned reuse to read the drift statistics back, and
 * once at the end.  Returns DC_ERR_NONFINITE if a drift statistic is not
 * finite and DC_ERR_DEVICE_TIMEOUT if a bounded device wait gave up. */
dc_status dc_denoise(dc_model* m, float* latents, const dc_cond* cond, const dc_sched* sched,
                     void* stream, dc_run_stats* stats);

/* dc_denoise on HOST latents: copies [B][N][C] fp32 to the device, runs the
 * sampler, copies the result back into host_latents, synchronises `stream`.
 * Page-locked host memory gives asynchronous copies; pageable also works. */
dc_status dc_denoise_host(dc_model* m, float* host_latents, const dc_cond* cond,
                          const dc_sched* sched, void* stream, dc_run_stats* stats);

/* ------------------------------------------------ sampler-state snapshots
 * A snapshot is the whole state of a sampler call after k_done of its K
 * steps (Sec. 3.2 controller + Eq. 1 cache): the latents x_{k_done+1}, every
 * scene's refresh latent x_j and cache row c = r + b_e + pos (both guidance
 * branches), the
 * plan of the remaining steps after any replans, the charge C, the last
 * refresh j and cache age of each scene, and the call's record so far.
 * Resuming from it (dc_denoise_steps) continues the call exactly: the final
 * latents and record equal the uninterrupted call's bit for bit.  Use:
 * preempting a long call, or moving it to another model instance or box.
 * Layout (caller-owned host memory, native byte order):
 *   header, 128 bytes: char magic[8] "DCSNAP01"; uint32 version (3);
 *     int32 B, K, cfg (0 or 1), k_done, dtype, n_tokens, d_model, channels;
 *     uint32 element bytes of c; uint64 digest; uint64 total bytes;
 *     int64 backbone_calls; 56 zero bytes
 *   B scene records of 48 bytes: double charge, D; int32 j, age, supported,
 *     n_compute, n_reuse, n_veto, n_replan, 0
 *   uint8 planned, plan, executed, checked: [B][K+1] each, each padded to
 *     a multiple of 8 bytes
 *   double d_obs, d_bar: [B][K+1] each
 *   at the next multiple of 256: float latents [B][N][C], float x_j [B][N][C]
 *   at the next multiple of 256: c [B_i][N][d] in the model dtype
 *     (B_i = 2B with guidance, else B)
 *   bf16 models with 16 channels only, at the next multiple of 256: float
 *     [B_i][N][2], the sum and the sum of squares of each cache row's values
 * digest: FNV-1a (64-bit) of the call's inputs (trajectories, sigmas, tau,
 * veto, cfg_scale, and the forced actions or the anchor responses). */

/* Bytes of a snapshot of B scenes and K steps for a model of this shape
 * (cfg: 1 with guidance); 0 for an invalid argument.  Shapes are bounded so
 * that no section size overflows: B <= 65536, K <= 100000, n_tokens <= 2^26,
 * d_model and channels <= 65536; a header outside these bounds is rejected by
 * dc_snapshot_info and dc_denoise_steps.  Host only. */
size_t dc_snapshot_bytes(const dc_model_desc* desc, int B, int K, int cfg);

typedef struct {
  int B, K, cfg, k_done, dtype, n_tokens, d_model, channels;
  unsigned long long digest;
  long long backbone_calls;
} dc_snapshot_desc;

/* Validate a snapshot's header and size (magic, version, field ranges,
 * bytes == the size its shape implies) and describe it.  Host only;
 * DC_ERR_INVALID_ARG on any mismatch. */
dc_status dc_snapshot_info(const void* snap, size_t bytes, dc_snapshot_desc* out);

/* dc_denoise over steps k0+1 .. k_stop only.  k0 = 0 when resume is NULL
 * (latents holds x_1); otherwise k0 = the snapshot's k_done and latents is
 * overwritten with its x_{k0+1} (the snapshot must come from a call with the
 * same inputs -- its digest is checked -- on a model of the same dtype and
 * shape, possibly another instance).  k0 < k_stop <= K.  save: NULL, or a
 * host buffer of dc_snapshot_bytes(...) bytes that receives the state after
 * step k_stop (the stream is synchronised before return).  stats: as for
 * dc_denoise, covering steps 1..k_stop (restored from the snapshot for steps
 * up to k0); launches counts this call's kernels only.  dc_denoise is
 * dc_denoise_steps with k_stop = K and no snapshots. */
dc_status dc_denoise_steps(dc_model* m, float* latents, const dc_cond* cond, const dc_sched* sched,
                           int k_stop, const void* resume, size_t resume_bytes, void* save,
                           size_t save_bytes, void* stream, dc_run_stats* stats);

/* Eq. 5 along one full trace: run all K steps as full evaluations from
 * `noise` (DEVICE fp32 [N][C], not modified) under `traj`, and write
 * d_out[j*(H_max+1)+h] = ||u_{j+h} - u_j|| / (||u_{j+h}|| + eps) for
 * j = 1..K-1, h = 1..min(H_max, K-j) (other entries 0).  Host d_out,
 * [K][H_max+1] doubles; 1 <= K <= max_steps, 1 <= H_max <= 4096. */
dc_status dc_anchor_drift(dc_model* m, const float* noise, const dc_trajectory* traj, int K,
                          const double* sigmas, int H_max, double eps, double* d_out, void* stream);

/* Eq. 6-7 along one full trace: the joint run responses of one anchor.
 * Runs all K steps as full evaluations from `noise` (DEVICE fp32 [N][C], not
 * modified) under `traj` (the anchor trace x_1..x_{K+1} with its cached
 * r_1..r_K), forms e_{j,l} = H_{j+l}(x_{j+l}, r_j) - H_{j+l}(x_{j+l}, r_{j+l})
 * with the reuse interface H (Eq. 6), carries each through the rest of the
 * run with Jacobian-vector products of the model along the frozen trace --
 * dx_{t+1} = dsig_t e, dx_{m+1} = dx_m + dsig_m J_m dx_m for m = t+1..K,
 * J_m = dv_m/dx_m -- and writes
 *   q_out[j*(H_max+1)+h] = ||sum_{l<=h} dx_{K+1}(e_{j,l})|| / (||x_{K+1}|| + eps)
 * for j = 1..K-1, h = 1..min(H_max, K-j), other entries 0 (host q_out, fp64
 * sums).  The tangents run in fp32 on the model's weights (any model dtype);
 * the calibration cost is O(K^2 H_max) tangent passes, batched per trace
 * point.  Device workspace is allocated and freed inside the call (about
 * 8 GB at most for the tangents plus the stored activations); the call
 * synchronises `stream`.  head_dim must be 8, 16, 32, 64, 72 or 128;
 * 1 <= K <= max_steps, 1 <= H_max <= 4096. */
dc_status dc_anchor_response(dc_model* m, const float* noise, const dc_trajectory* traj, int K,
                             const double* sigmas, int H_max, double eps, double* q_out,
                             void* stream);

/* Drift sums for Eq. 12 on B scenes: for each scene s, out[2s] =
 * sum ||u(x_now_s) - u(x_ref_s)||^2 = sum ||(x_now_s - x_ref_s) W_e^T||^2 and
 * out[2s+1] = sum ||u(x_now_s)||^2 with u(x) = x W_e^T + b_e + pos, summed
 * over all tokens and channels in fp32 in a fixed order (deterministic).
 * x_now, x_ref: DEVICE fp32 [B][N][C]; out: DEVICE fp32 [2B].  The sums use
 * the model's per-call workspace (B <= max_batch). */
dc_status dc_drift_sums(dc_model* m, const float* x_now, const float* x_ref, int B, float* out,
                        void* stream);

/* dc_drift_sums for callers that cannot allocate device memory while they
 * run (for example a planning loop whose memory budget is fixed at start-up,
 * or a host process that may not call cudaMalloc after initialisation,
 * since cudaMalloc can synchronise the device and can fail).  The paper has
 * no counterpart.  It returns the same sums as dc_drift_sums, from the
 * same inputs into the same outputs (x_now, x_ref: DEVICE
 * fp32 [B][N][C]; out: DEVICE fp32 [2B]), but the reduction scratch is a
 * fixed 32 KiB array in device memory that every GPU loading this library
 * holds until the process exits; no device memory is allocated or freed.
 * B must be in [1, min(max_batch, 64)]; larger B is rejected with
 * DC_ERR_INVALID_ARG before any launch.  The first call on a device looks up
 * the array's device address (with that device made current); make that
 * first call before capturing the stream into a graph.  All calls share the
 * one array: calls that can overlap on the GPU (different streams without
 * ordering) race on it and must be serialised by the caller.  Every scratch
 * entry a call reads is written earlier in the same call.  The cached
 * address does not survive a cudaDeviceReset, which also invalidates every
 * model on the device: destroy models before a reset, create them again
 * after it. */
dc_status dc_drift_sums_noalloc(dc_model* m, const float* x_now, const float* x_ref, int B,
                                float* out, void* stream);

/* Test hook for the failure detection of the device kernels.  Every wait of
 * the tensor-core kernels (TMA copies landing, MMAs completing, the stages of
 * the warp-specialised pipelines handing work to each other) gives up after
 * a limit, records a code in the model's error word, lets the rest of the
 * launch drain and return, and makes later tensor-core launches of the model
 * skip their work until the host has read the word: the call then returns
 * DC_ERR_DEVICE_TIMEOUT and clears the word, and the next call runs normally.
 * The limit is 2 s; this call sets it to `ns` nanoseconds for the waits on
 * work in progress of the model's later launches (0 restores 2 s), so that a
 * test can make them run out.  Waits that drain copies or MMAs a CTA has
 * already issued keep the 2 s limit.  Synchronises the device. */
dc_status dc_set_wait_limit(dc_model* m, unsigned int ns);

/* Write the cached backbone output r_j (Eq. 1: r = h_L - u of the scene's
 * last full evaluation) of `scene` (0 <= scene < max_batch) into DEVICE
 * memory dst, [N][d] elements of the model dtype (fp32 or bf16); `bytes`
 * must equal N * d * sizeof(element).  The cache itself holds c = h_L -
 * x W_e^T = r + b_e + pos (so that a reuse step rebuilds u + r from the
 * latent alone); this call returns c - b_e - pos, rounded to the model
 * dtype.  Asynchronous on `stream`.  Intended for inspection and tests. */
dc_status dc_cache_copy(dc_model* m, int scene, void* dst, size_t bytes, void* stream);

/* The attention kernel of the block stack on caller-provided operands:
 * o = softmax(q k^T / sqrt(head_dim)) v over all n_tokens of each
 * (slot, head).  qkv: DEVICE [3][slots][heads][n_tokens][dhp] (q, k, v
 * planes) with dhp = head_dim rounded up to a multiple of 16 for bf16 (pad
 * columns must be zero) and dhp = head_dim for fp32; out: DEVICE
 * [slots][n_tokens][heads * head_dim].  dtype DC_DTYPE_BF16 supports
 * head_dim 64, 72, 128 (and 16); DC_DTYPE_F32 supports 8, 16, 32, 64.
 * slots * heads <= 2^15 and n_tokens <= 2^22 (DC_ERR_UNSUPPORTED beyond). */
dc_status dc_attention(int dtype, const void* qkv, int slots, int heads, int n_tokens,
                       int head_dim, void* out, void* stream);

/* Per-kernel timing of dc_denoise: when enabled, every launch is bracketed
 * by CUDA events on the call's stream and, at the end of each dc_denoise
 * call, its device time is added to its category together with the
 * algorithmic work of the launch (flops for the contractions, bytes for the
 * memory-bound kernels).  dc_profile(m, 1) resets the totals and starts
 * recording; dc_profile(m, 0) stops.  dc_profile_read fills DC_PROF_N
 * entries per array (any may be NULL). */
enum {
  DC_PROF_CONDITION = 0, /* adaLN modulation table (activations split + product) */
  DC_PROF_EMBED,         /* u = x W_e^T + b_e + pos */
  DC_PROF_LN,            /* adaLN LayerNorm + modulation */
  DC_PROF_GEMM_QKV,      /* tcgen05 GEMM, QKV scatter epilogue */
  DC_PROF_ATTENTION,     /* full spatiotemporal attention */
  DC_PROF_GEMM_OUT,      /* out-projection GEMM + gated residual */
  DC_PROF_GEMM_MLP1,     /* MLP-up GEMM + GELU (bf16, d 384: the fused MLP, both projections) */
  DC_PROF_GEMM_MLP2,     /* MLP-down GEMM + gated residual (none where the MLP is fused) */
  DC_PROF_FINAL,         /* interface + Euler + cache write (compute steps) */
  DC_PROF_REUSE,         /* reuse step: cached r + interface + Euler */
  DC_PROF_DRIFT,         /* drift sums of Eq. 12 */
  DC_PROF_JVP_ATTENTION, /* dc_anchor_response: attention and its tangent (fp32) */
  DC_PROF_JVP_GEMM,      /* dc_anchor_response: linear layers and their tangents (fp32) */
  DC_PROF_JVP_OTHER,     /* dc_anchor_response: LayerNorm, embedding, interface, updates */
  DC_PROF_COND_MLP,      /* the rest of the conditioning: timestep/trajectory MLPs before the
                            adaLN table and the per-step head tables after it */
  DC_PROF_N
};
dc_status dc_profile(dc_model* m, int enable);
dc_status dc_profile_read(dc_model* m, double* ms, long long* launches, double* flops,
                          double* bytes);

const char* dc_status_string(dc_status s);
const char* dc_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* DRIVECACHE_H */
