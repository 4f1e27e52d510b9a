// Sampler-state snapshots: layout, input digest and header checks (host).
#include "runtime/snapshot.h"

#include <cstring>
#include <string>

#include "plan/planner.h"

namespace dc {

namespace {

size_t up8(size_t x) { return (x + 7) & ~size_t(7); }
size_t up256(size_t x) { return (x + 255) & ~size_t(255); }

struct Fnv {
  uint64_t h = 1469598103934665603ull;
  void bytes(const void* p, size_t n) {
    const unsigned char* c = static_cast<const unsigned char*>(p);
    for (size_t i = 0; i < n; ++i) {
      h ^= c[i];
      h *= 1099511628211ull;
    }
  }
  template <typename T>
  void val(const T& v) { bytes(&v, sizeof(T)); }
};

}  // namespace

SnapLayout snap_layout(int B, int K, int cfg, int N, int d, int C, size_t elt) {
  SnapLayout l;
  l.B = B; l.K = K; l.Bi = cfg ? 2 * B : B; l.N = N; l.d = d; l.C = C; l.elt = elt;
  l.W = (size_t)K + 1;
  const size_t bw = up8((size_t)B * l.W);
  l.scene = sizeof(SnapHeader);
  l.planned = l.scene + (size_t)B * sizeof(SnapScene);
  l.plan = l.planned + bw;
  l.executed = l.plan + bw;
  l.checked = l.executed + bw;
  l.d_obs = l.checked + bw;
  l.d_bar = l.d_obs + (size_t)B * l.W * sizeof(double);
  l.lat = up256(l.d_bar + (size_t)B * l.W * sizeof(double));
  l.xj = l.lat + (size_t)B * N * C * sizeof(float);
  l.r = up256(l.xj + (size_t)B * N * C * sizeof(float));
  l.cs = up256(l.r + (size_t)l.Bi * N * d * elt);
  // the row sums of the cache: bf16 models with 16 channels (tensor-core interface)
  l.cs_bytes = elt == 2 && C == 16 ? (size_t)l.Bi * N * 2 * sizeof(float) : 0;
  l.total = l.cs_bytes ? l.cs + l.cs_bytes : l.r + (size_t)l.Bi * N * d * elt;
  return l;
}

uint64_t call_digest(const dc_cond* cond, const dc_sched* sc) {
  Fnv f;
  f.val(cond->B);
  for (int s = 0; s < cond->B; ++s) {
    const dc_trajectory& t = cond->traj[s];
    f.val(t.n_poses);
    f.bytes(t.poses, (size_t)t.n_poses * sizeof(dc_pose));
  }
  f.val(sc->K);
  f.bytes(sc->sigmas, (size_t)(sc->K + 1) * sizeof(double));
  f.val(sc->tau);
  f.val(sc->veto);
  f.val(sc->cfg_scale);
  const size_t W = (size_t)sc->K + 1;
  if (sc->forced) {
    f.val(1);
    f.bytes(sc->forced, (size_t)cond->B * W);
  } else {
    f.val(0);
    const dc_anchor_responses* a = sc->anchors;
    f.val(a->K); f.val(a->H_max);
    f.val(a->L0); f.val(a->T0); f.val(a->L1); f.val(a->T1);
    f.val(a->valid); f.val(a->eps); f.val(a->variant);
    const size_t tab = (size_t)a->K * (a->H_max + 1);
    for (const double* q : {a->q0, a->q1, a->d0, a->d1}) f.bytes(q, tab * sizeof(double));
    f.val(a->legal ? 1 : 0);
    if (a->legal) f.bytes(a->legal, (size_t)(a->K + 1) * (a->H_max + 1));
  }
  return f.h;
}

dc_status read_header(const void* snap, size_t bytes, SnapHeader* h) {
  if (!snap || !h) { set_error("snapshot or header is NULL"); return DC_ERR_INVALID_ARG; }
  if (bytes < sizeof(SnapHeader)) {
    set_error("snapshot shorter than its 128-byte header");
    return DC_ERR_INVALID_ARG;
  }
  std::memcpy(h, snap, sizeof(SnapHeader));
  if (std::memcmp(h->magic, kSnapMagic, sizeof(kSnapMagic)) != 0) {
    set_error("not a sampler snapshot (magic)");
    return DC_ERR_INVALID_ARG;
  }
  if (h->version != kSnapVersion) {
    set_error("snapshot version " + std::to_string(h->version) + " is not supported");
    return DC_ERR_INVALID_ARG;
  }
  // shape bounds keep every section size far from size_t overflow
  if (h->B < 1 || h->B > (1 << 16) || h->K < 1 || h->K > 100000 || (h->cfg != 0 && h->cfg != 1) ||
      h->k_done < 1 || h->k_done > h->K || h->N < 1 || h->N > (1 << 26) || h->d < 1 ||
      h->d > (1 << 16) || h->C < 1 || h->C > (1 << 16) ||
      (h->dtype != DC_DTYPE_F32 && h->dtype != DC_DTYPE_BF16) ||
      h->elt != (h->dtype == DC_DTYPE_BF16 ? 2u : 4u) || h->backbone_calls < 0) {
    set_error("snapshot header fields out of range");
    return DC_ERR_INVALID_ARG;
  }
  const SnapLayout l = snap_layout(h->B, h->K, h->cfg, h->N, h->d, h->C, h->elt);
  if (h->bytes != l.total || bytes != l.total) {
    set_error("snapshot size " + std::to_string(bytes) + " does not match its shape (" +
              std::to_string(l.total) + " bytes)");
    return DC_ERR_INVALID_ARG;
  }
  return DC_OK;
}

}  // namespace dc

extern "C" {

size_t dc_snapshot_bytes(const dc_model_desc* desc, int B, int K, int cfg) {
  if (!desc || B < 1 || B > (1 << 16) || K < 1 || K > 100000 || (cfg != 0 && cfg != 1) ||
      desc->n_tokens < 1 || desc->n_tokens > (1 << 26) || desc->d_model < 1 ||
      desc->d_model > (1 << 16) || desc->channels < 1 || desc->channels > (1 << 16) ||
      (desc->dtype != DC_DTYPE_F32 && desc->dtype != DC_DTYPE_BF16))
    return 0;
  const size_t elt = desc->dtype == DC_DTYPE_BF16 ? 2 : 4;
  return dc::snap_layout(B, K, cfg, desc->n_tokens, desc->d_model, desc->channels, elt).total;
}

dc_status dc_snapshot_info(const void* snap, size_t bytes, dc_snapshot_desc* out) {
  dc::SnapHeader h;
  dc_status s = dc::read_header(snap, bytes, &h);
  if (s != DC_OK) return s;
  if (!out) { dc::set_error("out is NULL"); return DC_ERR_INVALID_ARG; }
  out->B = h.B;
  out->K = h.K;
  out->cfg = h.cfg;
  out->k_done = h.k_done;
  out->dtype = h.dtype;
  out->n_tokens = h.N;
  out->d_model = h.d;
  out->channels = h.C;
  out->digest = h.digest;
  out->backbone_calls = h.backbone_calls;
  return DC_OK;
}

}  // extern "C"
