// Sampler-state snapshots (host side): the byte layout declared in
// drivecache.h, the digest of a call's inputs, and header validation.  The
// sampler (model.cu) fills and consumes the blobs; nothing here touches the
// device.
#pragma once

#include <cstddef>
#include <cstdint>

#include "drivecache.h"

namespace dc {

constexpr char kSnapMagic[8] = {'D', 'C', 'S', 'N', 'A', 'P', '0', '1'};
constexpr uint32_t kSnapVersion = 3;  // 2: cache rows c = r + b_e + pos; 3: their row sums

struct SnapHeader {
  char magic[8];
  uint32_t version;
  int32_t B, K, cfg, k_done, dtype, N, d, C;
  uint32_t elt;
  uint64_t digest;
  uint64_t bytes;
  int64_t backbone_calls;
  uint8_t pad[56];
};
static_assert(sizeof(SnapHeader) == 128, "snapshot header is 128 bytes");

struct SnapScene {
  double charge, D;
  int32_t j, age, supported, n_compute, n_reuse, n_veto, n_replan, zero;
};
static_assert(sizeof(SnapScene) == 48, "snapshot scene record is 48 bytes");

// Offsets of every section for one call shape.
struct SnapLayout {
  int B = 0, K = 0, Bi = 0, N = 0, d = 0, C = 0;
  size_t elt = 0, W = 0;
  size_t scene = 0, planned = 0, plan = 0, executed = 0, checked = 0, d_obs = 0, d_bar = 0,
         lat = 0, xj = 0, r = 0, cs = 0, cs_bytes = 0, total = 0;
};
SnapLayout snap_layout(int B, int K, int cfg, int N, int d, int C, size_t elt);

// FNV-1a (64-bit) over the inputs that determine a call: trajectories,
// sigmas, tau, veto, cfg_scale, and the forced actions or the anchor
// responses (tables, legality mask, eps, variant).
uint64_t call_digest(const dc_cond* cond, const dc_sched* sc);

// Checks magic, version, field ranges and that `bytes` equals the size the
// header's shape implies; fills *h.
dc_status read_header(const void* snap, size_t bytes, SnapHeader* h);

}  // namespace dc
