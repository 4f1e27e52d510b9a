// Host planner internals (C++17, fp64, no device code).  The C entry points
// in planner.cpp and the sampler runtime both call these.
#pragma once

#include <string>
#include <vector>

#include "drivecache.h"

namespace dc {

constexpr unsigned char kCompute = DC_ACT_COMPUTE;
constexpr unsigned char kReuse = DC_ACT_REUSE;

void set_error(const std::string& msg);

// Eq. 2.
void motion_stats(const dc_pose* p, int n, double* L, double* T);

// Eq. 3 + support gate + Eq. 4: returns 1 and D when supported.
int scene_intensity(double L, double T, const dc_anchor_responses& a, double* D);

// Eq. 8-9 for one scene: c_hat and d_bar, row-major [K][H+1].
struct SceneTables {
  int K = 0, H = 0;
  std::vector<double> c, dbar;
  double at_c(int j, int h) const { return c[(size_t)j * (H + 1) + h]; }
  double at_d(int j, int h) const { return dbar[(size_t)j * (H + 1) + h]; }
};
void scene_tables(const dc_anchor_responses& a, double D, SceneTables* t);

// Eq. 10-11 + backtracking on steps k0..K from a full evaluation at k0.
// acts must hold K+1 entries; entries k0..K are written.  Returns B*.
int plan_suffix(const SceneTables& t, const unsigned char* legal, int k0, double budget,
                unsigned char* acts, double* cost);

// Cost curve m(n) = min_h J_K(n, h) from k0 = 1 (INF where infeasible).
void cost_curve(const SceneTables& t, const unsigned char* legal, std::vector<double>* m);

// The fixed variants' schedule: n reuses spread evenly over steps 2..T,
// an illegal age turning the reuse into a full evaluation.  acts[1..T].
void even_schedule(int n, int T, int H, const unsigned char* legal, unsigned char* acts);

// One scene's initial plan under anchors.variant (dc_plan and the sampler):
// fills acts[1..K], *n_reuse, *cost and *D, and *tabs when the variant uses
// scene tables; returns 1 when the scene is planned (supported).
int plan_scene(double L, double Th, const dc_anchor_responses& a, double budget,
               unsigned char* acts, int* n_reuse, double* cost, double* D, SceneTables* tabs);

dc_status check_anchors(const dc_anchor_responses* a);

// DC_VAR_FIXED_INTERVAL: the budget is a reuse count, an integer in [0, K-1].
dc_status check_reuse_count(const dc_anchor_responses& a, double budget);

}  // namespace dc
