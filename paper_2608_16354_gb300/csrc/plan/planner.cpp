// Host planner of DriveCache: motion statistics (Eq. 2), anchor selection
// (Sec. 3.1), support gate and intensity (Eq. 3-4), scene tables (Eq. 8-9),
// exact DP placement (Eq. 10-11) with backtracking, suffix replanning and
// budget calibration (Sec. 3.2).
//
// All arithmetic is IEEE binary64, evaluated left to right in step order and
// compiled without floating-point contraction, so every decision is a
// deterministic function of the inputs on any host.

#include "planner.h"

#include <algorithm>
#include <cmath>
#include <cstring>
#include <limits>
#include <set>
#include <string>
#include <vector>

namespace dc {

namespace {
const double kInf = std::numeric_limits<double>::infinity();
const double kPi = 3.141592653589793238462643383279502884;
thread_local std::string g_last_error;

// Angle difference wrapped into (-pi, pi] by the IEEE remainder (exact).
double wrap_angle(double a) {
  double r = std::remainder(a, 2.0 * kPi);
  if (r == -kPi) r = kPi;
  return r;
}

bool legal_at(const unsigned char* legal, int H, int k, int h) {
  if (h < 1 || h > H || k < 2) return false;
  return legal == nullptr || legal[(size_t)k * (H + 1) + h] != 0;
}

double median_of(std::vector<double> v) {
  std::sort(v.begin(), v.end());
  size_t n = v.size();
  if (n % 2 == 1) return v[n / 2];
  return (v[n / 2 - 1] + v[n / 2]) / 2.0;
}

// Sec. 3.2 tau rule on the cost curves of the calibration clips (entry n =
// min_h J_T(n, h), +inf where infeasible; an empty or all-infinite curve is a
// clip that counts zero reuses): the smallest finite curve value whose
// median B* reaches `target`, else the largest (*reached = 0); 0 without
// candidates.  The result does not depend on the order of the clips.
void budget_from_curves(const std::vector<std::vector<double>>& curves, int target, double* tau,
                        int* reached) {
  const int n = (int)curves.size();
  std::set<double> cands;
  for (const auto& c : curves)
    for (double v : c)
      if (v < kInf) cands.insert(v);
  if (cands.empty()) {
    *tau = 0.0;
    if (reached) *reached = 0;
    return;
  }
  std::vector<double> counts(n);
  for (double c : cands) {
    for (int i = 0; i < n; ++i) {
      int b = 0;
      for (size_t m = 0; m < curves[i].size(); ++m)
        if (curves[i][m] < kInf && curves[i][m] <= c) b = (int)m;
      counts[i] = (double)b;
    }
    if (median_of(counts) >= (double)target) {
      *tau = c;
      if (reached) *reached = 1;
      return;
    }
  }
  *tau = *cands.rbegin();
  if (reached) *reached = 0;
}

void zscores(const double* v, int n, std::vector<double>* z) {
  double s = 0.0;
  for (int i = 0; i < n; ++i) s = s + v[i];
  double mean = s / n;
  double ss = 0.0;
  for (int i = 0; i < n; ++i) ss = ss + (v[i] - mean) * (v[i] - mean);
  double sd = std::sqrt(ss / n);
  z->assign(n, 0.0);
  if (sd == 0.0) return;
  for (int i = 0; i < n; ++i) (*z)[i] = (v[i] - mean) / sd;
}

// Rolling DP of Eq. 10 from J_{k0}(0,0) = 0.  Fills the final row
// Jfin[n][h] (n = 0..K-k0) and the refresh argmin table arg[k][n].
struct DPResult {
  int nmax = 0, H = 0, k0 = 1, K = 0;
  std::vector<double> Jfin;  // [(nmax+1) * (H+1)]
  std::vector<int> arg;      // [(K+1) * (nmax+1)], refresh-state argmin
};

void run_dp(const SceneTables& t, const unsigned char* legal, int k0, DPResult* r) {
  const int K = t.K, H = t.H;
  const int nmax = K - k0;
  const int W = H + 1;
  r->nmax = nmax; r->H = H; r->k0 = k0; r->K = K;
  std::vector<double> cur((size_t)(nmax + 1) * W, kInf), nxt((size_t)(nmax + 1) * W);
  r->arg.assign((size_t)(K + 1) * (nmax + 1), -1);
  cur[0] = 0.0;
  for (int k = k0; k < K; ++k) {
    std::fill(nxt.begin(), nxt.end(), kInf);
    int* argk = &r->arg[(size_t)(k + 1) * (nmax + 1)];
    // J_{k+1}(n, 0) = min_h J_k(n, h), smallest h on ties
    for (int n = 0; n <= nmax; ++n) {
      double best = kInf;
      int bh = -1;
      for (int h = 0; h <= H; ++h) {
        double v = cur[(size_t)n * W + h];
        if (v < best) { best = v; bh = h; }
      }
      nxt[(size_t)n * W] = best;
      argk[n] = bh;
    }
    // J_{k+1}(n+1, h+1) = J_k(n, h) + c_hat_{k-h, h+1} when L(k+1, h+1)
    for (int n = 0; n < nmax; ++n) {
      for (int h = 0; h < H; ++h) {
        double v = cur[(size_t)n * W + h];
        if (v == kInf) continue;
        if (!legal_at(legal, H, k + 1, h + 1)) continue;
        double cand = v + t.at_c(k - h, h + 1);
        double& dst = nxt[(size_t)(n + 1) * W + h + 1];
        if (cand < dst) dst = cand;
      }
    }
    std::swap(cur, nxt);
  }
  r->Jfin = cur;
}

}  // namespace

void set_error(const std::string& msg) { g_last_error = msg; }
static const char* last_error_cstr() { return g_last_error.c_str(); }

void motion_stats(const dc_pose* p, int n, double* L, double* T) {
  double l = 0.0, th = 0.0;
  for (int t = 1; t < n; ++t) {
    double dx = p[t].x - p[t - 1].x;
    double dy = p[t].y - p[t - 1].y;
    l = l + std::sqrt(dx * dx + dy * dy);
    th = th + std::fabs(wrap_angle(p[t].psi - p[t - 1].psi));
  }
  *L = l;
  *T = th;
}

int scene_intensity(double L, double T, const dc_anchor_responses& a, double* D) {
  *D = 0.0;
  if (!a.valid) return 0;
  if (a.variant == DC_VAR_NO_MOTION_PRIOR) {  // no motion prior: one intensity for all
    *D = 0.5;
    return 1;
  }
  double zL = (L - a.L0) / std::max(a.L1 - a.L0, a.eps);
  double zT = (T - a.T0) / std::max(a.T1 - a.T0, a.eps);
  if (a.variant == DC_VAR_TRANSLATION_ONLY) {
    if (!(0.0 <= zL && zL <= 1.0)) return 0;
    *D = zL;
    return 1;
  }
  if (a.variant == DC_VAR_ROTATION_ONLY) {
    if (!(0.0 <= zT && zT <= 1.0)) return 0;
    *D = zT;
    return 1;
  }
  if (!(0.0 <= zL && zL <= 1.0 && 0.0 <= zT && zT <= 1.0)) return 0;
  *D = std::sqrt(zL * zL + zT * zT) / std::sqrt(2.0);  // Eq. 4
  return 1;
}

void even_schedule(int n, int T, int H, const unsigned char* legal, unsigned char* acts) {
  acts[1] = kCompute;
  int age = 0;
  for (int k = 2; k <= T; ++k) {
    const bool want =
        T > 1 && (long long)(k - 1) * n / (T - 1) > (long long)(k - 2) * n / (T - 1);
    if (want && legal_at(legal, H, k, age + 1)) {
      acts[k] = kReuse;
      ++age;
    } else {
      acts[k] = kCompute;
      age = 0;
    }
  }
}

namespace {
// Sum of c_hat_{j,h} over the reuses of a schedule, in step order.
double schedule_cost(const unsigned char* acts, const SceneTables& t) {
  double total = 0.0;
  int j = 1, age = 0;
  for (int k = 2; k <= t.K; ++k) {
    if (acts[k] == kReuse) {
      ++age;
      total = total + t.at_c(j, age);
    } else {
      j = k;
      age = 0;
    }
  }
  return total;
}
int count_reuse(const unsigned char* acts, int T) {
  int n = 0;
  for (int k = 1; k <= T; ++k) n += acts[k] == kReuse;
  return n;
}
}  // namespace

int plan_scene(double L, double Th, const dc_anchor_responses& a, double budget,
               unsigned char* acts, int* n_reuse, double* cost, double* D, SceneTables* tabs) {
  const int T = a.K;
  for (int k = 1; k <= T; ++k) acts[k] = kCompute;
  *n_reuse = 0;
  *cost = 0.0;
  *D = 0.0;
  if (a.variant == DC_VAR_FIXED_INTERVAL) {  // no motion, no budget: a fixed pattern
    even_schedule((int)budget, T, a.H_max, a.legal, acts);
    *n_reuse = count_reuse(acts, T);
    return 1;
  }
  if (!scene_intensity(L, Th, a, D)) return 0;
  scene_tables(a, *D, tabs);
  *n_reuse = plan_suffix(*tabs, a.legal, 1, budget, acts, cost);
  if (a.variant == DC_VAR_FIXED_PLACEMENT) {  // the DP's count, evenly placed
    even_schedule(*n_reuse, T, a.H_max, a.legal, acts);
    *n_reuse = count_reuse(acts, T);
    *cost = schedule_cost(acts, *tabs);
  }
  return 1;
}

void scene_tables(const dc_anchor_responses& a, double D, SceneTables* t) {
  const int K = a.K, H = a.H_max, W = H + 1;
  t->K = K; t->H = H;
  t->c.assign((size_t)K * W, 0.0);
  t->dbar.assign((size_t)K * W, 0.0);
  std::vector<double> Q(W);
  for (int j = 1; j < K; ++j) {
    const size_t row = (size_t)j * W;
    double run = -kInf;
    Q[0] = 0.0;
    for (int h = 1; h <= H; ++h) {
      double q0 = a.q0[row + h], q1 = a.q1[row + h];
      double qt = q0 + D * std::max(q1 - q0, 0.0);  // Eq. 8
      run = std::max(run, qt);                      // Eq. 9 envelope
      Q[h] = run;
    }
    for (int h = 1; h <= H; ++h) t->c[row + h] = Q[h] - Q[h - 1];
    for (int h = 1; h <= H; ++h) {
      double d0 = a.d0[row + h], d1 = a.d1[row + h];
      t->dbar[row + h] = d0 + D * std::max(d1 - d0, 0.0);
    }
  }
}

int plan_suffix(const SceneTables& t, const unsigned char* legal, int k0, double budget,
                unsigned char* acts, double* cost) {
  DPResult r;
  run_dp(t, legal, k0, &r);
  const int W = t.H + 1;
  // Eq. 11: largest n whose best cost is finite and within the budget
  int nstar = 0;
  for (int n = 0; n <= r.nmax; ++n) {
    double m = kInf;
    for (int h = 0; h <= t.H; ++h) m = std::min(m, r.Jfin[(size_t)n * W + h]);
    if (m < kInf && m <= budget) nstar = n;
  }
  int h = -1;
  double best = kInf;
  for (int hh = 0; hh <= t.H; ++hh) {
    double v = r.Jfin[(size_t)nstar * W + hh];
    if (v < best) { best = v; h = hh; }
  }
  int n = nstar;
  for (int k = t.K; k > k0; --k) {
    if (h > 0) {
      acts[k] = kReuse;
      --n; --h;
    } else {
      acts[k] = kCompute;
      h = r.arg[(size_t)k * (r.nmax + 1) + n];
    }
  }
  acts[k0] = kCompute;
  if (cost) *cost = best;
  return nstar;
}

void cost_curve(const SceneTables& t, const unsigned char* legal, std::vector<double>* m) {
  DPResult r;
  run_dp(t, legal, 1, &r);
  const int W = t.H + 1;
  m->assign(r.nmax + 1, kInf);
  for (int n = 0; n <= r.nmax; ++n)
    for (int h = 0; h <= t.H; ++h) (*m)[n] = std::min((*m)[n], r.Jfin[(size_t)n * W + h]);
}

dc_status check_reuse_count(const dc_anchor_responses& a, double budget) {
  if (a.variant != DC_VAR_FIXED_INTERVAL) return DC_OK;
  if (!(budget >= 0.0 && budget <= a.K - 1) || budget != std::floor(budget)) {
    set_error("fixed-interval variant: the budget is the reuse count, an integer in [0, K-1]");
    return DC_ERR_INVALID_ARG;
  }
  return DC_OK;
}

dc_status check_anchors(const dc_anchor_responses* a) {
  if (!a) { set_error("anchors is NULL"); return DC_ERR_INVALID_ARG; }
  if (a->K < 1 || a->K > 100000 || a->H_max < 1 || a->H_max > 4096) {
    set_error("anchors: K must be >= 1 and H_max in [1, 4096]");
    return DC_ERR_INVALID_ARG;
  }
  if (!(a->eps > 0.0) || !std::isfinite(a->eps)) {
    set_error("anchors: eps must be finite and > 0");
    return DC_ERR_INVALID_ARG;
  }
  if (a->variant < DC_VAR_DRIVECACHE || a->variant > DC_VAR_FIXED_INTERVAL) {
    set_error("anchors: variant must be one of DC_VAR_*");
    return DC_ERR_INVALID_ARG;
  }
  if (!a->valid) return DC_OK;
  if (!std::isfinite(a->L0) || !std::isfinite(a->T0) || !std::isfinite(a->L1) ||
      !std::isfinite(a->T1)) {
    set_error("anchors: non-finite anchor statistics");
    return DC_ERR_INVALID_ARG;
  }
  if (!a->q0 || !a->q1 || !a->d0 || !a->d1) {
    set_error("anchors: q0/q1/d0/d1 must be non-NULL when valid");
    return DC_ERR_INVALID_ARG;
  }
  const int W = a->H_max + 1;
  for (int j = 1; j < a->K; ++j)
    for (int h = 1; h <= a->H_max; ++h) {
      size_t i = (size_t)j * W + h;
      const double v[4] = {a->q0[i], a->q1[i], a->d0[i], a->d1[i]};
      for (double x : v)
        if (!std::isfinite(x) || x < 0.0) {
          set_error("anchors: response/drift tables must be finite and >= 0 (j=" +
                    std::to_string(j) + ", h=" + std::to_string(h) + ")");
          return DC_ERR_INVALID_ARG;
        }
    }
  return DC_OK;
}

}  // namespace dc

// ------------------------------------------------------------------ C ABI

namespace {

dc_status check_traj(const dc_trajectory* tr) {
  if (!tr || !tr->poses || tr->n_poses < 1) {
    dc::set_error("trajectory must have n_poses >= 1 and non-NULL poses");
    return DC_ERR_INVALID_ARG;
  }
  for (int i = 0; i < tr->n_poses; ++i) {
    const dc_pose& p = tr->poses[i];
    if (!std::isfinite(p.x) || !std::isfinite(p.y) || !std::isfinite(p.psi)) {
      dc::set_error("trajectory has a non-finite pose at index " + std::to_string(i));
      return DC_ERR_INVALID_ARG;
    }
  }
  return DC_OK;
}

}  // namespace

using namespace dc;

extern "C" {

dc_status dc_motion_stats(const dc_trajectory* traj, double* L, double* Theta) {
  dc_status s = check_traj(traj);
  if (s != DC_OK) return s;
  if (!L || !Theta) { dc::set_error("L/Theta output is NULL"); return DC_ERR_INVALID_ARG; }
  dc::motion_stats(traj->poses, traj->n_poses, L, Theta);
  return DC_OK;
}

dc_status dc_select_anchors(const double* L, const double* Theta, int n, double anchors_out[4],
                            int* valid, int* index_out) {
  if (!L || !Theta || !anchors_out || !valid || n < 1) {
    dc::set_error("dc_select_anchors: NULL pointer or n < 1");
    return DC_ERR_INVALID_ARG;
  }
  for (int i = 0; i < n; ++i)
    if (!std::isfinite(L[i]) || !std::isfinite(Theta[i])) {
      dc::set_error("dc_select_anchors: non-finite statistic");
      return DC_ERR_INVALID_ARG;
    }
  std::vector<double> zL, zT;
  zscores(L, n, &zL);
  zscores(Theta, n, &zT);
  int i0 = 0;
  double best = zL[0] + zT[0];
  for (int i = 1; i < n; ++i) {
    double s = zL[i] + zT[i];
    if (s < best) { best = s; i0 = i; }
  }
  const double L0 = L[i0], T0 = Theta[i0];
  const double med = median_of(std::vector<double>(Theta, Theta + n));
  int i1 = -1;
  double bestp = -kInf;
  for (int i = 0; i < n; ++i) {
    if (Theta[i] > med && L[i] > L0 && Theta[i] > T0) {
      double p = zL[i] * zT[i];
      if (i1 < 0 || p > bestp) { bestp = p; i1 = i; }
    }
  }
  anchors_out[0] = L0;
  anchors_out[1] = T0;
  anchors_out[2] = i1 >= 0 ? L[i1] : 0.0;
  anchors_out[3] = i1 >= 0 ? Theta[i1] : 0.0;
  *valid = i1 >= 0 ? 1 : 0;
  if (index_out) { index_out[0] = i0; index_out[1] = i1; }
  return DC_OK;
}

dc_status dc_plan(const dc_trajectory* traj, const dc_anchor_responses* anc, double budget, int T,
                  dc_schedule* out) {
  dc_status s = check_traj(traj);
  if (s != DC_OK) return s;
  if ((s = dc::check_anchors(anc)) != DC_OK) return s;
  if (!out || !out->action || T != anc->K || out->T != T || std::isnan(budget)) {
    dc::set_error("dc_plan: out/action NULL, T != anchors.K, out->T != T, or NaN budget");
    return DC_ERR_INVALID_ARG;
  }
  if ((s = dc::check_reuse_count(*anc, budget)) != DC_OK) return s;
  double L, Th, D;
  dc::motion_stats(traj->poses, traj->n_poses, &L, &Th);
  out->L = L;
  out->Theta = Th;
  out->action[0] = 0;
  dc::SceneTables t;
  out->supported = dc::plan_scene(L, Th, *anc, budget, out->action, &out->n_reuse, &out->cost,
                                  &D, &t);
  out->D = D;
  return DC_OK;
}

dc_status dc_replan(const dc_anchor_responses* anc, double D, int k_refresh, double remaining,
                    dc_schedule* inout) {
  dc_status s = dc::check_anchors(anc);
  if (s != DC_OK) return s;
  if (!inout || !inout->action || inout->T != anc->K || k_refresh < 1 || k_refresh > anc->K ||
      !(D >= 0.0 && D <= 1.0) || std::isnan(remaining)) {
    dc::set_error("dc_replan: bad schedule, k_refresh outside 1..K, D outside [0,1] or NaN budget");
    return DC_ERR_INVALID_ARG;
  }
  if (anc->variant == DC_VAR_FIXED_PLACEMENT || anc->variant == DC_VAR_FIXED_INTERVAL) {
    // the fixed variants keep their pattern
    int n = 0;
    for (int k = 1; k <= inout->T; ++k) n += inout->action[k] == dc::kReuse;
    inout->n_reuse = n;
    inout->cost = 0.0;
    return DC_OK;
  }
  if (!anc->valid) {
    dc::set_error("dc_replan: anchors are invalid (full inference, nothing to replan)");
    return DC_ERR_INVALID_ARG;
  }
  dc::SceneTables t;
  dc::scene_tables(*anc, D, &t);
  dc::plan_suffix(t, anc->legal, k_refresh, remaining, inout->action, &inout->cost);
  int n = 0;
  for (int k = 1; k <= inout->T; ++k) n += inout->action[k] == dc::kReuse;
  inout->n_reuse = n;
  return DC_OK;
}

dc_status dc_calibrate_budget(const dc_trajectory* clips, int n, const dc_anchor_responses* anc,
                              int target, int T, double* tau, int* reached) {
  dc_status s = dc::check_anchors(anc);
  if (s != DC_OK) return s;
  if (!clips || n < 1 || !tau || T != anc->K || target < 0) {
    dc::set_error("dc_calibrate_budget: NULL clips/tau, n < 1, T != anchors.K or target < 0");
    return DC_ERR_INVALID_ARG;
  }
  for (int i = 0; i < n; ++i)
    if ((s = check_traj(&clips[i])) != DC_OK) return s;
  if (anc->variant == DC_VAR_FIXED_INTERVAL) {
    // the reuse count is the budget itself
    if (target > T - 1) {
      dc::set_error("dc_calibrate_budget: fixed-interval target must be in [0, T-1]");
      return DC_ERR_INVALID_ARG;
    }
    std::vector<unsigned char> acts((size_t)T + 1, 0);
    dc::even_schedule(target, T, anc->H_max, anc->legal, acts.data());
    int got = 0;
    for (int k = 1; k <= T; ++k) got += acts[k] == dc::kReuse;
    *tau = (double)target;
    if (reached) *reached = got >= target ? 1 : 0;
    return DC_OK;
  }
  std::vector<std::vector<double>> curves(n);
  for (int i = 0; i < n; ++i) {
    double L, Th, D;
    dc::motion_stats(clips[i].poses, clips[i].n_poses, &L, &Th);
    if (!dc::scene_intensity(L, Th, *anc, &D)) continue;  // counts as zero reuses
    dc::SceneTables t;
    dc::scene_tables(*anc, D, &t);
    dc::cost_curve(t, anc->legal, &curves[i]);
  }
  budget_from_curves(curves, target, tau, reached);
  return DC_OK;
}

dc_status dc_cost_curve(const dc_trajectory* clip, const dc_anchor_responses* anc, int T,
                        double* m_out, int* supported) {
  dc_status s = dc::check_anchors(anc);
  if (s != DC_OK) return s;
  if (!clip || !m_out || T != anc->K) {
    dc::set_error("dc_cost_curve: NULL clip/m_out or T != anchors.K");
    return DC_ERR_INVALID_ARG;
  }
  if (anc->variant == DC_VAR_FIXED_INTERVAL) {
    dc::set_error("dc_cost_curve: the fixed-interval variant has no cost curve (its budget is the reuse count)");
    return DC_ERR_INVALID_ARG;
  }
  if ((s = check_traj(clip)) != DC_OK) return s;
  for (int m = 0; m < T; ++m) m_out[m] = kInf;
  double L, Th, D;
  dc::motion_stats(clip->poses, clip->n_poses, &L, &Th);
  const int sup = dc::scene_intensity(L, Th, *anc, &D);
  if (supported) *supported = sup;
  if (!sup) return DC_OK;
  dc::SceneTables t;
  dc::scene_tables(*anc, D, &t);
  std::vector<double> c;
  dc::cost_curve(t, anc->legal, &c);
  for (size_t m = 0; m < c.size() && m < (size_t)T; ++m) m_out[m] = c[m];
  return DC_OK;
}

dc_status dc_budget_from_curves(const double* curves, int n, int T, int target, double* tau,
                                int* reached) {
  if (!curves || n < 1 || T < 1 || target < 0 || !tau) {
    dc::set_error("dc_budget_from_curves: NULL curves/tau, n < 1, T < 1 or target < 0");
    return DC_ERR_INVALID_ARG;
  }
  std::vector<std::vector<double>> c(n);
  for (int i = 0; i < n; ++i) {
    c[i].assign(curves + (size_t)i * T, curves + (size_t)(i + 1) * T);
    for (double v : c[i])
      if (std::isnan(v) || v < 0.0) {
        dc::set_error("dc_budget_from_curves: curve entries must be >= 0 or +infinity");
        return DC_ERR_INVALID_ARG;
      }
  }
  budget_from_curves(c, target, tau, reached);
  return DC_OK;
}

dc_status dc_legal_mask(int K, int H_max, int expert_boundary, int segment_len,
                        int no_cache_until, unsigned char* out) {
  if (!out || K < 1 || K > 100000 || H_max < 1 || H_max > 4096 || expert_boundary < 0 ||
      segment_len < 0 || no_cache_until < 0) {
    dc::set_error("dc_legal_mask: NULL out, K or H_max out of range, or a negative rule");
    return DC_ERR_INVALID_ARG;
  }
  const int W = H_max + 1;
  for (int k = 0; k <= K; ++k)
    for (int h = 0; h <= H_max; ++h) {
      const int j = k - h;  // refresh step of the run this reuse extends
      bool ok = k >= 2 && h >= 1 && j >= 1;
      if (ok && expert_boundary > 0) ok = (j <= expert_boundary) == (k <= expert_boundary);
      if (ok && segment_len > 0) ok = (j - 1) / segment_len == (k - 1) / segment_len;
      if (ok && no_cache_until > 0) ok = k > no_cache_until;
      out[(size_t)k * W + h] = ok ? 1 : 0;
    }
  return DC_OK;
}

const char* dc_status_string(dc_status s) {
  switch (s) {
    case DC_OK: return "ok";
    case DC_ERR_INVALID_ARG: return "invalid argument";
    case DC_ERR_NOMEM: return "out of memory";
    case DC_ERR_CUDA: return "CUDA error";
    case DC_ERR_DEVICE_TIMEOUT: return "device wait timed out";
    case DC_ERR_NONFINITE: return "non-finite value";
    case DC_ERR_UNSUPPORTED: return "unsupported shape or dtype";
  }
  return "unknown status";
}

const char* dc_last_error(void) { return dc::last_error_cstr(); }

}  // extern "C"
