// Construction of the compressed cache (Alg. 1), layer by layer, on the
// caller's stream.  Every step is a kernel of construct_kernels.cuh; the host
// only validates, sizes the scratch buffers and sequences the launches.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <string>
#include <vector>

#include "construct_kernels.cuh"
#include "lloyd_pt.cuh"
#include "lloyd_tc.cuh"
#include "internal.h"

namespace reskv {

reskv_status alloc_handle(const reskv_config& cfg, cudaStream_t stream, reskv_cache** out);
void release_handle(reskv_cache* c);
reskv_status finalize_ragged_layout(reskv_cache* c);

namespace {

using namespace build;

reskv_status fail(reskv_status st, const std::string& msg) {
  set_error(msg);
  return st;
}

struct Scratch {
  std::vector<void*> ptrs;
  ~Scratch() {
    for (void* p : ptrs) cudaFree(p);
  }
  template <typename T>
  bool get(T** p, size_t count) {
    *p = nullptr;
    if (count == 0) count = 1;
    if (device_alloc(reinterpret_cast<void**>(p), count * sizeof(T)) != cudaSuccess) {
      cudaGetLastError();
      *p = nullptr;
      return false;
    }
    ptrs.push_back(*p);
    return true;
  }
};

#define RESKV_LAUNCH_CHECK(what)                                                      \
  do {                                                                               \
    cudaError_t e_ = cudaGetLastError();                                             \
    if (e_ != cudaSuccess)                                                           \
      return fail(RESKV_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e_)); \
  } while (0)

template <typename K>
cudaError_t set_smem(K kernel, size_t bytes) {
  return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(bytes));
}

int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Device time per construction stage: an event is recorded on the stream at
// every stage boundary of a layer; at the end of the layer the intervals are
// added to their stages (events are reused from layer to layer).
class StageTimer {
 public:
  explicit StageTimer(cudaStream_t s) : stream_(s) {}
  ~StageTimer() {
    for (cudaEvent_t e : pool_) cudaEventDestroy(e);
  }
  // the interval that starts now belongs to `stage` (-1: not timed)
  bool mark(int stage) {
    if (n_ == pool_.size()) {
      cudaEvent_t e;
      if (cudaEventCreate(&e) != cudaSuccess) return false;
      pool_.push_back(e);
    }
    stage_.resize(n_ + 1);
    stage_[n_] = stage;
    return cudaEventRecord(pool_[n_++], stream_) == cudaSuccess;
  }
  // close the layer: wait for its last event, accumulate, start over
  bool flush(float* ms) {
    if (n_ == 0) return true;
    if (cudaEventSynchronize(pool_[n_ - 1]) != cudaSuccess) return false;
    for (size_t i = 0; i + 1 < n_; ++i) {
      float t = 0.f;
      if (cudaEventElapsedTime(&t, pool_[i], pool_[i + 1]) != cudaSuccess) return false;
      if (stage_[i] >= 0) ms[stage_[i]] += t;
    }
    n_ = 0;
    return true;
  }

 private:
  cudaStream_t stream_;
  std::vector<cudaEvent_t> pool_;
  std::vector<int> stage_;
  size_t n_ = 0;
};

enum { kStScore = 0, kStRank, kStValTargets, kStLloyd, kStValLoss, kStPack };

}  // namespace

reskv_status build_all_layers(reskv_cache** out, const reskv_config& cfg,
                              const int32_t* override_host, const void* const* Kl,
                              const void* const* Vl, const void* const* Ql, cudaStream_t stream) {
  // ---------------- validation ----------------
  const int64_t s = cfg.seq_len;
  const int b = cfg.budget;
  if (cfg.recent_window < 0) return fail(RESKV_ERR_INVALID_ARG, "recent_window must be >= 0");
  const int P = int(std::min<int64_t>(cfg.recent_window, s));
  const int UL = cfg.batch * cfg.n_kv_heads;
  const int G = cfg.group;
  const int64_t U_all = int64_t(cfg.n_layers) * UL;
  if (cfg.budget_mode != RESKV_BUDGET_UNIFORM && cfg.budget_mode != RESKV_BUDGET_ADAKV)
    return fail(RESKV_ERR_INVALID_ARG, "unknown budget_mode");
  // AdaKV allocation across the KV heads of each (layer, batch element); with
  // b >= s nothing is evicted and the layout keeps one budget
  const bool adakv = cfg.budget_mode == RESKV_BUDGET_ADAKV && int64_t(b) < s;
  if (cfg.budget_mode == RESKV_BUDGET_ADAKV) {
    if (cfg.unit_budgets)
      return fail(RESKV_ERR_INVALID_ARG, "budget_mode ADAKV allocates the budgets: unit_budgets must be NULL");
    if (!(cfg.adakv_safeguard >= 0.f && cfg.adakv_safeguard <= 1.f))
      return fail(RESKV_ERR_INVALID_ARG, "adakv_safeguard must be in [0, 1]");
  }
  const bool per_unit = cfg.unit_budgets != nullptr || adakv;
  const int n_free_head = b - P;                       // selectable slots per head (AdaKV)
  const int ada_f = adakv ? std::min(n_free_head, std::max(0, int(std::floor(
                                double(cfg.adakv_safeguard) * double(n_free_head))))) : 0;
  if (adakv && double(cfg.n_kv_heads) * double(s) >= double(int64_t(1) << 31))
    return fail(RESKV_ERR_UNSUPPORTED, "AdaKV: n_kv_heads * seq_len must be < 2^31");
  if (adakv && n_free_head > kTopMax)
    return fail(RESKV_ERR_UNSUPPORTED, "AdaKV: budget - recent_window must be <= 8192");
  // the largest budget a unit can get (sizes the scratch), and whether any unit evicts
  int64_t b_hi = b;
  bool any_evict = int64_t(b) < s;
  if (cfg.unit_budgets) {
    b_hi = 0;
    any_evict = false;
    for (int64_t u = 0; u < U_all; ++u) {
      const int64_t bu = cfg.unit_budgets[u];
      if (std::min(bu, s) < P)
        return fail(RESKV_ERR_INVALID_ARG, "unit_budgets must be >= min(recent_window, seq_len)");
      b_hi = std::max(b_hi, bu);
      any_evict |= bu < s;
    }
  } else if (int64_t(std::min<int64_t>(b, s)) < P) {
    return fail(RESKV_ERR_INVALID_ARG, "budget must be >= min(recent_window, seq_len)");
  }
  if (adakv)   // |P| + f + every shared slot, within s and the ranking limit
    b_hi = std::min<int64_t>(std::min<int64_t>(s, int64_t(P) + kTopMax),
                             int64_t(P) + ada_f + int64_t(cfg.n_kv_heads) * (n_free_head - ada_f));
  const int n_top = int(std::min<int64_t>(b_hi, s)) - P;   // ranking width per unit
  if (n_top > kTopMax)
    return fail(RESKV_ERR_UNSUPPORTED, "budget - recent_window must be <= 8192");
  const bool all_main = !any_evict;
  const bool proxy = override_host == nullptr && !all_main;
  if (cfg.score_mode != RESKV_SCORE_OBS_POOL && cfg.score_mode != RESKV_SCORE_KEYNORM)
    return fail(RESKV_ERR_INVALID_ARG, "unknown score_mode");
  if (cfg.pool_kernel < 1 || cfg.pool_kernel % 2 == 0)
    return fail(RESKV_ERR_INVALID_ARG, "pool_kernel must be a positive odd number");
  const bool need_q = cfg.score_mode == RESKV_SCORE_OBS_POOL || proxy;
  if (need_q) {
    if (!Ql) return fail(RESKV_ERR_INVALID_ARG, "observation queries are required");
    for (int l = 0; l < cfg.n_layers; ++l)
      if (!Ql[l]) return fail(RESKV_ERR_INVALID_ARG, "NULL observation-query layer");
    if (cfg.score_mode == RESKV_SCORE_OBS_POOL && (cfg.n_fit < 1 || cfg.n_fit > cfg.n_obs))
      return fail(RESKV_ERR_INVALID_ARG, "need 1 <= n_fit <= n_obs");
    if (proxy) {
      const int used_fit = cfg.score_mode == RESKV_SCORE_OBS_POOL ? cfg.n_fit : 0;
      if (cfg.n_val < 1 || used_fit + cfg.n_val > cfg.n_obs)
        return fail(RESKV_ERR_INVALID_ARG, "need n_val >= 1 and n_fit + n_val <= n_obs");
    }
  }
  for (int l = 0; l < cfg.n_layers; ++l)
    if (!Kl[l] || !Vl[l]) return fail(RESKV_ERR_INVALID_ARG, "NULL K or V layer");
  if (cfg.lloyd_iters < 1 || cfg.lloyd_iters > 64)
    return fail(RESKV_ERR_INVALID_ARG, "lloyd_iters must be in [1, 64]");
  if (cfg.n_grid < 0 || cfg.n_grid > RESKV_MAX_GRID)
    return fail(RESKV_ERR_INVALID_ARG, "n_grid must be in [0, 8]");
  if (!(cfg.delta >= 0.f && cfg.delta < 1.f) || !std::isfinite(cfg.beta))
    return fail(RESKV_ERR_INVALID_ARG, "delta must be in [0, 1) and beta finite");

  // candidate budgets r = floor(ratio * b) > 0, distinct, ascending (App. B).
  // One budget: the columns are those r.  Per-unit budgets: the columns are
  // the distinct positive ratios, ascending; unit u's r in a column is
  // floor(ratio * b_u), dropped (0) when zero, equal to the previous column's,
  // or leaving less than |P| main slots (unit_cands).
  std::vector<int32_t> cands;          // one budget: r of every column
  std::vector<float> col_ratio;        // per-unit budgets: ratio of every column
  std::vector<int32_t> col_rmax;       // per column: the largest r any unit can have
  for (int i = 0; i < cfg.n_grid; ++i)
    if (!(cfg.grid_ratios[i] >= 0.f && cfg.grid_ratios[i] <= 1.f))
      return fail(RESKV_ERR_INVALID_ARG, "grid ratios must be in [0, 1]");
  if (proxy && !per_unit) {
    for (int i = 0; i < cfg.n_grid; ++i) {
      const int r = int(std::floor(double(cfg.grid_ratios[i]) * double(b)));
      if (r > 0 && b - r >= P && std::find(cands.begin(), cands.end(), r) == cands.end())
        cands.push_back(r);
    }
    std::sort(cands.begin(), cands.end());
    col_rmax = cands;
  } else if (proxy) {
    for (int i = 0; i < cfg.n_grid; ++i)
      if (cfg.grid_ratios[i] > 0.f &&
          std::find(col_ratio.begin(), col_ratio.end(), cfg.grid_ratios[i]) == col_ratio.end())
        col_ratio.push_back(cfg.grid_ratios[i]);
    std::sort(col_ratio.begin(), col_ratio.end());
    for (float ratio : col_ratio)
      col_rmax.push_back(int(std::floor(double(ratio) * double(b_hi))));
  }
  // r of every candidate column for the units of one layer ([ncol, UL], column 0 = 0)
  auto unit_candidates = [&](const int32_t* bl, std::vector<int32_t>& out) {
    const int nc = 1 + int(col_rmax.size());
    out.assign(size_t(nc) * UL, 0);
    for (int i = 0; i < UL; ++i) {
      const int64_t bu = bl ? bl[i] : b;
      int prev = 0;
      for (int c = 1; c < nc; ++c) {
        int r = cands.empty() ? int(std::floor(double(col_ratio[c - 1]) * double(bu))) : cands[c - 1];
        if (r <= 0 || r == prev || bu - r < P || bu >= s) r = 0;
        else prev = r;
        out[size_t(c) * UL + i] = r;
      }
    }
  };
  std::vector<int32_t> ovr;
  int rmax = 0;
  if (override_host) {
    ovr.assign(override_host, override_host + U_all);
    for (int64_t u = 0; u < U_all; ++u) {
      const int r = ovr[u];
      const int64_t bu = cfg.unit_budgets ? cfg.unit_budgets[u] : b;
      if (r < 0 || r >= bu) return fail(RESKV_ERR_INVALID_ARG, "residual_override out of [0, budget)");
      if (r > 0 && !adakv && (bu >= s || bu - r < P))
        return fail(RESKV_ERR_INVALID_ARG,
                    "residual_override needs budget < seq_len and budget - r >= recent_window");
      rmax = std::max(rmax, r);
    }
  }
  for (int32_t r : col_rmax) rmax = std::max(rmax, r);
  if (rmax > kMaxR) return fail(RESKV_ERR_UNSUPPORTED, "residual entries per unit must be <= 8192");

  // ---------------- handle and scratch ----------------
  reskv_cache* c = nullptr;
  reskv_status st;
  std::vector<int32_t> budgets_host;   // per-unit budgets (every layer)
  if (adakv) {
    // provisional layout with b per unit: the allocation keeps every
    // (layer, batch element)'s total, so only offsets inside it move
    budgets_host.assign(size_t(U_all), b);
    reskv_config lay = cfg;
    lay.unit_budgets = budgets_host.data();
    st = alloc_handle(lay, stream, &c);
  } else {
    if (cfg.unit_budgets) budgets_host.assign(cfg.unit_budgets, cfg.unit_budgets + U_all);
    st = alloc_handle(cfg, stream, &c);
  }
  if (st != RESKV_OK) return st;
  c->candidates = per_unit ? std::vector<int32_t>() : cands;
  c->n_candidates = int32_t(col_rmax.size());
  c->ranked_width = std::max(n_top, 0);
  if (proxy) c->unit_cands.assign(size_t(U_all) * col_rmax.size(), 0);
  const int ncol = 1 + int(col_rmax.size());         // run 0 = pure-main cache
  const int ntiles = int(cdiv(s, kTile));
  const int n_fit_rows = cfg.score_mode == RESKV_SCORE_OBS_POOL ? G * cfg.n_fit : 0;
  const int n_val_rows = proxy ? G * cfg.n_val : 0;
  const int nchunks = int(cdiv(s, int64_t(kTile) * kValChunkTiles));
  // entry storage: one slice per run with r > 0
  std::vector<int32_t> run_off(std::max(ncol, 2), 0);
  int64_t ent_stride = 0;
  if (proxy) {
    for (int i = 0; i < int(col_rmax.size()); ++i) {
      run_off[1 + i] = int32_t(ent_stride);
      ent_stride += col_rmax[i];
    }
  } else {
    ent_stride = rmax;
  }

  Scratch S;
  double* scores = nullptr;
  float* A = nullptr;
  float2* tstats = nullptr;
  float2* rstats = nullptr;
  int32_t *top = nullptr, *rank_pos = nullptr, *assign = nullptr, *hist = nullptr;
  int32_t *ccount = nullptr, *cbase = nullptr, *members = nullptr, *ecount = nullptr;
  int32_t *r_runs = nullptr, *r_final = nullptr, *chosen = nullptr, *run_off_d = nullptr;
  int32_t* budgets_d = nullptr;        // [U_all] per-unit budgets (per_unit only)
  float *centersT = nullptr, *cnorm = nullptr, *vpart = nullptr, *oS = nullptr;
  __nv_bfloat16* cplanes = nullptr;
  double* centers64 = nullptr;
  long long* msum = nullptr;
  uint32_t* mflag = nullptr;
  float* knorm2 = nullptr;
  int4* amb = nullptr;
  int* amb_count = nullptr;
  float* centers32 = nullptr;
  // the previous Lloyd iteration's assignment and member lists
  int32_t *assign2 = nullptr, *members2 = nullptr, *cbase2 = nullptr, *ccount2 = nullptr;
  uint32_t* moved = nullptr;
  __nv_bfloat16 *kbar = nullptr, *vbar = nullptr;
  double *rowerr = nullptr, *losses = nullptr;
  const size_t US = size_t(UL) * size_t(s);
  const int nruns = proxy ? ncol : 2;
  bool ok = S.get(&scores, US) && S.get(&top, size_t(UL) * std::max(n_top, 1)) &&
            S.get(&rank_pos, US) && S.get(&r_runs, size_t(nruns) * UL) &&
            S.get(&r_final, UL) && S.get(&chosen, UL) && S.get(&run_off_d, run_off.size()) &&
            (!per_unit || S.get(&budgets_d, size_t(U_all)));
  if (ok && n_fit_rows > 0)
    ok = S.get(&A, US) && S.get(&tstats, size_t(UL) * n_fit_rows * ntiles) &&
         S.get(&rstats, size_t(UL) * n_fit_rows);
  if (ok && rmax > 0)
    ok = S.get(&assign, US) && S.get(&hist, size_t(UL) * ntiles * rmax) &&
         S.get(&ccount, size_t(UL) * rmax) && S.get(&cbase, size_t(UL) * rmax) &&
         S.get(&members, US) && S.get(&centersT, size_t(UL) * kHeadDim * rmax) &&
         S.get(&centers64, size_t(UL) * kHeadDim * rmax) &&
         S.get(&cplanes, size_t(UL) * 2 * rmax * kHeadDim) &&
         S.get(&cnorm, size_t(UL) * rmax) && S.get(&kbar, size_t(UL) * ent_stride * kHeadDim) &&
         S.get(&vbar, size_t(UL) * ent_stride * kHeadDim) &&
         S.get(&ecount, size_t(UL) * ent_stride) &&
         S.get(&msum, size_t(UL) * rmax * 2 * kHeadDim) && S.get(&mflag, size_t(UL) * rmax) &&
         S.get(&knorm2, US) && S.get(&amb, US) && S.get(&amb_count, 1) &&
         S.get(&centers32, size_t(UL) * rmax * kHeadDim) && S.get(&assign2, US) &&
         S.get(&members2, US) && S.get(&cbase2, size_t(UL) * rmax) && S.get(&ccount2, size_t(UL) * rmax) &&
         S.get(&moved, (US + 31) / 32);
  // the member sums start at zero; each pass's k_lloyd_finish clears what it
  // read.  Assignments start at -1 (no centre) and per-tile counts at 0, so
  // that a tile a failed assignment never reached holds no index and no count
  if (ok && rmax > 0)
    ok = cudaMemsetAsync(assign, 0xff, US * sizeof(int32_t), stream) == cudaSuccess &&
         cudaMemsetAsync(assign2, 0xff, US * sizeof(int32_t), stream) == cudaSuccess &&
         cudaMemsetAsync(hist, 0, size_t(UL) * ntiles * rmax * sizeof(int32_t), stream) == cudaSuccess;
  if (ok && rmax > 0)
    ok = cudaMemsetAsync(msum, 0, size_t(UL) * rmax * 2 * kHeadDim * sizeof(long long), stream) ==
             cudaSuccess &&
         cudaMemsetAsync(mflag, 0, size_t(UL) * rmax * sizeof(uint32_t), stream) == cudaSuccess;
  if (ok && proxy)
    ok = S.get(&vpart, size_t(UL) * n_val_rows * nchunks * kValRec) &&
         S.get(&oS, size_t(UL) * n_val_rows * kHeadDim) &&
         S.get(&rowerr, size_t(UL) * n_val_rows) && S.get(&losses, size_t(UL) * ncol);
  if (ok && cfg.keep_debug) {
    const size_t U = size_t(c->n_units);
    cudaError_t e = device_alloc(reinterpret_cast<void**>(&c->dbg_scores), U * size_t(s) * 8);
    if (e == cudaSuccess)
      e = device_alloc(reinterpret_cast<void**>(&c->dbg_ranked), U * std::max(n_top, 1) * 4);
    if (e == cudaSuccess) e = device_alloc(reinterpret_cast<void**>(&c->dbg_losses), U * ncol * 8);
    if (e == cudaSuccess) e = cudaMemsetAsync(c->dbg_losses, 0, U * ncol * 8, stream);
    ok = e == cudaSuccess;
    c->dbg_n_top = n_top;
  }
  if (!ok) {
    cudaGetLastError();
    release_handle(c);
    return fail(RESKV_ERR_OOM, "construction scratch allocation failed");
  }

  auto cleanup_fail = [&](reskv_status e) {
    release_handle(c);
    return e;
  };

  // per-run r arrays [nruns, UL] (proxy: per layer from the units' budgets;
  // override: filled per layer)
  std::vector<int32_t> hr;
  if (proxy) unit_candidates(nullptr, hr);
  if (cudaMemcpyAsync(run_off_d, run_off.data(), run_off.size() * 4, cudaMemcpyHostToDevice,
                      stream) != cudaSuccess ||
      (cfg.unit_budgets && cudaMemcpyAsync(budgets_d, budgets_host.data(), size_t(U_all) * 4,
                                           cudaMemcpyHostToDevice, stream) != cudaSuccess) ||
      cudaStreamSynchronize(stream) != cudaSuccess)
    return cleanup_fail(fail(RESKV_ERR_CUDA, "copying run tables"));

  // kernel attributes
  const size_t sm_obs1 = size_t(kTile) * kAsgRowBytes;               // the key tile
  const size_t sm_obs2 = sm_obs1 + size_t(kThreads / 32) * kTile * 4;  // + per-warp sums
  const size_t sm_top = size_t(kTopMax) * 12 + (256 + 32 + 4) * 4;
  const size_t sm_assign = lloyd_tc_smem(rmax);
  if (set_smem(k_obs_pass1, sm_obs1) != cudaSuccess || set_smem(k_obs_pass2, sm_obs2) != cudaSuccess ||
      set_smem(k_topk, sm_top) != cudaSuccess || set_smem(k_lloyd_assign_tc, sm_assign) != cudaSuccess ||
      set_smem(k_lloyd_assign_pt, kPtSmemMax) != cudaSuccess ||
      set_smem(k_val_loss, kValSmem) != cudaSuccess ||
      set_smem(k_val_full, kValSmem) != cudaSuccess)
    return cleanup_fail(fail(RESKV_ERR_CUDA, "setting kernel shared-memory limits"));

  const double one_minus_delta = 1.0 - double(cfg.delta);
  StageTimer timer(stream);
  bool timing_ok = true;

  int test_fault = take_test_wait_fault() ? 1 : 0;   // test hook (reskv_test_inject)
  for (int l = 0; l < cfg.n_layers; ++l) {
    const __nv_bfloat16* K = static_cast<const __nv_bfloat16*>(Kl[l]);
    const __nv_bfloat16* V = static_cast<const __nv_bfloat16*>(Vl[l]);
    const __nv_bfloat16* Q = Ql ? static_cast<const __nv_bfloat16*>(Ql[l]) : nullptr;

    // ---- token scores ----
    timing_ok &= timer.mark(kStScore);
    if (cfg.score_mode == RESKV_SCORE_OBS_POOL) {
      ObsArgs oa{K, Q, s, G, cfg.n_obs, n_fit_rows, cfg.n_fit, ntiles, tstats, rstats, A};
      k_obs_pass1<<<dim3(ntiles, UL), kThreads, sm_obs1, stream>>>(oa);
      k_obs_rowstats<<<unsigned(cdiv(int64_t(UL) * n_fit_rows, 256)), 256, 0, stream>>>(oa, UL);
      k_obs_pass2<<<dim3(ntiles, UL), kThreads, sm_obs2, stream>>>(oa);
      k_pool<<<unsigned(cdiv(int64_t(US), 256)), 256, 0, stream>>>(A, scores, s, UL, cfg.pool_kernel);
    } else {
      k_score_keynorm<<<unsigned(cdiv(int64_t(US), 8)), 256, 0, stream>>>(K, scores, int64_t(US));
    }
    RESKV_LAUNCH_CHECK("scoring");
    timing_ok &= timer.mark(kStRank);
    int32_t* bl_d = per_unit ? budgets_d + size_t(l) * UL : nullptr;   // this layer's budgets
    const int32_t* bl_h = per_unit ? budgets_host.data() + size_t(l) * UL : nullptr;
    if (adakv) {
      // AdaKV: mark every head's safeguard (its top f), split the shared slots
      TopArgs tf{scores, s, P, ada_f, top, rank_pos, c->status, nullptr};
      k_topk<<<UL, kTopThreads, sm_top, stream>>>(tf);
      AdaArgs aa{scores, rank_pos, s, P, cfg.n_kv_heads, ada_f, P + ada_f,
                 int64_t(cfg.n_kv_heads) * (n_free_head - ada_f), bl_d};
      k_adakv<<<cfg.batch, kTopThreads, 0, stream>>>(aa);
      RESKV_LAUNCH_CHECK("AdaKV budgets");
      if (cudaMemcpyAsync(budgets_host.data() + size_t(l) * UL, bl_d, size_t(UL) * 4,
                          cudaMemcpyDeviceToHost, stream) != cudaSuccess ||
          cudaStreamSynchronize(stream) != cudaSuccess)
        return cleanup_fail(fail(RESKV_ERR_CUDA, "reading the AdaKV budgets"));
      // the layer's units keep their region; place them inside it
      const int64_t u0 = int64_t(l) * UL;
      for (int i = 0; i < UL; ++i) {
        const int64_t bu = bl_h[i];
        if (bu < P + ada_f || bu > b_hi)
          return cleanup_fail(fail(bu > b_hi ? RESKV_ERR_UNSUPPORTED : RESKV_ERR_CUDA,
                                   "AdaKV budget " + std::to_string(bu) + " of unit " +
                                       std::to_string(u0 + i) +
                                       " is outside what construction covers"));
        if (!ovr.empty() && ovr[size_t(u0 + i)] > 0 &&
            (bu >= s || bu - ovr[size_t(u0 + i)] < P))
          return cleanup_fail(fail(RESKV_ERR_INVALID_ARG,
                                   "residual_override of unit " + std::to_string(u0 + i) +
                                       " leaves less than recent_window main slots of its AdaKV budget"));
        c->h_offsets[size_t(u0 + i) + 1] = c->h_offsets[size_t(u0 + i)] + int32_t(bu) + c->append_capacity;
      }
      if (cudaMemcpyAsync(c->offsets + u0, c->h_offsets.data() + u0, size_t(UL + 1) * 4,
                          cudaMemcpyHostToDevice, stream) != cudaSuccess)
        return cleanup_fail(fail(RESKV_ERR_CUDA, "copying unit offsets"));
    }
    if (per_unit && n_top > 0 &&
        cudaMemsetAsync(top, 0xff, size_t(UL) * n_top * 4, stream) != cudaSuccess)
      return cleanup_fail(fail(RESKV_ERR_CUDA, "clearing the ranking"));
    TopArgs ta{scores, s, P, n_top, top, rank_pos, c->status, bl_d};
    k_topk<<<UL, kTopThreads, sm_top, stream>>>(ta);
    RESKV_LAUNCH_CHECK("ranking");
    // candidate r per unit of this layer
    int grid_r = rmax;
    if (proxy) {
      if (per_unit || l == 0) unit_candidates(bl_h, hr);
      for (int c2 = 1; c2 < ncol; ++c2)
        for (int i = 0; i < UL; ++i)
          c->unit_cands[(size_t(l) * UL + i) * (ncol - 1) + (c2 - 1)] = hr[size_t(c2) * UL + i];
      if ((per_unit || l == 0) &&
          cudaMemcpyAsync(r_runs, hr.data(), hr.size() * 4, cudaMemcpyHostToDevice, stream) != cudaSuccess)
        return cleanup_fail(fail(RESKV_ERR_CUDA, "copying candidate budgets"));
      grid_r = 0;
      for (int32_t r : hr) grid_r = std::max<int>(grid_r, r);
    }

    LloydArgs la{K, V, s, P, n_top, b, ntiles, rmax, top, rank_pos, nullptr, centersT, cnorm,
                 centers64, assign, hist, ccount, cbase, members, kbar, vbar, ecount,
                 ent_stride, 0, c->status, bl_d, cplanes, msum, mflag, knorm2, amb, amb_count, centers32,
                 assign2, members2, cbase2, ccount2, moved, 0};
    if (rmax > 0)
      k_key_norm2<<<unsigned(cdiv(int64_t(US), 8)), 256, 0, stream>>>(K, knorm2, int64_t(US));
    // the persistent assignment loads key tiles by TMA (a 16-byte aligned
    // base and at least one whole tile of rows); otherwise the streaming form
    CUtensorMap tmK;
    const bool pt_keys = rmax > 0 && US >= size_t(kTile) && encode_key_tiles(&tmK, K, uint64_t(US));
    auto lloyd_run = [&](const int32_t* r_unit, int ent_off, int r_hi) -> reskv_status {
      la.r_unit = r_unit;
      la.ent_off = ent_off;
      timing_ok &= timer.mark(kStLloyd);
      const unsigned gr = unsigned(std::max(r_hi, 1));
      const unsigned pt_grid = unsigned(std::min<int64_t>(c->num_sms, int64_t(UL) * ntiles));
      k_lloyd_init<<<dim3(gr, UL), kHeadDim, 0, stream>>>(la);
      // key sums in full for the first kDeltaFrom iterations, then updated
      // from the previous iteration's by the tokens that moved (a third of
      // the tokens move in the second iteration, about a tenth later)
      constexpr int kDeltaFrom = 2;
      int32_t* const abuf[2][4] = {{assign, members, cbase, ccount}, {assign2, members2, cbase2, ccount2}};
      for (int it = 0; it < cfg.lloyd_iters; ++it) {
        int32_t* const* cur = abuf[it & 1];
        int32_t* const* prv = abuf[(it + 1) & 1];
        la.assign = cur[0];
        la.members = cur[1];
        la.cbase = cur[2];
        la.ccount = cur[3];
        la.assign_prev = prv[0];
        la.members_prev = prv[1];
        la.cbase_prev = prv[2];
        la.ccount_prev = prv[3];
        if (pt_keys && r_hi <= kPtRmax) {   // the centres fit in shared memory: persistent form
          if (cudaMemsetAsync(amb_count, 0, sizeof(int), stream) != cudaSuccess)
            return fail(RESKV_ERR_CUDA, "clearing the ambiguous-token count");
          const int rp = (r_hi + 15) & ~15;
          la.test_fault = test_fault;     // an injected fault is taken by the first launch only
          test_fault = 0;
          k_lloyd_assign_pt<<<pt_grid, kPtThreads, lloyd_pt_smem(rp), stream>>>(la, UL, rp,
                                                                                 lloyd_pt_key_bufs(rp), tmK);
          la.test_fault = 0;
          k_lloyd_resolve<<<unsigned(4 * c->num_sms), kResWarps * 32, 0, stream>>>(la);
        } else {
          k_lloyd_assign_tc<<<dim3(ntiles, UL), kTcThreads, sm_assign, stream>>>(la);
        }
        k_lloyd_scan<<<dim3(UL, unsigned(cdiv(int64_t(gr), kScanCentres))), kScanCentres * kScanSegs, 0, stream>>>(la);
        k_lloyd_bases<<<UL, 256, 0, stream>>>(la);
        k_lloyd_scatter<<<dim3(ntiles, UL), kTile, 0, stream>>>(la);
        const int last = it == cfg.lloyd_iters - 1;
        const dim3 ga(unsigned(cdiv(s, int64_t(kAccRows))), UL);
        if (it >= kDeltaFrom) {
          k_lloyd_moved<<<unsigned(cdiv(int64_t(US), 256)), 256, 0, stream>>>(la, int64_t(US));
          k_lloyd_accum<false, 1><<<ga, kThreads, 0, stream>>>(la);
          k_lloyd_accum<false, -1><<<ga, kThreads, 0, stream>>>(la);
        } else {
          k_lloyd_accum<false, 0><<<ga, kThreads, 0, stream>>>(la);
        }
        if (last) k_lloyd_accum<true, 0><<<ga, kThreads, 0, stream>>>(la);
        const int keep = !last && it + 1 >= kDeltaFrom;     // the next pass updates these sums
        k_lloyd_finish<<<dim3(unsigned(cdiv(int64_t(gr), kFinWarps)), UL), kFinWarps * 32, 0, stream>>>(
            la, last, keep);
      }
      RESKV_LAUNCH_CHECK("residual entries");
      return RESKV_OK;
    };

    if (proxy) {
      // ---- validation targets, candidates, choice of r ----
      timing_ok &= timer.mark(kStValTargets);
      ValArgs va{K, V, Q, s, G, cfg.n_obs, cfg.n_val, n_val_rows, nchunks, vpart, oS};
      k_val_full<<<dim3(nchunks, unsigned(cdiv(n_val_rows, kRowBlk)), UL), kThreads, kValSmem, stream>>>(va);
      k_val_combine<<<dim3(n_val_rows, UL), kHeadDim, 0, stream>>>(va);
      RESKV_LAUNCH_CHECK("validation targets");
      for (int run = 0; run < ncol; ++run) {
        const int32_t* r_unit = r_runs + size_t(run) * UL;
        if (run > 0) {
          int r_hi = 0;
          for (int i = 0; i < UL; ++i) r_hi = std::max(r_hi, hr[size_t(run) * UL + i]);
          if (r_hi == 0) {           // no unit of the layer has this candidate
            k_loss_reduce<<<unsigned(cdiv(UL, 128)), 128, 0, stream>>>(rowerr, losses, 0, UL,
                                                                      ncol, run, r_unit);
            RESKV_LAUNCH_CHECK("validation loss");
            continue;
          }
          st = lloyd_run(r_unit, run_off[run], r_hi);
          if (st != RESKV_OK) return cleanup_fail(st);
        }
        timing_ok &= timer.mark(kStValLoss);
        LossArgs lo{K, V, Q, s, G, cfg.n_obs, cfg.n_val, n_val_rows, P, n_top, b, top, r_unit,
                    kbar, vbar, ecount, ent_stride, run_off[run], cfg.beta, cfg.gate_mode,
                    cfg.tau, cfg.alpha, cfg.g_min, cfg.g_fixed, oS, rowerr, cfg.softmax_mode,
                    bl_d};
        k_val_loss<<<dim3(unsigned(cdiv(n_val_rows, kRowBlk)), UL), kThreads, kValSmem, stream>>>(lo);
        k_loss_reduce<<<unsigned(cdiv(UL, 128)), 128, 0, stream>>>(rowerr, losses, n_val_rows, UL,
                                                                  ncol, run, r_unit);
        RESKV_LAUNCH_CHECK("validation loss");
      }
      k_choose<<<unsigned(cdiv(UL, 128)), 128, 0, stream>>>(losses, ncol, r_runs, UL,
                                                           one_minus_delta, r_final, chosen);
      RESKV_LAUNCH_CHECK("choosing r");
    } else {
      // fixed r per unit (or the budget covers every token: r = 0)
      timing_ok &= timer.mark(-1);
      std::vector<int32_t> rl(UL, 0), ch(UL, 0);
      bool any = false;
      if (!ovr.empty())
        for (int i = 0; i < UL; ++i) {
          rl[i] = ovr[size_t(l) * UL + i];
          ch[i] = rl[i] > 0 ? 1 : 0;
          any |= rl[i] > 0;
        }
      if (cudaMemcpyAsync(r_final, rl.data(), UL * 4, cudaMemcpyHostToDevice, stream) != cudaSuccess ||
          cudaMemcpyAsync(chosen, ch.data(), UL * 4, cudaMemcpyHostToDevice, stream) != cudaSuccess ||
          cudaStreamSynchronize(stream) != cudaSuccess)
        return cleanup_fail(fail(RESKV_ERR_CUDA, "copying residual counts"));
      if (any) {
        st = lloyd_run(r_final, 0, *std::max_element(rl.begin(), rl.end()));
        if (st != RESKV_OK) return cleanup_fail(st);
      }
    }

    // ---- pack the chosen cache ----
    timing_ok &= timer.mark(kStPack);
    PackArgs pa{K, V, s, P, b, c->stride, rank_pos, r_final, chosen, run_off_d, kbar, vbar, ecount,
                ent_stride, cfg.beta, int64_t(l) * UL, c->kslots, c->vslots, c->logc,
                c->slot_pos, c->counts, c->n_main, c->n_res, bl_d,
                per_unit ? c->offsets : nullptr};
    k_pack<<<UL, 1024, 0, stream>>>(pa);
    RESKV_LAUNCH_CHECK("packing");
    timing_ok &= timer.mark(-1);
    timing_ok &= timer.flush(c->build_ms);

    if (cfg.keep_debug) {
      cudaError_t e = cudaMemcpyAsync(c->dbg_scores + size_t(l) * US, scores, US * 8,
                                      cudaMemcpyDeviceToDevice, stream);
      if (e == cudaSuccess && n_top > 0)
        e = cudaMemcpyAsync(c->dbg_ranked + size_t(l) * UL * n_top, top, size_t(UL) * n_top * 4,
                            cudaMemcpyDeviceToDevice, stream);
      if (e == cudaSuccess && proxy)
        e = cudaMemcpyAsync(c->dbg_losses + size_t(l) * UL * ncol, losses, size_t(UL) * ncol * 8,
                            cudaMemcpyDeviceToDevice, stream);
      if (e != cudaSuccess) return cleanup_fail(fail(RESKV_ERR_CUDA, "keeping intermediates"));
    }
  }
  if (!timing_ok)                        // timing is reported, not needed: clear it
    for (float& t : c->build_ms) t = 0.f;
  if (adakv && (st = finalize_ragged_layout(c)) != RESKV_OK) return cleanup_fail(st);
  // scratch is freed (cudaFree synchronises) when S leaves scope
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return cleanup_fail(fail(RESKV_ERR_CUDA, std::string("construction: ") +
                                                                   cudaGetErrorString(e)));
  *out = c;
  return RESKV_OK;
}

}  // namespace reskv
