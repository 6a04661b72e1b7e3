// Host side of the C ABI declared in include/reskv.h: argument validation,
// ownership of the device layout, import/export, and decode launches.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <string>
#include <vector>

#include "internal.h"
#include "reskv.h"

namespace reskv {

static thread_local std::string g_last_error;

void set_error(const std::string& msg) { g_last_error = msg; }

// reskv_test_inject state: decode launches still to fail their first wait;
// allocations until the injected failure (0: none pending)
static std::atomic<int64_t> g_wait_faults{0};
static std::atomic<int64_t> g_alloc_countdown{0};

bool take_test_wait_fault() {
  int64_t n = g_wait_faults.load();
  while (n > 0 && !g_wait_faults.compare_exchange_weak(n, n - 1)) {
  }
  return n > 0;
}

cudaError_t device_alloc(void** p, size_t bytes) {
  int64_t n = g_alloc_countdown.load();
  while (n > 0 && !g_alloc_countdown.compare_exchange_weak(n, n - 1)) {
  }
  if (n == 1) {                        // the injected failure: nothing allocated
    *p = nullptr;
    return cudaErrorMemoryAllocation;
  }
  return cudaMalloc(p, bytes);
}

// construction (construct.cu)
reskv_status build_all_layers(reskv_cache** out, const reskv_config& cfg,
                              const int32_t* override_host, const void* const* K,
                              const void* const* V, const void* const* Qobs,
                              cudaStream_t stream);

namespace {

reskv_status fail(reskv_status st, const std::string& msg) {
  set_error(msg);
  return st;
}

reskv_status cuda_fail(cudaError_t err, const char* what) {
  return fail(err == cudaErrorMemoryAllocation ? RESKV_ERR_OOM : RESKV_ERR_CUDA,
              std::string(what) + ": " + cudaGetErrorString(err));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Shape and gate fields shared by build and import.
reskv_status validate_shape(const reskv_config* cfg) {
  if (!cfg) return fail(RESKV_ERR_INVALID_ARG, "cfg is NULL");
  if (cfg->batch < 1 || cfg->n_layers < 1 || cfg->n_kv_heads < 1)
    return fail(RESKV_ERR_INVALID_ARG, "batch, n_layers and n_kv_heads must be >= 1");
  if (cfg->group != 1 && cfg->group != 2 && cfg->group != 4)
    return fail(RESKV_ERR_UNSUPPORTED, "group (query heads per KV head) must be 1, 2 or 4");
  if (cfg->head_dim != kHeadDim) return fail(RESKV_ERR_UNSUPPORTED, "head_dim must be 128");
  if (cfg->seq_len < 1 || cfg->seq_len > (int64_t(1) << 30))
    return fail(RESKV_ERR_INVALID_ARG, "seq_len must be in [1, 2^30]");
  if (cfg->budget < 1 || cfg->budget > (1 << 20))
    return fail(RESKV_ERR_INVALID_ARG, "budget must be in [1, 2^20]");
  if (cfg->decode_warps < 0) return fail(RESKV_ERR_INVALID_ARG, "decode_warps must be >= 0");
  if (cfg->decode_kernel < RESKV_DECODE_AUTO || cfg->decode_kernel > RESKV_DECODE_LSE_MERGE)
    return fail(RESKV_ERR_INVALID_ARG, "unknown decode_kernel");
  if (cfg->softmax_mode != RESKV_SOFTMAX_SHARED && cfg->softmax_mode != RESKV_SOFTMAX_SEPARATE)
    return fail(RESKV_ERR_INVALID_ARG, "unknown softmax_mode");
  if (cfg->append_policy != RESKV_APPEND_FAIL && cfg->append_policy != RESKV_APPEND_RING_DROP &&
      cfg->append_policy != RESKV_APPEND_RING_FOLD)
    return fail(RESKV_ERR_INVALID_ARG, "unknown append_policy");
  if (cfg->append_capacity < 0 || cfg->append_capacity > (1 << 20))
    return fail(RESKV_ERR_INVALID_ARG, "append_capacity must be in [0, 2^20]");
  const int64_t n_units = int64_t(cfg->n_layers) * cfg->batch * cfg->n_kv_heads;
  double slots = double(n_units) * (double(cfg->budget) + cfg->append_capacity);
  if (cfg->unit_budgets) {
    slots = 0;
    for (int64_t u = 0; u < n_units; ++u) {
      if (cfg->unit_budgets[u] < 1 || cfg->unit_budgets[u] > (1 << 20))
        return fail(RESKV_ERR_INVALID_ARG, "unit_budgets must be in [1, 2^20]");
      slots += double(cfg->unit_budgets[u]) + cfg->append_capacity;
    }
  }
  if (slots + kLogcPad >= double(int64_t(1) << 31))
    return fail(RESKV_ERR_UNSUPPORTED, "at most 2^31 cache slots");
  if (cfg->gate_mode != RESKV_GATE_DYNAMIC && cfg->gate_mode != RESKV_GATE_FIXED)
    return fail(RESKV_ERR_INVALID_ARG, "unknown gate_mode");
  if (!std::isfinite(cfg->tau) || !std::isfinite(cfg->alpha) || !(cfg->g_min >= 0.f) ||
      !(cfg->g_min <= 1.f) || !(cfg->g_fixed >= 0.f) || !(cfg->g_fixed <= 1.f))
    return fail(RESKV_ERR_INVALID_ARG, "gate parameters out of range (g_min, g_fixed in [0,1])");
  const double units = double(cfg->n_layers) * cfg->batch * cfg->n_kv_heads;
  if (units * cfg->budget > double(int64_t(1) << 40))
    return fail(RESKV_ERR_INVALID_ARG, "cache too large");
  return RESKV_OK;
}

template <typename T>
reskv_status dalloc(T** p, size_t count, const char* what) {
  *p = nullptr;
  if (count == 0) count = 1;
  cudaError_t err = device_alloc(reinterpret_cast<void**>(p), count * sizeof(T));
  if (err != cudaSuccess) {
    *p = nullptr;
    cudaGetLastError();
    return cuda_fail(err, what);
  }
  return RESKV_OK;
}

// cuTensorMapEncodeTiled through the runtime's driver entry point (no -lcuda)
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  }
  return fn;
}


void free_handle(reskv_cache* c) {
  if (!c) return;
  cudaFree(c->kslots);
  cudaFree(c->vslots);
  cudaFree(c->logc);
  cudaFree(c->slot_pos);
  cudaFree(c->counts);
  cudaFree(c->n_main);
  cudaFree(c->n_res);
  cudaFree(c->n_app);
  cudaFree(c->n_total);
  cudaFree(c->offsets);
  cudaFree(c->partials);
  cudaFree(c->tickets);
  cudaFree(c->status);
  cudaFree(c->dbg_scores);
  cudaFree(c->dbg_ranked);
  cudaFree(c->dbg_losses);
  cudaFree(c->hio.q);
  cudaFree(c->hio.o);
  delete c;
}

// Warps per CTA of the cluster kernel for clusters of `cluster` CTAs: 8, or
// fewer when the unit has less than one 16-slot chunk per warp.
int cluster_warps(int64_t budget, int cluster) {
  const int64_t chunks = (budget + kDecodeChunk - 1) / kDecodeChunk + 1;
  return int(std::min<int64_t>(kDecodeWarpsPerCta,
                               std::max<int64_t>(1, (chunks + cluster - 1) / cluster)));
}

MmaPlan plan_mma(const reskv_cache* c, int64_t n_units, int64_t total_slots) {
  return plan_mma_shape(c->num_sms, c->max_warps, c->cfg.decode_warps, c->max_unit_slots,
                        c->ragged, n_units, total_slots);
}

// Cluster decode shape for launches of `units` units: the largest cluster
// (at most 8 CTAs, at most SMs / units) at which all of the launch's clusters
// are resident at once; cluster = 0 if not even single-CTA clusters are.
reskv_status plan_cluster(const reskv_cache* c, int64_t units, reskv_cache::ClusterPlan* out) {
  *out = reskv_cache::ClusterPlan{};
  if (units > c->num_sms) return RESKV_OK;
  for (int cs = int(std::min<int64_t>(8, c->num_sms / units)); cs >= 1; --cs) {
    const int wpc = cluster_warps(c->max_unit_slots, cs);
    const int fit = decode_cluster_max_active(c->cfg.group, cs, wpc);
    if (fit < 0) return fail(RESKV_ERR_CUDA, "querying cluster occupancy of the decode kernel");
    if (fit >= units) {
      out->cluster = cs;
      out->warps_per_cta = wpc;
      return RESKV_OK;
    }
  }
  return RESKV_OK;
}

}  // namespace

// Allocate a zeroed layout and decode workspace for cfg's shape.
reskv_status alloc_handle(const reskv_config& cfg, cudaStream_t stream, reskv_cache** out) {
  reskv_cache* c = new (std::nothrow) reskv_cache();
  if (!c) return fail(RESKV_ERR_OOM, "host allocation failed");
  c->cfg = cfg;
  c->cfg.residual_override = nullptr;
  cudaError_t err = cudaGetDevice(&c->device);
  if (err == cudaSuccess)
    err = cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device);
  if (err != cudaSuccess) {
    delete c;
    return cuda_fail(err, "device query");
  }
  c->n_units = int64_t(cfg.n_layers) * cfg.batch * cfg.n_kv_heads;
  c->budget = cfg.budget;
  c->append_capacity = cfg.append_capacity;
  c->stride = cfg.budget + cfg.append_capacity;
  c->n_app_max.assign(size_t(cfg.n_layers), 0);
  c->max_warps = c->num_sms * kDecodeWarpsPerCta;
  c->ragged = cfg.unit_budgets != nullptr;
  c->h_offsets.assign(size_t(c->n_units) + 1, 0);
  c->max_unit_slots = c->stride;
  for (int64_t u = 0; u < c->n_units; ++u) {
    const int32_t su = (c->ragged ? cfg.unit_budgets[u] : cfg.budget) + cfg.append_capacity;
    c->h_offsets[size_t(u) + 1] = c->h_offsets[size_t(u)] + su;
    if (c->ragged) c->max_unit_slots = u == 0 ? su : std::max(c->max_unit_slots, su);
  }
  c->total_slots = c->h_offsets.back();
  c->cfg.unit_budgets = nullptr;       // the host array is the caller's
  const size_t slots = size_t(c->total_slots);
  reskv_status st = RESKV_OK;
  if ((st = dalloc(&c->kslots, slots * kHeadDim, "cache keys")) != RESKV_OK ||
      (st = dalloc(&c->vslots, slots * kHeadDim, "cache values")) != RESKV_OK ||
      (st = dalloc(&c->logc, slots + kLogcPad, "log counts")) != RESKV_OK ||
      (st = dalloc(&c->slot_pos, slots, "slot positions")) != RESKV_OK ||
      (st = dalloc(&c->counts, slots, "slot counts")) != RESKV_OK ||
      (st = dalloc(&c->n_main, size_t(c->n_units), "n_main")) != RESKV_OK ||
      (st = dalloc(&c->n_res, size_t(c->n_units), "n_res")) != RESKV_OK ||
      (st = dalloc(&c->n_app, size_t(c->n_units), "n_app")) != RESKV_OK ||
      (st = dalloc(&c->n_total, size_t(c->n_units), "appended token counts")) != RESKV_OK ||
      (c->ragged &&
       (st = dalloc(&c->offsets, size_t(c->n_units) + 1, "unit offsets")) != RESKV_OK) ||
      (st = dalloc(&c->partials,
                   std::max({decode_partials_floats(c->n_units, c->max_warps, cfg.group),
                             decode_mma_partials_floats(c->n_units, c->max_warps, cfg.group),
                             decode_lse_scratch_floats(c->n_units, cfg.group)}),
                   "decode workspace")) != RESKV_OK ||
      (st = dalloc(&c->tickets, size_t(c->n_units), "decode tickets")) != RESKV_OK ||
      (st = dalloc(&c->status, 1, "status word")) != RESKV_OK) {
    free_handle(c);
    return st;
  }
  err = cudaMemsetAsync(c->kslots, 0, slots * kHeadDim * 2, stream);
  if (err == cudaSuccess) err = cudaMemsetAsync(c->vslots, 0, slots * kHeadDim * 2, stream);
  if (err == cudaSuccess) err = cudaMemsetAsync(c->logc, 0, (slots + kLogcPad) * 4, stream);
  if (err == cudaSuccess) err = cudaMemsetAsync(c->slot_pos, 0xff, slots * 4, stream);
  if (err == cudaSuccess) err = cudaMemsetAsync(c->counts, 0, slots * 4, stream);
  if (err == cudaSuccess) err = cudaMemsetAsync(c->n_app, 0, size_t(c->n_units) * 4, stream);
  if (err == cudaSuccess) err = cudaMemsetAsync(c->n_total, 0, size_t(c->n_units) * 4, stream);
  if (err == cudaSuccess && c->ragged)
    err = cudaMemcpyAsync(c->offsets, c->h_offsets.data(), c->h_offsets.size() * 4,
                          cudaMemcpyHostToDevice, stream);
  if (err == cudaSuccess && c->ragged) err = cudaStreamSynchronize(stream);   // h_offsets is pageable
  if (err == cudaSuccess) err = cudaMemsetAsync(c->tickets, 0, size_t(c->n_units) * 4, stream);
  if (err == cudaSuccess) err = cudaMemsetAsync(c->status, 0, 4, stream);
  if (err != cudaSuccess) {
    free_handle(c);
    return cuda_fail(err, "initialising the cache");
  }
  c->kv_rank = 3;                       // one copy per chunk, else two
  if (!encode_rows(&c->tmap_k, c->kslots, slots, 3) || !encode_rows(&c->tmap_v, c->vslots, slots, 3))
    c->kv_rank = 2;
  if (c->kv_rank == 2 &&
      (!encode_rows(&c->tmap_k, c->kslots, slots, 2) || !encode_rows(&c->tmap_v, c->vslots, slots, 2))) {
    free_handle(c);
    return fail(RESKV_ERR_CUDA, "creating the TMA tensor maps of the cache");
  }
  const int64_t per_layer = int64_t(cfg.batch) * cfg.n_kv_heads;
  if ((st = plan_cluster(c, per_layer, &c->cplan_layer)) != RESKV_OK ||
      (st = plan_cluster(c, c->n_units, &c->cplan_all)) != RESKV_OK) {
    free_handle(c);
    return st;
  }
  *out = c;
  return RESKV_OK;
}

void release_handle(reskv_cache* c) { free_handle(c); }

// After construction has placed units of a ragged layout (AdaKV budgets):
// the largest unit and the cluster plans follow the final budgets.
reskv_status finalize_ragged_layout(reskv_cache* c) {
  c->max_unit_slots = 0;
  for (int64_t u = 0; u < c->n_units; ++u)
    c->max_unit_slots = std::max<int32_t>(c->max_unit_slots,
                                          c->h_offsets[size_t(u) + 1] - c->h_offsets[size_t(u)]);
  const int64_t per_layer = int64_t(c->cfg.batch) * c->cfg.n_kv_heads;
  reskv_status st = plan_cluster(c, per_layer, &c->cplan_layer);
  if (st == RESKV_OK) st = plan_cluster(c, c->n_units, &c->cplan_all);
  return st;
}

bool encode_rows(CUtensorMap* map, const void* base, uint64_t rows, int rank) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint32_t estr[3] = {1, 1, 1};
  if (rank == 3) {
    const cuuint64_t dims[3] = {64, cuuint64_t(rows), 2};
    const cuuint64_t strides[2] = {cuuint64_t(kSlotRowBytes), 128};
    const cuuint32_t box[3] = {64, 16, 2};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
  }
  const cuuint64_t dims[2] = {cuuint64_t(kHeadDim), cuuint64_t(rows)};
  const cuuint64_t strides[1] = {cuuint64_t(kSlotRowBytes)};
  const cuuint32_t box[2] = {64, 16};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_key_tiles(CUtensorMap* map, const void* keys, uint64_t rows) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint32_t estr[3] = {1, 1, 1};
  const cuuint64_t dims[3] = {64, cuuint64_t(rows), 2};
  const cuuint64_t strides[2] = {cuuint64_t(kHeadDim) * 2, 128};
  const cuuint32_t box[3] = {64, 128, 2};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(keys), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// At most 7 warps per SM: 7 x 2 ring stages streamed the 32-layer 32K cache
// 1 % faster than 8 x 2 and 8 x 3.
constexpr int kMmaWarpsPerCta = 7;

MmaPlan plan_mma_shape(int num_sms, int64_t max_warps, int32_t user_warps, int64_t max_unit_slots,
                       bool ragged, int64_t n_units, int64_t total_slots) {
  MmaPlan m;
  int64_t W = 0;
  int wpc = kMmaWarpsPerCta;
  if (user_warps > 0) {
    W = user_warps;
  } else if (n_units >= num_sms && n_units <= 4 * int64_t(num_sms) &&
             max_unit_slots <= 256 && !ragged) {
    W = n_units;                      // one warp per unit: no partial records at all
  } else {
    wpc = int(std::min<int64_t>(kMmaWarpsPerCta,
                                std::max<int64_t>(1, total_slots / (int64_t(num_sms) * 200))));
    W = int64_t(num_sms) * wpc;
    if (total_slots < W * 32) W = std::max<int64_t>(1, total_slots / 32);
  }
  // every warp needs a 16-slot chunk of its own (pieces are whole chunks)
  if (W > total_slots / kDecodeChunk) W = total_slots / kDecodeChunk;
  if (W > max_warps) W = max_warps;
  if (W < 1) W = 1;
  // Short units (each at most an eighth of a warp's piece): every warp takes
  // k consecutive whole units, so no unit is cut and no partial record,
  // ticket or merge is needed; the warps' loads differ by at most one unit.
  if (user_warps == 0 && int64_t(max_unit_slots) * 8 * W <= total_slots) {
    const int64_t k = (n_units + W - 1) / W;
    W = (n_units + k - 1) / k;
    m.k = int32_t(k);
  }
  m.W = W;
  m.wpc = int(std::min<int64_t>(8, (W + num_sms - 1) / num_sms));
  // Ring depth: about 16 stages per SM in all.  On the 32-layer 32K cache
  // 8 warps x 2 stages stream faster than 8 x 3 (and 6 x 3 than 6 x 2):
  // more copies in flight only lengthen the loaded latency.
  m.stages = std::min(decode_mma_stages(m.wpc), std::max(2, (16 + m.wpc / 2) / m.wpc));
  return m;
}

}  // namespace reskv

using namespace reskv;

extern "C" {

void reskv_config_default(reskv_config* cfg) {
  if (!cfg) return;
  std::memset(cfg, 0, sizeof(*cfg));
  cfg->head_dim = kHeadDim;
  cfg->group = 4;
  cfg->recent_window = 64;
  cfg->n_obs = 128;
  cfg->n_fit = 96;
  cfg->n_val = 32;
  cfg->pool_kernel = 5;
  cfg->score_mode = RESKV_SCORE_OBS_POOL;
  cfg->n_grid = 5;
  const float grid[5] = {0.0f, 0.05f, 0.10f, 0.15f, 0.20f};
  for (int i = 0; i < 5; ++i) cfg->grid_ratios[i] = grid[i];
  cfg->lloyd_iters = 4;
  cfg->delta = 0.01f;
  cfg->beta = 1.0f;
  cfg->residual_override = nullptr;
  cfg->gate_mode = RESKV_GATE_DYNAMIC;
  cfg->tau = 0.25f;
  cfg->alpha = 12.0f;
  cfg->g_min = 0.0f;
  cfg->g_fixed = 1.0f;
  cfg->keep_debug = 0;
  cfg->budget_mode = RESKV_BUDGET_UNIFORM;
  cfg->adakv_safeguard = 0.2f;
  cfg->append_policy = RESKV_APPEND_RING_FOLD;
}

const char* reskv_last_error(void) { return g_last_error.c_str(); }

reskv_status reskv_build_cache(const reskv_config* cfg, const void* const* K_layers,
                               const void* const* V_layers, const void* const* Qobs_layers,
                               void* stream, reskv_cache** out) {
  g_last_error.clear();
  reskv_status st = validate_shape(cfg);
  if (st != RESKV_OK) return st;
  if (!out || !K_layers || !V_layers) return fail(RESKV_ERR_INVALID_ARG, "NULL argument");
  reskv_cache* c = nullptr;
  st = build_all_layers(&c, *cfg, cfg->residual_override, K_layers, V_layers, Qobs_layers,
                        static_cast<cudaStream_t>(stream));
  if (st == RESKV_OK) *out = c;
  return st;
}

reskv_status reskv_import_cache(const reskv_config* cfg, const reskv_host_cache* h, void* stream,
                                reskv_cache** out) {
  g_last_error.clear();
  reskv_status st = validate_shape(cfg);
  if (st != RESKV_OK) return st;
  if (!h || !out || !h->n_main || !h->n_res || !h->kslots || !h->vslots || !h->logc)
    return fail(RESKV_ERR_INVALID_ARG, "NULL argument");
  const int64_t U = int64_t(cfg->n_layers) * cfg->batch * cfg->n_kv_heads;
  for (int64_t u = 0; u < U; ++u) {
    const int32_t bu = cfg->unit_budgets ? cfg->unit_budgets[u] : cfg->budget;
    if (h->n_main[u] < 1 || h->n_res[u] < 0 || int64_t(h->n_main[u]) + h->n_res[u] > bu)
      return fail(RESKV_ERR_INVALID_ARG,
                  "unit " + std::to_string(u) + ": need 1 <= n_main and n_main + n_res <= budget");
    if (h->n_app && (h->n_app[u] < 0 || h->n_app[u] > cfg->append_capacity))
      return fail(RESKV_ERR_INVALID_ARG,
                  "unit " + std::to_string(u) + ": need 0 <= n_app <= append_capacity");
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  reskv_cache* c = nullptr;
  if ((st = alloc_handle(*cfg, s, &c)) != RESKV_OK) return st;
  if (h->n_app) {
    const int64_t per_layer = int64_t(cfg->batch) * cfg->n_kv_heads;
    for (int64_t u = 0; u < U; ++u)
      c->n_app_max[size_t(u / per_layer)] = std::max(c->n_app_max[size_t(u / per_layer)], h->n_app[u]);
  }
  const size_t slots = size_t(c->total_slots);
  cudaError_t err = cudaMemcpyAsync(c->kslots, h->kslots, slots * kHeadDim * 2,
                                    cudaMemcpyHostToDevice, s);
  if (err == cudaSuccess)
    err = cudaMemcpyAsync(c->vslots, h->vslots, slots * kHeadDim * 2, cudaMemcpyHostToDevice, s);
  if (err == cudaSuccess)
    err = cudaMemcpyAsync(c->logc, h->logc, slots * 4, cudaMemcpyHostToDevice, s);
  if (err == cudaSuccess)
    err = cudaMemcpyAsync(c->n_main, h->n_main, size_t(U) * 4, cudaMemcpyHostToDevice, s);
  if (err == cudaSuccess)
    err = cudaMemcpyAsync(c->n_res, h->n_res, size_t(U) * 4, cudaMemcpyHostToDevice, s);
  if (err == cudaSuccess && h->n_app)
    err = cudaMemcpyAsync(c->n_app, h->n_app, size_t(U) * 4, cudaMemcpyHostToDevice, s);
  if (err == cudaSuccess && h->n_app)      // imported appended rows: appended in slot order
    err = cudaMemcpyAsync(c->n_total, c->n_app, size_t(U) * 4, cudaMemcpyDeviceToDevice, s);
  if (err == cudaSuccess && h->slot_pos)
    err = cudaMemcpyAsync(c->slot_pos, h->slot_pos, slots * 4, cudaMemcpyHostToDevice, s);
  if (err == cudaSuccess && h->counts)
    err = cudaMemcpyAsync(c->counts, h->counts, slots * 4, cudaMemcpyHostToDevice, s);
  if (err == cudaSuccess) err = cudaStreamSynchronize(s);
  if (err != cudaSuccess) {
    release_handle(c);
    return cuda_fail(err, "importing the cache");
  }
  *out = c;
  return RESKV_OK;
}

reskv_status reskv_export_cache(const reskv_cache* c, reskv_host_cache* h, void* stream) {
  g_last_error.clear();
  if (!c || !h || !h->n_main || !h->n_res || !h->kslots || !h->vslots || !h->logc ||
      !h->slot_pos || !h->counts || !h->n_app)
    return fail(RESKV_ERR_INVALID_ARG, "NULL argument");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t U = size_t(c->n_units), slots = size_t(c->total_slots);
  cudaError_t err = cudaMemcpyAsync(h->kslots, c->kslots, slots * kHeadDim * 2,
                                    cudaMemcpyDeviceToHost, s);
  if (err == cudaSuccess)
    err = cudaMemcpyAsync(h->vslots, c->vslots, slots * kHeadDim * 2, cudaMemcpyDeviceToHost, s);
  if (err == cudaSuccess) err = cudaMemcpyAsync(h->logc, c->logc, slots * 4, cudaMemcpyDeviceToHost, s);
  if (err == cudaSuccess)
    err = cudaMemcpyAsync(h->slot_pos, c->slot_pos, slots * 4, cudaMemcpyDeviceToHost, s);
  if (err == cudaSuccess)
    err = cudaMemcpyAsync(h->counts, c->counts, slots * 4, cudaMemcpyDeviceToHost, s);
  if (err == cudaSuccess) err = cudaMemcpyAsync(h->n_main, c->n_main, U * 4, cudaMemcpyDeviceToHost, s);
  if (err == cudaSuccess) err = cudaMemcpyAsync(h->n_res, c->n_res, U * 4, cudaMemcpyDeviceToHost, s);
  if (err == cudaSuccess) err = cudaMemcpyAsync(h->n_app, c->n_app, U * 4, cudaMemcpyDeviceToHost, s);
  if (err == cudaSuccess) err = cudaStreamSynchronize(s);
  if (err != cudaSuccess) return cuda_fail(err, "exporting the cache");
  return RESKV_OK;
}

}  // extern "C"

namespace reskv {
namespace {

// Alg. 2 for layers [layer0, layer0 + n_layers) in one launch.
reskv_status decode_layers(const reskv_cache* c, int32_t layer0, int32_t n_layers,
                           const void* Q, void* O, void* stream) {
  if (!c || !Q || !O) return fail(RESKV_ERR_INVALID_ARG, "NULL argument");
  const reskv_config& cfg = c->cfg;
  if (layer0 < 0 || n_layers < 1 || int64_t(layer0) + n_layers > cfg.n_layers)
    return fail(RESKV_ERR_INVALID_ARG, "need 0 <= layer0 and 1 <= n_layers <= L - layer0");
  if (!aligned16(Q) || !aligned16(O))
    return fail(RESKV_ERR_INVALID_ARG, "Q and O must be 16-byte aligned");
  const int64_t per_layer = int64_t(cfg.batch) * cfg.n_kv_heads;
  const int32_t l_end = layer0 + n_layers;
  DecodeParams p{};
  p.kslots = c->kslots;
  p.vslots = c->vslots;
  p.logc = c->logc;
  p.n_main = c->n_main;
  p.n_res = c->n_res;
  p.n_app = c->append_capacity > 0 ? c->n_app : nullptr;
  p.offsets = c->ragged ? c->offsets : nullptr;
  p.kv_rank = c->kv_rank;
  p.Q = static_cast<const __nv_bfloat16*>(Q);
  p.O = static_cast<float*>(O);
  p.partials = c->partials;
  p.tickets = c->tickets;
  p.status = c->status;
  p.unit0 = int64_t(layer0) * per_layer;
  p.n_units = int32_t(int64_t(n_layers) * per_layer);
  p.stride = c->stride;
  int32_t app = 0;                     // most appended rows of a unit of the launch
  for (int l = layer0; l < l_end; ++l) app = std::max(app, c->n_app_max[size_t(l)]);
  p.tail_unused = c->append_capacity - app;
  p.n_kv_heads = cfg.n_kv_heads;
  p.total_slots = c->h_offsets[size_t(p.unit0 + p.n_units)] - c->h_offsets[size_t(p.unit0)];
  p.gate_mode = cfg.gate_mode;
  p.softmax_mode = cfg.softmax_mode;
  p.tau = cfg.tau;
  p.alpha = cfg.alpha;
  p.g_min = cfg.g_min;
  p.g_fixed = cfg.g_fixed;
  p.test_fault = take_test_wait_fault() ? 1 : 0;
  reskv_cache::ClusterPlan cp;
  if (n_layers == 1) {
    cp = c->cplan_layer;
  } else if (n_layers == cfg.n_layers) {
    cp = c->cplan_all;
  } else {                             // other layer counts: planned on first use
    if (c->cplan_range.empty()) c->cplan_range.assign(size_t(cfg.n_layers) + 1, {-1, 0});
    if (c->cplan_range[size_t(n_layers)].cluster < 0) {
      reskv_status st = plan_cluster(c, p.n_units, &c->cplan_range[size_t(n_layers)]);
      if (st != RESKV_OK) return st;
    }
    cp = c->cplan_range[size_t(n_layers)];
  }
  int kernel = cfg.decode_kernel;
  if (kernel == RESKV_DECODE_AUTO)
    kernel = (cp.cluster > 0 && cfg.decode_warps == 0) ? RESKV_DECODE_CLUSTER : RESKV_DECODE_MMA;
  if (kernel == RESKV_DECODE_CLUSTER || kernel == RESKV_DECODE_LSE_MERGE) {
    // one cluster per unit; a launch too large for one wave runs single-CTA
    // clusters in several waves
    const int cs = cp.cluster > 0 ? cp.cluster : 1;
    const int wpc = cp.cluster > 0 ? cp.warps_per_cta : cluster_warps(c->max_unit_slots, 1);
    p.n_warps = int32_t(int64_t(cs) * wpc);
    // ring depth: as deep as shared memory allows, but 2 stages per warp in
    // clusters of 2 or more CTAs (one-layer launches of 32 units, b = 2048,
    // 4-CTA clusters: 7.55 us against 7.64 with 3 stages; of 64 units,
    // b = 1024, 2-CTA clusters, alternating on one GPU: 7.70-7.73 us against
    // 7.74-7.76)
    p.n_stages = decode_cluster_stages(wpc, cs);
    if (cs >= 2) p.n_stages = std::min(p.n_stages, 2);
    cudaError_t err =
        kernel == RESKV_DECODE_CLUSTER
            ? launch_decode_cluster(p, c->tmap_k, c->tmap_v, cfg.group, cs, wpc,
                                    static_cast<cudaStream_t>(stream))
            : launch_decode_lse(p, c->tmap_k, c->tmap_v, cfg.group, cs, wpc,
                                static_cast<cudaStream_t>(stream));
    if (err != cudaSuccess) return cuda_fail(err, "decode launch");
    return RESKV_OK;
  }
  // Split plan.  CUDA-core kernel: one warp per >= 32 slots, at most 8 warps
  // per SM.  Tensor-core stream-K kernel: one warp per unit when the launch
  // has between 1 and 4 short units (at most 16 tiles of 16 slots) per SM, so
  // that no unit is cut; otherwise (a lone warp on a long unit is bound by
  // the latency of its tile chain) one CTA per SM with 1..8
  // warps so that every warp streams >= ~200 slots (fewer, longer pieces for
  // small launches, with a deeper ring in the shared memory that fewer warps
  // leave free).
  const bool mma = kernel == RESKV_DECODE_MMA;
  int64_t W = 0;
  int wpc = kDecodeWarpsPerCta;
  if (mma) {
    const MmaPlan mp = plan_mma(c, p.n_units, p.total_slots);
    W = mp.W;
    wpc = mp.wpc;
    p.units_per_warp = mp.k;
    p.n_stages = mp.stages;
  } else {
    W = cfg.decode_warps > 0 ? cfg.decode_warps : p.total_slots / 32;
    if (W > p.total_slots) W = p.total_slots;
    if (W < 1) W = 1;
    if (W > c->max_warps) W = c->max_warps;
  }
  if (W < 1) W = 1;
  p.n_warps = int32_t(W);
  if (!mma) p.n_stages = 0;
  cudaError_t err =
      mma ? launch_decode_mma(p, c->tmap_k, c->tmap_v, cfg.group, int((W + wpc - 1) / wpc), wpc,
                              static_cast<cudaStream_t>(stream))
          : launch_decode(p, cfg.group, int((W + kDecodeWarpsPerCta - 1) / kDecodeWarpsPerCta),
                          static_cast<cudaStream_t>(stream));
  if (err != cudaSuccess) return cuda_fail(err, "decode launch");
  return RESKV_OK;
}

}  // namespace
}  // namespace reskv

extern "C" {

reskv_status reskv_decode_attn(const reskv_cache* c, int32_t layer, const void* Q, void* O,
                               void* stream) {
  if (!c) return fail(RESKV_ERR_INVALID_ARG, "NULL argument");
  if (layer < -1 || layer >= c->cfg.n_layers)
    return fail(RESKV_ERR_INVALID_ARG, "layer must be -1 or in [0, n_layers)");
  return layer < 0 ? decode_layers(c, 0, c->cfg.n_layers, Q, O, stream)
                   : decode_layers(c, layer, 1, Q, O, stream);
}

reskv_status reskv_decode_attn_layers(const reskv_cache* c, int32_t layer0, int32_t n_layers,
                                      const void* Q, void* O, void* stream) {
  return decode_layers(c, layer0, n_layers, Q, O, stream);
}

reskv_status reskv_append(reskv_cache* c, int32_t layer, const void* K_new, const void* V_new,
                          void* stream) {
  if (!c || !K_new || !V_new) return fail(RESKV_ERR_INVALID_ARG, "NULL argument");
  const reskv_config& cfg = c->cfg;
  if (layer < -1 || layer >= cfg.n_layers)
    return fail(RESKV_ERR_INVALID_ARG, "layer must be -1 or in [0, n_layers)");
  if (!aligned16(K_new) || !aligned16(V_new))
    return fail(RESKV_ERR_INVALID_ARG, "K_new and V_new must be 16-byte aligned");
  const int l0 = layer < 0 ? 0 : layer, l1 = layer < 0 ? cfg.n_layers : layer + 1;
  if (c->append_capacity == 0)
    return fail(RESKV_ERR_UNSUPPORTED, "the cache has no append region (append_capacity 0)");
  if (cfg.append_policy == RESKV_APPEND_FAIL)
    for (int l = l0; l < l1; ++l)
      if (c->n_app_max[size_t(l)] >= c->append_capacity)
        return fail(RESKV_ERR_UNSUPPORTED, "layer " + std::to_string(l) + ": the append region (" +
                                               std::to_string(c->append_capacity) +
                                               " slots per unit) is full");
  const int64_t per_layer = int64_t(cfg.batch) * cfg.n_kv_heads;
  cudaError_t err = launch_append(c, int64_t(l0) * per_layer, int64_t(l1 - l0) * per_layer,
                                  static_cast<const __nv_bfloat16*>(K_new),
                                  static_cast<const __nv_bfloat16*>(V_new),
                                  static_cast<cudaStream_t>(stream));
  if (err != cudaSuccess) return cuda_fail(err, "append launch");
  for (int l = l0; l < l1; ++l)
    c->n_app_max[size_t(l)] = std::min(c->n_app_max[size_t(l)] + 1, c->append_capacity);
  return RESKV_OK;
}

// The device address of host memory the current device can access (page-locked
// and mapped, as cudaHostAlloc / cudaMallocHost / cudaHostRegister give under
// unified addressing), or NULL.
static void* device_view(const void* host) {
  cudaPointerAttributes a{};
  if (cudaPointerGetAttributes(&a, host) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return a.type == cudaMemoryTypeHost ? a.devicePointer : nullptr;
}

reskv_status reskv_decode_attn_host(const reskv_cache* c, const void* Q_host, void* O_host,
                                    void* stream) {
  if (!c || !Q_host || !O_host) return fail(RESKV_ERR_INVALID_ARG, "NULL argument");
  const reskv_config& cfg = c->cfg;
  const int L = cfg.n_layers;
  const size_t rows = size_t(cfg.batch) * cfg.n_kv_heads * cfg.group;   // query rows per layer
  const size_t q_bytes = L * rows * kHeadDim * 2, o_bytes = L * rows * kHeadDim * 4;
  {
    const uint8_t* qa = static_cast<const uint8_t*>(Q_host);
    const uint8_t* oa = static_cast<const uint8_t*>(O_host);
    if (oa < qa + q_bytes && qa < oa + o_bytes)
      return fail(RESKV_ERR_INVALID_ARG, "O_host overlaps Q_host");
  }
  // Page-locked buffers: the decode kernel reads Q from and writes O to host
  // memory itself (over the host link), so the transfers overlap the
  // streaming of the cache and no copy sits before or after the launch.
  void* qv = device_view(Q_host);
  void* ov = device_view(O_host);
  if (qv && ov) return reskv_decode_attn_layers(c, 0, L, qv, ov, stream);
  // Otherwise stage through device buffers owned by the handle.
  reskv_cache::HostIo& io = c->hio;
  if (!io.q) {
    void* q = nullptr;
    void* o = nullptr;
    cudaError_t err = device_alloc(&q, q_bytes);
    if (err == cudaSuccess) err = device_alloc(&o, o_bytes);
    if (err != cudaSuccess) {
      cudaGetLastError();
      cudaFree(q);
      return err == cudaErrorMemoryAllocation ? fail(RESKV_ERR_OOM, "staging buffers")
                                              : cuda_fail(err, "staging buffers");
    }
    io.o = o;
    io.q = q;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t err = cudaMemcpyAsync(io.q, Q_host, q_bytes, cudaMemcpyHostToDevice, s);
  if (err != cudaSuccess) return cuda_fail(err, "copying Q in");
  const reskv_status st = reskv_decode_attn_layers(c, 0, L, io.q, io.o, s);
  if (st != RESKV_OK) return st;
  err = cudaMemcpyAsync(O_host, io.o, o_bytes, cudaMemcpyDeviceToHost, s);
  if (err != cudaSuccess) return cuda_fail(err, "copying O out");
  return RESKV_OK;
}

void reskv_free(reskv_cache* c) {
  if (!c) return;
  cudaDeviceSynchronize();
  free_handle(c);
}

reskv_status reskv_check_status(const reskv_cache* c) {
  if (!c) return fail(RESKV_ERR_INVALID_ARG, "NULL handle");
  uint32_t word = 0;
  cudaError_t err = cudaDeviceSynchronize();
  if (err == cudaSuccess) err = cudaMemcpy(&word, c->status, 4, cudaMemcpyDeviceToHost);
  if (err != cudaSuccess) return cuda_fail(err, "reading the status word");
  if (word != 0)
    return fail(RESKV_ERR_DEVICE_STATUS, "kernel status word " + std::to_string(word) +
                                             " (1 = bounded wait timed out, 2 = index out of range)");
  return RESKV_OK;
}

reskv_status reskv_get_info(const reskv_cache* c, reskv_cache_info* info) {
  if (!c || !info) return fail(RESKV_ERR_INVALID_ARG, "NULL argument");
  info->n_units = c->n_units;
  info->budget = c->budget;
  info->head_dim = kHeadDim;
  info->slot_bytes = 2 * kSlotRowBytes;
  info->cache_bytes = c->total_slots * (2 * kSlotRowBytes + 4);
  const bool auto_plan = c->cfg.decode_kernel == RESKV_DECODE_AUTO && c->cfg.decode_warps == 0;
  const bool cluster = c->cfg.decode_kernel == RESKV_DECODE_CLUSTER;
  info->layer_cluster = auto_plan ? c->cplan_layer.cluster
                                  : cluster ? std::max(1, c->cplan_layer.cluster) : 0;
  info->layer_cluster_warps =
      info->layer_cluster ? (c->cplan_layer.cluster ? c->cplan_layer.warps_per_cta
                                                    : cluster_warps(c->max_unit_slots, 1))
                          : 0;
  info->all_cluster = auto_plan ? c->cplan_all.cluster
                                : cluster ? std::max(1, c->cplan_all.cluster) : 0;
  for (int i = 0; i < 6; ++i) info->build_ms[i] = c->build_ms[i];
  info->append_capacity = c->append_capacity;
  info->stride = c->ragged ? 0 : c->stride;
  info->total_slots = c->total_slots;
  info->max_appended = 0;
  for (int32_t a : c->n_app_max) info->max_appended = std::max(info->max_appended, a);
  info->ragged = c->ragged ? 1 : 0;
  info->all_cluster_warps =
      info->all_cluster ? (c->cplan_all.cluster ? c->cplan_all.warps_per_cta
                                                : cluster_warps(c->max_unit_slots, 1))
                        : 0;
  const int64_t per_layer = int64_t(c->cfg.batch) * c->cfg.n_kv_heads;
  const bool mma_all = c->cfg.decode_kernel == RESKV_DECODE_MMA ||
                       (auto_plan && c->cplan_all.cluster == 0);
  const bool mma_layer = c->cfg.decode_kernel == RESKV_DECODE_MMA ||
                         (auto_plan && c->cplan_layer.cluster == 0);
  info->all_units_per_warp = mma_all ? plan_mma(c, c->n_units, c->total_slots).k : 0;
  info->layer_units_per_warp =
      mma_layer ? plan_mma(c, per_layer, c->h_offsets[size_t(per_layer)]).k : 0;
  info->n_candidates = c->n_candidates;
  info->ranked_width = int32_t(c->dbg_ranked ? c->dbg_n_top : c->ranked_width);
  info->kv_copy_rank = c->kv_rank;
  info->reserved0 = 0;
  return RESKV_OK;
}

reskv_status reskv_test_inject(int32_t what, int64_t n) {
  if (n < 0) return fail(RESKV_ERR_INVALID_ARG, "n must be >= 0");
  switch (what) {
    case RESKV_TEST_FAIL_FIRST_WAIT: g_wait_faults.store(n); return RESKV_OK;
    case RESKV_TEST_FAIL_ALLOC: g_alloc_countdown.store(n); return RESKV_OK;
    default: return fail(RESKV_ERR_INVALID_ARG, "unknown fault to inject");
  }
}

reskv_status reskv_get_unit_budgets(const reskv_cache* c, int32_t* host_budgets, int64_t n_units) {
  if (!c || !host_budgets) return fail(RESKV_ERR_INVALID_ARG, "NULL argument");
  if (n_units != c->n_units) return fail(RESKV_ERR_INVALID_ARG, "n_units does not match the handle");
  for (int64_t u = 0; u < n_units; ++u)
    host_budgets[u] = c->h_offsets[size_t(u) + 1] - c->h_offsets[size_t(u)] - c->append_capacity;
  return RESKV_OK;
}

reskv_status reskv_export_debug(const reskv_cache* c, int32_t what, void* host_dst, size_t bytes) {
  if (!c || !host_dst) return fail(RESKV_ERR_INVALID_ARG, "NULL argument");
  const void* src = nullptr;
  size_t need = 0;
  const size_t U = size_t(c->n_units);
  const size_t ncand = c->candidates.size();
  switch (what) {
    case RESKV_DEBUG_SCORES:
      src = c->dbg_scores;
      need = U * size_t(c->cfg.seq_len) * 8;
      break;
    case RESKV_DEBUG_RANKED:
      src = c->dbg_ranked;
      need = U * size_t(c->dbg_n_top) * 4;
      break;
    case RESKV_DEBUG_LOSSES:
      src = c->dbg_losses;
      need = U * (1 + size_t(c->n_candidates)) * 8;
      break;
    case RESKV_DEBUG_CANDIDATES:
      if (c->n_candidates > 0 && c->candidates.empty())
        return fail(RESKV_ERR_INVALID_ARG,
                    "per-unit budgets: read RESKV_DEBUG_UNIT_CANDIDATES instead");
      if (bytes != ncand * 4) return fail(RESKV_ERR_INVALID_ARG, "size mismatch");
      if (ncand) std::memcpy(host_dst, c->candidates.data(), bytes);
      return RESKV_OK;
    case RESKV_DEBUG_UNIT_CANDIDATES:
      if (bytes != U * size_t(c->n_candidates) * 4)
        return fail(RESKV_ERR_INVALID_ARG, "size mismatch: need " +
                                               std::to_string(U * size_t(c->n_candidates) * 4) +
                                               " bytes");
      if (bytes && c->unit_cands.size() * 4 != bytes)
        return fail(RESKV_ERR_INVALID_ARG, "no candidates were kept (the proxy did not run)");
      if (bytes) std::memcpy(host_dst, c->unit_cands.data(), bytes);
      return RESKV_OK;
    default:
      return fail(RESKV_ERR_INVALID_ARG, "unknown debug array");
  }
  if (!src) return fail(RESKV_ERR_INVALID_ARG, "intermediate not kept (keep_debug was 0)");
  if (bytes != need)
    return fail(RESKV_ERR_INVALID_ARG, "size mismatch: need " + std::to_string(need) + " bytes");
  cudaError_t err = cudaDeviceSynchronize();
  if (err == cudaSuccess) err = cudaMemcpy(host_dst, src, bytes, cudaMemcpyDeviceToHost);
  if (err != cudaSuccess) return cuda_fail(err, "exporting an intermediate");
  return RESKV_OK;
}

}  // extern "C"
