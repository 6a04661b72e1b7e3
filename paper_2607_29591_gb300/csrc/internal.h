// Internal declarations shared by the host ABI and the kernels.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <string>
#include <vector>

#include "reskv.h"

namespace reskv {

constexpr int kHeadDim = 128;          // d (only 128 is built)
constexpr int kSlotRowBytes = kHeadDim * 2;
constexpr float kLog2e = 1.4426950408889634f;

// Decode split: every launch streams the concatenated slot range of its units
// ("flat" index x = local_unit * stride + j) and cuts it into n_warps pieces,
// one per warp (equal slot pieces in the CUDA-core kernel, equal pieces of
// whole 16-slot chunks or whole units in the tensor-core stream-K kernel).  A
// unit covered by one warp is finished by that warp; a unit cut between warps
// is finished by the last of them to arrive, from per-(unit, warp) partial
// records.
//
// Unit u owns slots [u*stride, u*stride + stride), stride = budget + append
// capacity, or with per-unit budgets [offsets[u], offsets[u+1]) of size
// budget_u + append capacity: n_main exact main rows, n_res residual entries,
// then n_app exact rows appended at decode time (main rows too); the rest is
// unused.
struct DecodeParams {
  const __nv_bfloat16* kslots;  // [U, budget, d] whole cache
  const __nv_bfloat16* vslots;  // [U, budget, d]
  const float* logc;            // [U, budget]  beta*ln c at residual slots
  const int32_t* n_main;        // [U]
  const int32_t* n_res;         // [U]
  const int32_t* n_app;         // [U] appended rows, or NULL (none)
  const int32_t* offsets;       // [U+1] first slot of each unit, or NULL (uniform stride)
  const __nv_bfloat16* Q;       // [n_units / H_kv, H_kv*G, d] for this launch
  float* O;                     // same shape as Q, fp32
  float* partials;              // [(n_units + n_warps) * 2 * G * (d + 2)]
  int32_t* tickets;             // [U], zero between launches
  uint32_t* status;             // device status word
  int64_t unit0;                // first unit of the launch
  int64_t total_slots;          // n_units * stride
  int32_t n_units;
  int32_t stride;               // slots per unit (uniform layout)
  int32_t tail_unused;          // append capacity - max n_app over the launch's
                                // units: rows at the end of every unit that are
                                // certainly unused
  int32_t n_kv_heads;
  int32_t n_warps;              // W
  int32_t n_stages;             // ring stages per warp (tensor-core kernel)
  int32_t gate_mode;
  int32_t softmax_mode;         // RESKV_SOFTMAX_*
  float tau, alpha, g_min, g_fixed;
  int32_t kv_rank;              // rank of the K and V TMA maps: 3 (one copy per
                                // 16-row chunk) or 2 (two copies)
  int32_t units_per_warp;       // tensor-core stream-K kernel: 0 cuts the slot
                                // range into n_warps equal pieces; k > 0 gives
                                // warp w the whole units [w k, (w + 1) k) of the
                                // launch instead (short units: no unit is cut)
  // testing only (reskv_test_inject): nonzero makes every warp of the launch
  // give up its first ring wait as if its bound had run out (status word
  // set, copies in flight drained, output incomplete)
  int32_t test_fault;
};

constexpr int kDecodeWarpsPerCta = 8;

// Launch the CUDA-core decode kernel for `group` (1, 2 or 4) query heads per KV head.
cudaError_t launch_decode(const DecodeParams& p, int group, int n_ctas, cudaStream_t stream);
size_t decode_partials_floats(int64_t n_units, int n_warps, int group);
// Launch the tensor-core decode kernel (K/V rows through the given TMA maps).
cudaError_t launch_decode_mma(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                              int group, int n_ctas, int warps_per_cta, cudaStream_t stream);
int decode_mma_stages(int warps_per_cta);
size_t decode_mma_partials_floats(int64_t n_units, int n_warps, int group);
// Launch the cluster decode kernel: one cluster of `cluster` CTAs (1..8) of
// `warps_per_cta` warps per unit, p.n_stages <= decode_cluster_stages(warps, cluster).
cudaError_t launch_decode_cluster(const DecodeParams& p, const CUtensorMap& tk,
                                  const CUtensorMap& tv, int group, int cluster,
                                  int warps_per_cta, cudaStream_t stream);
int decode_cluster_stages(int warps_per_cta, int cluster);
int decode_cluster_smem_bytes(int warps_per_cta, int stages, int cluster);
// The paper-style comparison path: main-branch pass, residual-branch pass (both
// the cluster kernel on one branch's rows) and a log-sum-exp merge kernel; the
// branch records go to p.partials, which must hold decode_lse_scratch_floats().
cudaError_t launch_decode_lse(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                              int group, int cluster, int warps_per_cta, cudaStream_t stream);
size_t decode_lse_scratch_floats(int64_t n_units, int group);
// How many clusters of that shape the current device holds at once (0: none).
int decode_cluster_max_active(int group, int cluster, int warps_per_cta);
// Slots per tensor-core tile and per TMA chunk of the decode kernels.
constexpr int kDecodeChunk = 16;
// Slots of zero padding after the log-count array (16-slot chunk copies).
constexpr int kLogcPad = 16;

void set_error(const std::string& msg);

// Fault injection for tests (reskv_test_inject): whether the next decode
// launch is to report a timed-out first wait (consumes one pending launch),
// and every device allocation of the library, which fails as cudaMalloc out
// of memory when an injected failure is due.
bool take_test_wait_fault();
cudaError_t device_alloc(void** p, size_t bytes);

// Split plan of the tensor-core stream-K kernel for a launch of `n_units`
// units holding `total_slots` slots (largest unit `max_unit_slots`): W warps,
// wpc per CTA, k > 0 when every warp takes k whole units instead of an equal
// piece of chunks, and the ring stages per warp.  user_warps > 0 fixes W.
struct MmaPlan {
  int64_t W = 1;
  int wpc = kDecodeWarpsPerCta;
  int32_t k = 0;
  int stages = 0;
};
MmaPlan plan_mma_shape(int num_sms, int64_t max_warps, int32_t user_warps, int64_t max_unit_slots,
                       bool ragged, int64_t n_units, int64_t total_slots);
// TMA map of [rows, 128] bf16 rows (base 16-byte aligned) for 16-row chunk
// copies into the 128-byte swizzled stage layout [dims 0..63 of the 16 rows |
// dims 64..127 of the 16 rows].  rank 3: one copy per chunk, box {64 dims,
// 16 rows, 2 halves} over dims {64, rows, 2} whose halves lie 128 bytes apart;
// rank 2: two copies, box {64 dims, 16 rows} at dims 0 and 64.  False if the
// driver refuses the map.
bool encode_rows(CUtensorMap* map, const void* base, uint64_t rows, int rank);
// 128-row tiles of a [rows, 128] bf16 key array, both 64-dim halves in one
// copy, 128-byte swizzle (the Lloyd assignment's key tiles)
bool encode_key_tiles(CUtensorMap* map, const void* keys, uint64_t rows);

}  // namespace reskv

struct reskv_cache;
namespace reskv {
// Append one K and V row to each of `n` units starting at global unit `unit0`
// (K_new, V_new: [n, d] bf16); append.cu.
cudaError_t launch_append(reskv_cache* c, int64_t unit0, int64_t n, const __nv_bfloat16* K_new,
                          const __nv_bfloat16* V_new, cudaStream_t stream);
}  // namespace reskv

// The opaque handle of the C ABI.
struct reskv_cache {
  reskv_config cfg;             // residual_override cleared
  int device = 0;
  int num_sms = 0;
  int64_t n_units = 0;
  int32_t budget = 0;
  int32_t append_capacity = 0;
  int32_t stride = 0;           // budget + append_capacity (uniform layout)
  bool ragged = false;          // per-unit budgets: units at offsets[u]
  std::vector<int32_t> h_offsets;   // [U+1] first slot of every unit (host)
  int64_t total_slots = 0;
  int32_t max_unit_slots = 0;   // largest b_u + A
  std::vector<int32_t> n_app_max;   // per layer: max appended rows of its units (host copy)
  // layout (device)
  __nv_bfloat16* kslots = nullptr;
  __nv_bfloat16* vslots = nullptr;
  float* logc = nullptr;
  int32_t* slot_pos = nullptr;
  int32_t* counts = nullptr;
  int32_t* n_main = nullptr;
  int32_t* n_res = nullptr;
  int32_t* n_app = nullptr;
  int32_t* n_total = nullptr;   // [U] tokens appended since construction (ring order)
  int32_t* offsets = nullptr;   // [U+1]
  // decode workspace (device)
  float* partials = nullptr;
  int32_t* tickets = nullptr;
  uint32_t* status = nullptr;
  int max_warps = 0;
  // cluster decode shape for one-layer and all-layer launches; cluster = 0
  // when the launch's units do not fit on the device in one wave
  struct ClusterPlan {
    int cluster = 0;
    int warps_per_cta = 0;
  } cplan_layer, cplan_all;
  // plans of calls over other layer counts (reskv_decode_attn_layers), by
  // count; cluster = -1 until planned
  mutable std::vector<ClusterPlan> cplan_range;
  // reskv_decode_attn_host with pageable buffers: device staging of Q and O
  // for all layers (made by the first such call)
  struct HostIo {
    void* q = nullptr;
    void* o = nullptr;
  };
  mutable HostIo hio;
  // TMA maps of kslots / vslots over [U * budget rows, 128 dims] for 16-row
  // chunk copies with the 128-byte swizzle: rank 3 (one copy per chunk) or 2
  // (two 64-dim copies), see encode_rows
  CUtensorMap tmap_k;
  CUtensorMap tmap_v;
  int32_t kv_rank = 2;          // rank of both maps (encode_rows)
  // construction intermediates kept for reskv_export_debug (device)
  double* dbg_scores = nullptr;
  int32_t* dbg_ranked = nullptr;
  double* dbg_losses = nullptr;
  int64_t dbg_n_top = 0;
  std::vector<int32_t> candidates;   // one budget: r of every candidate column
  int32_t n_candidates = 0;          // candidate columns of the validation proxy
  int32_t ranked_width = 0;          // entries per unit of the kept ranking
  std::vector<int32_t> unit_cands;   // [U, n_candidates] r per column and unit (0: none)
  // device time of the construction stages (ms): scores, ranking, validation
  // targets, Lloyd, validation losses + choice of r, packing
  float build_ms[6] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
};
