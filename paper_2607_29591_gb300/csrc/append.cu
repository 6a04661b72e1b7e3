// Decode-time growth of the cache (Sec. 3.1: each decode step appends the new
// token's key and value): one exact K row and V row per (batch, KV head) unit
// goes after the unit's main and residual slots and counts as a main-cache
// token from then on.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "device_utils.cuh"
#include "internal.h"

namespace reskv {
namespace {

struct AppendArgs {
  const __nv_bfloat16* K_new;   // [n, d]
  const __nv_bfloat16* V_new;
  __nv_bfloat16* kslots;
  __nv_bfloat16* vslots;
  float* logc;
  int32_t* slot_pos;
  int32_t* counts;
  const int32_t* n_main;
  const int32_t* n_res;
  int32_t* n_app;
  const int32_t* offsets;       // [U+1] unit starts, or NULL (uniform stride)
  int64_t unit0;
  int32_t stride;
  int32_t capacity;
  int64_t seq_len;
  uint32_t* status;
};

// One 16-thread block per unit; thread t copies dims 8t..8t+7 of K and V.
__global__ void __launch_bounds__(16) k_append(AppendArgs a) {
  const int64_t i = blockIdx.x, u = a.unit0 + i;
  const int t = threadIdx.x;
  const int na = a.n_app[u];
  if (na >= a.capacity) {              // the host checks capacity first
    if (t == 0) report_status(a.status, kStatusBadIndex);
    return;
  }
  const int64_t ubase = a.offsets ? int64_t(a.offsets[u]) : u * a.stride;
  const int64_t row = ubase + a.n_main[u] + a.n_res[u] + na;
  reinterpret_cast<uint4*>(a.kslots + row * kHeadDim)[t] =
      reinterpret_cast<const uint4*>(a.K_new + i * kHeadDim)[t];
  reinterpret_cast<uint4*>(a.vslots + row * kHeadDim)[t] =
      reinterpret_cast<const uint4*>(a.V_new + i * kHeadDim)[t];
  __syncthreads();                     // every thread has read n_app[u]
  if (t == 0) {
    a.slot_pos[row] = int32_t(a.seq_len + na);   // position of the token in the sequence
    a.counts[row] = 0;
    a.logc[row] = 0.f;
    a.n_app[u] = na + 1;
  }
  // The rows are visible device-wide before this grid completes: decode
  // kernels launched after it read the cache before their own grid
  // dependency wait.
  __threadfence();
}

}  // namespace

cudaError_t launch_append(reskv_cache* c, int64_t unit0, int64_t n, const __nv_bfloat16* K_new,
                          const __nv_bfloat16* V_new, cudaStream_t stream) {
  AppendArgs a{K_new, V_new, c->kslots, c->vslots, c->logc, c->slot_pos, c->counts,
               c->n_main, c->n_res, c->n_app, c->ragged ? c->offsets : nullptr, unit0,
               c->stride, c->append_capacity,
               c->cfg.seq_len, c->status};
  k_append<<<unsigned(n), 16, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace reskv
