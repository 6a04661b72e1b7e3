// Construction kernels (Alg. 1) -- token scoring, ranking, Lloyd residual
// entries, validation proxy and packing.  Included once, by construct.cu.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cfloat>
#include <climits>
#include <cstdint>

#include "device_utils.cuh"
#include "internal.h"

namespace reskv {
namespace build {

constexpr int kTile = 128;          // tokens per tile
constexpr int kRowBlk = 32;         // query rows per block
constexpr int kThreads = 256;       // 8 warps

// ---------------------------------------------------------------------------
// Shared-memory tiles
// ---------------------------------------------------------------------------

// Keys of a 128-token tile, fp32, dim-major, with the float4 column swizzled
// by (dim / 8) so that the transposing stores spread over banks.
__device__ __forceinline__ int kt_index(int k, int tok) {
  return k * kTile + ((((tok >> 2) ^ ((k >> 3) & 7)) << 2) | (tok & 3));
}

// Load rows [tok0, tok0 + 128) of a [s, d] bf16 matrix into Kt (zeros past s).
__device__ __forceinline__ void load_kt(float* Kt, const __nv_bfloat16* K, int64_t s, int64_t tok0) {
  for (int it = 0; it < 8; ++it) {
    const int idx = it * kThreads + threadIdx.x;
    const int tok = idx >> 4, dc = idx & 15;
    uint4 w = make_uint4(0, 0, 0, 0);
    if (tok0 + tok < s) w = __ldg(reinterpret_cast<const uint4*>(K + (tok0 + tok) * kHeadDim) + dc);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = bf16x2_to_float2(ws[j]);
      Kt[kt_index(8 * dc + 2 * j, tok)] = f.x;
      Kt[kt_index(8 * dc + 2 * j + 1, tok)] = f.y;
    }
  }
}

// Load 32 query rows (scaled) into Qt[k][row]; rows >= n_rows are zero.
// row r of the block is global row rowbase + r, read from rowptr(r).
template <typename RowPtr>
__device__ __forceinline__ void load_qt(float* Qt, int n_rows, float scale, RowPtr rowptr) {
  for (int it = 0; it < 2; ++it) {
    const int idx = it * kThreads + threadIdx.x;
    const int row = idx >> 4, dc = idx & 15;
    uint4 w = make_uint4(0, 0, 0, 0);
    if (row < n_rows) w = __ldg(reinterpret_cast<const uint4*>(rowptr(row)) + dc);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = bf16x2_to_float2(ws[j]);
      Qt[(8 * dc + 2 * j) * kRowBlk + row] = f.x * scale;
      Qt[(8 * dc + 2 * j + 1) * kRowBlk + row] = f.y * scale;
    }
  }
}

// S[4 rows][4 tokens] for warp w (rows 4w..4w+3) and lane (tokens 4l..4l+3).
__device__ __forceinline__ void tile_logits(const float* Qt, const float* Kt, float S[4][4]) {
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) S[i][j] = 0.f;
#pragma unroll 8
  for (int k = 0; k < kHeadDim; ++k) {
    const float4 q = *reinterpret_cast<const float4*>(Qt + k * kRowBlk + 4 * w);
    const float4 kk = *reinterpret_cast<const float4*>(Kt + k * kTile + ((lane ^ ((k >> 3) & 7)) << 2));
    const float qa[4] = {q.x, q.y, q.z, q.w};
    const float ka[4] = {kk.x, kk.y, kk.z, kk.w};
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) S[i][j] = fmaf(qa[i], ka[j], S[i][j]);
  }
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// ---------------------------------------------------------------------------
// Token scores (App. B.2 SnapKV rule; Alg. 1 step 2)
// ---------------------------------------------------------------------------

struct ObsArgs {
  const __nv_bfloat16* K;      // layer keys [UL, s, d]
  const __nv_bfloat16* Qobs;   // layer observation queries [UL*G, n_obs, d]
  int64_t s;
  int32_t G, n_obs, n_rows;    // n_rows = G * n_fit, row = g * n_fit + t
  int32_t n_fit;
  int32_t ntiles;
  float2* tile_stats;          // [UL, n_rows, ntiles] (max, sum) per tile, log2 domain
  float2* row_stats;           // [UL, n_rows] (max, 1/sum)
  float* A;                    // [UL, s] attention summed over fit rows, averaged over G
};

// Pass 1: per (row, tile) max and sum of 2^{a log2e} over the tile's tokens.
__global__ void __launch_bounds__(kThreads, 2) k_obs_pass1(ObsArgs p) {
  extern __shared__ __align__(16) float sm[];
  float* Kt = sm;
  float* Qt = sm + kHeadDim * kTile;
  const int tile = blockIdx.x, ul = blockIdx.y;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t tok0 = int64_t(tile) * kTile;
  load_kt(Kt, p.K + int64_t(ul) * p.s * kHeadDim, p.s, tok0);
  const float scale = kLog2e * rsqrtf(float(kHeadDim));
  for (int rb = 0; rb < p.n_rows; rb += kRowBlk) {
    __syncthreads();
    load_qt(Qt, min(kRowBlk, p.n_rows - rb), scale, [&](int r) {
      const int row = rb + r, g = row / p.n_fit, t = row % p.n_fit;
      return p.Qobs + ((int64_t(ul) * p.G + g) * p.n_obs + t) * kHeadDim;
    });
    __syncthreads();
    float S[4][4];
    tile_logits(Qt, Kt, S);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int row = rb + 4 * w + i;
      float mx = -INFINITY;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (tok0 + 4 * lane + j < p.s) mx = fmaxf(mx, S[i][j]);
      mx = warp_max(mx);
      float sum = 0.f;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (tok0 + 4 * lane + j < p.s) sum += exp2f(S[i][j] - mx);
      sum = warp_sum(sum);
      if (lane == 0 && row < p.n_rows)
        p.tile_stats[(int64_t(ul) * p.n_rows + row) * p.ntiles + tile] = make_float2(mx, sum);
    }
  }
}

// Row statistics over all tiles (in tile order).
__global__ void k_obs_rowstats(ObsArgs p, int UL) {
  const int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= int64_t(UL) * p.n_rows) return;
  const float2* t = p.tile_stats + i * p.ntiles;
  float mx = -INFINITY;
  for (int k = 0; k < p.ntiles; ++k) mx = fmaxf(mx, t[k].x);
  float sum = 0.f;
  for (int k = 0; k < p.ntiles; ++k) sum += t[k].y * exp2f(t[k].x - mx);
  p.row_stats[i] = make_float2(mx, 1.0f / sum);
}

// Pass 2: A_p = (1/G) sum over fit rows of the softmax weight of token p.
__global__ void __launch_bounds__(kThreads, 2) k_obs_pass2(ObsArgs p) {
  extern __shared__ __align__(16) float sm[];
  float* Kt = sm;
  float* Qt = sm + kHeadDim * kTile;
  float* red = Qt + kHeadDim * kRowBlk;        // [8 warps][128 tokens]
  const int tile = blockIdx.x, ul = blockIdx.y;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t tok0 = int64_t(tile) * kTile;
  load_kt(Kt, p.K + int64_t(ul) * p.s * kHeadDim, p.s, tok0);
  const float scale = kLog2e * rsqrtf(float(kHeadDim));
  float col[4] = {0.f, 0.f, 0.f, 0.f};
  for (int rb = 0; rb < p.n_rows; rb += kRowBlk) {
    __syncthreads();
    load_qt(Qt, min(kRowBlk, p.n_rows - rb), scale, [&](int r) {
      const int row = rb + r, g = row / p.n_fit, t = row % p.n_fit;
      return p.Qobs + ((int64_t(ul) * p.G + g) * p.n_obs + t) * kHeadDim;
    });
    __syncthreads();
    float S[4][4];
    tile_logits(Qt, Kt, S);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int row = rb + 4 * w + i;
      if (row >= p.n_rows) continue;
      const float2 st = p.row_stats[int64_t(ul) * p.n_rows + row];
#pragma unroll
      for (int j = 0; j < 4; ++j) col[j] += exp2f(S[i][j] - st.x) * st.y;
    }
  }
  __syncthreads();
#pragma unroll
  for (int j = 0; j < 4; ++j) red[w * kTile + 4 * lane + j] = col[j];
  __syncthreads();
  if (threadIdx.x < kTile) {
    float a = 0.f;
    for (int ww = 0; ww < kThreads / 32; ++ww) a += red[ww * kTile + threadIdx.x];
    const int64_t tok = tok0 + threadIdx.x;
    if (tok < p.s) p.A[int64_t(ul) * p.s + tok] = a / float(p.G);
  }
}

// Zero-padded average pooling of width `pool` (odd), summed in fp64.
__global__ void k_pool(const float* A, double* scores, int64_t s, int UL, int pool) {
  const int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= int64_t(UL) * s) return;
  const int64_t ul = i / s, pidx = i % s;
  const int half = pool / 2;
  double acc = 0.0;
  for (int j = -half; j <= half; ++j) {
    const int64_t q = pidx + j;
    if (q >= 0 && q < s) acc += double(A[ul * s + q]);
  }
  scores[i] = acc / double(pool);
}

// Query-free score ||k_p||^2, summed in fp64 over dims in order (no FMA).
__global__ void k_score_keynorm(const __nv_bfloat16* K, double* scores, int64_t n_rows) {
  const int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (i >= n_rows) return;
  const uint4* row = reinterpret_cast<const uint4*>(K + i * kHeadDim);
  double acc = 0.0;
  for (int c = 0; c < 16; ++c) {
    const uint4 w = __ldg(row + c);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = bf16x2_to_float2(ws[j]);
      acc = __dadd_rn(acc, __dmul_rn(double(f.x), double(f.x)));
      acc = __dadd_rn(acc, __dmul_rn(double(f.y), double(f.y)));
    }
  }
  scores[i] = acc;
}

// ---------------------------------------------------------------------------
// Ranking of S \ P (Sec. 5.2, Eq. main_selection): the top n_top positions by
// score, highest first, ties to the lower position.  One CTA per unit: radix
// select of the n_top-th largest key, order-preserving compaction, bitonic sort.
// ---------------------------------------------------------------------------

constexpr int kTopThreads = 1024;
constexpr int kTopMax = 8192;

struct TopArgs {
  const double* scores;   // [UL, s]
  int64_t s;
  int32_t recent;         // |P|
  int32_t n_top;          // entries to rank
  int32_t* top;           // [UL, n_top] positions in rank order
  int32_t* rank_pos;      // [UL, s]: rank, INT_MAX (never main) or -1 (protected)
  uint32_t* status;
};

__device__ __forceinline__ uint64_t score_key(double v) {
  // non-negative doubles order like their bit patterns; clamp -0 and negatives to 0
  return v > 0.0 ? static_cast<uint64_t>(__double_as_longlong(v)) : 0ull;
}

__device__ __forceinline__ int block_exclusive_scan(int v, int* warp_sums, int* total) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[w] = x;
  __syncthreads();
  if (w == 0) {
    int ws = lane < nw ? warp_sums[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, ws, o);
      if (lane >= o) ws += y;
    }
    if (lane < nw) warp_sums[lane] = ws;
  }
  __syncthreads();
  const int excl = x - v + (w > 0 ? warp_sums[w - 1] : 0);
  if (total) *total = warp_sums[nw - 1];
  __syncthreads();
  return excl;
}

__global__ void __launch_bounds__(kTopThreads, 1) k_topk(TopArgs p) {
  extern __shared__ __align__(16) uint8_t smraw[];
  uint64_t* skey = reinterpret_cast<uint64_t*>(smraw);                   // [kTopMax]
  int32_t* sidx = reinterpret_cast<int32_t*>(skey + kTopMax);            // [kTopMax]
  int* hist = reinterpret_cast<int*>(sidx + kTopMax);                     // [256]
  int* warp_sums = hist + 256;                                            // [32]
  int* bcast = warp_sums + 32;                                            // [4]
  const int ul = blockIdx.x;
  const int64_t s = p.s;
  const int64_t n_ev = s > p.recent ? s - p.recent : 0;
  const double* sc = p.scores + int64_t(ul) * s;
  int32_t* rp = p.rank_pos + int64_t(ul) * s;
  const int K = p.n_top;
  // protected window and default ranks
  for (int64_t i = threadIdx.x; i < s; i += blockDim.x) rp[i] = (i < n_ev) ? INT_MAX : -1;
  if (K <= 0) return;

  // radix select: threshold key tau with count(> tau) < K <= count(>= tau)
  uint64_t prefix = 0, mask = 0;
  int k_rem = K;
  for (int shift = 56; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int64_t i = threadIdx.x; i < n_ev; i += blockDim.x) {
      const uint64_t key = score_key(sc[i]);
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 0xff], 1);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int cum = 0, digit = 0;
      for (int d = 255; d >= 0; --d) {
        if (cum + hist[d] >= k_rem) {
          digit = d;
          break;
        }
        cum += hist[d];
      }
      bcast[0] = digit;
      bcast[1] = k_rem - cum;
    }
    __syncthreads();
    prefix |= uint64_t(bcast[0]) << shift;
    mask |= uint64_t(0xff) << shift;
    k_rem = bcast[1];
    __syncthreads();
  }
  const uint64_t tau = prefix;      // k_rem keys equal to tau are taken, lowest positions first

  // order-preserving compaction of the selected positions (contiguous chunks per thread)
  const int64_t chunk = (n_ev + blockDim.x - 1) / blockDim.x;
  const int64_t lo = int64_t(threadIdx.x) * chunk;
  const int64_t hi = lo + chunk < n_ev ? lo + chunk : n_ev;
  int n_gt = 0, n_eq = 0;
  for (int64_t i = lo; i < hi; ++i) {
    const uint64_t key = score_key(sc[i]);
    n_gt += key > tau;
    n_eq += key == tau;
  }
  const int eq_before = block_exclusive_scan(n_eq, warp_sums, nullptr);
  int take_eq = k_rem - eq_before;
  take_eq = take_eq < 0 ? 0 : (take_eq > n_eq ? n_eq : take_eq);
  int out = block_exclusive_scan(n_gt + take_eq, warp_sums, nullptr);
  for (int64_t i = lo; i < hi; ++i) {
    const uint64_t key = score_key(sc[i]);
    bool sel = key > tau;
    if (key == tau && take_eq > 0) {
      sel = true;
      --take_eq;
    }
    if (sel) {
      if (out < K) {
        skey[out] = key;
        sidx[out] = int32_t(i);
      } else if (p.status) {
        report_status(p.status, kStatusBadIndex);
      }
      ++out;
    }
  }
  int np2 = 1;
  while (np2 < K) np2 <<= 1;
  for (int i = K + threadIdx.x; i < np2; i += blockDim.x) {
    skey[i] = 0;
    sidx[i] = INT_MAX;      // padding sorts last
  }
  __syncthreads();
  // bitonic sort by (key descending, position ascending)
  for (int size = 2; size <= np2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int t = threadIdx.x; t < np2 / 2; t += blockDim.x) {
        const int i = 2 * t - (t & (stride - 1));
        const int j = i + stride;
        const bool up = ((i & size) == 0);
        const uint64_t ki = skey[i], kj = skey[j];
        const int32_t ii = sidx[i], ij = sidx[j];
        // "i before j" in the final order: larger key, then smaller position
        const bool i_first = (ki > kj) || (ki == kj && ii < ij);
        if (i_first != up) {
          skey[i] = kj;
          skey[j] = ki;
          sidx[i] = ij;
          sidx[j] = ii;
        }
      }
      __syncthreads();
    }
  }
  for (int i = threadIdx.x; i < K; i += blockDim.x) {
    const int32_t pos = sidx[i];
    p.top[int64_t(ul) * K + i] = pos;
    rp[pos] = i;
  }
}

}  // namespace build
}  // namespace reskv
