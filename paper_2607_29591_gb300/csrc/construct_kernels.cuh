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
#include "mma_tile.cuh"

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

constexpr int kAsgRowBytes = kHeadDim * 2;  // one bf16 row of 128 dims

// byte offset of 16-byte chunk `ch` of row `row` in a [rows][256 B] bf16 tile;
// chunks XOR-swizzled by row so that ldmatrix reads of 8 rows are conflict free
__device__ __forceinline__ uint32_t asg_swz(int row, int ch) {
  return uint32_t(row) * kAsgRowBytes + uint32_t((ch ^ (row & 7)) << 4);
}

// 16-byte asynchronous copy global -> shared; src_bytes = 0 writes zeros
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(src_bytes)
               : "memory");
}

// Stage the bf16 keys of tokens tok0..tok0+127 as a swizzled [128][256 B]
// tile (zeros past s); the copies complete at the caller's wait.
__device__ __forceinline__ void stage_key_tile(uint32_t ks_s, const __nv_bfloat16* Ku, int64_t s,
                                               int64_t tok0) {
  for (int idx = threadIdx.x; idx < kTile * 16; idx += blockDim.x) {
    const int row = idx >> 4, ch = idx & 15;
    const bool in = tok0 + row < s;
    cp_async16(ks_s + asg_swz(row, ch), Ku + (in ? (tok0 + row) * kHeadDim : 0) + 8 * ch,
               in ? 16u : 0u);
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
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
// Token scores (App. B.2 SnapKV rule; Alg. 1)
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

// Logits of fit rows against a 128-token tile on the tensor cores: a warp
// takes 16 query rows at a time (rows 16 rb .. 16 rb + 15, A fragments straight
// from global memory), the keys are the B operand from the swizzled tile.
// Products of the bf16 rows and keys are exact, accumulated in fp32, then
// scaled by log2(e)/sqrt(d) (the logits in log2 units).  The accumulator of
// n-tile nt holds rows g (entries 0, 1) and g + 8 (entries 2, 3) at tokens
// 8 nt + 2 t4 (+1), with g = lane / 4, t4 = lane % 4.
__device__ __forceinline__ const uint32_t* obs_row(const ObsArgs& p, int ul, int row) {
  const int g = row / p.n_fit, t = row % p.n_fit;
  return reinterpret_cast<const uint32_t*>(p.Qobs +
                                           ((int64_t(ul) * p.G + g) * p.n_obs + t) * kHeadDim);
}

__device__ __forceinline__ void obs_afrag(const ObsArgs& p, int ul, int rb, int lane,
                                          uint32_t (&A)[8][4]) {
  const int g = lane >> 2, t4 = lane & 3;
  const int r0 = rb * 16 + g, r1 = r0 + 8;
  const uint32_t* q0 = r0 < p.n_rows ? obs_row(p, ul, r0) : nullptr;
  const uint32_t* q1 = r1 < p.n_rows ? obs_row(p, ul, r1) : nullptr;
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    A[ks][0] = q0 ? __ldg(q0 + 8 * ks + t4) : 0u;
    A[ks][1] = q1 ? __ldg(q1 + 8 * ks + t4) : 0u;
    A[ks][2] = q0 ? __ldg(q0 + 8 * ks + 4 + t4) : 0u;
    A[ks][3] = q1 ? __ldg(q1 + 8 * ks + 4 + t4) : 0u;
  }
}

// logits of the 16 rows against tokens 64 h .. 64 h + 63 of the tile
__device__ __forceinline__ void obs_half_logits(uint32_t ks_s, int h, int lane,
                                                const uint32_t (&A)[8][4], float (&S)[8][4]) {
  const int mi = lane >> 3;
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) S[nt][0] = S[nt][1] = S[nt][2] = S[nt][3] = 0.f;
#pragma unroll
  for (int np = 0; np < 4; ++np) {
    const int trow = 64 * h + 16 * np + (mi >> 1) * 8 + (lane & 7);
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      uint32_t b0, b1, b2, b3;
      ldsm_x4(ks_s + asg_swz(trow, 2 * ks + (mi & 1)), b0, b1, b2, b3);
      mma16816(S[2 * np], A[ks][0], A[ks][1], A[ks][2], A[ks][3], b0, b1);
      mma16816(S[2 * np + 1], A[ks][0], A[ks][1], A[ks][2], A[ks][3], b2, b3);
    }
  }
  const float scale = kLog2e * rsqrtf(float(kHeadDim));
#pragma unroll
  for (int nt = 0; nt < 8; ++nt)
#pragma unroll
    for (int e = 0; e < 4; ++e) S[nt][e] *= scale;
}

// Pass 1: per (row, tile) max and sum of 2^{a log2e} over the tile's tokens.
__global__ void __launch_bounds__(kThreads, 2) k_obs_pass1(ObsArgs p) {
  extern __shared__ __align__(128) uint8_t obs_raw[];
  const int tile = blockIdx.x, ul = blockIdx.y;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t4 = lane & 3;
  const int64_t tok0 = int64_t(tile) * kTile;
  const uint32_t ks_s = smem_u32(obs_raw);
  stage_key_tile(ks_s, p.K + int64_t(ul) * p.s * kHeadDim, p.s, tok0);
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  __syncthreads();
  for (int rb = w; rb * 16 < p.n_rows; rb += kThreads / 32) {
    uint32_t A[8][4];
    obs_afrag(p, ul, rb, lane, A);
    float M[2] = {-INFINITY, -INFINITY}, Lsum[2] = {0.f, 0.f};    // rows g, g + 8
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      float S[8][4];
      obs_half_logits(ks_s, h, lane, A, S);
#pragma unroll
      for (int a = 0; a < 2; ++a) {
        float mx = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt)
#pragma unroll
          for (int c = 0; c < 2; ++c)
            if (tok0 + 64 * h + 8 * nt + 2 * t4 + c < p.s) mx = fmaxf(mx, S[nt][2 * a + c]);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
        float sum = 0.f;
        if (mx != -INFINITY) {
#pragma unroll
          for (int nt = 0; nt < 8; ++nt)
#pragma unroll
            for (int c = 0; c < 2; ++c)
              if (tok0 + 64 * h + 8 * nt + 2 * t4 + c < p.s) sum += exp2f(S[nt][2 * a + c] - mx);
        }
        sum += __shfl_xor_sync(0xffffffffu, sum, 1);
        sum += __shfl_xor_sync(0xffffffffu, sum, 2);
        if (mx != -INFINITY) {                    // fold the half into the row's (max, sum)
          const float nm = fmaxf(M[a], mx);
          Lsum[a] = Lsum[a] * exp2f(M[a] - nm) + sum * exp2f(mx - nm);
          M[a] = nm;
        }
      }
    }
    if (t4 == 0) {
#pragma unroll
      for (int a = 0; a < 2; ++a) {
        const int row = rb * 16 + g + 8 * a;
        if (row < p.n_rows)
          p.tile_stats[(int64_t(ul) * p.n_rows + row) * p.ntiles + tile] =
              make_float2(M[a], Lsum[a]);
      }
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
  for (int k = 0; k < p.ntiles; ++k)
    if (t[k].y > 0.f) sum += t[k].y * exp2f(t[k].x - mx);
  p.row_stats[i] = make_float2(mx, 1.0f / sum);
}

// Pass 2: A_p = (1/G) sum over fit rows of the softmax weight of token p.
__global__ void __launch_bounds__(kThreads, 2) k_obs_pass2(ObsArgs p) {
  extern __shared__ __align__(128) uint8_t obs_raw[];
  float* red = reinterpret_cast<float*>(obs_raw + kTile * kAsgRowBytes);   // [8 warps][128 tokens]
  const int tile = blockIdx.x, ul = blockIdx.y;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t4 = lane & 3;
  const int64_t tok0 = int64_t(tile) * kTile;
  const uint32_t ks_s = smem_u32(obs_raw);
  stage_key_tile(ks_s, p.K + int64_t(ul) * p.s * kHeadDim, p.s, tok0);
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  __syncthreads();
  for (int h = 0; h < 2; ++h) {                  // tokens 64 h .. 64 h + 63
    float col[8][2];                             // this lane's column sums
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) col[nt][0] = col[nt][1] = 0.f;
    for (int rb = w; rb * 16 < p.n_rows; rb += kThreads / 32) {
      uint32_t A[8][4];
      obs_afrag(p, ul, rb, lane, A);
      float2 st[2];
#pragma unroll
      for (int a = 0; a < 2; ++a) {
        const int row = rb * 16 + g + 8 * a;
        st[a] = row < p.n_rows ? p.row_stats[int64_t(ul) * p.n_rows + row] : make_float2(0.f, 0.f);
      }
      float S[8][4];
      obs_half_logits(ks_s, h, lane, A, S);
#pragma unroll
      for (int nt = 0; nt < 8; ++nt)
#pragma unroll
        for (int c = 0; c < 2; ++c)
#pragma unroll
          for (int a = 0; a < 2; ++a)
            if (st[a].y > 0.f) col[nt][c] += exp2f(S[nt][2 * a + c] - st[a].x) * st[a].y;
    }
    // sum over the eight row groups of the warp (the warps are summed below)
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        float v = col[nt][c];
        v += __shfl_xor_sync(0xffffffffu, v, 4);
        v += __shfl_xor_sync(0xffffffffu, v, 8);
        v += __shfl_xor_sync(0xffffffffu, v, 16);
        if (g == 0) red[w * kTile + 64 * h + 8 * nt + 2 * t4 + c] = v;
      }
  }
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

// Query-free score ||k_p||^2 (a build choice; the paper defines none): the
// exact sum of the squares, rounded once to the nearest fp64 value (ties to
// even), so it does not depend on any summation order.
//
// A bf16 value is M 2^e with an integer M < 2^8 (M = 128 + mantissa field for
// normal values, the mantissa field for subnormals), so its square is
// M^2 2^t with M^2 < 2^16 and t = 2e even, t in [-266, 242].  One warp per
// row, four dims per lane.  With tmax the largest t of the row's nonzero
// squares, every square with t >= tmax - 104 is an exact integer multiple of
// 2^(tmax - 104) below 2^120, and 128 of them sum below 2^127: the warp adds
// them as 128-bit integers and one lane rounds the sum.  A row with a
// nonzero square below that window (its values span more than 52 binades)
// goes to an exact 576-bit accumulator in one lane.

using u128 = unsigned __int128;

// Correctly rounded fp64 value of a 2^base, a > 0; `sticky`: a positive
// amount below a's last bit is to be added as well.
__device__ inline double round_u128(u128 a, int base, bool sticky) {
  const uint64_t hi = uint64_t(a >> 64), lo = uint64_t(a);
  const int p = hi ? 127 - __clzll((long long)hi) : 63 - __clzll((long long)lo);
  if (p <= 52) return ldexp(double(lo), base);            // exact (sticky never set here)
  const int sh = p - 52;
  uint64_t mant = uint64_t(a >> sh);
  const u128 one = 1;
  const u128 rem = a & ((one << sh) - 1), half = one << (sh - 1);
  if (rem > half || (rem == half && (sticky || (mant & 1u)))) ++mant;
  return ldexp(double(mant), base + sh);
}

// The square of one bf16 value as (M^2, t); M^2 = 0 for zero.
__device__ inline void bf16_square(uint32_t b, uint32_t& m2, int& t, bool& finite) {
  const uint32_t ef = (b >> 7) & 0xffu, mf = b & 0x7fu;
  const uint32_t M = ef ? 128u + mf : mf;
  m2 = M * M;
  t = 2 * (int(ef ? ef : 1u) - 134);
  finite = ef != 0xffu;
}

// Exact sum of a row's squares in 32-bit digits (bit q = t + 266 of the sum
// in digit q / 32), then the correctly rounded fp64 value.  One thread.
__device__ double keynorm_wide(const __nv_bfloat16* rowp) {
  const uint16_t* bits = reinterpret_cast<const uint16_t*>(rowp);
  uint64_t dig[18];
#pragma unroll
  for (int j = 0; j < 18; ++j) dig[j] = 0;
  for (int i = 0; i < kHeadDim; ++i) {
    uint32_t m2;
    int t;
    bool fin;
    bf16_square(bits[i], m2, t, fin);
    if (!m2) continue;
    const int q = t + 266;
    const uint64_t v = uint64_t(m2) << (q & 31);
    dig[q >> 5] += v & 0xffffffffu;
    dig[(q >> 5) + 1] += v >> 32;
  }
  for (int j = 0; j < 17; ++j) {
    dig[j + 1] += dig[j] >> 32;
    dig[j] &= 0xffffffffu;
  }
  int top = 17;
  while (top > 0 && dig[top] == 0) --top;
  u128 a = 0;
  for (int j = top; j > top - 4; --j) a = (a << 32) | (j >= 0 ? dig[j] : 0u);
  bool sticky = false;
  for (int j = 0; j < top - 3; ++j) sticky |= dig[j] != 0;
  return a ? round_u128(a, (top - 3) * 32 - 266, sticky) : 0.0;
}

// One warp per row; the grid covers n_rows warps (blockDim a multiple of 32).
__global__ void k_score_keynorm(const __nv_bfloat16* K, double* scores, int64_t n_rows) {
  const int64_t row = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= n_rows) return;                              // whole warps leave together
  const uint2 w = __ldg(reinterpret_cast<const uint2*>(K + row * kHeadDim) + lane);
  const uint32_t b[4] = {w.x & 0xffffu, w.x >> 16, w.y & 0xffffu, w.y >> 16};
  uint32_t m2[4];
  int t[4];
  bool finite = true;
  int tmax = INT_MIN;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    bool f;
    bf16_square(b[j], m2[j], t[j], f);
    finite &= f;
    if (m2[j]) tmax = max(tmax, t[j]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) tmax = max(tmax, __shfl_xor_sync(0xffffffffu, tmax, o));
  if (!__all_sync(0xffffffffu, finite)) {                 // inf or NaN: the fp64 sum is too
    double acc = 0.0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const double x = double(__uint_as_float(b[j] << 16));
      acc += x * x;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) scores[row] = acc;
    return;
  }
  if (tmax == INT_MIN) {                                  // every value is zero
    if (lane == 0) scores[row] = 0.0;
    return;
  }
  bool wide = false;
#pragma unroll
  for (int j = 0; j < 4; ++j) wide |= m2[j] != 0 && t[j] < tmax - 104;
  if (__any_sync(0xffffffffu, wide)) {
    if (lane == 0) scores[row] = keynorm_wide(K + row * kHeadDim);
    return;
  }
  u128 a = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j)
    if (m2[j]) a += u128(m2[j]) << (t[j] - tmax + 104);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t hi = __shfl_xor_sync(0xffffffffu, uint64_t(a >> 64), o);
    const uint64_t lo = __shfl_xor_sync(0xffffffffu, uint64_t(a), o);
    a += (u128(hi) << 64) | lo;
  }
  if (lane == 0) scores[row] = round_u128(a, tmax - 104, false);
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
  const int32_t* budgets; // [UL] per-unit budgets (rank min(b_u, s) - |P| each,
                          // at stride n_top), or NULL: rank n_top for every unit
};

// Budget of unit ul of the layer: its own, or the shared one.
__device__ __forceinline__ int64_t unit_budget(const int32_t* budgets, int ul, int64_t b) {
  return budgets ? int64_t(budgets[ul]) : b;
}

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
  int K = p.n_top;
  if (p.budgets) {
    const int64_t keep = (p.budgets[ul] < s ? int64_t(p.budgets[ul]) : s) - p.recent;
    K = keep < 0 ? 0 : int(keep);
    if (K > p.n_top) {
      if (threadIdx.x == 0 && p.status) report_status(p.status, kStatusBadIndex);
      K = p.n_top;
    }
  }
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
    p.top[int64_t(ul) * p.n_top + i] = pos;
    rp[pos] = i;
  }
}

// ---------------------------------------------------------------------------
// AdaKV budgets across the KV heads of one (layer, batch element) (App. B,
// "AdaKV": token scores as importance, safeguard coefficient).  Every head
// keeps |P| + f slots (its window and its f best-ranked tokens, which a
// ranking of the top f has marked in rank_pos); the n_free other slots go to
// the highest-scored remaining evictable tokens of all heads, ordered by
// (score desc, head asc, position asc).  One CTA per batch element: a radix
// select of the n_free-th largest key over the heads' remaining tokens, then
// per-head counts above and at the threshold.
// ---------------------------------------------------------------------------

struct AdaArgs {
  const double* scores;      // [UL, s]
  const int32_t* rank_pos;   // [UL, s]: rank < f marks a head's safeguard tokens
  int64_t s;
  int32_t recent;            // |P| (clamped to s)
  int32_t n_heads;           // H_kv; unit ul = batch * H_kv + h
  int32_t f;                 // safeguard tokens per head
  int32_t base;              // |P| + f
  int64_t n_free;            // H_kv * (b - |P| - f)
  int32_t* budgets;          // [UL] out
};

__global__ void __launch_bounds__(kTopThreads, 1) k_adakv(AdaArgs p) {
  __shared__ int hist[256];
  __shared__ int bcast[2];
  __shared__ int cnt[2];
  const int grp = blockIdx.x, H = p.n_heads;
  const int64_t s = p.s, n_ev = s > p.recent ? s - p.recent : 0;
  const int ul0 = grp * H;
  if (p.n_free <= 0) {
    for (int h = threadIdx.x; h < H; h += blockDim.x) p.budgets[ul0 + h] = p.base;
    return;
  }
  // radix select: threshold key tau with count(> tau) < n_free <= count(>= tau)
  uint64_t prefix = 0, mask = 0;
  int64_t k_rem = p.n_free;
  for (int shift = 56; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    for (int h = 0; h < H; ++h) {
      const double* sc = p.scores + int64_t(ul0 + h) * s;
      const int32_t* rp = p.rank_pos + int64_t(ul0 + h) * s;
      for (int64_t i = threadIdx.x; i < n_ev; i += blockDim.x) {
        if (rp[i] < p.f) continue;                       // the head's safeguard token
        const uint64_t key = score_key(sc[i]);
        if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 0xff], 1);
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int64_t cum = 0;
      int digit = 0;
      for (int d = 255; d >= 0; --d) {
        if (cum + hist[d] >= k_rem) {
          digit = d;
          break;
        }
        cum += hist[d];
      }
      bcast[0] = digit;
      bcast[1] = int(k_rem - cum);
    }
    __syncthreads();
    prefix |= uint64_t(bcast[0]) << shift;
    mask |= uint64_t(0xff) << shift;
    k_rem = bcast[1];
    __syncthreads();
  }
  const uint64_t tau = prefix;   // k_rem keys equal to tau are taken: lower heads first
  int64_t eq_before = 0;
  for (int h = 0; h < H; ++h) {
    if (threadIdx.x == 0) cnt[0] = cnt[1] = 0;
    __syncthreads();
    const double* sc = p.scores + int64_t(ul0 + h) * s;
    const int32_t* rp = p.rank_pos + int64_t(ul0 + h) * s;
    int gt = 0, eq = 0;
    for (int64_t i = threadIdx.x; i < n_ev; i += blockDim.x) {
      if (rp[i] < p.f) continue;
      const uint64_t key = score_key(sc[i]);
      gt += key > tau;
      eq += key == tau;
    }
    if (gt) atomicAdd(&cnt[0], gt);
    if (eq) atomicAdd(&cnt[1], eq);
    __syncthreads();
    if (threadIdx.x == 0) {
      int64_t take_eq = k_rem - eq_before;
      take_eq = take_eq < 0 ? 0 : (take_eq > cnt[1] ? cnt[1] : take_eq);
      p.budgets[ul0 + h] = p.base + cnt[0] + int32_t(take_eq);
    }
    eq_before += cnt[1];
    __syncthreads();
  }
}


// ---------------------------------------------------------------------------
// Residual entries by Lloyd's algorithm (Sec. 5.3, Eqs. residual_partition,
// summary; App. B: 4 iterations, initial centres = the highest-scored evicted
// keys).  One "run" builds r_unit[ul] entries for every unit of the layer.
// E = S \ M_r = { p < s - |P| : rank_pos[p] >= m - |P| },  m = b - r.
// Deterministic: assignments by (distance, centre index); member sums in
// fp64 in token order (stable counting sort); no float atomics.
// ---------------------------------------------------------------------------

constexpr int kMaxR = 8192;

struct LloydArgs {
  const __nv_bfloat16* K;      // layer keys [UL, s, d]
  const __nv_bfloat16* V;      // layer values
  int64_t s;
  int32_t recent;              // |P| (already clamped to s)
  int32_t n_top;
  int32_t budget;
  int32_t ntiles;
  int32_t rmax;
  const int32_t* top;          // [UL, n_top]
  const int32_t* rank_pos;     // [UL, s]
  const int32_t* r_unit;       // [UL]
  float* centersT;             // [UL, d, rmax]  fp32 copy (dim-major) for the fast path
  float* cnorm;                // [UL, rmax]     ||c||^2 of the fp32 copy
  double* centers64;           // [UL, rmax, d]  the centres (fp64 means)
  int32_t* assign;             // [UL, s] centre index, -1 outside E
  int32_t* hist;               // [UL, ntiles, rmax] per-tile counts, then offsets
  int32_t* ccount;             // [UL, rmax] members per centre
  int32_t* cbase;              // [UL, rmax] first member slot per centre
  int32_t* members;            // [UL, s] token positions grouped by centre
  __nv_bfloat16* kbar;         // [UL, ent_stride, d] entries of this run at ent_off
  __nv_bfloat16* vbar;
  int32_t* ecount;             // [UL, ent_stride]
  int64_t ent_stride;
  int32_t ent_off;
  uint32_t* status;
  const int32_t* budgets;      // [UL] per-unit budgets, or NULL (budget)
  __nv_bfloat16* cplanes;      // [UL, 2, rmax, d] the fp32 centres split into
                               // two bf16 planes c1 + c2 (tensor-core operands)
  long long* msum;             // [UL, rmax, 2, d] fixed-point member sums (K, V); zero between passes
  uint32_t* mflag;             // [UL, rmax] set when a member value is outside the fixed-point range
  float* knorm2;               // [UL, s] fp32 ||k||^2 of every key (the persistent assignment's bound)
  int4* amb;                   // [UL * s] tokens the persistent assignment leaves to k_lloyd_resolve
  int* amb_count;              // their number (zeroed before each assignment)
  float* centers32;            // [UL, rmax, d] row-major fp32 copy of the centres
  // the previous iteration's assignment and member lists (delta accumulation)
  const int32_t* assign_prev;
  const int32_t* members_prev;
  const int32_t* cbase_prev;
  const int32_t* ccount_prev;
  uint32_t* moved;             // [UL * s / 32] bit per token: its centre changed (delta accumulation)
  int32_t test_fault;          // test hook: CTA 0's certifier gives up its first wait
};

__device__ __forceinline__ bool in_evicted(const LloydArgs& p, int ul, int64_t pos, int r) {
  const int32_t rk = p.rank_pos[int64_t(ul) * p.s + pos];
  const int32_t keep = int32_t(unit_budget(p.budgets, ul, p.budget)) - r - p.recent;  // ranked main
  return rk >= 0 && rk >= keep;
}

// The bf16 planes of centre j, dim d: c = c1 + c2 + e, |e| <= 2^-16 |c| (the
// remainder c - c1 is exact in fp32; each plane keeps 8 significant bits).
__device__ __forceinline__ void write_planes(const LloydArgs& p, int ul, int j, int d, float c) {
  const __nv_bfloat16 c1 = __float2bfloat16_rn(c);
  const __nv_bfloat16 c2 = __float2bfloat16_rn(c - __bfloat162float(c1));
  __nv_bfloat16* b = p.cplanes + (int64_t(ul) * 2 * p.rmax + j) * kHeadDim + d;
  b[0] = c1;
  b[int64_t(p.rmax) * kHeadDim] = c2;
}

// centre j = key of the (m - |P| + j)-th ranked token
__global__ void k_lloyd_init(LloydArgs p) {
  __shared__ float red[kHeadDim];
  const int j = blockIdx.x, ul = blockIdx.y, d = threadIdx.x;
  const int r = p.r_unit[ul];
  if (j >= r) return;
  const int32_t keep = int32_t(unit_budget(p.budgets, ul, p.budget)) - r - p.recent;
  const int32_t pos = p.top[int64_t(ul) * p.n_top + keep + j];
  const float c = __bfloat162float(p.K[(int64_t(ul) * p.s + pos) * kHeadDim + d]);
  p.centersT[(int64_t(ul) * kHeadDim + d) * p.rmax + j] = c;
  write_planes(p, ul, j, d, c);
  p.centers64[(int64_t(ul) * p.rmax + j) * kHeadDim + d] = double(c);
  p.centers32[(int64_t(ul) * p.rmax + j) * kHeadDim + d] = c;
  red[d] = c * c;
  __syncthreads();
  if (d == 0) {
    float n = 0.f;
    for (int i = 0; i < kHeadDim; ++i) n += red[i];
    p.cnorm[int64_t(ul) * p.rmax + j] = n;
  }
}

// Lloyd assignment (k_lloyd_assign_tc, lloyd_tc.cuh): best (d0, j0), second
// best (d1, j1) and third-best distance d2 of the centres seen so far for one
// token; centres arrive in increasing index, so strict comparisons keep the
// lower index on ties
__device__ __forceinline__ void top3_insert(float& d0, int& j0, float& d1, int& j1, float& d2,
                                            float x, int jx) {
  const bool c0 = x < d0, c1 = x < d1, c2 = x < d2;
  d2 = c1 ? d1 : (c2 ? x : d2);
  d1 = c0 ? d0 : (c1 ? x : d1);
  j1 = c0 ? j0 : (c1 ? jx : j1);
  d0 = c0 ? x : d0;
  j0 = c0 ? jx : j0;
}

// Per centre: the member count of each tile becomes the tile's offset within
// the centre's members (an exclusive prefix over tiles, in place), and the
// total its count.  A CTA takes 32 centres of a unit; its 8 warps split the
// tiles into 8 segments (coalesced over the 32 centres), sum them, and
// rewrite their segment from the prefix of the segments before.
constexpr int kScanCentres = 32;
constexpr int kScanSegs = 8;

__global__ void __launch_bounds__(kScanCentres * kScanSegs) k_lloyd_scan(LloydArgs p) {
  __shared__ int seg[kScanSegs][kScanCentres];
  const int ul = blockIdx.x;
  const int r = p.r_unit[ul];
  if (int(blockIdx.y) * kScanCentres >= r) return;
  const int lane = threadIdx.x & 31, sg = threadIdx.x >> 5;
  const int c = blockIdx.y * kScanCentres + lane;
  const bool live = c < r;
  const int T = p.ntiles, t0 = T * sg / kScanSegs, t1 = T * (sg + 1) / kScanSegs;
  int32_t* h = p.hist + int64_t(ul) * T * p.rmax + c;
  int sum = 0;
  if (live) {
    int t = t0;
    for (; t + 16 <= t1; t += 16) {            // 16 independent loads in flight
      int v[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) v[u] = h[int64_t(t + u) * p.rmax];
#pragma unroll
      for (int u = 0; u < 16; ++u) sum += v[u];
    }
    for (; t < t1; ++t) sum += h[int64_t(t) * p.rmax];
  }
  seg[sg][lane] = sum;
  __syncthreads();
  int run = 0;
  for (int k = 0; k < sg; ++k) run += seg[k][lane];
  if (live) {
    int t = t0;
    for (; t + 16 <= t1; t += 16) {
      int v[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) v[u] = h[int64_t(t + u) * p.rmax];
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        h[int64_t(t + u) * p.rmax] = run;
        run += v[u];
      }
    }
    for (; t < t1; ++t) {
      const int v = h[int64_t(t) * p.rmax];
      h[int64_t(t) * p.rmax] = run;
      run += v;
    }
    if (sg == kScanSegs - 1) p.ccount[int64_t(ul) * p.rmax + c] = run;
  }
}

// Per unit: centre j's members start at cbase[j], the exclusive prefix of
// the counts.
__global__ void k_lloyd_bases(LloydArgs p) {
  __shared__ int warp_sums[32];
  const int ul = blockIdx.x;
  const int r = p.r_unit[ul];
  if (r == 0) return;
  const int per = (r + blockDim.x - 1) / blockDim.x;      // centres per thread (contiguous)
  const int32_t* cc = p.ccount + int64_t(ul) * p.rmax;
  int mine = 0;
  for (int q = 0; q < per; ++q) {
    const int j = threadIdx.x * per + q;
    if (j < r) mine += cc[j];
  }
  int base = block_exclusive_scan(mine, warp_sums, nullptr);
  for (int q = 0; q < per; ++q) {
    const int j = threadIdx.x * per + q;
    if (j < r) {
      p.cbase[int64_t(ul) * p.rmax + j] = base;
      base += cc[j];
    }
  }
}

// stable scatter of evicted tokens into per-centre member lists
__global__ void k_lloyd_scatter(LloydArgs p) {
  __shared__ int a_s[kTile];
  const int tile = blockIdx.x, ul = blockIdx.y;
  const int r = p.r_unit[ul];
  if (r == 0) return;
  const int t = threadIdx.x;
  const int64_t pos = int64_t(tile) * kTile + t;
  const int a = pos < p.s ? p.assign[int64_t(ul) * p.s + pos] : -1;
  a_s[t] = a;
  __syncthreads();
  if (a < 0) return;
  if (a >= r) {                        // only after a failed assignment
    report_status(p.status, kStatusBadIndex);
    return;
  }
  int rank = 0;
  for (int i = 0; i < t; ++i) rank += (a_s[i] == a);
  const int64_t off = p.cbase[int64_t(ul) * p.rmax + a] +
                      p.hist[(int64_t(ul) * p.ntiles + tile) * p.rmax + a] + rank;
  if (off < 0 || off >= p.s) {         // counts inconsistent with the assignment: the same
    report_status(p.status, kStatusBadIndex);
    return;
  }
  p.members[int64_t(ul) * p.s + off] = int32_t(pos);
}

// New centre = mean key of its members; on the last iteration also the mean
// value, and the stored bf16 entry (Eq. summary).  The member sums are exact
// fixed-point integers, so they are free of summation order, and the
// conversion of the total to fp64 is the exact sum rounded once; mean = that
// sum / count.  If a member value is outside the fixed-point range the centre
// is summed in fp64 in member order instead.
//
// Two kernels.  k_lloyd_accum sweeps the member list (grouped by centre)
// token-parallel: each warp takes kAccRowsPerWarp consecutive member slots,
// gathers their rows, keeps running sums for the centre it is in, and adds
// them into msum[ul][j] with 64-bit integer atomics when the centre changes.
// Integer addition is associative, so the totals do not depend on the order
// the atomics land in.  k_lloyd_finish then forms the means, one CTA per
// centre, and clears msum / mflag for the next pass.
//
// The running sums split every member value on the FP32 pipe, with two
// magic-number roundings (no integer shifts, which would bound the kernel on
// the integer ALU).  For |x| < 128 and x a multiple of 2^-32:
//   s = x + C1 (C1 = 1.5 * 2^8; s lies in [256, 512), whose ulp is 2^-15),
//   h = s - C1 (x rounded to a multiple of 2^-15; exact), l = x - h (exact,
//   |l| <= 2^-16), t = l + C2 (C2 = 1.5 * 2^-9; t lies in [2^-9, 2^-8), ulp
//   2^-32, so t is exact).
// Then bits(s) - bits(C1) = h * 2^15 and bits(t) - bits(C2) = l * 2^32 as
// integers, so a lane adds bits(s) and bits(t) into 32-bit sums (mod 2^32)
// and the flush subtracts n * bits(C) for the n rows added: the exact
// |sum h * 2^15| < 2^28 and |sum l * 2^32| <= 2^22 for n <= 64.  The flush
// joins them into the 64-bit total (sum h * 2^15) * 2^17 + sum l * 2^32
// (unit 2^-32).  A value outside the window shows as t - C2 != l (inexact:
// a subnormal, a tail below 2^-32, inf, NaN) or as |x| >= 128; the centre is
// then summed in fp64 instead.  Below 128 a sum of 2^17 terms stays under 2^63.
constexpr int kAccRowsPerWarp = 64;
constexpr int kAccRows = kAccRowsPerWarp * (kThreads / 32);   // member slots per CTA
static_assert(kAccRowsPerWarp <= 64, "the mod-2^32 lane sums must stay below 2^31");
constexpr float kFixC1 = 384.0f;
constexpr float kFixC2 = 0x1.8p-9f;

struct FixSum {
  uint32_t hi[4], lo[4];
};

struct FixState {
  float err, mx;                 // sum of |t - C2 - l|, max |x|: exact iff 0 and < 128
};

__device__ __forceinline__ void fix_add(float x, uint32_t& hi, uint32_t& lo, FixState& st) {
  const float s = __fadd_rn(x, kFixC1);
  const float h = __fadd_rn(s, -kFixC1);
  const float l = __fadd_rn(x, -h);
  const float t = __fadd_rn(l, kFixC2);
  st.err = __fadd_rn(st.err, fabsf(__fadd_rn(__fadd_rn(t, -kFixC2), -l)));
  st.mx = fmaxf(st.mx, fabsf(x));
  hi += __float_as_uint(s);
  lo += __float_as_uint(t);
}

// four consecutive bf16 (two words, low half first) into the lane sums
__device__ __forceinline__ void acc_row(uint2 w, FixSum& a, FixState& st) {
  fix_add(__uint_as_float(w.x << 16), a.hi[0], a.lo[0], st);
  fix_add(__uint_as_float(w.x & 0xffff0000u), a.hi[1], a.lo[1], st);
  fix_add(__uint_as_float(w.y << 16), a.hi[2], a.lo[2], st);
  fix_add(__uint_as_float(w.y & 0xffff0000u), a.hi[3], a.lo[3], st);
}

// dim q's 64-bit fixed-point total of n added rows; the lane sums are cleared
__device__ __forceinline__ unsigned long long fix_total(FixSum& a, int q, uint32_t n) {
  const int32_t h = int32_t(a.hi[q] - n * __float_as_uint(kFixC1));
  const int32_t l = int32_t(a.lo[q] - n * __float_as_uint(kFixC2));
  a.hi[q] = 0u;
  a.lo[q] = 0u;
  return static_cast<unsigned long long>(((long long)h << 17) + (long long)l);
}

// values = false: the key sums (every pass); values = true: the value sums
// (the last pass), a launch of their own so each keeps 8 rows in flight per
// warp at full occupancy.
// delta = 0: every member of the current lists.  Once few tokens move, the
// key sums are updated instead (integer sums: the update is exact):
// delta = +1 adds the members of the current lists whose centre changed, and
// delta = -1 subtracts the members of the previous lists whose centre changed
// (a bit of the moved-token bitmap per member; rows of movers only).  An
// inexact value that joins raises the centre's flag; flags are kept while the
// sums are (a flagged centre is summed again in fp64 from its members).
// the moved-token bitmap of the iteration: token t's bit in word t / 32
__global__ void k_lloyd_moved(LloydArgs p, int64_t n_tok) {
  const int64_t t = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  const bool mv = t < n_tok && p.assign[t] != p.assign_prev[t];
  const unsigned b = __ballot_sync(0xffffffffu, mv);
  if ((threadIdx.x & 31) == 0 && t < n_tok) p.moved[t >> 5] = b;
}

template <bool values, int delta>
__global__ void __launch_bounds__(kThreads) k_lloyd_accum(LloydArgs p) {
  static_assert(delta == 0 || !values, "value sums are taken in full");
  const int ul = blockIdx.y;
  const int r = p.r_unit[ul];
  if (r <= 0) return;
  const int32_t* cb = (delta < 0 ? p.cbase_prev : p.cbase) + int64_t(ul) * p.rmax;
  const int32_t* cc = (delta < 0 ? p.ccount_prev : p.ccount) + int64_t(ul) * p.rmax;
  // (the clamps below only act after a failed assignment, whose status is raised)
  const int n_mem = min(cb[r - 1] + cc[r - 1], int(p.s));
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int lo = blockIdx.x * kAccRows + w * kAccRowsPerWarp;
  if (lo >= n_mem) return;
  const int hi = min(n_mem, lo + kAccRowsPerWarp);
  // the centre holding slot lo: the last j with cbase[j] <= lo (it is never
  // empty: an empty centre shares its cbase with the next one)
  int j = 0;
  for (int step = 1 << (31 - __clz(max(r - 1, 1))); step > 0; step >>= 1)
    if (j + step < r && cb[j + step] <= lo) j += step;
  int bnd = cb[j] + cc[j];
  const int32_t* mem = (delta < 0 ? p.members_prev : p.members) + int64_t(ul) * p.s;
  const __nv_bfloat16* Xb = (values ? p.V : p.K) + int64_t(ul) * p.s * kHeadDim + 4 * lane;
  unsigned long long* ms = reinterpret_cast<unsigned long long*>(p.msum) +
                           int64_t(ul) * p.rmax * 2 * kHeadDim + (values ? kHeadDim : 0) + 4 * lane;
  FixSum sk = {};
  FixState st = {0.0f, 0.0f};
  uint32_t n = 0;                 // rows in the lane sums
  auto flush = [&](int jj) {
    unsigned long long* m = ms + int64_t(jj) * 2 * kHeadDim;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const unsigned long long v = fix_total(sk, q, n);
      atomicAdd(m + q, delta < 0 ? 0ull - v : v);
    }
    const bool ok = st.err == 0.0f && st.mx < 128.0f;
    if (delta >= 0 && __any_sync(0xffffffffu, !ok) && lane == 0)
      atomicOr(p.mflag + int64_t(ul) * p.rmax + jj, 1u);
    st = FixState{0.0f, 0.0f};
    n = 0;
  };
  for (int i32 = lo; i32 < hi; i32 += 32) {
    // a member position outside the unit only follows a failed assignment
    // (its status is raised): read row 0 instead of leaving the array
    int my = i32 + lane < hi ? mem[i32 + lane] : 0;
    my = uint32_t(my) < uint32_t(p.s) ? my : 0;
    if constexpr (delta != 0) {
      // the block's movers, in list order, 8 rows at a time
      bool mv = false;
      if (i32 + lane < hi) {
        const int64_t t = int64_t(ul) * p.s + my;
        mv = (p.moved[t >> 5] >> (t & 31)) & 1u;
      }
      unsigned take = __ballot_sync(0xffffffffu, mv);
      while (take) {
        int idx[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          idx[q] = take ? __ffs(take) - 1 : -1;
          take &= take - 1;
        }
        uint2 kw[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const int64_t pos = __shfl_sync(0xffffffffu, my, idx[q] < 0 ? 0 : idx[q]);
          if (idx[q] >= 0) kw[q] = __ldg(reinterpret_cast<const uint2*>(Xb + pos * kHeadDim));
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          if (idx[q] >= 0) {
            const int i = i32 + idx[q];
            while (i >= bnd && j < r - 1) {   // warp-uniform: the next centre starts here
              flush(j);
              ++j;
              bnd = cb[j] + cc[j];
            }
            acc_row(kw[q], sk, st);
            ++n;
          }
        }
      }
    } else {
#pragma unroll 1
      for (int i8 = 0; i8 < 32 && i32 + i8 < hi; i8 += 8) {
        uint2 kw[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const int64_t pos = __shfl_sync(0xffffffffu, my, i8 + q);
          if (i32 + i8 + q < hi) kw[q] = __ldg(reinterpret_cast<const uint2*>(Xb + pos * kHeadDim));
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const int i = i32 + i8 + q;
          if (i < hi) {
            while (i >= bnd && j < r - 1) {   // warp-uniform: the next centre starts here
              flush(j);
              ++j;
              bnd = cb[j] + cc[j];
            }
            acc_row(kw[q], sk, st);
            ++n;
          }
        }
      }
    }
  }
  flush(j);
}

// One warp per centre, lane l on dims 4l..4l+3 (coalesced sums, centres and
// entries); ||c||^2 of the fp32 centre by a butterfly (the certification
// bounds its rounding for any summation order).
constexpr int kFinWarps = 8;

// keep: the key sums and flags stay for the next pass's update (delta
// accumulation); otherwise both halves of the sums and the flag are cleared.
__global__ void __launch_bounds__(kFinWarps * 32) k_lloyd_finish(LloydArgs p, int final_pass, int keep) {
  const int lane = threadIdx.x & 31;
  const int j = blockIdx.x * kFinWarps + (threadIdx.x >> 5), ul = blockIdx.y;
  const int r = p.r_unit[ul];
  if (j >= r) return;
  const int64_t uj = int64_t(ul) * p.rmax + j;
  const int cnt = p.ccount[uj];
  const bool exact = p.mflag[uj] == 0u;
  long long* ms = p.msum + uj * 2 * kHeadDim + 4 * lane;
  // mean = RN(sum / cnt) with sum = RN(S * 2^-32) for the integer sum S: by
  // Markstein's correction with the rounded reciprocal y = RN(1 / (cnt 2^32)),
  // q0 = RN(S y), r = S - q0 cnt 2^32 (exact in one fma), q = RN(q0 + r y) is
  // the correctly rounded quotient -- two fp64 fmas and a product per
  // dimension instead of a division (fp64 is scarce on this part)
  double tk[4], tv[4], mk[4], mv[4];
  const double cd = double(cnt);
  if (exact) {
    const double y = cnt > 0 ? (1.0 / cd) * 0x1p-32 : 0.0;
    const double bd = cd * 0x1p32;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const double sk = double(ms[q]);
      const double qk = sk * y;
      mk[q] = fma(fma(-qk, bd, sk), y, qk);
      mv[q] = 0.0;
      if (final_pass) {
        const double sv = double(ms[kHeadDim + q]);
        const double qv = sv * y;
        mv[q] = fma(fma(-qv, bd, sv), y, qv);
      }
    }
  } else {
    // fp64 sums in member order
#pragma unroll
    for (int q = 0; q < 4; ++q) tk[q] = tv[q] = 0.0;
    const int64_t mb = p.cbase[uj];
    const int cnt_in = (mb >= 0 && mb + cnt <= p.s) ? cnt : 0;   // see k_lloyd_accum
    const int32_t* mem = p.members + int64_t(ul) * p.s + (cnt_in > 0 ? mb : 0);
    const __nv_bfloat16* Kd = p.K + int64_t(ul) * p.s * kHeadDim + 4 * lane;
    const __nv_bfloat16* Vd = p.V + int64_t(ul) * p.s * kHeadDim + 4 * lane;
    for (int i = 0; i < cnt_in; ++i) {
      const int64_t pos = uint32_t(mem[i]) < uint32_t(p.s) ? mem[i] : 0;   // see k_lloyd_accum
      const uint2 kw = *reinterpret_cast<const uint2*>(Kd + pos * kHeadDim);
      const float2 k01 = bf16x2_to_float2(kw.x), k23 = bf16x2_to_float2(kw.y);
      tk[0] += double(k01.x);
      tk[1] += double(k01.y);
      tk[2] += double(k23.x);
      tk[3] += double(k23.y);
      if (final_pass) {
        const uint2 vw = *reinterpret_cast<const uint2*>(Vd + pos * kHeadDim);
        const float2 v01 = bf16x2_to_float2(vw.x), v23 = bf16x2_to_float2(vw.y);
        tv[0] += double(v01.x);
        tv[1] += double(v01.y);
        tv[2] += double(v23.x);
        tv[3] += double(v23.y);
      }
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      mk[q] = tk[q] / cd;
      mv[q] = final_pass ? tv[q] / cd : 0.0;
    }
  }
  if (!keep) {
#pragma unroll
    for (int q = 0; q < 4; ++q) ms[q] = ms[kHeadDim + q] = 0;
  }
  double* c64 = p.centers64 + uj * kHeadDim + 4 * lane;
  float* c32 = p.centers32 + uj * kHeadDim + 4 * lane;
  float cf[4];
  if (cnt > 0) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int d = 4 * lane + q;
      cf[q] = float(mk[q]);
      c64[q] = mk[q];
      c32[q] = cf[q];
      p.centersT[(int64_t(ul) * kHeadDim + d) * p.rmax + j] = cf[q];
      write_planes(p, ul, j, d, cf[q]);
    }
  } else {                            // an empty centre keeps its place
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      mk[q] = c64[q];
      cf[q] = c32[q];
    }
  }
  float n = fmaf(cf[3], cf[3], fmaf(cf[2], cf[2], fmaf(cf[1], cf[1], cf[0] * cf[0])));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
  if (final_pass) {
    const int64_t e = int64_t(ul) * p.ent_stride + p.ent_off + j;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      p.kbar[e * kHeadDim + 4 * lane + q] = __double2bfloat16(mk[q]);
      p.vbar[e * kHeadDim + 4 * lane + q] = __double2bfloat16(cnt > 0 ? mv[q] : 0.0);
    }
    if (lane == 0) p.ecount[e] = cnt;
  }
  __syncwarp();                       // every lane has read mflag
  if (lane == 0) {
    p.cnorm[uj] = n;
    if (!keep) p.mflag[uj] = 0u;
  }
}

// ---------------------------------------------------------------------------
// Validation proxy (Sec. 5.5.1, Eqs. valloss, valproxy; Alg. 1)
// ---------------------------------------------------------------------------

constexpr int kValChunkTiles = 16;           // 2048 tokens per CTA
constexpr int kValRec = kHeadDim + 4;        // m, l, 2 pad, acc[d]: acc 16-byte aligned

struct ValArgs {
  const __nv_bfloat16* K;
  const __nv_bfloat16* V;
  const __nv_bfloat16* Qobs;   // [UL*G, n_obs, d]
  int64_t s;
  int32_t G, n_obs, n_val, n_rows;     // n_rows = G * n_val, row = g * n_val + t
  int32_t nchunks;
  float* part;                 // [UL, n_rows, nchunks, kValRec]  (m, l, pad, acc)
  float* oS;                   // [UL, n_rows, d]
};

__device__ __forceinline__ const __nv_bfloat16* val_row(const ValArgs& p, int ul, int row) {
  const int g = row / p.n_val, t = row % p.n_val;
  return p.Qobs + ((int64_t(ul) * p.G + g) * p.n_obs + (p.n_obs - p.n_val) + t) * kHeadDim;
}

// Shared memory of the validation kernels (k_val_full, k_val_loss): the key
// tile (bf16, 256-byte rows with the 16-byte chunks XOR-swizzled for
// ldmatrix), the value tile (bf16 rows), the logits of the CTA's 32 query rows
// (fp32, rows padded to 136 floats: the fragment stores are conflict free)
// and P^T (fp32, swizzled).  Under 113 KB: two CTAs per SM.
constexpr int kValSRow = kTile + 8;
constexpr size_t kValOffV = size_t(kTile) * kAsgRowBytes;
constexpr size_t kValOffS = kValOffV + size_t(kTile) * kAsgRowBytes;
constexpr size_t kValOffP = kValOffS + size_t(kRowBlk) * kValSRow * 4;
constexpr size_t kValSmem = kValOffP + size_t(kTile) * kRowBlk * 4;

// A fragments (m16n8k16) of 16 query rows: row g and g + 8 of lane g = lane / 4
// from rowptr(i) (nullptr: a zero row), unscaled bf16
template <typename RowPtr>
__device__ __forceinline__ void val_afrag(RowPtr rowptr, int lane, uint32_t (&A)[8][4]) {
  const int g = lane >> 2, t4 = lane & 3;
  const uint32_t* q0 = reinterpret_cast<const uint32_t*>(rowptr(g));
  const uint32_t* q1 = reinterpret_cast<const uint32_t*>(rowptr(g + 8));
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    A[ks][0] = q0 ? __ldg(q0 + 8 * ks + t4) : 0u;
    A[ks][1] = q1 ? __ldg(q1 + 8 * ks + t4) : 0u;
    A[ks][2] = q0 ? __ldg(q0 + 8 * ks + 4 + t4) : 0u;
    A[ks][3] = q1 ? __ldg(q1 + 8 * ks + 4 + t4) : 0u;
  }
}

// The scaled logits (log2 domain) of the CTA's 32 rows against the staged key
// tile into St: warp w < 4 takes rows 16 (w / 2).. and tokens 64 (w % 2)..
// (tensor cores: exact bf16 products, fp32 sums); the other warps wait.
__device__ __forceinline__ void val_tile_logits(uint32_t ks_s, const uint32_t (&A)[8][4], float* St) {
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (w >= 4) return;
  float S[8][4];
  obs_half_logits(ks_s, w & 1, lane, A, S);
  const int g = lane >> 2, t4 = lane & 3, r0 = 16 * (w >> 1) + g;
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) {
    const int tk = 64 * (w & 1) + 8 * nt + 2 * t4;
    *reinterpret_cast<float2*>(St + r0 * kValSRow + tk) = make_float2(S[nt][0], S[nt][1]);
    *reinterpret_cast<float2*>(St + (r0 + 8) * kValSRow + tk) = make_float2(S[nt][2], S[nt][3]);
  }
}

// this thread's logits: rows 4w..4w+3, tokens 4l..4l+3
__device__ __forceinline__ void val_read_logits(const float* St, float (&S)[4][4]) {
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float4 v = *reinterpret_cast<const float4*>(St + (4 * w + i) * kValSRow + 4 * lane);
    S[i][0] = v.x;
    S[i][1] = v.y;
    S[i][2] = v.z;
    S[i][3] = v.w;
  }
}

// 128 rows of 256 bytes into a bf16 tile (rows swizzled for ldmatrix or
// plain) by cp.async, one 16-byte chunk per copy; rowptr(i) = nullptr: zeros
// (the copy then reads nothing from `any`, a valid global address)
template <bool swz, typename RowPtr>
__device__ __forceinline__ void val_stage_rows(uint32_t dst, RowPtr rowptr, const __nv_bfloat16* any) {
  for (int idx = threadIdx.x; idx < kTile * 16; idx += blockDim.x) {
    const int row = idx >> 4, ch = idx & 15;
    const __nv_bfloat16* src = rowptr(row);
    cp_async16(dst + (swz ? asg_swz(row, ch) : uint32_t(row * kAsgRowBytes + ch * 16)),
               src ? src + 8 * ch : any, src ? 16u : 0u);
  }
}

// acc[i][d] += P^T[tok][row 4w + i] * V[tok][dim 4l + d] over the tile
__device__ __forceinline__ void val_pv(const float* Pt, const __nv_bfloat16* Vb, float (&acc)[4][4]) {
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll 4
  for (int tok = 0; tok < kTile; ++tok) {
    const float4 pp = *reinterpret_cast<const float4*>(Pt + tok * kRowBlk + ((w ^ ((tok >> 2) & 7)) << 2));
    const uint2 vw = *reinterpret_cast<const uint2*>(Vb + tok * kHeadDim + 4 * lane);
    const float2 v01 = bf16x2_to_float2(vw.x), v23 = bf16x2_to_float2(vw.y);
    const float pa[4] = {pp.x, pp.y, pp.z, pp.w};
    const float va[4] = {v01.x, v01.y, v23.x, v23.y};
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int d = 0; d < 4; ++d) acc[i][d] = fmaf(pa[i], va[d], acc[i][d]);
  }
}

// o_S(q) over all s tokens for the validation queries (Eq. attn), per chunk
__global__ void __launch_bounds__(kThreads, 2) k_val_full(ValArgs p) {
  extern __shared__ __align__(1024) uint8_t vraw[];
  const uint32_t ks_s = smem_u32(vraw), vb_s = ks_s + uint32_t(kValOffV);
  const __nv_bfloat16* Vb = reinterpret_cast<const __nv_bfloat16*>(vraw + kValOffV);
  float* St = reinterpret_cast<float*>(vraw + kValOffS);
  float* Pt = reinterpret_cast<float*>(vraw + kValOffP);
  const int chunk = blockIdx.x, rb = blockIdx.y * kRowBlk, ul = blockIdx.z;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint32_t A[8][4];
  if (w < 4) {
    const int r16 = rb + 16 * (w >> 1);
    val_afrag([&](int i) { return r16 + i < p.n_rows ? val_row(p, ul, r16 + i) : nullptr; }, lane, A);
  }
  float m[4], l[4], acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    m[i] = -INFINITY;
    l[i] = 0.f;
#pragma unroll
    for (int d = 0; d < 4; ++d) acc[i][d] = 0.f;
  }
  const __nv_bfloat16* Ku = p.K + int64_t(ul) * p.s * kHeadDim;
  const __nv_bfloat16* Vu = p.V + int64_t(ul) * p.s * kHeadDim;
  for (int tt = 0; tt < kValChunkTiles; ++tt) {
    const int64_t tok0 = (int64_t(chunk) * kValChunkTiles + tt) * kTile;
    if (tok0 >= p.s) break;
    __syncthreads();
    auto krow = [&](int i) { return tok0 + i < p.s ? Ku + (tok0 + i) * kHeadDim : nullptr; };
    auto vrow = [&](int i) { return tok0 + i < p.s ? Vu + (tok0 + i) * kHeadDim : nullptr; };
    val_stage_rows<true>(ks_s, krow, Ku);
    val_stage_rows<false>(vb_s, vrow, Vu);
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    val_tile_logits(ks_s, A, St);
    __syncthreads();
    float S[4][4];
    val_read_logits(St, S);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float tmax = -INFINITY;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (tok0 + 4 * lane + j >= p.s) S[i][j] = -INFINITY;
        tmax = fmaxf(tmax, S[i][j]);
      }
      tmax = warp_max(tmax);
      const float mn = fmaxf(m[i], tmax);
      const float sc = exp2f(m[i] - mn);
      l[i] *= sc;
#pragma unroll
      for (int d = 0; d < 4; ++d) acc[i][d] *= sc;
      m[i] = mn;
      float ps = 0.f;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        S[i][j] = exp2f(S[i][j] - mn);
        ps += S[i][j];
      }
      l[i] += warp_sum(ps);
    }
    // P^T into shared memory: Pt[tok][rows], float4 column swizzled by (tok / 4)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int tok = 4 * lane + j;
      *reinterpret_cast<float4*>(Pt + tok * kRowBlk + ((w ^ (lane & 7)) << 2)) =
          make_float4(S[0][j], S[1][j], S[2][j], S[3][j]);
    }
    __syncthreads();
    val_pv(Pt, Vb, acc);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int row = rb + 4 * w + i;
    if (row >= p.n_rows) continue;
    float* out = p.part + ((int64_t(ul) * p.n_rows + row) * p.nchunks + chunk) * kValRec;
    if (lane == 0) {
      out[0] = m[i];
      out[1] = l[i];
    }
    *reinterpret_cast<float4*>(out + 4 + 4 * lane) = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
  }
}

__global__ void k_val_combine(ValArgs p) {
  const int row = blockIdx.x, ul = blockIdx.y, d = threadIdx.x;
  const float* base = p.part + (int64_t(ul) * p.n_rows + row) * p.nchunks * kValRec;
  float m = -INFINITY, l = 0.f, a = 0.f;
  for (int c = 0; c < p.nchunks; ++c) {
    const float* q = base + int64_t(c) * kValRec;
    const float cm = q[0], cl = q[1];
    if (cl <= 0.f) continue;
    const float mn = fmaxf(m, cm);
    const float s0 = exp2f(m - mn), s1 = exp2f(cm - mn);
    l = l * s0 + cl * s1;
    a = a * s0 + q[4 + d] * s1;
    m = mn;
  }
  p.oS[(int64_t(ul) * p.n_rows + row) * kHeadDim + d] = a / l;
}

struct LossArgs {
  const __nv_bfloat16* K;
  const __nv_bfloat16* V;
  const __nv_bfloat16* Qobs;
  int64_t s;
  int32_t G, n_obs, n_val, n_rows;
  int32_t recent, n_top, budget;
  const int32_t* top;          // [UL, n_top]
  const int32_t* r_unit;       // [UL]
  const __nv_bfloat16* kbar;   // [UL, ent_stride, d]
  const __nv_bfloat16* vbar;
  const int32_t* ecount;
  int64_t ent_stride;
  int32_t ent_off;
  float beta;
  int32_t gate_mode;
  float tau, alpha, g_min, g_fixed;
  const float* oS;             // [UL, n_rows, d]
  double* rowerr;              // [UL, n_rows]
  int32_t softmax_mode;        // decode rule of the losses (RESKV_SOFTMAX_*)
  const int32_t* budgets;      // [UL] per-unit budgets, or NULL (budget)
};

// ||o^(r)(q) - o_S(q)||^2 per validation query, with the decode rule of
// Sec. 5.4 and the gate.  Tiled like k_val_full: a CTA takes 32 query rows of
// a unit and walks the candidate's main slots (the kept ranked tokens, then
// the recent window), then its residual entries (logit + beta ln c), each
// gathered into shared memory once for all 32 rows (logits on the tensor
// cores), with one online-softmax state per branch.  Dynamic shared memory:
// kValSmem.
struct LossState {
  float m[4], l[4], acc[4][4];
};

// One 128-token tile (logits in St, V in Vb) into state st: logits + bias[j]
// for this lane's tokens 4l + j (-inf: no token)
__device__ __forceinline__ void loss_tile(const float* St, float* Pt, const __nv_bfloat16* Vb,
                                          const float (&bias)[4], LossState& st) {
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float S[4][4];
  val_read_logits(St, S);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float tmax = -INFINITY;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      S[i][j] += bias[j];
      tmax = fmaxf(tmax, S[i][j]);
    }
    tmax = warp_max(tmax);
    const float mn = fmaxf(st.m[i], tmax);
    // a tile with no token leaves the state as it is (mn = -inf)
    const float sc = mn == -INFINITY ? 1.0f : exp2f(st.m[i] - mn);
    st.l[i] *= sc;
#pragma unroll
    for (int d = 0; d < 4; ++d) st.acc[i][d] *= sc;
    st.m[i] = mn;
    float ps = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      S[i][j] = mn == -INFINITY ? 0.f : exp2f(S[i][j] - mn);
      ps += S[i][j];
    }
    st.l[i] += warp_sum(ps);
  }
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int tok = 4 * lane + j;
    *reinterpret_cast<float4*>(Pt + tok * kRowBlk + ((w ^ (lane & 7)) << 2)) =
        make_float4(S[0][j], S[1][j], S[2][j], S[3][j]);
  }
  __syncthreads();
  val_pv(Pt, Vb, st.acc);
}

__global__ void __launch_bounds__(kThreads, 1) k_val_loss(LossArgs p) {
  extern __shared__ __align__(1024) uint8_t vraw[];
  const uint32_t ks_s = smem_u32(vraw), vb_s = ks_s + uint32_t(kValOffV);
  const __nv_bfloat16* Vb = reinterpret_cast<const __nv_bfloat16*>(vraw + kValOffV);
  float* St = reinterpret_cast<float*>(vraw + kValOffS);
  float* Pt = reinterpret_cast<float*>(vraw + kValOffP);
  const int rb = blockIdx.x * kRowBlk, ul = blockIdx.y;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = p.r_unit[ul];
  const int64_t bu = unit_budget(p.budgets, ul, p.budget);
  const int64_t m = r == 0 ? (bu < p.s ? bu : p.s) : bu - r;
  const int64_t keep = m - p.recent;
  uint32_t A[8][4];
  if (w < 4) {
    const int r16 = rb + 16 * (w >> 1);
    val_afrag([&](int i) -> const __nv_bfloat16* {
      const int row = r16 + i;
      if (row >= p.n_rows) return nullptr;
      const int g = row / p.n_val, t = row % p.n_val;
      return p.Qobs + ((int64_t(ul) * p.G + g) * p.n_obs + (p.n_obs - p.n_val) + t) * kHeadDim;
    }, lane, A);
  }
  LossState sM, sR;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    sM.m[i] = sR.m[i] = -INFINITY;
    sM.l[i] = sR.l[i] = 0.f;
#pragma unroll
    for (int d = 0; d < 4; ++d) sM.acc[i][d] = sR.acc[i][d] = 0.f;
  }
  const __nv_bfloat16* Ku = p.K + int64_t(ul) * p.s * kHeadDim;
  const __nv_bfloat16* Vu = p.V + int64_t(ul) * p.s * kHeadDim;
  const int32_t* top = p.top + int64_t(ul) * p.n_top;
  // main slots: the ranked tokens kept, then the recent window
  for (int64_t j0 = 0; j0 < m; j0 += kTile) {
    auto pos = [&](int tok) -> int64_t {
      const int64_t j = j0 + tok;
      return j >= m ? -1 : (j < keep ? top[j] : (p.s - p.recent) + (j - keep));
    };
    __syncthreads();
    val_stage_rows<true>(ks_s, [&](int tok) {
      const int64_t q = pos(tok);
      return q < 0 ? static_cast<const __nv_bfloat16*>(nullptr) : Ku + q * kHeadDim;
    }, Ku);
    val_stage_rows<false>(vb_s, [&](int tok) {
      const int64_t q = pos(tok);
      return q < 0 ? static_cast<const __nv_bfloat16*>(nullptr) : Vu + q * kHeadDim;
    }, Vu);
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    val_tile_logits(ks_s, A, St);
    __syncthreads();
    float bias[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) bias[j] = j0 + 4 * lane + j < m ? 0.f : -INFINITY;
    loss_tile(St, Pt, Vb, bias, sM);
  }
  // residual entries: logit + beta ln c (log2 units); an empty entry is inert
  const int64_t e0 = int64_t(ul) * p.ent_stride + p.ent_off;
  for (int j0 = 0; j0 < r; j0 += kTile) {
    __syncthreads();
    val_stage_rows<true>(ks_s, [&](int tok) {
      return j0 + tok < r ? p.kbar + (e0 + j0 + tok) * kHeadDim : static_cast<const __nv_bfloat16*>(nullptr);
    }, Ku);
    val_stage_rows<false>(vb_s, [&](int tok) {
      return j0 + tok < r ? p.vbar + (e0 + j0 + tok) * kHeadDim : static_cast<const __nv_bfloat16*>(nullptr);
    }, Vu);
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    val_tile_logits(ks_s, A, St);
    __syncthreads();
    float bias[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int e = j0 + 4 * lane + j;
      const int c = e < r ? p.ecount[e0 + e] : 0;
      bias[j] = c > 0 ? p.beta * logf(float(c)) * kLog2e : -INFINITY;
    }
    loss_tile(St, Pt, Vb, bias, sR);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int row = rb + 4 * w + i;
    float g_val = p.g_fixed;
    if (p.gate_mode == RESKV_GATE_DYNAMIC) {
      const float pmax = 1.0f / sM.l[i];
      g_val = fmaxf(p.g_min, 1.0f / (1.0f + expf(-p.alpha * (p.tau - pmax))));
    }
    const float2 coef = branch_coefs(p.softmax_mode, g_val, sM.m[i], sM.l[i], sR.m[i], sR.l[i]);
    float e = 0.f;
    if (row < p.n_rows) {
      const float* os = p.oS + (int64_t(ul) * p.n_rows + row) * kHeadDim + 4 * lane;
#pragma unroll
      for (int d = 0; d < 4; ++d) {
        const float o = coef.x * sM.acc[i][d] + coef.y * sR.acc[i][d];
        const float df = o - os[d];
        e += df * df;
      }
    }
    e = warp_sum(e);
    if (lane == 0 && row < p.n_rows) p.rowerr[int64_t(ul) * p.n_rows + row] = double(e);
  }
}

// L_r = mean of the per-query errors (rows in order, fp64); +inf for a unit
// without a candidate in this column (r_unit = 0 in a column c > 0)
__global__ void k_loss_reduce(const double* rowerr, double* losses, int n_rows, int UL, int ncol,
                              int col, const int32_t* r_unit) {
  const int ul = blockIdx.x * blockDim.x + threadIdx.x;
  if (ul >= UL) return;
  double acc = 0.0;
  for (int i = 0; i < n_rows; ++i) acc += rowerr[int64_t(ul) * n_rows + i];
  losses[int64_t(ul) * ncol + col] = (col > 0 && r_unit[ul] == 0) ? INFINITY : acc / double(n_rows);
}

// r* = argmin_{r>0} L_r (ties -> smaller r: columns hold ascending r); keep it
// only if L_r* < (1 - delta) L_0.  r_runs: [ncol, UL] r of every column.
__global__ void k_choose(const double* losses, int ncol, const int32_t* r_runs, int UL,
                         double one_minus_delta, int32_t* r_final, int32_t* chosen) {
  const int ul = blockIdx.x * blockDim.x + threadIdx.x;
  if (ul >= UL) return;
  const double* L = losses + int64_t(ul) * ncol;
  int best = 0;
  for (int c = 1; c < ncol; ++c)
    if (r_runs[int64_t(c) * UL + ul] > 0 && (best == 0 || L[c] < L[best])) best = c;
  const bool use = best > 0 && L[best] < one_minus_delta * L[0];
  r_final[ul] = use ? r_runs[int64_t(best) * UL + ul] : 0;
  chosen[ul] = use ? best : 0;
}

// ---------------------------------------------------------------------------
// Packing into the ragged layout (end of Alg. 1): main rows in position
// order, then the chosen run's residual entries.
// ---------------------------------------------------------------------------

struct PackArgs {
  const __nv_bfloat16* K;
  const __nv_bfloat16* V;
  int64_t s;
  int32_t recent, budget;
  int32_t stride;              // slots per unit in the cache (budget + append capacity)
  const int32_t* rank_pos;     // [UL, s]
  const int32_t* r_final;      // [UL]
  const int32_t* chosen;       // [UL] run index of the chosen entries (0 = none)
  const int32_t* run_off;      // [n_runs] entry offset of each run
  const __nv_bfloat16* kbar;
  const __nv_bfloat16* vbar;
  const int32_t* ecount;
  int64_t ent_stride;
  float beta;
  int64_t unit0;               // global unit index of ul = 0
  __nv_bfloat16* kslots;
  __nv_bfloat16* vslots;
  float* logc;
  int32_t* slot_pos;
  int32_t* counts;
  int32_t* n_main;
  int32_t* n_res;
  const int32_t* budgets;      // [UL] per-unit budgets, or NULL (budget)
  const int32_t* offsets;      // [U + 1] first slot of every unit, or NULL (u * stride)
};

__global__ void __launch_bounds__(1024) k_pack(PackArgs p) {
  __shared__ int warp_sums[32];
  const int ul = blockIdx.x;
  const int64_t u = p.unit0 + ul;
  const int r = p.r_final[ul];
  const int64_t bu = unit_budget(p.budgets, ul, p.budget);
  const int64_t m = r == 0 ? (bu < p.s ? bu : p.s) : bu - r;
  const int64_t keep = m - p.recent;
  const int32_t* rp = p.rank_pos + int64_t(ul) * p.s;
  const int64_t base = p.offsets ? int64_t(p.offsets[u]) : u * p.stride;   // first slot of u
  int32_t* spos = p.slot_pos + base;
  const int64_t chunk = (p.s + blockDim.x - 1) / blockDim.x;
  const int64_t lo = int64_t(threadIdx.x) * chunk, hi = lo + chunk < p.s ? lo + chunk : p.s;
  int mine = 0;
  for (int64_t i = lo; i < hi; ++i) {
    const int32_t rk = rp[i];
    mine += (rk < 0 || rk < keep);
  }
  int out = block_exclusive_scan(mine, warp_sums, nullptr);
  for (int64_t i = lo; i < hi; ++i) {
    const int32_t rk = rp[i];
    if (rk < 0 || rk < keep) {
      if (out < m) spos[out] = int32_t(i);
      ++out;
    }
  }
  __syncthreads();
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  const __nv_bfloat16* Ku = p.K + int64_t(ul) * p.s * kHeadDim;
  const __nv_bfloat16* Vu = p.V + int64_t(ul) * p.s * kHeadDim;
  for (int64_t j = w; j < m; j += nw) {
    const int64_t pos = spos[j];
    const uint2 kw = __ldg(reinterpret_cast<const uint2*>(Ku + pos * kHeadDim) + lane);
    const uint2 vw = __ldg(reinterpret_cast<const uint2*>(Vu + pos * kHeadDim) + lane);
    reinterpret_cast<uint2*>(p.kslots + (base + j) * kHeadDim)[lane] = kw;
    reinterpret_cast<uint2*>(p.vslots + (base + j) * kHeadDim)[lane] = vw;
    if (lane == 0) {
      p.counts[base + j] = 0;
      p.logc[base + j] = 0.f;
    }
  }
  const int c = p.chosen[ul];
  for (int j = w; j < r; j += nw) {
    const int64_t e = int64_t(ul) * p.ent_stride + p.run_off[c] + j;
    const int64_t slot = base + m + j;
    reinterpret_cast<uint2*>(p.kslots + slot * kHeadDim)[lane] =
        reinterpret_cast<const uint2*>(p.kbar + e * kHeadDim)[lane];
    reinterpret_cast<uint2*>(p.vslots + slot * kHeadDim)[lane] =
        reinterpret_cast<const uint2*>(p.vbar + e * kHeadDim)[lane];
    if (lane == 0) {
      const int cnt = p.ecount[e];
      p.counts[slot] = cnt;
      p.logc[slot] = cnt > 0 ? p.beta * logf(float(cnt)) : -INFINITY;
      spos[m + j] = -1;
    }
  }
  if (threadIdx.x == 0) {
    p.n_main[u] = int32_t(m);
    p.n_res[u] = r;
  }
}

}  // namespace build
}  // namespace reskv
