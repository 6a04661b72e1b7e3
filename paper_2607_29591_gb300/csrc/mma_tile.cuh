// The 16-slot tensor-core tile of the shared-softmax decode (Alg. 2; Sec. 5.4
// Eqs. residual_logit, reskv_den, reskv_num) and the pieces around it, shared
// by the two tensor-core decode kernels (decode_mma.cu: stream-K over the
// launch's whole slot range; decode_cluster.cu: one thread-block cluster per
// unit).
//
// One tile step covers 16 consecutive slots staged in shared memory with
// legacy tensor-core MMAs (mma.sync m16n8k16, bf16 in, fp32 accumulate):
//
//   logits  S[16 x 8 slots]  = Q[16 x 128] K^T        rows 0..G-1 = query heads
//   output  O[16 x 8 dims]  += P[16 x 16 slots] V      rows 0..G-1: main-cache
//                                                       weights, rows 8..8+G-1:
//                                                       residual weights
//
// The mma tile has 16 rows for G <= 4 heads; the unused rows 8..15 carry the
// residual branch, so the main and residual numerators (which the gate scales
// differently) accumulate side by side in one fragment with no extra MMA.
// P is split into bf16 hi + lo parts (two MMAs) so that the weights keep
// ~16 significant bits; logits are exact bf16 products summed in fp32.
//
// A stage holds the tile's K and V rows as four 2-D TMA boxes of 64 dims x 16
// rows with the 128-byte swizzle (K dims 0..63 | K dims 64..127 | V lo | V hi),
// so that ldmatrix reads of eight rows at one column are bank-conflict free.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "device_utils.cuh"
#include "internal.h"

namespace reskv {

constexpr int kMmaMaxW = 8;                // warps per CTA (at most)
constexpr int kMmaMaxSt = 12;              // ring stages per warp (at most)
constexpr int kCh = kDecodeChunk;          // slots per stage (= one MMA tile)
constexpr int kBox = kCh * 128;            // one 64-dim half of 16 rows, bytes
constexpr int kStageBytes = 4 * kBox;      // K lo | K hi | V lo | V hi
constexpr int kRec = kHeadDim + 4;         // partial record: m, l, pad, pad, acc[d]
constexpr int kSmemLimit = 227 * 1024;     // dynamic shared memory per CTA

// A warp's ring of `stages` stages plus its 16-slot log-count copies and
// mbarriers; each warp's region starts 1024-byte aligned (128-byte swizzle).
__host__ __device__ constexpr int warp_bytes(int stages) { return stages * kStageBytes + 1024; }
__host__ __device__ constexpr int warp_logc_offset(int stages) { return stages * kStageBytes; }
__host__ __device__ constexpr int warp_bars_offset(int stages) {
  return stages * kStageBytes + kMmaMaxSt * kCh * 4;
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// D += A * B, m16n8k16, bf16 inputs, fp32 accumulators
__device__ __forceinline__ void mma16816(float* d, uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ float2 unpack_bf16(uint32_t w) { return bf16x2_to_float2(w); }

// Eq. gate with p_max = 1 / lM: lM is the main-cache softmax sum relative to
// the largest main weight (which is 2^0).
__device__ __forceinline__ float gate_of(const DecodeParams& p, float lM) {
  if (p.gate_mode == RESKV_GATE_FIXED) return p.g_fixed;
  const float p_max = 1.0f / lM;
  return fmaxf(p.g_min, 1.0f / (1.0f + expf(-p.alpha * (p.tau - p_max))));
}

// ldmatrix row addresses of this lane (byte offsets inside a stage): for Q K^T
// the four 32-dim groups of K rows, for P V the eight 16-dim groups of V rows
// (transposed loads).
__device__ __forceinline__ void tile_offsets(int lane, uint32_t (&off_qk)[4], uint32_t (&off_pv)[8]) {
  const int r8 = lane & 7, mi = lane >> 3;
#pragma unroll
  for (int j = 0; j < 4; ++j) {                 // dims 32j..32j+31, matrix mi = 8-dim chunk
    const int cg = 4 * j + mi, half = cg >> 3, cc = cg & 7;
    off_qk[j] = half * kBox + r8 * 128 + ((cc ^ r8) << 4);
  }
#pragma unroll
  for (int q = 0; q < 8; ++q) {                 // dims 16q..16q+15
    const int cg = 2 * q + (mi >> 1), half = cg >> 3, cc = cg & 7, nt = mi & 1;
    off_pv[q] = 2 * kBox + half * kBox + nt * 1024 + r8 * 128 + ((cc ^ r8) << 4);
  }
}

// A operand of Q K^T for query row `qrow` of this lane's head: the words at
// dims 16kk + 2qp (+1) and 16kk + 8 + 2qp (+1); zero for rows >= G.
__device__ __forceinline__ void load_q_frag(const __nv_bfloat16* Q, int64_t qrow, bool hv, int qp,
                                            uint32_t (&dst)[16]) {
  const uint32_t* qw = reinterpret_cast<const uint32_t*>(Q + qrow * kHeadDim);
#pragma unroll
  for (int kk = 0; kk < 8; ++kk) {
    dst[2 * kk] = hv ? __ldg(qw + 8 * kk + qp) : 0u;
    dst[2 * kk + 1] = hv ? __ldg(qw + 8 * kk + 4 + qp) : 0u;
  }
}

// Online-softmax state of one unit in the fragment layout of the m16n8
// accumulator: O[dt][0..1] = main numerator of head h = lane/4 at dims
// 8dt + 2qp (+1), O[dt][2..3] = residual numerator of the same head; the
// running maxima are in log2 units and shared by the quad, the sums are this
// lane's share (summed over the quad when the unit finishes).
struct TileState {
  float O[16][4];
  float mM, lM, mR, lR;

  __device__ __forceinline__ void reset() {
#pragma unroll
    for (int dt = 0; dt < 16; ++dt) O[dt][0] = O[dt][1] = O[dt][2] = O[dt][3] = 0.f;
    mM = mR = -INFINITY;
    lM = lR = 0.f;
  }
};

// Fold the 16-slot tile staged at `st` (first global slot t0; residual
// log-counts at lc[0..15]) into `S`.  Slots y in [rlo, rhi) are residual
// entries (folded into the residual state when kResidual; a main-only pass
// skips them), the other slots in [mlo, mhi) are exact main rows (selected
// tokens and rows appended at decode time); every other row is masked.
template <bool kResidual = true>
__device__ __forceinline__ void tile_update(TileState& S, uint32_t st, const float* lc, int64_t t0,
                                            int64_t mlo, int64_t mhi, int64_t rlo, int64_t rhi,
                                            const uint32_t (&qa)[16], const uint32_t (&off_qk)[4],
                                            const uint32_t (&off_pv)[8], float qscale, bool hv,
                                            int qp) {
  // ---- logits S = Q K^T for the 16 slots (two 8-slot n-tiles) ----
  float S0[4] = {0.f, 0.f, 0.f, 0.f}, S1[4] = {0.f, 0.f, 0.f, 0.f};
  float S0b[4] = {0.f, 0.f, 0.f, 0.f}, S1b[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    uint32_t b0, b1, b2, b3, c0, c1, c2, c3;
    ldsm_x4(st + off_qk[j], b0, b1, b2, b3);             // slots 0..7
    ldsm_x4(st + off_qk[j] + 1024, c0, c1, c2, c3);      // slots 8..15
    mma16816(S0, qa[4 * j], 0u, qa[4 * j + 1], 0u, b0, b1);
    mma16816(S1, qa[4 * j], 0u, qa[4 * j + 1], 0u, c0, c1);
    mma16816(S0b, qa[4 * j + 2], 0u, qa[4 * j + 3], 0u, b2, b3);
    mma16816(S1b, qa[4 * j + 2], 0u, qa[4 * j + 3], 0u, c2, c3);
  }
  // this thread's slots: t0 + 8n + 2qp + i
  float sM[4], sR[4];
  const float sv[4] = {(S0[0] + S0b[0]) * qscale, (S0[1] + S0b[1]) * qscale,
                       (S1[0] + S1b[0]) * qscale, (S1[1] + S1b[1]) * qscale};
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const int rowi = (e >> 1) * 8 + 2 * qp + (e & 1);
    const int64_t y = t0 + rowi;
    const bool in_r = y >= rlo && y < rhi;
    const bool im = hv && y >= mlo && y < mhi && !in_r;
    const bool ir = kResidual && hv && in_r;
    sM[e] = im ? sv[e] : -INFINITY;
    sR[e] = ir ? sv[e] + lc[rowi] * kLog2e : -INFINITY;   // + beta log c_j
  }
  float tM = fmaxf(fmaxf(sM[0], sM[1]), fmaxf(sM[2], sM[3]));
  float tR = fmaxf(fmaxf(sR[0], sR[1]), fmaxf(sR[2], sR[3]));
  tM = fmaxf(tM, __shfl_xor_sync(0xffffffffu, tM, 1));
  tM = fmaxf(tM, __shfl_xor_sync(0xffffffffu, tM, 2));
  tR = fmaxf(tR, __shfl_xor_sync(0xffffffffu, tR, 1));
  tR = fmaxf(tR, __shfl_xor_sync(0xffffffffu, tR, 2));
  if (tM > S.mM) {                                   // rescale the main rows
    const float sc = exp2f(S.mM - tM);
    S.lM *= sc;
#pragma unroll
    for (int dt = 0; dt < 16; ++dt) {
      S.O[dt][0] *= sc;
      S.O[dt][1] *= sc;
    }
    S.mM = tM;
  }
  if (tR > S.mR) {                                   // rescale the residual rows
    const float sc = exp2f(S.mR - tR);
    S.lR *= sc;
#pragma unroll
    for (int dt = 0; dt < 16; ++dt) {
      S.O[dt][2] *= sc;
      S.O[dt][3] *= sc;
    }
    S.mR = tR;
  }
  float pM[4], pR[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    pM[e] = sM[e] > -INFINITY ? exp2f(sM[e] - S.mM) : 0.f;   // masked rows weigh 0
    pR[e] = sR[e] > -INFINITY ? exp2f(sR[e] - S.mR) : 0.f;
    S.lM += pM[e];
    S.lR += pR[e];
  }
  // A = P (rows 0..7 main, rows 8..15 residual), hi + lo bf16 parts
  const uint32_t h0 = pack_bf16(pM[0], pM[1]), h1 = pack_bf16(pR[0], pR[1]);
  const uint32_t h2 = pack_bf16(pM[2], pM[3]), h3 = pack_bf16(pR[2], pR[3]);
  const float2 f0 = unpack_bf16(h0), f1 = unpack_bf16(h1), f2 = unpack_bf16(h2), f3 = unpack_bf16(h3);
  const uint32_t l0 = pack_bf16(pM[0] - f0.x, pM[1] - f0.y), l1 = pack_bf16(pR[0] - f1.x, pR[1] - f1.y);
  const uint32_t l2 = pack_bf16(pM[2] - f2.x, pM[3] - f2.y), l3 = pack_bf16(pR[2] - f3.x, pR[3] - f3.y);
  // ---- O += P V ----
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    uint32_t v0, v1, v2, v3;
    ldsm_x4_t(st + off_pv[q], v0, v1, v2, v3);
    mma16816(S.O[2 * q], h0, h1, h2, h3, v0, v1);
    mma16816(S.O[2 * q + 1], h0, h1, h2, h3, v2, v3);
    mma16816(S.O[2 * q], l0, l1, l2, l3, v0, v1);
    mma16816(S.O[2 * q + 1], l0, l1, l2, l3, v2, v3);
  }
}

}  // namespace reskv
