// The 16-slot tensor-core tile of the shared-softmax decode (Alg. 2; Sec. 5.4
// Eqs. residual_logit, reskv_den, reskv_num) and the pieces around it, shared
// by the two tensor-core decode kernels (decode_mma.cu: stream-K over the
// launch's whole slot range; decode_cluster.cu: one thread-block cluster per
// unit).
//
// One tile step covers 16 consecutive slots staged in shared memory with
// legacy tensor-core MMAs (mma.sync m16n8k16, bf16 in, fp32 accumulate), in
// transposed form:
//
//   logits  S^T[16 slots x 8 columns] = K[16 x 128] Q^T      8 MMAs
//   output  O[16 rows x 8 dims]      += P[16 x 16 slots] V   16 MMAs
//
// Column c of S^T is query head c for c < G (main branch) and head c - G for
// G <= c < 2G (residual branch, whose logits add beta log c_j); columns from
// 2G on are unused.  The logits of a column are its head's, masked to the
// branch's slots, so one MMA gives both branches.  After the softmax the
// weights are split into bf16 hi and lo parts (~16 significant bits together)
// and moved into the A layout with movmatrix: rows 0..7 hold the hi part of
// columns 0..7, rows 8..15 the lo part, so accumulator row g plus row g + 8 is
// the numerator of column g.
//
// A stage holds the tile's K and V rows as four 2 KB blocks of 16 rows x 64
// dims with the 128-byte swizzle (K dims 0..63 | K dims 64..127 | V lo | V hi;
// one 3-D TMA copy fills both blocks of K, one both of V), so that ldmatrix
// reads of eight rows at one column are bank-conflict free.
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
constexpr int kRec = kHeadDim + 4;         // partial record: m, l, mt, pad, acc[d]
constexpr int kSmemLimit = 227 * 1024;     // dynamic shared memory per CTA

// A column's reference maximum before its first logit: finite, so that
// exponents of masked (-inf) logits stay -inf and never become NaN.
constexpr float kMInit = -1e30f;
// A column's reference maximum is raised only when a logit exceeds it by more
// than kLazy (log2 units): its weights stay below 2^kLazy and most tiles skip
// the rescale of the accumulators.  Any reference gives the same softmax; the
// column's largest logit is kept apart for the gate's p_max.
constexpr float kLazy = 8.0f;

// Shared memory of a CTA of `warps` warps with rings of `stages` stages: from
// a 1024-byte aligned base (128-byte swizzle), the warps' rings one after the
// other, then the 16 log-counts of every stage, then every stage's mbarrier
// (rounded up to 16 bytes).  Keeping the small parts out of the rings lets a
// CTA hold 28 stages in 227 KB.
constexpr int kStageExtra = kCh * 4 + 8;
__host__ __device__ constexpr int ring_smem_bytes(int warps, int stages) {
  return (warps * stages * (kStageBytes + kStageExtra) + 15) & ~15;
}
// Ring depth that fits `warps` warps next to `extra` more bytes.
__host__ __device__ constexpr int ring_stages(int warps, int extra) {
  return (kSmemLimit - 1024 - 16 - extra) / (warps * (kStageBytes + kStageExtra)) < kMmaMaxSt
             ? (kSmemLimit - 1024 - 16 - extra) / (warps * (kStageBytes + kStageExtra))
             : kMmaMaxSt;
}

struct WarpRing {
  uint8_t* cta;         // the CTA's aligned base (generic)
  uint32_t base;        // shared address of this warp's first stage
  uint8_t* ptr;         // the same, generic
  float* logc;          // [stages][16]
  uint64_t* bars;       // [stages]
};

__device__ __forceinline__ WarpRing warp_ring(uint8_t* smem_raw, int warps, int stages, int warp) {
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t abase = (raw + 1023u) & ~1023u;
  uint8_t* a = smem_raw + (abase - raw);
  const int nst = warps * stages;
  WarpRing r;
  r.cta = a;
  r.base = abase + uint32_t(warp * stages * kStageBytes);
  r.ptr = a + warp * stages * kStageBytes;
  r.logc = reinterpret_cast<float*>(a + nst * kStageBytes) + warp * stages * kCh;
  r.bars = reinterpret_cast<uint64_t*>(a + nst * (kStageBytes + kCh * 4)) + warp * stages;
  return r;
}

// L2 policy of the ring's cache copies: every slot is read once per decode
// call, so its lines are the first the L2 gives up (measured: one-layer
// launches 3-4 % shorter than with the default policy).
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            uint64_t* bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar)), "l"(pol)
      : "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, int x, int y, int z,
                                            uint64_t* bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, %3, %4}], [%5], %6;" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar)), "l"(pol)
      : "memory");
}

// The copies of one stage (one thread): K and V rows [row, row + 16) into st
// (K dims 0..63 | K dims 64..127 | V dims 0..63 | V dims 64..127) and, with
// with_logc, their 16 log-counts into lc, all completing on bar.  kv_rank:
// that of the maps; pol: the L2 policy of the K and V copies.  A chunk known
// to hold no residual rows skips the log-counts (the tile step reads them only
// at residual rows).
__device__ __forceinline__ void issue_stage(uint32_t st, float* lc, const CUtensorMap* tmK,
                                            const CUtensorMap* tmV, const float* logc, int row,
                                            int kv_rank, bool with_logc, uint64_t* bar,
                                            uint64_t pol) {
  mbar_arrive_expect_tx(bar, kStageBytes + (with_logc ? kCh * 4 : 0));
  if (kv_rank == 3) {
    tma_load_3d(st, tmK, 0, row, 0, bar, pol);
    tma_load_3d(st + 2 * kBox, tmV, 0, row, 0, bar, pol);
  } else {
    tma_load_2d(st, tmK, 0, row, bar, pol);
    tma_load_2d(st + kBox, tmK, 64, row, bar, pol);
    tma_load_2d(st + 2 * kBox, tmV, 0, row, bar, pol);
    tma_load_2d(st + 3 * kBox, tmV, 64, row, bar, pol);
  }
  if (with_logc) bulk_g2s(lc, logc + row, kCh * 4, bar);
}

// Whether the 16 rows from r0 are all main or appended rows of a unit whose
// used rows are [ub, ub + nt) with residual rows [ub + nm, ub + nm + nr).
__device__ __forceinline__ bool chunk_main_only(int r0, int ub, int nm, int nr, int nt) {
  return r0 >= ub && r0 + kCh <= ub + nt && (r0 + kCh <= ub + nm || r0 >= ub + nm + nr);
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

// The transpose of an 8x8 b16 matrix held in the m8n8 fragment layout (lane
// l: row l / 4, columns 2 (l % 4) and 2 (l % 4) + 1).
__device__ __forceinline__ uint32_t movm_t(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
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

// 2^x with the hardware approximation (ex2.approx.ftz, PTX ISA): 2^-inf = +0.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
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

// ldmatrix row addresses of this lane (byte offsets inside a stage): for
// K Q^T the A fragments of slots 0..15 x dims 16j..16j+15 (j = 0..3; dims
// 64..127 one box further), for P V the eight 16-dim groups of V rows
// (transposed loads).
__device__ __forceinline__ void tile_offsets(int lane, uint32_t (&off_k)[4], uint32_t (&off_pv)[8]) {
  const int r8 = lane & 7, mi = lane >> 3;
#pragma unroll
  for (int j = 0; j < 4; ++j) {                 // matrix mi: slots 8 (mi & 1).., dims 16j + 8 (mi >> 1)..
    const int cc = 2 * j + (mi >> 1);
    off_k[j] = (mi & 1) * 1024 + r8 * 128 + ((cc ^ r8) << 4);
  }
#pragma unroll
  for (int q = 0; q < 8; ++q) {                 // dims 16q..16q+15
    const int cg = 2 * q + (mi >> 1), half = cg >> 3, cc = cg & 7, nt = mi & 1;
    off_pv[q] = 2 * kBox + half * kBox + nt * 1024 + r8 * 128 + ((cc ^ r8) << 4);
  }
}

// B operand of K Q^T for column g = lane / 4 (query head g % G; zero from
// column 2G on): the words at dims 16kk + 2qp (+1) and 16kk + 8 + 2qp (+1) of
// Q row `qrow0 + (g % G)`.
template <int G>
__device__ __forceinline__ void load_q_frag(const __nv_bfloat16* Q, int64_t qrow0, int lane,
                                            uint32_t (&dst)[16]) {
  const int g = lane >> 2, qp = lane & 3;
  const bool hv = g < 2 * G;
  const uint32_t* qw = reinterpret_cast<const uint32_t*>(Q + (qrow0 + g % G) * kHeadDim);
#pragma unroll
  for (int kk = 0; kk < 8; ++kk) {
    dst[2 * kk] = hv ? __ldg(qw + 8 * kk + qp) : 0u;
    dst[2 * kk + 1] = hv ? __ldg(qw + 8 * kk + 4 + qp) : 0u;
  }
}

// Per-warp staging of a unit's query rows and output rows (stream-K kernel):
// the G query rows arrive by 16-byte cp.async copies into one of two buffers
// (the current unit and the next), the G output rows leave as whole 512-byte
// rows.  Rows are padded so that the fragment reads and the output writes hit
// distinct banks.  Whole-row transfers matter most when Q and O sit in host
// memory and cross the host link.
constexpr int kQRowBytes = kHeadDim * 2 + 16;                        // 272
constexpr int kORowFloats = kHeadDim + 8;                            // 136
constexpr int kIoBytes = 2 * 4 * kQRowBytes + 4 * kORowFloats * 4;   // G <= 4

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}

// Online-softmax state of one unit.  O[dt][0..1] = accumulator row g (hi
// weights of column g) and O[dt][2..3] = row g + 8 (lo weights of the same
// column) at dims 8dt + 2qp (+1).  The lane's softmax columns are 2qp and
// 2qp + 1: m = their reference maxima (equal in the column's 8 lanes), l and
// mt = this lane's share of their sums and largest logits (over slots g and
// g + 8 of every tile), reduced when the unit finishes.  Logits in log2 units.
struct TileState {
  float O[16][4];
  float m[2], l[2], mt[2];

  __device__ __forceinline__ void reset() {
#pragma unroll
    for (int dt = 0; dt < 16; ++dt) O[dt][0] = O[dt][1] = O[dt][2] = O[dt][3] = 0.f;
    m[0] = m[1] = kMInit;
    l[0] = l[1] = 0.f;
    mt[0] = mt[1] = -INFINITY;
  }
};

// A staged 16-slot tile in registers: the A fragments of K (slots x dims
// 16kk..16kk+15) for K Q^T, the B fragments of V (slots x dims 16q..16q+15)
// for P V, and the log-counts of slots g and g + 8.  Once a warp holds them
// it may refill the stage: the copy into it overlaps the tile's softmax and
// P V.
struct TileFrags {
  uint32_t k[8][4];
  uint32_t v[8][4];
  float lc[2];
};

__device__ __forceinline__ void tile_load(uint32_t st, const float* lc, const uint32_t (&off_k)[4],
                                          const uint32_t (&off_pv)[8], int lane, TileFrags& F) {
#pragma unroll
  for (int kk = 0; kk < 8; ++kk)
    ldsm_x4(st + off_k[kk & 3] + (kk >> 2) * kBox, F.k[kk][0], F.k[kk][1], F.k[kk][2], F.k[kk][3]);
#pragma unroll
  for (int q = 0; q < 8; ++q) ldsm_x4_t(st + off_pv[q], F.v[q][0], F.v[q][1], F.v[q][2], F.v[q][3]);
  const int g = lane >> 2;
  F.lc[0] = lc[g];
  F.lc[1] = lc[g + 8];
}

// Fold a 16-slot tile (first global slot t0) into `S`.  Slots y in
// [rlo, rhi) are residual entries (folded into the residual columns when
// kResidual; a main-only pass skips them), the other slots in [mlo, mhi) are
// exact main rows (selected tokens and rows appended at decode time); every
// other row is masked.  kPureMain: the caller has checked that all 16 slots
// are main rows (no bounds are read).  Slot indices fit in 32 bits (a cache
// holds fewer than 2^31 slots).
template <int G, bool kPureMain, bool kResidual = true>
__device__ __forceinline__ void tile_update(TileState& S, const TileFrags& F, int t0, int mlo,
                                            int mhi, int rlo, int rhi, const uint32_t (&qb)[16],
                                            float qscale, int lane) {
  const int g = lane >> 2, qp = lane & 3;
  // ---- logits S^T = K Q^T: four accumulator chains of two 16-dim steps ----
  float Sc[4][4];
#pragma unroll
  for (int c = 0; c < 4; ++c) Sc[c][0] = Sc[c][1] = Sc[c][2] = Sc[c][3] = 0.f;
#pragma unroll
  for (int kk = 0; kk < 8; ++kk)
    mma16816(Sc[kk & 3], F.k[kk][0], F.k[kk][1], F.k[kk][2], F.k[kk][3], qb[2 * kk], qb[2 * kk + 1]);
  float sv[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) sv[j] = ((Sc[0][j] + Sc[1][j]) + (Sc[2][j] + Sc[3][j])) * qscale;
  // x[i][e]: slot g + 8i, column 2qp + e
  float x[2][2] = {{sv[0], sv[1]}, {sv[2], sv[3]}};
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int c = 2 * qp + e;
    const bool cM = c < G, cR = kResidual && c >= G && c < 2 * G;
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      if constexpr (kPureMain) {
        x[i][e] = cM ? x[i][e] : -INFINITY;
      } else {
        const int y = t0 + g + 8 * i;
        const bool inR = y >= rlo && y < rhi;
        const bool sM = y >= mlo && y < mhi && !inR;
        x[i][e] = (cM && sM) ? x[i][e]
                  : (cR && inR) ? x[i][e] + F.lc[i] * kLog2e   // + beta log c_j
                                : -INFINITY;
      }
    }
  }
#pragma unroll
  for (int e = 0; e < 2; ++e) S.mt[e] = fmaxf(S.mt[e], fmaxf(x[0][e], x[1][e]));
  // ---- raise the reference maxima when a logit passes them by more than kLazy ----
  const bool up = fmaxf(x[0][0], x[1][0]) > S.m[0] + kLazy || fmaxf(x[0][1], x[1][1]) > S.m[1] + kLazy;
  if (__any_sync(0xffffffffu, up)) {
    float sc[2];
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      float t = fmaxf(x[0][e], x[1][e]);
      t = fmaxf(t, __shfl_xor_sync(0xffffffffu, t, 4));
      t = fmaxf(t, __shfl_xor_sync(0xffffffffu, t, 8));
      t = fmaxf(t, __shfl_xor_sync(0xffffffffu, t, 16));
      const float mn = fmaxf(S.m[e], t);
      sc[e] = exp2f(S.m[e] - mn);
      S.l[e] *= sc[e];
      S.m[e] = mn;
    }
    // accumulator rows g and g + 8 belong to column g, held by lane 4g + g/2
    const float rs = __shfl_sync(0xffffffffu, (g & 1) ? sc[1] : sc[0], 4 * g + (g >> 1));
#pragma unroll
    for (int dt = 0; dt < 16; ++dt) {
      S.O[dt][0] *= rs;
      S.O[dt][1] *= rs;
      S.O[dt][2] *= rs;
      S.O[dt][3] *= rs;
    }
  }
  float pr[2][2];
#pragma unroll
  for (int i = 0; i < 2; ++i)
#pragma unroll
    for (int e = 0; e < 2; ++e) pr[i][e] = ex2_approx(x[i][e] - S.m[e]);   // masked: 0
  S.l[0] += pr[0][0] + pr[1][0];
  S.l[1] += pr[0][1] + pr[1][1];
  // P^T (slots x columns) as bf16 hi + lo parts, transposed into the A layout
  const uint32_t ha = pack_bf16(pr[0][0], pr[0][1]), hb = pack_bf16(pr[1][0], pr[1][1]);
  const float2 fa = unpack_bf16(ha), fb = unpack_bf16(hb);
  const uint32_t la = pack_bf16(pr[0][0] - fa.x, pr[0][1] - fa.y);
  const uint32_t lb = pack_bf16(pr[1][0] - fb.x, pr[1][1] - fb.y);
  const uint32_t a0 = movm_t(ha), a1 = movm_t(la), a2 = movm_t(hb), a3 = movm_t(lb);
  // ---- O += P V ----
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    mma16816(S.O[2 * q], a0, a1, a2, a3, F.v[q][0], F.v[q][1]);
    mma16816(S.O[2 * q + 1], a0, a1, a2, a3, F.v[q][2], F.v[q][3]);
  }
}

// Whether the 16 slots from t0 are all main rows of the given bounds.
__device__ __forceinline__ bool tile_pure_main(int t0, int mlo, int mhi, int rlo, int rhi) {
  return t0 >= mlo && t0 + kCh <= mhi && (rhi <= t0 || rlo >= t0 + kCh || rlo >= rhi);
}

// Statistics of the softmax column g = lane / 4 (accumulator rows g, g + 8):
// reference max m, sum l and largest logit mt over the unit's slots so far.
// Every lane of the warp calls it.
struct RowStats {
  float m, l, mt;
};

__device__ __forceinline__ RowStats tile_row_stats(const TileState& S, int lane) {
  float l0 = S.l[0], l1 = S.l[1], t0 = S.mt[0], t1 = S.mt[1];
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, o);
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
    t0 = fmaxf(t0, __shfl_xor_sync(0xffffffffu, t0, o));
    t1 = fmaxf(t1, __shfl_xor_sync(0xffffffffu, t1, o));
  }
  const int g = lane >> 2, src = 4 * g + (g >> 1);   // lane holding column g
  const bool odd = g & 1;
  RowStats r;
  r.m = __shfl_sync(0xffffffffu, odd ? S.m[1] : S.m[0], src);
  r.l = __shfl_sync(0xffffffffu, odd ? l1 : l0, src);
  r.mt = __shfl_sync(0xffffffffu, odd ? t1 : t0, src);
  return r;
}

// Numerator of column g at dims 8dt + 2qp (+1): hi row plus lo row.
__device__ __forceinline__ float2 tile_row_value(const TileState& S, int dt) {
  return make_float2(S.O[dt][0] + S.O[dt][2], S.O[dt][1] + S.O[dt][3]);
}

// The sum relative to the largest weight (what gate_of takes for the main
// branch), from a (reference max, sum, largest logit) triple; 0 when empty.
__device__ __forceinline__ float sum_rel_max(float m, float l, float mt) {
  return l > 0.f ? l * exp2f(m - mt) : 0.f;
}

}  // namespace reskv
