// Shared-softmax residual decode (Alg. 2; Sec. 5.4 Eqs. residual_logit,
// reskv_den, reskv_num, reskv; Sec. 5.5.2 Eq. gate) on the tensor cores.
//
// Same split of work as the CUDA-core kernel (decode_kernel.cu): a launch
// streams the flat slot range of its units, cut into W equal contiguous
// pieces, one per warp; units cut between warps are merged by the last warp
// to arrive.  What changes is the inner loop, which is instruction-bound on
// CUDA cores (about 50 warp instructions per 512-byte slot).  Here one warp
// step covers a 16-slot tile with legacy tensor-core MMAs (mma.sync
// m16n8k16, bf16 in, fp32 accumulate):
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
// K and V rows reach shared memory through 2-D TMA tensor copies with the
// 128-byte swizzle (boxes of 64 dims x 16 slots), so that ldmatrix reads of
// eight rows at one column are bank-conflict free; the residual log-counts of
// each 16-slot chunk ride along as a 64-byte bulk copy.  Chunks are aligned to
// 16 global slots; rows outside the warp's piece are masked.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdint>

#include "device_utils.cuh"
#include "internal.h"

namespace reskv {
namespace {

constexpr int kMaxW = 8;                // warps per CTA (at most)
constexpr int kMaxSt = 12;              // ring stages per warp (at most)
constexpr int kCh = 16;                 // slots per stage (= one MMA tile)
constexpr int kBox = kCh * 128;         // one 64-dim half of 16 rows, bytes
constexpr int kStageBytes = 4 * kBox;   // K lo | K hi | V lo | V hi
constexpr int kRec = kHeadDim + 4;      // m, l, pad, pad, acc[d]
constexpr int kSmemLimit = 227 * 1024;  // dynamic shared memory per CTA

__host__ __device__ constexpr int warp_bytes(int stages) { return stages * kStageBytes + 1024; }

__device__ __forceinline__ int64_t warp_begin(int64_t w, int64_t T, int64_t W) { return (w * T) / W; }
__device__ __forceinline__ int64_t warp_of(int64_t x, int64_t T, int64_t W) { return ((x + 1) * W - 1) / T; }

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

__device__ __forceinline__ float gate_of(const DecodeParams& p, float lM) {
  if (p.gate_mode == RESKV_GATE_FIXED) return p.g_fixed;
  const float p_max = 1.0f / lM;                  // the largest main weight (2^0 / sum)
  return fmaxf(p.g_min, 1.0f / (1.0f + expf(-p.alpha * (p.tau - p_max))));
}

template <int G>
__global__ void __launch_bounds__(kMaxW * 32, 1)
    reskv_decode_mma_kernel(const DecodeParams p, const __grid_constant__ CUtensorMap tmK,
                            const __grid_constant__ CUtensorMap tmV) {
  extern __shared__ uint8_t smem_raw[];
  const int kW = blockDim.x >> 5;       // warps per CTA of this launch
  const int kSt = p.n_stages;           // ring stages per warp of this launch
  const int kWarpBytes = warp_bytes(kSt);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = lane >> 2;              // query head (row of the mma tile)
  const int qp = lane & 3;              // position in the quad
  const bool hv = h < G;
  const int64_t gw = int64_t(blockIdx.x) * kW + warp;
  if (gw >= p.n_warps) return;
  const int64_t T = p.total_slots, W = p.n_warps;
  const int64_t b = p.budget;
  const int64_t gbase = p.unit0 * b;
  const int64_t ga = gbase + warp_begin(gw, T, W), ge = gbase + warp_begin(gw + 1, T, W);
  if (ga >= ge) return;
  // first unit with used slots in [ga, ge): the piece may start in the unused
  // tail slots of a unit (n_main + n_res < budget), which this warp must skip
  int64_t u = ga / b;
  if (u * b + p.n_main[u] + p.n_res[u] <= ga) ++u;
  if (u * b >= ge) return;

  // per-warp shared memory, 1024-byte aligned for the 128-byte swizzle
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = ((raw + 1023u) & ~1023u) + uint32_t(warp) * kWarpBytes;
  uint8_t* base_ptr = smem_raw + (base - raw);
  float* logc_s = reinterpret_cast<float*>(base_ptr + kSt * kStageBytes);        // [kSt][16]
  uint64_t* bars = reinterpret_cast<uint64_t*>(base_ptr + kSt * kStageBytes + kMaxSt * kCh * 4);

  const int64_t cb = ga & ~int64_t(kCh - 1);              // first chunk, 16-slot aligned
  const int64_t nchunks = (ge - cb + kCh - 1) / kCh;

  if (lane == 0) {
    for (int s = 0; s < kSt; ++s) mbar_init(&bars[s], 1);
    fence_mbar_init();
  }
  __syncwarp();

  auto issue = [&](int64_t k) {        // lane 0
    const int s = int(k % kSt);
    const int row = int(cb + k * kCh);
    const uint32_t st = base + s * kStageBytes;
    mbar_arrive_expect_tx(&bars[s], kStageBytes + kCh * 4);
    tma_load_2d(st, &tmK, 0, row, &bars[s]);
    tma_load_2d(st + kBox, &tmK, 64, row, &bars[s]);
    tma_load_2d(st + 2 * kBox, &tmV, 0, row, &bars[s]);
    tma_load_2d(st + 3 * kBox, &tmV, 64, row, &bars[s]);
    bulk_g2s(logc_s + s * kCh, p.logc + row, kCh * 4, &bars[s]);
  };
  if (lane == 0)
    for (int64_t k = 0; k < nchunks && k < kSt; ++k) issue(k);

  // ldmatrix row addresses of this lane (byte offsets inside a stage)
  const int r8 = lane & 7, mi = lane >> 3;
  uint32_t off_qk[4], off_pv[8];
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

  const float qscale = kLog2e * rsqrtf(float(kHeadDim));
  bool failed = false;

  // unit cursor and its query fragments (A operand of Q K^T: words of head h
  // at dims 16kk + 2qp (+1) and 16kk + 8 + 2qp (+1))
  uint32_t qa[16], qn[16];
  int32_t nm = 0, nr = 0, nm_n = 0, nr_n = 0;
  auto load_q = [&](int64_t uu, uint32_t* dst, int32_t& m_out, int32_t& r_out) {
    const int64_t ul = uu - p.unit0;
    const int64_t qrow = (ul / p.n_kv_heads) * int64_t(p.n_kv_heads) * G + (ul % p.n_kv_heads) * G + h;
    const uint32_t* qw = reinterpret_cast<const uint32_t*>(p.Q + qrow * kHeadDim);
#pragma unroll
    for (int kk = 0; kk < 8; ++kk) {
      dst[2 * kk] = hv ? __ldg(qw + 8 * kk + qp) : 0u;
      dst[2 * kk + 1] = hv ? __ldg(qw + 8 * kk + 4 + qp) : 0u;
    }
    m_out = p.n_main[uu];
    r_out = p.n_res[uu];
  };
  load_q(u, qa, nm, nr);
  if ((u + 1) * b < ge) load_q(u + 1, qn, nm_n, nr_n);

  float O[16][4];
  float mM = -INFINITY, lM = 0.f, mR = -INFINITY, lR = 0.f;
  auto reset = [&]() {
#pragma unroll
    for (int dt = 0; dt < 16; ++dt) O[dt][0] = O[dt][1] = O[dt][2] = O[dt][3] = 0.f;
    mM = mR = -INFINITY;
    lM = lR = 0.f;
  };
  reset();

  // Finish unit uu: write o^ (whole unit in this warp) or a partial record.
  auto finish = [&](int64_t uu, int32_t um, int32_t ur) {
    float lMt = lM + __shfl_xor_sync(0xffffffffu, lM, 1);
    lMt += __shfl_xor_sync(0xffffffffu, lMt, 2);
    float lRt = lR + __shfl_xor_sync(0xffffffffu, lR, 1);
    lRt += __shfl_xor_sync(0xffffffffu, lRt, 2);
    const int64_t ubase = uu * b, uend = ubase + um + ur;
    const int64_t ul = uu - p.unit0;
    const int64_t orow = (ul / p.n_kv_heads) * int64_t(p.n_kv_heads) * G + (ul % p.n_kv_heads) * G + h;
    if (ga <= ubase && ge >= uend) {
      if (hv) {
        const float g = gate_of(p, lMt);
        float wM = 1.f, wR = 0.f;
        if (lRt > 0.f && g > 0.f) {
          const float mx = fmaxf(mM, mR);
          wM = exp2f(mM - mx);
          wR = g * exp2f(mR - mx);
        }
        const float inv = 1.0f / (wM * lMt + wR * lRt);
        float* op = p.O + orow * kHeadDim + 2 * qp;
#pragma unroll
        for (int dt = 0; dt < 16; ++dt)
          *reinterpret_cast<float2*>(op + dt * 8) =
              make_float2((wM * O[dt][0] + wR * O[dt][2]) * inv, (wM * O[dt][1] + wR * O[dt][3]) * inv);
      }
      return;
    }
    const int64_t flat0 = ubase - gbase;
    const int64_t w0 = warp_of(flat0, T, W), w1 = warp_of(uend - 1 - gbase, T, W);
    float* rec = p.partials + (ul + gw) * (2 * G * kRec);
    if (hv) {
      float* rm = rec + (0 * G + h) * kRec;
      float* rr = rec + (1 * G + h) * kRec;
      if (qp == 0) {
        rm[0] = mM;
        rm[1] = lMt;
        rr[0] = mR;
        rr[1] = lRt;
      }
#pragma unroll
      for (int dt = 0; dt < 16; ++dt) {
        *reinterpret_cast<float2*>(rm + 4 + dt * 8 + 2 * qp) = make_float2(O[dt][0], O[dt][1]);
        *reinterpret_cast<float2*>(rr + 4 + dt * 8 + 2 * qp) = make_float2(O[dt][2], O[dt][3]);
      }
    }
    __threadfence();
    __syncwarp();
    int ticket = 0;
    if (lane == 0) ticket = atomicAdd(p.tickets + uu, 1);
    ticket = __shfl_sync(0xffffffffu, ticket, 0);
    if (ticket != int(w1 - w0)) return;
    __threadfence();
    if (hv) {
      // one pass over the records in warp order (online log-sum-exp merge)
      float Ms[2] = {-INFINITY, -INFINITY}, Ls[2] = {0.f, 0.f};
      float acc[2][32];
#pragma unroll
      for (int sg = 0; sg < 2; ++sg)
#pragma unroll
        for (int i = 0; i < 32; ++i) acc[sg][i] = 0.f;
      for (int64_t w = w0; w <= w1; ++w) {
        const float* rr = p.partials + (ul + w) * (2 * G * kRec);
#pragma unroll
        for (int sg = 0; sg < 2; ++sg) {
          const float* r = rr + (sg * G + h) * kRec;
          const float rm = __ldcg(r), rl = __ldcg(r + 1);
          float2 v[16];
#pragma unroll
          for (int dt = 0; dt < 16; ++dt)
            v[dt] = __ldcg(reinterpret_cast<const float2*>(r + 4 + dt * 8 + 2 * qp));
          if (rl > 0.f) {
            const float mx = fmaxf(Ms[sg], rm);
            const float sa = exp2f(Ms[sg] - mx), sb = exp2f(rm - mx);
            Ls[sg] = Ls[sg] * sa + rl * sb;
#pragma unroll
            for (int dt = 0; dt < 16; ++dt) {
              acc[sg][2 * dt] = acc[sg][2 * dt] * sa + v[dt].x * sb;
              acc[sg][2 * dt + 1] = acc[sg][2 * dt + 1] * sa + v[dt].y * sb;
            }
            Ms[sg] = mx;
          }
        }
      }
      const float g = gate_of(p, Ls[0]);
      float wM = 1.f, wR = 0.f;
      if (Ls[1] > 0.f && g > 0.f) {
        const float mx = fmaxf(Ms[0], Ms[1]);
        wM = exp2f(Ms[0] - mx);
        wR = g * exp2f(Ms[1] - mx);
      }
      const float inv = 1.0f / (wM * Ls[0] + wR * Ls[1]);
      float* op = p.O + orow * kHeadDim + 2 * qp;
#pragma unroll
      for (int dt = 0; dt < 16; ++dt)
        *reinterpret_cast<float2*>(op + dt * 8) =
            make_float2((wM * acc[0][2 * dt] + wR * acc[1][2 * dt]) * inv,
                        (wM * acc[0][2 * dt + 1] + wR * acc[1][2 * dt + 1]) * inv);
    }
    __syncwarp();
    if (lane == 0) p.tickets[uu] = 0;
  };

  bool done = false;
  int64_t issued = nchunks < kSt ? nchunks : kSt;     // chunks [0, issued) requested
  int64_t waited = 0;                                 // chunks [0, waited) completed
  for (int64_t k = 0; k < nchunks && !done; ++k) {
    const int s = int(k % kSt);
    if (!mbar_wait_bounded(&bars[s], uint32_t((k / kSt) & 1))) {
      failed = true;
      if (lane == 0) report_status(p.status, kStatusWaitTimeout);
      break;
    }
    waited = k + 1;
    const int64_t t0 = cb + k * kCh;
    const uint32_t st = base + s * kStageBytes;
    const float* lc = logc_s + s * kCh;
    // every unit with rows in this tile
    while (true) {
      const int64_t ubase = u * b;
      const int64_t mlo = ubase > ga ? ubase : ga;
      const int64_t mhi = (ubase + nm < ge) ? ubase + nm : ge;
      const int64_t rlo = (ubase + nm > ga) ? ubase + nm : ga;
      const int64_t rhi = (ubase + nm + nr < ge) ? ubase + nm + nr : ge;
      const bool any = (mlo < mhi && mlo < t0 + kCh && mhi > t0) ||
                       (rlo < rhi && rlo < t0 + kCh && rhi > t0);
      if (any) {
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
          const bool im = hv && y >= mlo && y < mhi;
          const bool ir = hv && y >= rlo && y < rhi;
          sM[e] = im ? sv[e] : -INFINITY;
          sR[e] = ir ? sv[e] + lc[rowi] * kLog2e : -INFINITY;   // + beta log c_j
        }
        float tM = fmaxf(fmaxf(sM[0], sM[1]), fmaxf(sM[2], sM[3]));
        float tR = fmaxf(fmaxf(sR[0], sR[1]), fmaxf(sR[2], sR[3]));
        tM = fmaxf(tM, __shfl_xor_sync(0xffffffffu, tM, 1));
        tM = fmaxf(tM, __shfl_xor_sync(0xffffffffu, tM, 2));
        tR = fmaxf(tR, __shfl_xor_sync(0xffffffffu, tR, 1));
        tR = fmaxf(tR, __shfl_xor_sync(0xffffffffu, tR, 2));
        if (tM > mM) {                                   // rescale the main rows
          const float sc = exp2f(mM - tM);
          lM *= sc;
#pragma unroll
          for (int dt = 0; dt < 16; ++dt) {
            O[dt][0] *= sc;
            O[dt][1] *= sc;
          }
          mM = tM;
        }
        if (tR > mR) {                                   // rescale the residual rows
          const float sc = exp2f(mR - tR);
          lR *= sc;
#pragma unroll
          for (int dt = 0; dt < 16; ++dt) {
            O[dt][2] *= sc;
            O[dt][3] *= sc;
          }
          mR = tR;
        }
        float pM[4], pR[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          pM[e] = sM[e] > -INFINITY ? exp2f(sM[e] - mM) : 0.f;   // masked rows weigh 0
          pR[e] = sR[e] > -INFINITY ? exp2f(sR[e] - mR) : 0.f;
          lM += pM[e];
          lR += pR[e];
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
          mma16816(O[2 * q], h0, h1, h2, h3, v0, v1);
          mma16816(O[2 * q + 1], h0, h1, h2, h3, v2, v3);
          mma16816(O[2 * q], l0, l1, l2, l3, v0, v1);
          mma16816(O[2 * q + 1], l0, l1, l2, l3, v2, v3);
        }
      }
      // does unit u end inside this tile (or at the end of the piece)?
      const int64_t uend = u * b + nm + nr;
      const int64_t stop = uend < ge ? uend : ge;
      if (stop > t0 + kCh) break;                        // continues in the next tile
      finish(u, nm, nr);
      reset();
      ++u;
      if (u * b >= ge) {
        done = true;
        break;
      }
#pragma unroll
      for (int i = 0; i < 16; ++i) qa[i] = qn[i];
      nm = nm_n;
      nr = nr_n;
      if ((u + 1) * b < ge) load_q(u + 1, qn, nm_n, nr_n);
    }
    if (done) break;
    __syncwarp();
    if (k + kSt < nchunks) {
      if (lane == 0) {
        fence_proxy_async_smem();
        issue(k + kSt);
      }
      issued = k + kSt + 1;
    }
  }
  // never leave with a copy in flight into this warp's ring (bounded waits)
  for (int64_t kk = waited; kk < issued; ++kk)
    mbar_wait_bounded(&bars[kk % kSt], uint32_t((kk / kSt) & 1));
  (void)failed;
}

}  // namespace

template <int G>
static cudaError_t launch_mma_g(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                                int n_ctas, int warps_per_cta, cudaStream_t stream) {
  static std::atomic<unsigned long long> configured{0};
  const int smem = warps_per_cta * warp_bytes(p.n_stages) + 1024;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  const unsigned long long bit = 1ull << (dev & 63);
  if (!(configured.load() & bit)) {
    err = cudaFuncSetAttribute(reskv_decode_mma_kernel<G>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit);
    if (err != cudaSuccess) return err;
    configured.fetch_or(bit);
  }
  reskv_decode_mma_kernel<G><<<n_ctas, warps_per_cta * 32, smem, stream>>>(p, tk, tv);
  return cudaGetLastError();
}

cudaError_t launch_decode_mma(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                              int group, int n_ctas, int warps_per_cta, cudaStream_t stream) {
  switch (group) {
    case 1: return launch_mma_g<1>(p, tk, tv, n_ctas, warps_per_cta, stream);
    case 2: return launch_mma_g<2>(p, tk, tv, n_ctas, warps_per_cta, stream);
    case 4: return launch_mma_g<4>(p, tk, tv, n_ctas, warps_per_cta, stream);
    default: return cudaErrorInvalidValue;
  }
}

// Ring depth for `warps_per_cta` warps sharing one SM's shared memory.
int decode_mma_stages(int warps_per_cta) {
  int st = ((kSmemLimit - 1024) / warps_per_cta - 1024) / kStageBytes;
  return st > kMaxSt ? kMaxSt : st;
}

size_t decode_mma_partials_floats(int64_t n_units, int n_warps, int group) {
  return size_t(n_units + n_warps) * 2 * group * kRec;
}

}  // namespace reskv
