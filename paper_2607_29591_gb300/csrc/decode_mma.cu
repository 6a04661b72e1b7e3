// Shared-softmax residual decode (Alg. 2; Sec. 5.4 Eqs. residual_logit,
// reskv_den, reskv_num, reskv; Sec. 5.5.2 Eq. gate) on the tensor cores,
// stream-K over the whole slot range of a launch.
//
// Launches are programmatic dependent launches (a kernel streams its first
// ring of cache chunks while the previous kernel on the stream finishes).
//
// Same split of work as the CUDA-core kernel (decode_kernel.cu): a launch
// streams the flat slot range of its units, cut into W equal contiguous
// pieces, one per warp; units cut between warps are merged by the last warp
// to arrive.  What changes is the inner loop, which is instruction-bound on
// CUDA cores (about 50 warp instructions per 512-byte slot).  Here one warp
// step covers a 16-slot tile with legacy tensor-core MMAs (mma_tile.cuh).
//
// K and V rows reach shared memory through 2-D TMA tensor copies with the
// 128-byte swizzle; the residual log-counts of each 16-slot chunk ride along
// as a 64-byte bulk copy.  Chunks are aligned to 16 global slots; rows outside
// the warp's piece are masked.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdint>

#include "device_utils.cuh"
#include "internal.h"
#include "mma_tile.cuh"

namespace reskv {
namespace {

constexpr int kMaxW = kMmaMaxW;
constexpr int kMaxSt = kMmaMaxSt;

__device__ __forceinline__ int64_t warp_begin(int64_t w, int64_t T, int64_t W) { return (w * T) / W; }
__device__ __forceinline__ int64_t warp_of(int64_t x, int64_t T, int64_t W) { return ((x + 1) * W - 1) / T; }

// kRagged: units at p.offsets[u] (per-unit budgets); otherwise at u * stride.
template <int G, bool kRagged>
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
  const int64_t b = p.stride;
  // first slot of unit uu
  auto ustart = [&](int64_t uu) -> int64_t {
    if constexpr (kRagged) return p.offsets[uu];
    else return uu * b;
  };
  const int64_t gbase = ustart(p.unit0);
  int64_t ga, ge;
  if (p.units_per_warp > 0) {            // whole units [gw k, (gw + 1) k)
    const int64_t k = p.units_per_warp;
    const int64_t u_lo = gw * k, u_hi = u_lo + k < p.n_units ? u_lo + k : p.n_units;
    if (u_lo >= u_hi) return;
    ga = ustart(p.unit0 + u_lo);
    ge = ustart(p.unit0 + u_hi);
  } else {                               // equal slot pieces
    ga = gbase + warp_begin(gw, T, W);
    ge = gbase + warp_begin(gw + 1, T, W);
  }
  if (ga >= ge) return;
  // first unit with used slots in [ga, ge): the piece may start in the unused
  // tail slots of a unit (past its n_main + n_res + n_app used rows), which
  // this warp must skip
  int64_t u;
  if constexpr (kRagged) {              // last unit starting at or before ga
    int64_t lo = p.unit0, hi = p.unit0 + p.n_units;
    while (hi - lo > 1) {
      const int64_t mid = (lo + hi) >> 1;
      if (p.offsets[mid] <= ga) lo = mid;
      else hi = mid;
    }
    u = lo;
  } else {
    u = ga / b;
  }
  if (ustart(u) + p.n_main[u] + p.n_res[u] + (p.n_app ? p.n_app[u] : 0) <= ga) ++u;
  if (ustart(u) >= ge) return;

  // per-warp shared memory, 1024-byte aligned for the 128-byte swizzle
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = ((raw + 1023u) & ~1023u) + uint32_t(warp) * kWarpBytes;
  uint8_t* base_ptr = smem_raw + (base - raw);
  float* logc_s = reinterpret_cast<float*>(base_ptr + warp_logc_offset(kSt));   // [kSt][16]
  uint64_t* bars = reinterpret_cast<uint64_t*>(base_ptr + warp_bars_offset(kSt));

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
  // Programmatic dependent launch: the next kernel on the stream may start
  // now and overlap its prologue and first cache copies with this kernel.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  uint32_t off_qk[4], off_pv[8];
  tile_offsets(lane, off_qk, off_pv);

  const float qscale = kLog2e * rsqrtf(float(kHeadDim));
  bool failed = false;

  // unit cursor and its query fragments (the next unit's are loaded ahead)
  uint32_t qa[16], qn[16];
  int32_t nm = 0, nr = 0, nt = 0, nm_n = 0, nr_n = 0, nt_n = 0;   // main, residual, used rows
  auto load_q = [&](int64_t uu, uint32_t (&dst)[16], int32_t& m_out, int32_t& r_out,
                    int32_t& t_out) {
    const int64_t ul = uu - p.unit0;
    const int64_t qrow = (ul / p.n_kv_heads) * int64_t(p.n_kv_heads) * G + (ul % p.n_kv_heads) * G + h;
    load_q_frag(p.Q, qrow, hv, qp, dst);
    m_out = p.n_main[uu];
    r_out = p.n_res[uu];
    t_out = m_out + r_out + (p.n_app ? p.n_app[uu] : 0);
  };
  // Q, O, the partial records and the tickets only after the previous kernel
  // on the stream has completed (before: the cache alone, which no kernel
  // that may run concurrently writes)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  load_q(u, qa, nm, nr, nt);
  if (ustart(u + 1) < ge) load_q(u + 1, qn, nm_n, nr_n, nt_n);

  TileState S;
  S.reset();
  float(&O)[16][4] = S.O;
  float &mM = S.mM, &lM = S.lM, &mR = S.mR, &lR = S.lR;

  // Finish unit uu: write o^ (whole unit in this warp) or a partial record.
  auto finish = [&](int64_t uu, int32_t ut) {
    float lMt = lM + __shfl_xor_sync(0xffffffffu, lM, 1);
    lMt += __shfl_xor_sync(0xffffffffu, lMt, 2);
    float lRt = lR + __shfl_xor_sync(0xffffffffu, lR, 1);
    lRt += __shfl_xor_sync(0xffffffffu, lRt, 2);
    const int64_t ubase = ustart(uu), uend = ubase + ut;
    const int64_t ul = uu - p.unit0;
    const int64_t orow = (ul / p.n_kv_heads) * int64_t(p.n_kv_heads) * G + (ul % p.n_kv_heads) * G + h;
    if (ga <= ubase && ge >= uend) {
      if (hv) {
        const float2 w = branch_coefs(p.softmax_mode, gate_of(p, lMt), mM, lMt, mR, lRt);
        float* op = p.O + orow * kHeadDim + 2 * qp;
#pragma unroll
        for (int dt = 0; dt < 16; ++dt)
          *reinterpret_cast<float2*>(op + dt * 8) =
              make_float2(w.x * O[dt][0] + w.y * O[dt][2], w.x * O[dt][1] + w.y * O[dt][3]);
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
      const float2 w = branch_coefs(p.softmax_mode, gate_of(p, Ls[0]), Ms[0], Ls[0], Ms[1], Ls[1]);
      float* op = p.O + orow * kHeadDim + 2 * qp;
#pragma unroll
      for (int dt = 0; dt < 16; ++dt)
        *reinterpret_cast<float2*>(op + dt * 8) =
            make_float2(w.x * acc[0][2 * dt] + w.y * acc[1][2 * dt],
                        w.x * acc[0][2 * dt + 1] + w.y * acc[1][2 * dt + 1]);
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
      const int64_t ubase = ustart(u);
      const int64_t mlo = ubase > ga ? ubase : ga;
      const int64_t mhi = (ubase + nt < ge) ? ubase + nt : ge;   // main + appended rows
      const int64_t rlo = (ubase + nm > ga) ? ubase + nm : ga;
      const int64_t rhi = (ubase + nm + nr < ge) ? ubase + nm + nr : ge;
      const bool any = (mlo < mhi && mlo < t0 + kCh && mhi > t0) ||
                       (rlo < rhi && rlo < t0 + kCh && rhi > t0);
      if (any)
        tile_update(S, st, lc, t0, mlo, mhi, rlo, rhi, qa, off_qk, off_pv,
                    qscale, hv, qp);
      // does unit u end inside this tile (or at the end of the piece)?
      const int64_t uend = ubase + nt;
      const int64_t stop = uend < ge ? uend : ge;
      if (stop > t0 + kCh) break;                        // continues in the next tile
      finish(u, nt);
      S.reset();
      ++u;
      if (ustart(u) >= ge) {
        done = true;
        break;
      }
#pragma unroll
      for (int i = 0; i < 16; ++i) qa[i] = qn[i];
      nm = nm_n;
      nr = nr_n;
      nt = nt_n;
      if (ustart(u + 1) < ge) load_q(u + 1, qn, nm_n, nr_n, nt_n);
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

template <int G, bool kRagged>
static cudaError_t launch_mma_g(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                                int n_ctas, int warps_per_cta, cudaStream_t stream) {
  static std::atomic<unsigned long long> configured{0};
  const int smem = warps_per_cta * warp_bytes(p.n_stages) + 1024;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  const unsigned long long bit = 1ull << (dev & 63);
  if (!(configured.load() & bit)) {
    err = cudaFuncSetAttribute(reskv_decode_mma_kernel<G, kRagged>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit);
    if (err != cudaSuccess) return err;
    configured.fetch_or(bit);
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(n_ctas), 1, 1);
  cfg.blockDim = dim3(unsigned(warps_per_cta) * 32u, 1, 1);
  cfg.dynamicSmemBytes = size_t(smem);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // see griddepcontrol
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  err = cudaLaunchKernelEx(&cfg, reskv_decode_mma_kernel<G, kRagged>, p, tk, tv);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

cudaError_t launch_decode_mma(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                              int group, int n_ctas, int warps_per_cta, cudaStream_t stream) {
  const bool ragged = p.offsets != nullptr;
  switch (group) {
    case 1: return ragged ? launch_mma_g<1, true>(p, tk, tv, n_ctas, warps_per_cta, stream)
                          : launch_mma_g<1, false>(p, tk, tv, n_ctas, warps_per_cta, stream);
    case 2: return ragged ? launch_mma_g<2, true>(p, tk, tv, n_ctas, warps_per_cta, stream)
                          : launch_mma_g<2, false>(p, tk, tv, n_ctas, warps_per_cta, stream);
    case 4: return ragged ? launch_mma_g<4, true>(p, tk, tv, n_ctas, warps_per_cta, stream)
                          : launch_mma_g<4, false>(p, tk, tv, n_ctas, warps_per_cta, stream);
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
