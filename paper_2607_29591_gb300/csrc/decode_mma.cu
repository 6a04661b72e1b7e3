// Shared-softmax residual decode (Alg. 2; Sec. 5.4 Eqs. residual_logit,
// reskv_den, reskv_num, reskv; Sec. 5.5.2 Eq. gate) on the tensor cores,
// stream-K over the whole slot range of a launch.
//
// Launches are programmatic dependent launches (a kernel streams its first
// ring of cache chunks while the previous kernel on the stream finishes).
//
// A launch streams the flat slot range of its units as 16-slot chunks
// (aligned to 16 global slots), cut into W equal pieces of whole chunks, one
// per warp (or, for short units, k whole units per warp); units cut between
// warps are merged by the last warp to arrive.  The CUDA-core kernel
// (decode_kernel.cu) splits the same range by slots and is instruction-bound
// (about 50 warp instructions per 512-byte slot); here one warp step covers a
// 16-slot tile with legacy tensor-core MMAs (mma_tile.cuh).
//
// K and V rows reach shared memory through TMA tensor copies with the
// 128-byte swizzle; the residual log-counts of each chunk ride along as a
// 64-byte bulk copy.  Rows of a chunk outside the warp's units are masked.
// Each warp stages its units' query rows and output rows through shared
// memory as whole rows, which matters when Q and O sit in host memory.
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

// Warp w of W takes chunks [w N / W, (w + 1) N / W) of N; chunk c is in the
// piece of warp ((c + 1) W - 1) / N.
__device__ __forceinline__ int64_t piece_begin(int64_t w, int64_t N, int64_t W) { return (w * N) / W; }
__device__ __forceinline__ int64_t piece_of(int64_t c, int64_t N, int64_t W) { return ((c + 1) * W - 1) / N; }

// kRagged: units at p.offsets[u] (per-unit budgets); otherwise at u * stride.
// Slot and unit indices fit in 32 bits (a cache holds fewer than 2^31 slots).
template <int G, bool kRagged>
__global__ void __launch_bounds__(kMaxW * 32, 1)
    reskv_decode_mma_kernel(const DecodeParams p, const __grid_constant__ CUtensorMap tmK,
                            const __grid_constant__ CUtensorMap tmV) {
  extern __shared__ uint8_t smem_raw[];
  const int kW = blockDim.x >> 5;       // warps per CTA of this launch
  const int kSt = p.n_stages;           // ring stages per warp of this launch
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2;              // softmax column / accumulator row of this lane
  const int qp = lane & 3;              // position in the quad
  const int gw = int(blockIdx.x) * kW + warp;
  if (gw >= p.n_warps) return;
  const int64_t T = p.total_slots, W = p.n_warps;
  const int unit0 = int(p.unit0);
  // first slot of unit uu
  auto ustart = [&](int uu) -> int {
    if constexpr (kRagged) return p.offsets[uu];
    else return uu * p.stride;
  };
  const int gbase = ustart(unit0);
  // the launch's 16-slot chunks, aligned to global multiples of 16 like the
  // copies: equal pieces of whole chunks, so that no chunk is read twice
  const int base16 = gbase & ~(kCh - 1);
  const int64_t NC = (int64_t(gbase) + T - base16 + kCh - 1) / kCh;
  auto warp_of_slot = [&](int y) -> int64_t { return piece_of((y - base16) / kCh, NC, W); };
  int ga, ge;
  if (p.units_per_warp > 0) {            // whole units [gw k, (gw + 1) k)
    const int k = p.units_per_warp;
    const int u_lo = gw * k, u_hi = u_lo + k < p.n_units ? u_lo + k : p.n_units;
    if (u_lo >= u_hi) return;
    ga = ustart(unit0 + u_lo);
    ge = ustart(unit0 + u_hi);
  } else {                               // equal pieces of whole chunks
    const int64_t end = int64_t(gbase) + T;
    ga = int(max(int64_t(gbase), base16 + piece_begin(gw, NC, W) * kCh));
    ge = int(min(end, base16 + piece_begin(gw + 1, NC, W) * kCh));
  }
  if (ga >= ge) return;
  // first unit with used slots in [ga, ge): the piece may start in the unused
  // tail slots of a unit (past its n_main + n_res + n_app used rows), which
  // this warp must skip
  int u;
  if constexpr (kRagged) {              // last unit starting at or before ga
    int lo = unit0, hi = unit0 + p.n_units;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (p.offsets[mid] <= ga) lo = mid;
      else hi = mid;
    }
    u = lo;
  } else {
    u = ga / p.stride;
  }
  if (ustart(u) + p.n_main[u] + p.n_res[u] + (p.n_app ? p.n_app[u] : 0) <= ga) ++u;
  if (ustart(u) >= ge) return;

  // this warp's ring, log-count copies and mbarriers
  const WarpRing ring = warp_ring(smem_raw, kW, kSt, warp);
  const uint32_t base = ring.base;
  float* logc_s = ring.logc;           // [kSt][16]
  uint64_t* bars = ring.bars;

  const int cb = ga & ~(kCh - 1);                        // first chunk, 16-slot aligned
  const int nchunks = (ge - cb + kCh - 1) / kCh;

  if (lane == 0) {
    for (int s = 0; s < kSt; ++s) mbar_init(&bars[s], 1);
    fence_mbar_init();
  }
  __syncwarp();

  const uint64_t pol = l2_evict_first_policy();
  auto issue = [&](int k, int s, bool with_logc) {   // lane 0: chunk k into stage s
    issue_stage(base + s * kStageBytes, logc_s + s * kCh, &tmK, &tmV, p.logc, cb + k * kCh, p.kv_rank,
                with_logc, &bars[s], pol);
  };
  // the first ring goes out before the unit's counts are read: with log-counts
  if (lane == 0)
    for (int k = 0; k < nchunks && k < kSt; ++k) issue(k, k, true);
  // Programmatic dependent launch: the next kernel on the stream may start
  // now and overlap its prologue and first cache copies with this kernel.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  uint32_t off_k[4], off_pv[8];
  tile_offsets(lane, off_k, off_pv);

  const float qscale = kLog2e * rsqrtf(float(kHeadDim));

  // this warp's staging of query rows (two buffers) and output rows
  uint8_t* io = ring.cta + ring_smem_bytes(kW, kSt) + warp * kIoBytes;
  const uint32_t io_s = smem_u32(io);
  float* obuf = reinterpret_cast<float*>(io + 2 * 4 * kQRowBytes);

  // unit cursor: unit u from slot ub (the next unit from ub1), its main,
  // residual and used rows, its query fragments; the next unit's query rows
  // and counts are requested ahead
  uint32_t qa[16];
  int nm = 0, nr = 0, nt = 0, nm_n = 0, nr_n = 0, nt_n = 0;
  auto qrow0_of = [&](int uu) -> int64_t {
    const int ul = uu - unit0;
    return int64_t(ul / p.n_kv_heads) * p.n_kv_heads * G + int64_t(ul % p.n_kv_heads) * G;
  };
  auto load_q = [&](int uu, int b, int& m_out, int& r_out, int& t_out) {
    const __nv_bfloat16* src = p.Q + qrow0_of(uu) * kHeadDim;
    for (int i = lane; i < G * 16; i += 32)    // G rows of sixteen 16-byte pieces
      cp_async16(io_s + b * 4 * kQRowBytes + (i >> 4) * kQRowBytes + (i & 15) * 16,
                 src + (i >> 4) * kHeadDim + (i & 15) * 8);
    asm volatile("cp.async.commit_group;" ::: "memory");
    m_out = p.n_main[uu];
    r_out = p.n_res[uu];
    t_out = m_out + r_out + (p.n_app ? p.n_app[uu] : 0);
  };
  // B operand of K Q^T for column g (query head g % G; zero from 2G on),
  // once buffer b holds the unit's rows
  auto q_frags = [&](int b) {
    const uint32_t* w = reinterpret_cast<const uint32_t*>(io + b * 4 * kQRowBytes + (g % G) * kQRowBytes);
    const bool hv = g < 2 * G;
#pragma unroll
    for (int kk = 0; kk < 8; ++kk) {
      qa[2 * kk] = hv ? w[8 * kk + qp] : 0u;
      qa[2 * kk + 1] = hv ? w[8 * kk + 4 + qp] : 0u;
    }
  };
  // the G output rows staged in obuf to O, whole rows per store
  auto write_out = [&](int64_t orow0) {
    __syncwarp();
    for (int i = lane; i < G * 32; i += 32) {
      const int r = i >> 5, c = i & 31;
      *reinterpret_cast<float4*>(p.O + (orow0 + r) * kHeadDim + 4 * c) =
          *reinterpret_cast<const float4*>(obuf + r * kORowFloats + 4 * c);
    }
    __syncwarp();
  };
  // Q, O, the partial records and the tickets only after the previous kernel
  // on the stream has completed (before: the cache alone, which no kernel
  // that may run concurrently writes)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // The next unit's rows are requested once the current unit has at most
  // kQAheadSlots rows left in the piece, not at once: when Q sits in host
  // memory, every warp asking for two units' rows at the start queues the
  // whole of Q on the host link before the first tile.
  constexpr int kQAheadSlots = 64;
  int ub = ustart(u), ub1 = ustart(u + 1);
  int qb = 0;                                       // query buffer of unit u
  bool next_asked = false;                          // unit u + 1's rows requested
  load_q(u, 0, nm, nr, nt);
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  __syncwarp();
  q_frags(0);

  TileState S;
  S.reset();

  // Finish unit uu (first slot ubase, ut used rows): write o^ (whole unit in
  // this warp) or a partial record; the last warp of a cut unit merges them.
  auto finish = [&](int uu, int ubase, int ut) {
    const RowStats rs = tile_row_stats(S, lane);
    const int uend = ubase + ut;
    const int64_t orow0 = qrow0_of(uu);
    const int ul = uu - unit0;
    float* ob = obuf + (g < G ? g : 0) * kORowFloats + 2 * qp;
    if (ga <= ubase && ge >= uend) {
      // the residual column of head g is column g + G, 4G lanes up
      const float mR = __shfl_down_sync(0xffffffffu, rs.m, 4 * G);
      const float lR = __shfl_down_sync(0xffffffffu, rs.l, 4 * G);
      const float2 w = branch_coefs(p.softmax_mode, gate_of(p, sum_rel_max(rs.m, rs.l, rs.mt)),
                                    rs.m, rs.l, mR, lR);
#pragma unroll
      for (int dt = 0; dt < 16; ++dt) {
        const float2 vm = tile_row_value(S, dt);
        const float rx = __shfl_down_sync(0xffffffffu, vm.x, 4 * G);
        const float ry = __shfl_down_sync(0xffffffffu, vm.y, 4 * G);
        if (g < G)
          *reinterpret_cast<float2*>(ob + dt * 8) =
              make_float2(w.x * vm.x + w.y * rx, w.x * vm.y + w.y * ry);
      }
      write_out(orow0);
      return;
    }
    // record of column g (< 2G): reference max, sum, largest logit, numerator
    const int64_t w0 = warp_of_slot(ubase), w1 = warp_of_slot(uend - 1);
    if (g < 2 * G) {
      float* r = p.partials + (int64_t(ul) + gw) * (2 * G * kRec) + g * kRec;
      if (qp == 0) *reinterpret_cast<float4*>(r) = make_float4(rs.m, rs.l, rs.mt, 0.f);
#pragma unroll
      for (int dt = 0; dt < 16; ++dt)
        *reinterpret_cast<float2*>(r + 4 + dt * 8 + 2 * qp) = tile_row_value(S, dt);
    }
    __threadfence();
    __syncwarp();
    int ticket = 0;
    if (lane == 0) ticket = atomicAdd(p.tickets + uu, 1);
    ticket = __shfl_sync(0xffffffffu, ticket, 0);
    if (ticket != int(w1 - w0)) return;
    __threadfence();
    // one pass over the records in warp order (online log-sum-exp merge),
    // column g per lane, then main and residual columns combined
    float M = kMInit, L = 0.f, MT = -INFINITY;
    float acc[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) acc[i] = 0.f;
    if (g < 2 * G) {
      for (int64_t w = w0; w <= w1; ++w) {
        const float* r = p.partials + (int64_t(ul) + w) * (2 * G * kRec) + g * kRec;
        const float4 hd = __ldcg(reinterpret_cast<const float4*>(r));
        float2 v[16];
#pragma unroll
        for (int dt = 0; dt < 16; ++dt)
          v[dt] = __ldcg(reinterpret_cast<const float2*>(r + 4 + dt * 8 + 2 * qp));
        if (hd.y > 0.f) {
          const float mx = fmaxf(M, hd.x);
          const float sa = exp2f(M - mx), sb = exp2f(hd.x - mx);
          L = L * sa + hd.y * sb;
#pragma unroll
          for (int dt = 0; dt < 16; ++dt) {
            acc[2 * dt] = acc[2 * dt] * sa + v[dt].x * sb;
            acc[2 * dt + 1] = acc[2 * dt + 1] * sa + v[dt].y * sb;
          }
          M = mx;
          MT = fmaxf(MT, hd.z);
        }
      }
    }
    const float mR = __shfl_down_sync(0xffffffffu, M, 4 * G);
    const float lR = __shfl_down_sync(0xffffffffu, L, 4 * G);
    const float2 w = branch_coefs(p.softmax_mode, gate_of(p, sum_rel_max(M, L, MT)), M, L, mR, lR);
#pragma unroll
    for (int dt = 0; dt < 16; ++dt) {
      const float rx = __shfl_down_sync(0xffffffffu, acc[2 * dt], 4 * G);
      const float ry = __shfl_down_sync(0xffffffffu, acc[2 * dt + 1], 4 * G);
      if (g < G)
        *reinterpret_cast<float2*>(ob + dt * 8) =
            make_float2(w.x * acc[2 * dt] + w.y * rx, w.x * acc[2 * dt + 1] + w.y * ry);
    }
    write_out(orow0);
    if (lane == 0) p.tickets[uu] = 0;
  };

  bool done = false;
  int issued = nchunks < kSt ? nchunks : kSt;         // chunks [0, issued) requested
  int waited = 0;                                     // chunks [0, waited) completed
  int s = 0;                                          // stage of chunk k
  uint32_t phase = 0;                                 // parity of its current use
  for (int k = 0; k < nchunks && !done; ++k) {
    if ((k == 0 && p.test_fault) || !mbar_wait_bounded(&bars[s], phase)) {
      if (lane == 0) report_status(p.status, kStatusWaitTimeout);
      break;
    }
    waited = k + 1;
    const int t0 = cb + k * kCh;
    TileFrags F;
    tile_load(base + s * kStageBytes, logc_s + s * kCh, off_k, off_pv, lane, F);
    // every unit with rows in this tile
    while (true) {
      const int mlo = ub > ga ? ub : ga;
      const int mhi = ub + nt < ge ? ub + nt : ge;              // main + appended rows
      const int rlo = ub + nm > ga ? ub + nm : ga;
      const int rhi = ub + nm + nr < ge ? ub + nm + nr : ge;
      if (tile_pure_main(t0, mlo, mhi, rlo, rhi))
        tile_update<G, true>(S, F, t0, mlo, mhi, rlo, rhi, qa, qscale, lane);
      else if ((mlo < mhi && mlo < t0 + kCh && mhi > t0) || (rlo < rhi && rlo < t0 + kCh && rhi > t0))
        tile_update<G, false>(S, F, t0, mlo, mhi, rlo, rhi, qa, qscale, lane);
      // does unit u end inside this tile (or at the end of the piece)?
      if (mhi > t0 + kCh) break;                              // continues in the next tile
      finish(u, ub, nt);
      S.reset();
      ++u;
      ub = ub1;
      if (ub >= ge) {
        done = true;
        break;
      }
      if (!next_asked) load_q(u, qb ^ 1, nm_n, nr_n, nt_n);   // a short unit
      qb ^= 1;
      asm volatile("cp.async.wait_group 0;" ::: "memory");   // unit u's rows
      __syncwarp();
      q_frags(qb);
      nm = nm_n;
      nr = nr_n;
      nt = nt_n;
      ub1 = ustart(u + 1);
      next_asked = false;
    }
    if (done) break;
    // refill the stage once the tile is done (measured faster here than a
    // refill right after the register loads, which the cluster kernel uses)
    __syncwarp();
    if (k + kSt < nchunks) {
      if (lane == 0) {
        fence_proxy_async_smem();
        issue(k + kSt, s, !chunk_main_only(cb + (k + kSt) * kCh, ub, nm, nr, nt));
      }
      issued = k + kSt + 1;
    }
    if (++s == kSt) {
      s = 0;
      phase ^= 1u;
    }
    if (!next_asked && ub1 < ge && min(ub + nt, ge) - (t0 + kCh) <= kQAheadSlots) {
      __syncwarp();
      load_q(u + 1, qb ^ 1, nm_n, nr_n, nt_n);
      next_asked = true;
    }
  }
  // never leave with a copy in flight into this warp's ring (bounded waits)
  // or with query rows still arriving (after a timed-out wait)
  for (int kk = waited; kk < issued; ++kk)
    mbar_wait_bounded(&bars[kk % kSt], uint32_t((kk / kSt) & 1));
  asm volatile("cp.async.wait_all;" ::: "memory");
}

}  // namespace

template <int G, bool kRagged>
static cudaError_t launch_mma_g(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                                int n_ctas, int warps_per_cta, cudaStream_t stream) {
  static std::atomic<unsigned long long> configured{0};
  const int smem = 1024 + ring_smem_bytes(warps_per_cta, p.n_stages) + warps_per_cta * kIoBytes;
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
int decode_mma_stages(int warps_per_cta) { return ring_stages(warps_per_cta, warps_per_cta * kIoBytes); }

size_t decode_mma_partials_floats(int64_t n_units, int n_warps, int group) {
  return size_t(n_units + n_warps) * 2 * group * kRec;
}

}  // namespace reskv
