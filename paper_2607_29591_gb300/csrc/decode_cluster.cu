// Shared-softmax residual decode (Alg. 2; Sec. 5.4 Eqs. residual_logit,
// reskv_den, reskv_num, reskv; Sec. 5.5.2 Eq. gate) on the tensor cores, one
// thread-block cluster per unit.
//
// The stream-K kernel (decode_mma.cu) cuts a launch's whole slot range into
// equal warp pieces.  When a launch holds few units -- one layer of a decode
// step, a few dozen (batch, KV head) units -- nearly every unit is then cut
// between many warps, and merging their partial results through global
// records and an arrival ticket costs more than streaming the unit.  Here a
// unit is given to a cluster of CS CTAs (CS = 1..8) on as many SMs; the
// cluster's CS x kW warps each stream an equal run of the unit's 16-slot
// chunks with the tile step of mma_tile.cuh, and the partial results never
// leave the chip:
//
//   1. every warp writes its record (per query head and branch: reference max,
//      sum, numerator) into its own, drained, ring buffer;
//   2. after a CTA barrier, the CTA's threads merge its warps' records in
//      warp order and store the CTA record into rank 0's shared memory
//      (distributed shared memory, slot = rank);
//   3. after one cluster barrier, rank 0 merges the CS CTA records in rank
//      order, applies the gate and writes o^; the other CTAs are done.
//
// A cluster barrier phase opened at the start (arrive) and closed before the
// first remote store (wait) makes sure rank 0 is running before it is written.
// Launches are programmatic dependent launches: a kernel streams its first
// ring of cache chunks while the previous kernel on the stream finishes, and
// waits for it before touching Q or O.
// The result does not depend on timing: both merges run in a fixed order.
//
// The same kernel, instantiated per branch, also gives the paper's own
// decode structure as a measured comparison (launch_decode_lse): main-cache
// attention and the residual branch as two passes that write (max, sum,
// normalised output) per query row, and a merge kernel that combines them
// through those log-sum-exp statistics and the gate.
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

constexpr int kMaxCluster = 8;                              // portable cluster size
constexpr int kCtaRecFloats = 2 * 4 * kRec;                // 2 branches x G <= 4 heads

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}

__device__ __forceinline__ uint32_t cluster_size() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}

// Every thread of every CTA of the cluster arrives; shared-memory writes
// before it are visible to every thread of the cluster after it.
__device__ __forceinline__ void cluster_sync() {
  asm volatile(
      "barrier.cluster.arrive.release.aligned;\n\t"
      "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// The two halves of a cluster barrier phase with no memory ordering: after
// the wait, every CTA of the cluster has started.
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}

__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
}

// Store into the shared memory of CTA `rank` of the cluster, at the address
// that `local` has in this CTA.
__device__ __forceinline__ uint32_t map_rank(uint32_t local, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(rank));
  return remote;
}

__device__ __forceinline__ void st_cluster(uint32_t local, uint32_t rank, float4 v) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(map_rank(local, rank)),
               "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w)
               : "memory");
}

// What one launch computes: the fused decode (o^ of Eq. reskv, the library's
// path), or one branch of the paper-style comparison path (Sec. 6.1, App. B:
// main-cache attention and residual branch as separate passes merged through
// log-sum-exp statistics), which writes per query row the branch's running
// max m, sum l and normalised output o = acc / l to a branch record.
enum : int { kFused = 0, kMainBranch = 1, kResBranch = 2 };
constexpr int kBrRec = kHeadDim + 4;    // branch record: m, l, pad, pad, o[d]

// Step 3 of the cluster kernel, in rank 0: merge the n <= CS CTA records
// (crec, [CS][2 branches][G heads][kRec]) in rank order, apply the gate and
// write o^ (or, on a branch pass, the branch record).  One thread per two dims
// of one head: every thread of the CTA takes part, and with CS equal to the
// cluster size no record is read twice.
template <int G, int kMode, int CS>
__device__ __forceinline__ void rank0_merge(const DecodeParams& p, const float* crec,
                                            int64_t orow0, int n) {
  for (int idx = threadIdx.x; idx < G * (kHeadDim / 2); idx += blockDim.x) {
    const int hh = idx / (kHeadDim / 2), d2 = 2 * (idx % (kHeadDim / 2));
    float4 ml[2][CS];
    float2 ac[2][CS];
#pragma unroll
    for (int sg = 0; sg < 2; ++sg)
#pragma unroll
      for (int c = 0; c < CS; ++c) {
        const int cc = c < n ? c : 0;
        const float* r = crec + cc * kCtaRecFloats + (sg * G + hh) * kRec;
        ml[sg][c] = *reinterpret_cast<const float4*>(r);
        ac[sg][c] = *reinterpret_cast<const float2*>(r + 4 + d2);
      }
    float Ms[2], Ls[2], Mt[2];
    float2 As[2];
#pragma unroll
    for (int sg = 0; sg < 2; ++sg) {
      float mx = -INFINITY, mt = -INFINITY;
#pragma unroll
      for (int c = 0; c < CS; ++c)
        if (c < n && ml[sg][c].y > 0.f) {
          mx = fmaxf(mx, ml[sg][c].x);
          mt = fmaxf(mt, ml[sg][c].z);
        }
      float l = 0.f;
      float2 a = make_float2(0.f, 0.f);
#pragma unroll
      for (int c = 0; c < CS; ++c)
        if (c < n && ml[sg][c].y > 0.f) {
          const float sc = exp2f(ml[sg][c].x - mx);
          l += ml[sg][c].y * sc;
          a.x += ac[sg][c].x * sc;
          a.y += ac[sg][c].y * sc;
        }
      Ms[sg] = mx;
      Ls[sg] = l;
      Mt[sg] = mt;
      As[sg] = a;
    }
    if constexpr (kMode == kFused) {
      const float2 w = branch_coefs(p.softmax_mode, gate_of(p, sum_rel_max(Ms[0], Ls[0], Mt[0])),
                                    Ms[0], Ls[0], Ms[1], Ls[1]);
      *reinterpret_cast<float2*>(p.O + (orow0 + hh) * kHeadDim + d2) =
          make_float2(w.x * As[0].x + w.y * As[1].x, w.x * As[0].y + w.y * As[1].y);
    } else {
      constexpr int sg = kMode == kMainBranch ? 0 : 1;
      const float inv = Ls[sg] > 0.f ? 1.0f / Ls[sg] : 0.f;
      float* br = p.partials + (orow0 + hh) * kBrRec;
      *reinterpret_cast<float2*>(br + 4 + d2) = make_float2(As[sg].x * inv, As[sg].y * inv);
      // (m, l) relative to the branch's largest logit, as the merge's gate takes it
      if (d2 == 0)
        *reinterpret_cast<float2*>(br) =
            Ls[sg] > 0.f ? make_float2(Mt[sg], sum_rel_max(Ms[sg], Ls[sg], Mt[sg]))
                         : make_float2(Ms[sg], Ls[sg]);
    }
  }
}

template <int G, int kMode>
__global__ void __launch_bounds__(kMmaMaxW * 32, 1)
    reskv_decode_cluster_kernel(const DecodeParams p, const __grid_constant__ CUtensorMap tmK,
                                const __grid_constant__ CUtensorMap tmV) {
  extern __shared__ uint8_t smem_raw[];
  const int kW = blockDim.x >> 5;       // warps per CTA of this launch
  const int kSt = p.n_stages;           // ring stages per warp of this launch
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2;              // softmax column / accumulator row of this lane
  const int qp = lane & 3;              // position in the quad
  const uint32_t cs = cluster_size(), rank = cluster_rank();

  // this cluster's unit, slots [ub, ub + stride).  Slot indices fit in 32
  // bits (a cache holds fewer than 2^31 slots), so no 64-bit division is needed.
  const int ul = int(blockIdx.x / cs);
  const int u = int(p.unit0) + ul;
  const int ub = p.offsets ? p.offsets[u] : u * p.stride;
  const int usize = p.offsets ? p.offsets[u + 1] - ub : p.stride;
  // the 16-slot chunks (aligned to 16 global slots) of the unit's rows that
  // may be in use, [ub, ub + usize - tail_unused), split evenly over the
  // cluster's warps.
  // The fused split does not wait for n_main / n_res / n_app: the first copies
  // are in flight before those loads return (unused rows, present only when
  // s < b or when units of the launch hold fewer appended rows than others,
  // are streamed and masked).  A branch pass streams only its own rows.
  int nm = 0, nr = 0, na = 0, lo = ub, hi = ub + usize - p.tail_unused;
  if constexpr (kMode != kFused) {
    nm = p.n_main[u];
    nr = p.n_res[u];
    na = p.n_app ? p.n_app[u] : 0;
    lo = kMode == kMainBranch ? ub : ub + nm;
    hi = kMode == kMainBranch ? ub + nm + nr + na : ub + nm + nr;
  }
  const int cb = lo & ~(kCh - 1);
  const int nch = hi > lo ? (hi - cb + kCh - 1) / kCh : 0;
  const int NW = int(cs) * kW, iw = int(rank) * kW + warp;
  const int k0 = (iw * nch) / NW, k1 = ((iw + 1) * nch) / NW;
  const int nchunks = k1 - k0;
  const int wcb = cb + k0 * kCh;                           // first row of this warp's run

  // per-warp shared memory, 1024-byte aligned for the 128-byte swizzle
  const WarpRing ring = warp_ring(smem_raw, kW, kSt, warp);
  uint8_t* abase_ptr = ring.cta;
  const uint32_t abase = smem_u32(abase_ptr);
  const uint32_t base = ring.base;
  uint8_t* base_ptr = ring.ptr;
  float* logc_s = ring.logc;           // [kSt][16]
  uint64_t* bars = ring.bars;
  // CTA records [cs][2][G][kRec] after the rings (read only in rank 0)
  float* crec = reinterpret_cast<float*>(abase_ptr + ring_smem_bytes(kW, kSt));
  const uint32_t crec_s = abase + uint32_t(ring_smem_bytes(kW, kSt));

  cluster_arrive_relaxed();             // closed by cluster_wait() before step 2
  if (lane == 0) {
    for (int s = 0; s < kSt; ++s) mbar_init(&bars[s], 1);
    fence_mbar_init();
  }
  __syncwarp();

  const uint64_t pol = l2_evict_first_policy();
  auto issue = [&](int k, int s, bool with_logc) {   // lane 0: chunk k into stage s
    issue_stage(base + s * kStageBytes, logc_s + s * kCh, &tmK, &tmV, p.logc, wcb + k * kCh, p.kv_rank,
                with_logc, &bars[s], pol);
  };
  const int issued0 = nchunks < kSt ? nchunks : kSt;
  if (lane == 0)
    for (int k = 0; k < issued0; ++k) issue(k, k, true);   // before the counts are read
  // Programmatic dependent launch: the next kernel on the stream may start
  // now (its own prologue and cache copies overlap this kernel's tail) ...
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if constexpr (kMode == kFused) {
    nm = p.n_main[u];
    nr = p.n_res[u];
    na = p.n_app ? p.n_app[u] : 0;
  }
  const int ue = ub + nm + nr + na;                        // used slots [ub, ue)
  // main rows: [m_lo, m_hi) minus the residual rows [r_lo, r_hi) (selected
  // tokens, then rows appended at decode time); a residual pass has none
  const int m_lo = kMode == kResBranch ? 0 : ub, m_hi = kMode == kResBranch ? 0 : ue;
  const int r_lo = ub + nm, r_hi = ub + nm + nr;
  uint32_t off_k[4], off_pv[8];
  tile_offsets(lane, off_k, off_pv);
  const float qscale = kLog2e * rsqrtf(float(kHeadDim));
  const int64_t orow0 = int64_t(ul / p.n_kv_heads) * p.n_kv_heads * G + (ul % p.n_kv_heads) * G;
  uint32_t qa[16];
  // ... and this kernel reads Q and writes O only after the previous kernel
  // has completed and its memory is visible.  Before this point it reads
  // only the cache (K, V, log-counts, n_main, n_res), which no kernel that
  // may run concurrently writes.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  load_q_frag<G>(p.Q, orow0, lane, qa);

  TileState S;
  S.reset();
  int issued = issued0;                 // chunks [0, issued) requested
  int waited = 0;                       // chunks [0, waited) completed
  int s = 0;                            // stage of chunk k
  uint32_t phase = 0;                   // parity of its current use
  for (int k = 0; k < nchunks; ++k) {
    if ((k == 0 && p.test_fault) || !mbar_wait_bounded(&bars[s], phase)) {
      if (lane == 0) report_status(p.status, kStatusWaitTimeout);
      break;
    }
    waited = k + 1;
    const int t0 = wcb + k * kCh;
    // the tile into registers, then its stage is refilled at once (the copy
    // overlaps this tile's softmax and P V)
    TileFrags F;
    tile_load(base + s * kStageBytes, logc_s + s * kCh, off_k, off_pv, lane, F);
    __syncwarp();
    if (k + kSt < nchunks) {
      if (lane == 0) {
        fence_proxy_async_smem();
        // a main-only pass never reads log-counts; otherwise only chunks
        // with residual rows need them
        issue(k + kSt, s,
              kMode != kMainBranch && !chunk_main_only(wcb + (k + kSt) * kCh, ub, nm, nr, nm + nr + na));
      }
      issued = k + kSt + 1;
    }
    if (++s == kSt) {
      s = 0;
      phase ^= 1u;
    }
    if (tile_pure_main(t0, m_lo, m_hi, r_lo, r_hi))
      tile_update<G, true>(S, F, t0, m_lo, m_hi, r_lo, r_hi, qa, qscale, lane);
    else
      tile_update<G, false, kMode != kMainBranch>(S, F, t0, m_lo, m_hi, r_lo, r_hi, qa, qscale,
                                                  lane);
  }
  // never reuse the ring while a copy is in flight into it (bounded waits)
  for (int kk = waited; kk < issued; ++kk)
    mbar_wait_bounded(&bars[kk % kSt], uint32_t((kk / kSt) & 1));
  __syncwarp();

  // 1. this warp's record, in the first bytes of its own ring: per softmax
  //    column g < 2G (branch g / G, head g % G) its reference max, sum,
  //    largest logit and numerator
  const RowStats rs = tile_row_stats(S, lane);
  if (g < 2 * G) {
    float* r = reinterpret_cast<float*>(base_ptr) + g * kRec;
    if (qp == 0) *reinterpret_cast<float4*>(r) = make_float4(rs.m, rs.l, rs.mt, 0.f);
#pragma unroll
    for (int dt = 0; dt < 16; ++dt)
      *reinterpret_cast<float2*>(r + 4 + dt * 8 + 2 * qp) = tile_row_value(S, dt);
  }
  __syncthreads();
  cluster_wait();                        // every CTA of the cluster is running

  // 2. CTA record: merge the kW warp records in warp order; a thread takes
  //    four dims of one (branch, head) record and issues all of its loads
  //    before the first use.  The record goes straight into slot `rank` of
  //    rank 0's CTA records (distributed shared memory).
  for (int idx = threadIdx.x; idx < 2 * G * (kHeadDim / 4); idx += blockDim.x) {
    const int rec = idx / (kHeadDim / 4), d4 = 4 * (idx % (kHeadDim / 4));
    float4 ml[kMmaMaxW];
    float4 ac[kMmaMaxW];
#pragma unroll
    for (int w = 0; w < kMmaMaxW; ++w) {
      const int ws = w < kW ? w : 0;           // in-range address; weight masked below
      const float* r = reinterpret_cast<const float*>(abase_ptr + ws * kSt * kStageBytes) + rec * kRec;
      ml[w] = *reinterpret_cast<const float4*>(r);
      ac[w] = *reinterpret_cast<const float4*>(r + 4 + d4);
    }
    float mx = -INFINITY, mt = -INFINITY;
#pragma unroll
    for (int w = 0; w < kMmaMaxW; ++w)
      if (w < kW && ml[w].y > 0.f) {
        mx = fmaxf(mx, ml[w].x);
        mt = fmaxf(mt, ml[w].z);
      }
    float l = 0.f;
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int w = 0; w < kMmaMaxW; ++w)
      if (w < kW && ml[w].y > 0.f) {
        const float sc = exp2f(ml[w].x - mx);
        l += ml[w].y * sc;
        a.x += ac[w].x * sc;
        a.y += ac[w].y * sc;
        a.z += ac[w].z * sc;
        a.w += ac[w].w * sc;
      }
    const uint32_t dst = crec_s + uint32_t(rank * kCtaRecFloats + rec * kRec) * 4u;
    st_cluster(dst + uint32_t(4 + d4) * 4u, 0, a);
    if (d4 == 0) st_cluster(dst, 0, make_float4(mx, l, mt, 0.f));
  }
  cluster_sync();
  if (rank != 0) return;                 // nobody reads this CTA's shared memory

  // 3. rank 0: merge the CS CTA records in rank order, gate, write o^
  switch (cs) {
    case 1: rank0_merge<G, kMode, 1>(p, crec, orow0, 1); break;
    case 2: rank0_merge<G, kMode, 2>(p, crec, orow0, 2); break;
    case 4: rank0_merge<G, kMode, 4>(p, crec, orow0, 4); break;
    default: rank0_merge<G, kMode, kMaxCluster>(p, crec, orow0, int(cs)); break;
  }
}

// Paper-style path, last step: merge the two branch records of every query
// row through their log-sum-exp statistics and the gate.  With the branch
// states (m, l, o = acc / l), o^ = a l_M o_M + c l_R o_R for the coefficients
// (a, c) of branch_coefs: Eq. reskv, or the ablation's rule.  Four rows per
// 128-thread block, four dims per thread.
__global__ void __launch_bounds__(128) reskv_lse_merge_kernel(const DecodeParams p,
                                                              int64_t n_rows) {
  const int64_t row = int64_t(blockIdx.x) * 4 + (threadIdx.x >> 5);
  if (row >= n_rows) return;
  const int d4 = 4 * (threadIdx.x & 31);
  const float* bm = p.partials + row * kBrRec;
  const float* br = p.partials + (n_rows + row) * kBrRec;
  const float2 sm = *reinterpret_cast<const float2*>(bm);
  const float2 sr = *reinterpret_cast<const float2*>(br);
  const float4 om = *reinterpret_cast<const float4*>(bm + 4 + d4);
  const float4 orr = *reinterpret_cast<const float4*>(br + 4 + d4);
  const float2 w = branch_coefs(p.softmax_mode, gate_of(p, sm.y), sm.x, sm.y, sr.x, sr.y);
  const float a = w.x * sm.y, c = w.y * sr.y;
  *reinterpret_cast<float4*>(p.O + row * kHeadDim + d4) =
      make_float4(a * om.x + c * orr.x, a * om.y + c * orr.y, a * om.z + c * orr.z,
                  a * om.w + c * orr.w);
}

}  // namespace

template <int G, int kMode>
static cudaError_t configure_cluster_g() {
  static std::atomic<unsigned long long> configured{0};
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  const unsigned long long bit = 1ull << (dev & 63);
  if (!(configured.load() & bit)) {
    err = cudaFuncSetAttribute(reskv_decode_cluster_kernel<G, kMode>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemLimit);
    if (err != cudaSuccess) return err;
    configured.fetch_or(bit);
  }
  return cudaSuccess;
}

static cudaLaunchConfig_t cluster_config(int64_t n_units, int cluster, int warps_per_cta,
                                         cudaStream_t stream, cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(n_units) * unsigned(cluster), 1, 1);
  cfg.blockDim = dim3(unsigned(warps_per_cta) * 32u, 1, 1);
  cfg.dynamicSmemBytes =
      size_t(decode_cluster_smem_bytes(warps_per_cta, decode_cluster_stages(warps_per_cta, cluster),
                                       cluster));
  cfg.stream = stream;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = unsigned(cluster);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

template <int G, int kMode>
static int max_active_g(int cluster, int warps_per_cta) {
  if (configure_cluster_g<G, kMode>() != cudaSuccess) return -1;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = cluster_config(cluster, cluster, warps_per_cta, nullptr, attr);
  int n = 0;
  const cudaError_t err =
      cudaOccupancyMaxActiveClusters(&n, reinterpret_cast<const void*>(reskv_decode_cluster_kernel<G, kMode>), &cfg);
  if (err != cudaSuccess) {
    (void)cudaGetLastError();
    return 0;                          // this shape cannot be launched at all
  }
  return n;
}

template <int G, int kMode>
static cudaError_t launch_cluster_g(const DecodeParams& p, const CUtensorMap& tk,
                                    const CUtensorMap& tv, int cluster, int warps_per_cta,
                                    cudaStream_t stream) {
  cudaError_t err = configure_cluster_g<G, kMode>();
  if (err != cudaSuccess) return err;
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = cluster_config(p.n_units, cluster, warps_per_cta, stream, attr);
  cfg.dynamicSmemBytes = size_t(decode_cluster_smem_bytes(warps_per_cta, p.n_stages, cluster));
  // may start before the previous kernel on the stream has finished (see
  // griddepcontrol.wait in the kernel)
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.numAttrs = 2;
  err = cudaLaunchKernelEx(&cfg, reskv_decode_cluster_kernel<G, kMode>, p, tk, tv);
  if (err != cudaSuccess) return err;
  return cudaGetLastError();
}

cudaError_t launch_decode_cluster(const DecodeParams& p, const CUtensorMap& tk,
                                  const CUtensorMap& tv, int group, int cluster,
                                  int warps_per_cta, cudaStream_t stream) {
  if (cluster < 1 || cluster > kMaxCluster || warps_per_cta < 1 || warps_per_cta > kMmaMaxW ||
      p.n_stages < 1 || p.n_stages > decode_cluster_stages(warps_per_cta, cluster))
    return cudaErrorInvalidValue;
  switch (group) {
    case 1: return launch_cluster_g<1, kFused>(p, tk, tv, cluster, warps_per_cta, stream);
    case 2: return launch_cluster_g<2, kFused>(p, tk, tv, cluster, warps_per_cta, stream);
    case 4: return launch_cluster_g<4, kFused>(p, tk, tv, cluster, warps_per_cta, stream);
    default: return cudaErrorInvalidValue;
  }
}

int decode_cluster_max_active(int group, int cluster, int warps_per_cta) {
  if (cluster < 1 || cluster > kMaxCluster || warps_per_cta < 1 || warps_per_cta > kMmaMaxW)
    return 0;
  switch (group) {
    case 1: return max_active_g<1, kFused>(cluster, warps_per_cta);
    case 2: return max_active_g<2, kFused>(cluster, warps_per_cta);
    case 4: return max_active_g<4, kFused>(cluster, warps_per_cta);
    default: return 0;
  }
}

template <int G>
static cudaError_t launch_lse_g(const DecodeParams& p, const CUtensorMap& tk,
                                const CUtensorMap& tv, int cluster, int warps_per_cta,
                                cudaStream_t stream) {
  const int64_t n_rows = int64_t(p.n_units) * G;
  DecodeParams pr = p;
  pr.partials = p.partials + n_rows * kBrRec;
  cudaError_t err = launch_cluster_g<G, kMainBranch>(p, tk, tv, cluster, warps_per_cta, stream);
  if (err == cudaSuccess)
    err = launch_cluster_g<G, kResBranch>(pr, tk, tv, cluster, warps_per_cta, stream);
  if (err != cudaSuccess) return err;
  reskv_lse_merge_kernel<<<unsigned((n_rows + 3) / 4), 128, 0, stream>>>(p, n_rows);
  return cudaGetLastError();
}

cudaError_t launch_decode_lse(const DecodeParams& p, const CUtensorMap& tk, const CUtensorMap& tv,
                              int group, int cluster, int warps_per_cta, cudaStream_t stream) {
  if (cluster < 1 || cluster > kMaxCluster || warps_per_cta < 1 || warps_per_cta > kMmaMaxW ||
      p.n_stages < 1 || p.n_stages > decode_cluster_stages(warps_per_cta, cluster))
    return cudaErrorInvalidValue;
  switch (group) {
    case 1: return launch_lse_g<1>(p, tk, tv, cluster, warps_per_cta, stream);
    case 2: return launch_lse_g<2>(p, tk, tv, cluster, warps_per_cta, stream);
    case 4: return launch_lse_g<4>(p, tk, tv, cluster, warps_per_cta, stream);
    default: return cudaErrorInvalidValue;
  }
}

size_t decode_lse_scratch_floats(int64_t n_units, int group) {
  return size_t(2) * size_t(n_units) * size_t(group) * kBrRec;
}

// Ring depth for `warps_per_cta` warps next to `cluster` CTA records.
int decode_cluster_stages(int warps_per_cta, int cluster) {
  return ring_stages(warps_per_cta, cluster * kCtaRecFloats * 4);
}

int decode_cluster_smem_bytes(int warps_per_cta, int stages, int cluster) {
  return 1024 + ring_smem_bytes(warps_per_cta, stages) + cluster * kCtaRecFloats * 4;
}

}  // namespace reskv
