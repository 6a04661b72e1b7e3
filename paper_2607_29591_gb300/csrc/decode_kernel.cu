// Shared-softmax residual decode (Alg. 2; Sec. 5.4 Eqs. residual_logit,
// reskv_den, reskv_num, reskv; Sec. 5.5.2 Eq. gate) on sm_103a.
//
// One launch covers n_units consecutive (layer, batch, KV head) units of the
// ragged cache.  Their slots are contiguous in HBM (unit u owns the slots from
// u*stride, or offsets[u] with per-unit budgets: n_main exact main rows, then
// n_res residual rows, then rows appended at decode time), so the launch
// reads one flat range of K rows and one of V rows.  That range is cut
// into W equal contiguous pieces, one per warp (stream-K at warp grain: every
// warp streams the same number of bytes whatever the ragged main/residual
// split).  Each warp
//   * streams its piece through a private ring of shared-memory stages filled
//     by 1-D TMA bulk copies (cp.async.bulk + mbarrier, 16-byte aligned rows),
//   * computes, per slot, the logits of the G query heads of the unit with
//     packed fp32x2 FMAs on bf16 rows unpacked in registers (8 lanes per slot,
//     4 slots per warp step, 16 dims per lane),
//   * keeps two online-softmax states in the log2 domain -- main slots and
//     residual slots (whose logits add beta*log c_j) -- because the gate g(q)
//     depends on the main-only sharpness p_max = 1 / sum_M 2^{a_p - max} and is
//     known only once every main slot has been seen; log g is a constant shift
//     of every residual logit, so the residual state is scaled by g at the end,
//   * finishes units it covers alone: Z^ = 2^{mM} lM + g 2^{mR} lR,
//     N^ likewise, o^ = N^ / Z^ (fp32 out).
// Units cut between warps are finished by the last warp to arrive (atomic
// ticket, no spinning); it merges the per-warp records in warp order, so the
// result does not depend on arrival order.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdint>

#include "device_utils.cuh"
#include "internal.h"

namespace reskv {
namespace {

constexpr int kStages = 4;            // ring depth per warp
constexpr int kChunk = 8;             // slots per stage
constexpr int kLogcBatch = 128;       // residual log-counts staged per batch
constexpr int kRingBytes = kStages * kChunk * kSlotRowBytes;   // per tensor
constexpr int kWarpSmem = 2 * kRingBytes + kStages * 8 + kLogcBatch * 4;
constexpr int kRecordFloats = kHeadDim + 2;                    // m, l, acc[d]

__device__ __forceinline__ int64_t warp_begin(int64_t w, int64_t T, int64_t W) {
  return (w * T) / W;
}
// The warp whose piece contains flat slot x: largest w with begin(w) <= x.
__device__ __forceinline__ int64_t warp_of(int64_t x, int64_t T, int64_t W) {
  return ((x + 1) * W - 1) / T;
}

struct SegState {
  float m, l;          // running max (log2 domain) and sum of 2^{a - m}
  float acc[16];       // sum of 2^{a - m} v over this lane's 16 dims
};

__device__ __forceinline__ float gate_value(const DecodeParams& p, float lM) {
  if (p.gate_mode == RESKV_GATE_FIXED) return p.g_fixed;
  const float p_max = 1.0f / lM;       // the max slot contributes 2^0 = 1
  const float sg = 1.0f / (1.0f + expf(-p.alpha * (p.tau - p_max)));
  return fmaxf(p.g_min, sg);
}

// o^ for one head over this lane's 16 dims from the main and residual states.
__device__ __forceinline__ void finalize(const DecodeParams& p, const SegState& M,
                                         const SegState& R, float* out16) {
  const float2 w = branch_coefs(p.softmax_mode, gate_value(p, M.l), M.m, M.l, R.m, R.l);
#pragma unroll
  for (int i = 0; i < 16; ++i) out16[i] = w.x * M.acc[i] + w.y * R.acc[i];
}

// Combine state b into a (both in the log2 domain).
__device__ __forceinline__ void merge_into(SegState& a, float bm, float bl, const float* bacc) {
  if (bl <= 0.0f) return;
  if (a.l <= 0.0f) {
    a.m = bm;
    a.l = bl;
#pragma unroll
    for (int i = 0; i < 16; ++i) a.acc[i] = bacc[i];
    return;
  }
  const float mx = fmaxf(a.m, bm);
  const float sa = exp2f(a.m - mx), sb = exp2f(bm - mx);
  a.m = mx;
  a.l = a.l * sa + bl * sb;
#pragma unroll
  for (int i = 0; i < 16; ++i) a.acc[i] = a.acc[i] * sa + bacc[i] * sb;
}

// Offsets of this lane's dims: dims [8*sub, 8*sub+8) and [64+8*sub, 64+8*sub+8).
__device__ __forceinline__ int dim_of(int sub, int i) { return (i < 8) ? 8 * sub + i : 64 + 8 * sub + (i - 8); }

template <int G>
__global__ void __launch_bounds__(kDecodeWarpsPerCta * 32, 1)
    reskv_decode_kernel(const DecodeParams p) {
  extern __shared__ __align__(128) uint8_t smem[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int grp = lane >> 3;       // slot within a 4-slot step / head in epilogues
  const int sub = lane & 7;        // 16 dims: [8sub, 8sub+8) u [64+8sub, 64+8sub+8)
  const int64_t gw = int64_t(blockIdx.x) * kDecodeWarpsPerCta + warp;
  if (gw >= p.n_warps) return;

  const int64_t T = p.total_slots, W = p.n_warps;
  const int64_t a = warp_begin(gw, T, W), e = warp_begin(gw + 1, T, W);
  if (a >= e) return;

  uint8_t* wbase = smem + warp * kWarpSmem;
  uint8_t* kring = wbase;
  uint8_t* vring = wbase + kRingBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(wbase + 2 * kRingBytes);
  float* logc_s = reinterpret_cast<float*>(wbase + 2 * kRingBytes + kStages * 8);

  const int64_t b = p.stride;
  // global slot of flat index 0, and the flat index where local unit uu starts
  const int64_t gbase = p.offsets ? int64_t(p.offsets[p.unit0]) : p.unit0 * b;
  auto uflat = [&](int64_t uu) -> int64_t {
    return p.offsets ? int64_t(p.offsets[p.unit0 + uu]) - gbase : uu * b;
  };
  const int64_t nchunks = (e - a + kChunk - 1) / kChunk;

  if (lane == 0) {
    for (int st = 0; st < kStages; ++st) mbar_init(&full[st], 1);
    fence_mbar_init();
  }
  __syncwarp();

  auto issue = [&](int64_t k) {        // lane 0 only
    const int64_t x0 = a + k * kChunk;
    const int64_t n = (e - x0 < kChunk) ? (e - x0) : kChunk;
    const int st = int(k % kStages);
    const uint32_t bytes = uint32_t(n) * kSlotRowBytes;
    mbar_arrive_expect_tx(&full[st], 2 * bytes);
    bulk_g2s(kring + st * kChunk * kSlotRowBytes, p.kslots + (gbase + x0) * kHeadDim, bytes,
             &full[st]);
    bulk_g2s(vring + st * kChunk * kSlotRowBytes, p.vslots + (gbase + x0) * kHeadDim, bytes,
             &full[st]);
  };

  if (lane == 0) {
    for (int64_t k = 0; k < nchunks && k < kStages; ++k) issue(k);
  }
  int64_t ready = -1;        // chunks [0, ready] have completed
  int64_t released = 0;      // chunks [0, released) handed back to the producer
  bool failed = false;

  auto wait_upto = [&](int64_t k) {
    while (ready < k && !failed) {
      ++ready;
      if ((ready == 0 && p.test_fault) ||
          !mbar_wait_bounded(&full[ready % kStages], uint32_t((ready / kStages) & 1))) {
        failed = true;
        if (lane == 0) report_status(p.status, kStatusWaitTimeout);
      }
    }
  };
  // Hand back every chunk that ends at or before flat slot `pos`.
  auto release_upto = [&](int64_t pos) {
    while (released < nchunks && a + (released + 1) * kChunk <= pos && !failed) {
      wait_upto(released);               // keep the barrier phases in order
      __syncwarp();
      if (lane == 0 && released + kStages < nchunks) {
        fence_proxy_async_smem();
        issue(released + kStages);
      }
      ++released;
    }
  };

  const float qscale = kLog2e * rsqrtf(float(kHeadDim));

  int64_t u_first = 0;                 // last unit starting at or before a
  if (p.offsets) {
    int64_t lo = 0, hi = p.n_units;
    while (hi - lo > 1) {
      const int64_t mid = (lo + hi) >> 1;
      if (uflat(mid) <= a) lo = mid;
      else hi = mid;
    }
    u_first = lo;
  } else {
    u_first = a / b;
  }
  for (int64_t u = u_first; u < p.n_units && uflat(u) < e && !failed; ++u) {
    const int64_t ubase = uflat(u);
    const int32_t nm = p.n_main[p.unit0 + u];
    const int32_t nr = p.n_res[p.unit0 + u];
    const int32_t na = p.n_app ? p.n_app[p.unit0 + u] : 0;
    const int64_t main_lo = ubase > a ? ubase : a;
    const int64_t main_hi = (ubase + nm < e) ? ubase + nm : e;
    const int64_t res_lo = (ubase + nm > a) ? ubase + nm : a;
    const int64_t res_hi = (ubase + nm + nr < e) ? ubase + nm + nr : e;
    const int64_t app_lo = (ubase + nm + nr > a) ? ubase + nm + nr : a;
    const int64_t app_hi = (ubase + nm + nr + na < e) ? ubase + nm + nr + na : e;
    if (main_lo >= main_hi && res_lo >= res_hi && app_lo >= app_hi)
      continue;                                             // only unused tail slots here

    // queries of the G heads of this unit, over this lane's 16 dims, scaled
    // by log2(e)/sqrt(d) so that 2^{s} = e^{a}
    float2 q2[G][8];
    {
      const int64_t qrow0 = (u / p.n_kv_heads) * int64_t(p.n_kv_heads) * G +
                            (u % p.n_kv_heads) * G;
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const uint4* qp = reinterpret_cast<const uint4*>(p.Q + (qrow0 + g) * kHeadDim);
        const uint4 c0 = __ldg(qp + sub), c1 = __ldg(qp + 8 + sub);
        const uint32_t w[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float2 f = bf16x2_to_float2(w[i]);
          q2[g][i] = make_float2(f.x * qscale, f.y * qscale);
        }
      }
    }

    // [0] main, [1] residual, [2] rows appended at decode time (main rows,
    // folded into [0] below): head `grp`, this lane's dims
    SegState segs[3];
#pragma unroll
    for (int sgi = 0; sgi < 3; ++sgi) {
      segs[sgi].m = -INFINITY;
      segs[sgi].l = 0.0f;
#pragma unroll
      for (int i = 0; i < 16; ++i) segs[sgi].acc[i] = 0.0f;
    }

#pragma unroll
    for (int sgi = 0; sgi < 3; ++sgi) {
      const int64_t lo = sgi == 0 ? main_lo : sgi == 1 ? res_lo : app_lo;
      const int64_t hi = sgi == 0 ? main_hi : sgi == 1 ? res_hi : app_hi;
      if (lo >= hi || failed) continue;
      const bool is_res = sgi == 1;
      release_upto(lo);

      float m[G], l[G];
      float2 acc[G][8];
#pragma unroll
      for (int g = 0; g < G; ++g) {
        m[g] = -INFINITY;
        l[g] = 0.0f;
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[g][i] = make_float2(0.f, 0.f);
      }

      int64_t logc_lo = lo;
#pragma unroll 1
      for (int64_t x = lo; x < hi && !failed; x += 4) {
        if (is_res && ((x - lo) % kLogcBatch) == 0) {
          logc_lo = x;
          __syncwarp();
#pragma unroll
          for (int t = 0; t < kLogcBatch / 32; ++t) {
            const int64_t y = x + t * 32 + lane;
            logc_s[t * 32 + lane] = (y < hi) ? __ldg(p.logc + gbase + y) * kLog2e : 0.0f;
          }
          __syncwarp();
        }
        const int64_t last = (x + 3 < hi) ? x + 3 : hi - 1;
        wait_upto((last - a) / kChunk);
        if (failed) break;
        const int64_t y = x + grp;
        const bool valid = y < hi;
        uint4 k0 = make_uint4(0, 0, 0, 0), k1 = k0, v0 = k0, v1 = k0;
        if (valid) {
          const int64_t off = y - a;
          const int st = int((off / kChunk) % kStages);
          const int row = int(off % kChunk);
          const uint4* kr = reinterpret_cast<const uint4*>(kring + (st * kChunk + row) * kSlotRowBytes);
          const uint4* vr = reinterpret_cast<const uint4*>(vring + (st * kChunk + row) * kSlotRowBytes);
          k0 = kr[sub];
          k1 = kr[8 + sub];
          v0 = vr[sub];
          v1 = vr[8 + sub];
        }
        const uint32_t kw[8] = {k0.x, k0.y, k0.z, k0.w, k1.x, k1.y, k1.z, k1.w};
        float s[G];
#pragma unroll
        for (int g = 0; g < G; ++g) {
          float2 t = make_float2(0.f, 0.f);
#pragma unroll
          for (int i = 0; i < 8; ++i) t = ffma2(q2[g][i], bf16x2_to_float2(kw[i]), t);
          s[g] = t.x + t.y;
        }
        // sum the 8 partial dot products of the slot's lane group (all lanes)
#pragma unroll
        for (int off2 = 1; off2 < 8; off2 <<= 1) {
#pragma unroll
          for (int g = 0; g < G; ++g) s[g] += __shfl_xor_sync(0xffffffffu, s[g], off2);
        }
        if (valid) {
          if (is_res) {
            const float lc = logc_s[y - logc_lo];
#pragma unroll
            for (int g = 0; g < G; ++g) s[g] += lc;     // + beta*log c_j (log2 units)
          }
          const uint32_t vw[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
#pragma unroll
          for (int g = 0; g < G; ++g) {
            if (s[g] == -INFINITY) continue;           // empty residual entry (c = 0)
            if (s[g] > m[g]) {
              const float sc = exp2f(m[g] - s[g]);
              l[g] *= sc;
#pragma unroll
              for (int i = 0; i < 8; ++i) acc[g][i] = fmul2(acc[g][i], make_float2(sc, sc));
              m[g] = s[g];
            }
            const float pr = exp2f(s[g] - m[g]);
            l[g] += pr;
            const float2 pr2 = make_float2(pr, pr);
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[g][i] = ffma2(pr2, bf16x2_to_float2(vw[i]), acc[g][i]);
          }
        }
        // never past the segment end: the next segment may start in the same stage
        release_upto((x + 4 < hi) ? x + 4 : hi);
      }
      if (failed) break;

      // combine the 4 lane groups (each saw a quarter of the slots)
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float mx = fmaxf(m[g], __shfl_xor_sync(0xffffffffu, m[g], 8));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
        const float sc = (l[g] > 0.0f) ? exp2f(m[g] - mx) : 0.0f;
        float lg = l[g] * sc;
        lg += __shfl_xor_sync(0xffffffffu, lg, 8);
        lg += __shfl_xor_sync(0xffffffffu, lg, 16);
        float ag[16];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          ag[2 * i] = acc[g][i].x * sc;
          ag[2 * i + 1] = acc[g][i].y * sc;
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          ag[i] += __shfl_xor_sync(0xffffffffu, ag[i], 8);
          ag[i] += __shfl_xor_sync(0xffffffffu, ag[i], 16);
        }
        if (g == grp) {                  // lane group `grp` keeps head `grp`
          segs[sgi].m = mx;
          segs[sgi].l = lg;
#pragma unroll
          for (int i = 0; i < 16; ++i) segs[sgi].acc[i] = ag[i];
        }
      }
    }
    if (failed) break;
    if (segs[2].l > 0.0f) {            // appended rows join the main softmax state
      const float mx = fmaxf(segs[0].m, segs[2].m);
      const float s0 = segs[0].l > 0.0f ? exp2f(segs[0].m - mx) : 0.0f;
      const float s2 = exp2f(segs[2].m - mx);
      segs[0].l = segs[0].l * s0 + segs[2].l * s2;
#pragma unroll
      for (int i = 0; i < 16; ++i) segs[0].acc[i] = segs[0].acc[i] * s0 + segs[2].acc[i] * s2;
      segs[0].m = mx;
    }

    // ---- finish the unit, or leave a partial record for the last warp ----
    const int64_t uend = ubase + nm + nr + na;
    const bool whole = (a <= ubase) && (e >= uend);
    const int64_t orow = (u / p.n_kv_heads) * int64_t(p.n_kv_heads) * G + (u % p.n_kv_heads) * G;
    if (whole) {
      if (grp < G) {
        float o[16];
        finalize(p, segs[0], segs[1], o);
        float* op = p.O + (orow + grp) * kHeadDim;
        *reinterpret_cast<float4*>(op + 8 * sub) = make_float4(o[0], o[1], o[2], o[3]);
        *reinterpret_cast<float4*>(op + 8 * sub + 4) = make_float4(o[4], o[5], o[6], o[7]);
        *reinterpret_cast<float4*>(op + 64 + 8 * sub) = make_float4(o[8], o[9], o[10], o[11]);
        *reinterpret_cast<float4*>(op + 64 + 8 * sub + 4) = make_float4(o[12], o[13], o[14], o[15]);
      }
      continue;
    }
    // partial record (u + gw): [seg][head][m, l, acc[d]]
    const int64_t w0 = warp_of(ubase, T, W);
    const int64_t w1 = warp_of(uend - 1, T, W);
    float* rec = p.partials + (u + gw) * (2 * G * kRecordFloats);
    if (grp < G) {
#pragma unroll
      for (int sgi = 0; sgi < 2; ++sgi) {
        float* r = rec + (sgi * G + grp) * kRecordFloats;
        if (sub == 0) {
          r[0] = segs[sgi].m;
          r[1] = segs[sgi].l;
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) r[2 + dim_of(sub, i)] = segs[sgi].acc[i];
      }
    }
    __threadfence();
    __syncwarp();
    int ticket = 0;
    if (lane == 0) ticket = atomicAdd(p.tickets + p.unit0 + u, 1);
    ticket = __shfl_sync(0xffffffffu, ticket, 0);
    if (ticket != int(w1 - w0)) continue;          // not the last to arrive
    __threadfence();
    if (grp < G) {
      SegState acc2[2];
#pragma unroll
      for (int sgi = 0; sgi < 2; ++sgi) {
        acc2[sgi].m = -INFINITY;
        acc2[sgi].l = 0.0f;
#pragma unroll
        for (int i = 0; i < 16; ++i) acc2[sgi].acc[i] = 0.0f;
      }
      for (int64_t w = w0; w <= w1; ++w) {
        const float* rr = p.partials + (u + w) * (2 * G * kRecordFloats);
#pragma unroll
        for (int sgi = 0; sgi < 2; ++sgi) {
          const float* r = rr + (sgi * G + grp) * kRecordFloats;
          const float bm = __ldcg(r), bl = __ldcg(r + 1);
          float bacc[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) bacc[i] = __ldcg(r + 2 + dim_of(sub, i));
          merge_into(acc2[sgi], bm, bl, bacc);
        }
      }
      float o[16];
      finalize(p, acc2[0], acc2[1], o);
      float* op = p.O + (orow + grp) * kHeadDim;
      *reinterpret_cast<float4*>(op + 8 * sub) = make_float4(o[0], o[1], o[2], o[3]);
      *reinterpret_cast<float4*>(op + 8 * sub + 4) = make_float4(o[4], o[5], o[6], o[7]);
      *reinterpret_cast<float4*>(op + 64 + 8 * sub) = make_float4(o[8], o[9], o[10], o[11]);
      *reinterpret_cast<float4*>(op + 64 + 8 * sub + 4) = make_float4(o[12], o[13], o[14], o[15]);
    }
    __syncwarp();
    if (lane == 0) p.tickets[p.unit0 + u] = 0;      // ready for the next launch
  }

  // never leave with a bulk copy in flight into this warp's ring (bounded
  // waits, also after a failure)
  const int64_t issued = (released + kStages < nchunks) ? released + kStages : nchunks;
  for (int64_t k = ready + 1; k < issued; ++k) {
    mbar_wait_bounded(&full[k % kStages], uint32_t((k / kStages) & 1));
  }
}

}  // namespace

size_t decode_partials_floats(int64_t n_units, int n_warps, int group) {
  return size_t(n_units + n_warps) * 2 * group * kRecordFloats;
}

template <int G>
static cudaError_t launch_g(const DecodeParams& p, int n_ctas, cudaStream_t stream) {
  // the shared-memory opt-in is set once per device, so that launches made
  // during CUDA-graph capture issue nothing but the launch itself
  static std::atomic<unsigned long long> configured{0};
  const int smem = kDecodeWarpsPerCta * kWarpSmem;
  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return err;
  const unsigned long long bit = 1ull << (dev & 63);
  if (!(configured.load() & bit)) {
    err = cudaFuncSetAttribute(reskv_decode_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               smem);
    if (err != cudaSuccess) return err;
    configured.fetch_or(bit);
  }
  reskv_decode_kernel<G><<<n_ctas, kDecodeWarpsPerCta * 32, smem, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_decode(const DecodeParams& p, int group, int n_ctas, cudaStream_t stream) {
  switch (group) {
    case 1: return launch_g<1>(p, n_ctas, stream);
    case 2: return launch_g<2>(p, n_ctas, stream);
    case 4: return launch_g<4>(p, n_ctas, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace reskv
