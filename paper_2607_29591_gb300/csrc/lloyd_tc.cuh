// Lloyd assignment (Sec. 5.3, Eq. residual_partition) on the 5th-generation
// tensor cores: every evicted token of a 128-token tile to its nearest centre.
//
// The distances d_j = ||c_j||^2 - 2 <c_j, k> (the ||k||^2 term is common)
// need the dot products of the tile's 128 bf16 keys with every centre: a
// [128 x 128] x [128 x r] contraction.  Each fp32 centre is split exactly into
// two bf16 planes c = c1 + c2 + e, |e_i| <= 2^-16 |c_i| (write_planes), so
// <c, k> = <c1, k> + <c2, k> up to e: one tcgen05.mma chain per 64-centre
// chunk (2 planes x 8 K-steps of 16 dims, M = 128 tokens, N = 64 centres)
// accumulates both planes in fp32 in tensor memory (TMEM), thread t of the CTA
// owns TMEM lane t = token t (threads t and t + 128 read its row's columns
// 0..31 and 32..63 of each chunk with tcgen05.ld).
//
// Pipeline (one CTA of 8 warps per tile): the keys are staged once; centre
// chunks stream through two shared-memory buffers and two 64-column TMEM
// blocks, so the MMAs of chunk c run while the threads reduce chunk c - 1:
//
//   iteration c:  wait for chunk c's planes; thread 0 issues its MMAs into
//                 TMEM block c & 1 and commits them to mbarrier c & 1;
//                 wait for chunk c - 1's MMAs (its buffer is then free:
//                 chunk c + 1's planes go there) and reduce its 64 distances.
//
// Operands are K-major with the 128-byte swizzle (the canonical layout of the
// shared-memory matrix descriptors): per 64-dim half, rows of 128 bytes, the
// 16-byte chunk c of row r at ((c ^ (r & 7)) << 4), 8-row groups 1024 bytes
// apart; the K-steps inside a half advance the descriptor's start by 32 bytes.
//
// Assignments must equal the fp64 oracle's, so every choice is certified: each
// thread sees every centre of its token and keeps the best and second-best
// centre and the third-best distance (top3_insert, branch-free); a bound on
// the computed distances' error decides whether the kept candidates, or all
// centres (when the third best is within the bound), could in truth be
// nearest, and those are re-evaluated as sum_i (k_i - c_i)^2 in fp64 against
// the fp64 centres by the whole warp, one token at a time (fp64 is scarce on
// this part).  Ties go to the lower centre index.
// Error bound of the dot product, u = 2^-24, P = sum_i |c_i k_i|: one MMA step
// adds 16 exact products to the fp32 accumulator with an error of at most
// 17 * 2^-22 times the largest partial magnitude (<= P) even if it truncates
// to 24 bits; 16 chained steps (both planes) give 272 * 2^-22 P = 1088u P,
// the split e adds 256u P: taken as 2048u P.
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

namespace reskv {
namespace build {

constexpr int kTcThreads = 256;              // 8 warps: warps w and w + 4 read TMEM lanes
                                             // 32 (w % 4).. = tokens, each half the columns
constexpr int kTcNC = 64;                    // centres per chunk (MMA N)
constexpr int kTcHalf = kTile * 128;         // one 64-dim half of the key tile, bytes
constexpr int kTcBHalf = kTcNC * 128;        // one 64-dim half of a chunk plane, bytes
constexpr int kTcBBuf = 2 * 2 * kTcBHalf;    // a chunk: 2 planes x 2 halves
constexpr uint32_t kTcCols = 2 * kTcNC;      // TMEM columns: two 64-column blocks
constexpr long long kTcWaitCycles = 4000000000LL;

// Shared memory: [keys 2 halves][2 chunk buffers][norms of every centre,
// padded to whole chunks][per-centre counts][2 mbarriers][TMEM address].
inline size_t lloyd_tc_smem(int rmax) {
  const size_t nch = size_t((rmax + kTcNC - 1) / kTcNC > 0 ? (rmax + kTcNC - 1) / kTcNC : 1);
  return 1024 + 2 * size_t(kTcHalf) + 2 * size_t(kTcBBuf) + nch * kTcNC * 4 +
         size_t(rmax > 0 ? rmax : 1) * 4 + 15 + 16 + 4 + 13;   // align, 2 mbarriers, TMEM slot
}

__device__ __forceinline__ uint32_t tc_sw128(int r, int c) {
  return uint32_t(r) * 128u + uint32_t((c ^ (r & 7)) << 4);
}

// Shared-memory matrix descriptor: start address (16-byte units), leading
// byte offset 1 (unused by swizzled K-major layouts), stride byte offset
// 1024 (8-row groups), descriptor version 1, 128-byte swizzle.
__device__ __forceinline__ uint64_t tc_desc(uint32_t saddr) {
  return uint64_t((saddr & 0x3FFFFu) >> 4) | (uint64_t(1) << 16) | (uint64_t(1024 >> 4) << 32) |
         (uint64_t(1) << 46) | (uint64_t(2) << 61);
}

// Instruction descriptor of kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, N = kTcNC, M = 128.
constexpr uint32_t kTcIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(kTcNC >> 3) << 17) |
                              (uint32_t(kTile >> 4) << 24);

__device__ __forceinline__ void tc_mma(uint32_t tmem_d, uint64_t ad, uint64_t bd, bool accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(ad), "l"(bd), "r"(kTcIdesc), "r"(accumulate ? 1 : 0));
}

__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}

// 32 consecutive fp32 columns of this thread's TMEM lane from column address ta
__device__ __forceinline__ void tc_ld32(uint32_t ta, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
      "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(ta));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Wait for phase `parity` of bar; false after the bound.
__device__ __forceinline__ bool tc_wait(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity))
    if (clock64() - t0 > kTcWaitCycles) return false;
  return true;
}


// Nearest centre of every evicted token of tile blockIdx.x of unit blockIdx.y
// (assign: centre index, -1 for tokens outside E), and the tile's count of
// members per centre (hist).
__global__ void __launch_bounds__(kTcThreads, 2) k_lloyd_assign_tc(LloydArgs p) {
  extern __shared__ uint8_t tc_raw[];
  uint8_t* base = tc_raw + ((1024u - (smem_u32(tc_raw) & 1023u)) & 1023u);   // 1024-aligned
  uint8_t* As = base;                                            // [2 halves][128 rows][128 B]
  uint8_t* Bs = As + 2 * kTcHalf;                                // [2 bufs][2 planes][2 halves][64][128 B]
  const int tile = blockIdx.x, ul = blockIdx.y;
  const int r = p.r_unit[ul];
  if (r == 0) return;
  const int nch = (r + kTcNC - 1) / kTcNC;
  float* cn_s = reinterpret_cast<float*>(Bs + 2 * kTcBBuf);    // [nch * 64], +inf past r
  int* cnt = reinterpret_cast<int*>(cn_s + nch * kTcNC);         // [r]
  uint64_t* bars = reinterpret_cast<uint64_t*>((reinterpret_cast<uintptr_t>(cnt + r) + 15) & ~uintptr_t(15));
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 2);
  __shared__ unsigned int cnmax_bits;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t tok0 = int64_t(tile) * kTile;
  const __nv_bfloat16* Ku = p.K + int64_t(ul) * p.s * kHeadDim;
  const __nv_bfloat16* planes = p.cplanes + int64_t(ul) * 2 * p.rmax * kHeadDim;
  const float* cnorm = p.cnorm + int64_t(ul) * p.rmax;
  const uint32_t as_s = smem_u32(As), bs_s = smem_u32(Bs);

  // centre chunk c's two planes into buffer c & 1 (zeros past r)
  auto stage_chunk = [&](int c) {
    const int cb = c * kTcNC;
    const uint32_t dst = bs_s + uint32_t(c & 1) * kTcBBuf;
    for (int i = tid; i < 2 * kTcNC * 16; i += kTcThreads) {
      const int pl = i / (kTcNC * 16), rem = i % (kTcNC * 16), row = rem >> 4, ch = rem & 15;
      const bool in = cb + row < r;
      const __nv_bfloat16* src = planes + (int64_t(pl) * p.rmax + (in ? cb + row : 0)) * kHeadDim + 8 * ch;
      cp_async16(dst + uint32_t(pl * 2 * kTcBHalf + (ch >> 3) * kTcBHalf) + tc_sw128(row, ch & 7), src,
                 in ? 16u : 0u);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  // the key tile (zeros past s), the first chunk, every centre norm
  for (int i = tid; i < kTile * 16; i += kTcThreads) {
    const int row = i >> 4, ch = i & 15;
    const bool in = tok0 + row < p.s;
    cp_async16(as_s + uint32_t((ch >> 3) * kTcHalf) + tc_sw128(row, ch & 7),
               Ku + (in ? (tok0 + row) * kHeadDim : 0) + 8 * ch, in ? 16u : 0u);
  }
  stage_chunk(0);
  if (tid == 0) cnmax_bits = 0u;
  for (int i = tid; i < nch * kTcNC; i += kTcThreads) cn_s[i] = i < r ? cnorm[i] : INFINITY;
  for (int i = tid; i < r; i += kTcThreads) cnt[i] = 0;
  if (tid == 0) {
    mbar_init(&bars[0], 1);
    mbar_init(&bars[1], 1);
    fence_mbar_init();
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tslot)),
                 "r"(kTcCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  __syncthreads();
  float cmx = 0.f;
  for (int i = tid; i < r; i += kTcThreads) cmx = fmaxf(cmx, cn_s[i]);
  atomicMax(&cnmax_bits, __float_as_uint(cmx));       // non-negative: bit order = value order
  tc_fence_after();
  const uint32_t tmem = *tslot;

  // this thread's token: best (d0, j0), second best (d1, j1), third-best d2
  float d0 = INFINITY, d1 = INFINITY, d2 = INFINITY;
  int j0 = INT_MAX, j1 = INT_MAX;
  bool failed = false;
  for (int c = 0; c <= nch; ++c) {
    if (c < nch) {
      // chunk c (and, at c = 0, the keys) in shared memory, visible to the tensor cores
      asm volatile("cp.async.wait_group 0;" ::: "memory");
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      tc_fence_before();
      __syncthreads();
      tc_fence_after();
      if (tid == 0 && !failed) {
        const uint32_t buf = bs_s + uint32_t(c & 1) * kTcBBuf;
        const uint32_t d_tmem = tmem + uint32_t((c & 1) * kTcNC);
#pragma unroll
        for (int pl = 0; pl < 2; ++pl)
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t half = uint32_t(k >> 2), kk = uint32_t(k & 3) * 32u;
            tc_mma(d_tmem, tc_desc(as_s + half * kTcHalf + kk),
                   tc_desc(buf + uint32_t(pl) * 2 * kTcBHalf + half * kTcBHalf + kk), pl + k > 0);
          }
        tc_commit(&bars[c & 1]);
      }
    }
    if (c >= 1) {
      const int cp = c - 1;                               // the chunk to reduce
      // a bounded wait; the verdict is made warp-uniform (tcgen05.ld below is
      // a warp-wide instruction)
      const bool ok = failed || tc_wait(&bars[cp & 1], uint32_t((cp >> 1) & 1));
      if (__any_sync(0xffffffffu, !ok) && !failed) {
        failed = true;
        if (lane == 0) report_status(p.status, kStatusWaitTimeout);
      }
      tc_fence_after();
      if (c + 1 < nch) stage_chunk(c + 1);               // into chunk cp's buffer, now free
      if (!failed) {
        // this thread's 32 columns of the chunk: lane quarter warp % 4,
        // column half warp / 4
        const int wq = warp & 3, wg = warp >> 2;
        const uint32_t ta = tmem + (uint32_t(32 * wq) << 16) + uint32_t((cp & 1) * kTcNC + 32 * wg);
        float acc[32];
        tc_ld32(ta, acc);
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int col = cp * kTcNC + 32 * wg + i;
          top3_insert(d0, j0, d1, j1, d2, fmaf(-2.0f, acc[i], cn_s[col]), col);
        }
      }
    } else if (nch > 1) {
      stage_chunk(1);
    }
  }

  // the two halves' lists of token t meet in thread t (warps 0..3): the
  // second half's best two join by (distance, index), its third best bounds
  // the centres neither list kept.  The chunk buffers are free by now.
  float* mrg = reinterpret_cast<float*>(Bs);                     // [128 tokens][5]
  if (warp >= 4) {
    float* m = mrg + (tid - kTile) * 5;
    m[0] = d0;
    m[1] = __int_as_float(j0);
    m[2] = d1;
    m[3] = __int_as_float(j1);
    m[4] = d2;
  }
  __syncthreads();
  if (warp < 4) {
    const float* m = mrg + tid * 5;
    const float od0 = m[0], od1 = m[2], od2 = m[4];
    const int oj0 = __float_as_int(m[1]), oj1 = __float_as_int(m[3]);
    d2 = fminf(d2, od2);
    float e[4] = {d0, d1, od0, od1};
    int je[4] = {j0, j1, oj0, oj1};
    // the two least (distance, index) of the four, the third least into d2
#pragma unroll
    for (int a = 0; a < 3; ++a)
#pragma unroll
      for (int b = 3; b > a; --b)
        if (e[b] < e[b - 1] || (e[b] == e[b - 1] && je[b] < je[b - 1])) {
          const float tf = e[b]; e[b] = e[b - 1]; e[b - 1] = tf;
          const int ti = je[b]; je[b] = je[b - 1]; je[b - 1] = ti;
        }
    d0 = e[0]; j0 = je[0];
    d1 = e[1]; j1 = je[1];
    d2 = fminf(d2, e[2]);
  }

  // certification: err(d) = 2 x (dot product
  // 2 gam_tc ||c|| ||k|| + norm sum 2 gam ||c||^2 + fp32 centre 4u ||k|| ||c||
  // + final subtraction 2u |d|), ||c|| <= max ||c|| over the unit
  const int64_t pos = tok0 + tid;
  const bool mine = warp < 4 && pos < p.s;                // thread t < 128: token t
  const bool ev = mine && !failed && in_evicted(p, ul, pos, r);
  unsigned cmask = 0u;                                    // bit 0: j0, bit 1: j1
  bool full = false;
  if (ev) {
    float s2 = 0.f;
#pragma unroll
    for (int ch = 0; ch < 16; ++ch) {
      const uint4 v = *reinterpret_cast<const uint4*>(As + (ch >> 3) * kTcHalf + tc_sw128(tid, ch & 7));
      const uint32_t wd[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float2 f = bf16x2_to_float2(wd[q]);
        s2 = fmaf(f.x, f.x, s2);
        s2 = fmaf(f.y, f.y, s2);
      }
    }
    const float u = 5.9604645e-8f, gam = 130.0f * u, gam_tc = 2048.0f * u;
    const float kn = sqrtf(s2) * (1.0f + gam), cm = sqrtf(__uint_as_float(cnmax_bits));
    const float e0 = 2.0f * (2.0f * gam_tc * cm * kn + 2.0f * gam * cm * cm + 4.0f * u * kn * cm);
    const float err0 = e0 + 4.0f * u * fabsf(d0);
    full = d2 - d0 <= err0 + e0 + 4.0f * u * fabsf(d2);   // the third best could win too
    if (j1 < r && d1 - d0 <= err0 + e0 + 4.0f * u * fabsf(d1)) cmask = 3u;
    if (j0 >= r) {                                        // only a NaN distance gets here
      report_status(p.status, kStatusBadIndex);
      j0 = 0;
      cmask = 0u;
      full = false;
    }
  }
  // fp64 re-evaluation, one ambiguous token at a time by the whole warp: lane
  // i holds dims 4i..4i+3, the distance is reduced over the warp (lane 0's sum
  // decides); ties -> lower index
  unsigned amb = __ballot_sync(0xffffffffu, ev && (full || cmask != 0u));   // 0 in warps 4..7
  const double* c64 = p.centers64 + int64_t(ul) * p.rmax * kHeadDim + 4 * lane;
  while (amb) {
    const int src = __ffs(amb) - 1;
    amb &= amb - 1;
    const int ts = 32 * warp + src;
    const bool fs = __shfl_sync(0xffffffffu, full ? 1 : 0, src) != 0;
    const int js0 = __shfl_sync(0xffffffffu, j0, src), js1 = __shfl_sync(0xffffffffu, j1, src);
    const uint2 kw = *reinterpret_cast<const uint2*>(As + (lane >> 4) * kTcHalf +
                                                     tc_sw128(ts, (lane & 15) >> 1) + 8 * (lane & 1));
    const float2 k01 = bf16x2_to_float2(kw.x), k23 = bf16x2_to_float2(kw.y);
    const double kx[4] = {k01.x, k01.y, k23.x, k23.y};
    double bd = INFINITY;
    int bj = INT_MAX;
    // fp64 distances of four centres (index < 0: none), reduced over the warp
    auto eval4 = [&](const int (&jq)[4]) {
      double a[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const double4_32a c =
            *reinterpret_cast<const double4_32a*>(c64 + int64_t(jq[q] < 0 ? 0 : jq[q]) * kHeadDim);
        double t = (kx[0] - c.x) * (kx[0] - c.x);
        t = fma(kx[1] - c.y, kx[1] - c.y, t);
        t = fma(kx[2] - c.z, kx[2] - c.z, t);
        a[q] = fma(kx[3] - c.w, kx[3] - c.w, t);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1)
#pragma unroll
        for (int q = 0; q < 4; ++q) a[q] += __shfl_xor_sync(0xffffffffu, a[q], o);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const double dd = __shfl_sync(0xffffffffu, a[q], 0);
        if (jq[q] >= 0 && (dd < bd || (dd == bd && jq[q] < bj))) {
          bd = dd;
          bj = jq[q];
        }
      }
    };
    if (fs) {                                             // every centre
      for (int jb = 0; jb < r; jb += 4) {
        const int jq[4] = {jb, jb + 1 < r ? jb + 1 : -1, jb + 2 < r ? jb + 2 : -1,
                           jb + 3 < r ? jb + 3 : -1};
        eval4(jq);
      }
    } else {                                              // the two kept candidates
      const int jq[4] = {js0, js1, -1, -1};
      eval4(jq);
    }
    if (lane == src) j0 = bj;
  }
  if (ev) {
    p.assign[int64_t(ul) * p.s + pos] = j0;
    atomicAdd(&cnt[j0], 1);
  } else if (mine) {
    p.assign[int64_t(ul) * p.s + pos] = -1;
  }
  tc_fence_before();
  __syncthreads();
  int32_t* h = p.hist + (int64_t(ul) * p.ntiles + tile) * p.rmax;
  for (int i = tid; i < r; i += kTcThreads) h[i] = cnt[i];
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTcCols));
  }
}

}  // namespace build
}  // namespace reskv
