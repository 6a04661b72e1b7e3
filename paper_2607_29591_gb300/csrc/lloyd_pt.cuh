// Lloyd assignment (Sec. 5.3, Eq. residual_partition), persistent form for
// units with at most 256 centres: one CTA per SM walks a contiguous range of
// (unit, 128-token tile) pairs, with the unit's centre planes resident in
// shared memory, so a tile costs one key-tile load and one tcgen05.mma chain.
// Four roles run decoupled, linked by mbarrier rings:
//
//   loader warp      loads key tiles by TMA (both 64-dim halves, 128-byte
//                    swizzle, one 32 KB copy) into a ring of nk buffers, as far
//                    ahead as the buffers allow, across unit changes too
//                    (key_full[]; a buffer is refilled once key_free[] says
//                    its MMAs are done).
//   MMA warp         for each tile issues the MMA chain of all the unit's
//                    centres (2 planes x 8 K-steps, M = 128 tokens, N = r
//                    rounded up to 16) into TMEM columns 256 (t & 1) ..,
//                    committed to full[] and to the key buffer's key_free[].
//                    At a change of unit it waits for every earlier MMA and
//                    for the column warps to be done with the old centre
//                    norms, then stages the new planes (cp.async).
//   8 column warps   warp w reads TMEM lanes 32 (w % 4).. (its tokens) and the
//                    16-column chunks w / 4, w / 4 + 2, .. of the distances,
//                    keeping each token's best three as fp32 keys with the
//                    centre index in the low 8 significand bits (two lists
//                    per thread, even and odd columns, each a fminf/fmaxf
//                    network), frees the TMEM buffer (tmem_empty[]), merges
//                    the two column halves and posts the tile's lists, with
//                    each token's rank and key norm, in a ring of kPtRing
//                    slots (list_full[]).
//   4 certifier      decide each evicted token from a rigorous bound on the
//   warps            tensor-core distance error: the best centre is certified,
//                    or the token joins a list that k_lloyd_resolve decides
//                    (direct fp32 distances, then fp64 where those still
//                    overlap).  They write assign, count the certified members
//                    per centre, write the tile's counts and free the slot
//                    (list_empty[]).
//
// Certification needs no global memory and no fp64 (scarce on this part),
// so the certifiers keep pace with the column warps.  Every wait is bounded;
// a wait that gives up raises kStatusWaitTimeout and an abort flag, and each
// role leaves its loop at a tile boundary agreed by a barrier reduction over
// the role's threads.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cfloat>
#include <cstdint>

#include "lloyd_tc.cuh"

namespace reskv {
namespace build {

constexpr int kPtColWarps = 8;
constexpr int kPtColThreads = kPtColWarps * 32;
constexpr int kPtCertWarps = 4;
constexpr int kPtCertThreads = kPtCertWarps * 32;
constexpr int kPtProducer = kPtColWarps + kPtCertWarps;        // the MMA-issuing warp's index
constexpr int kPtLoader = kPtProducer + 1;                      // the key-loading warp's index
constexpr int kPtThreads = (kPtLoader + 1) * 32;
constexpr int kPtRmax = 256;                                    // centres held resident
constexpr int kPtRing = 4;                                      // list slots
constexpr int kPtKeys = 2 * kTcHalf;                            // one key tile
constexpr uint32_t kPtBufCols = 256;                            // TMEM columns per buffer
constexpr uint32_t kPtCols = 2 * kPtBufCols;
constexpr int kPtXch = kTile * 3;                               // a token's three best keys
constexpr int kPtList = kTile * 5;                              // the same, + rank, ||k||^2

// Shared memory, from a 1024-aligned base: the planes of rp = r rounded up
// to 16 centres ([plane][64-dim half][rp rows][128 B], 512 rp bytes), nk key
// tiles of 32 KB, then a tail of fixed size: centre norms, 2 x the column
// halves' exchange keys, the ring (lists, counts, info), 2 x TMEM tile info,
// the abort flag, the mbarriers and the TMEM address.
constexpr int kPtMaxKeyBufs = 4;
constexpr size_t kPtOffNorm = 0;
constexpr size_t kPtOffXch = kPtOffNorm + kPtRmax * 4;
constexpr size_t kPtOffList = kPtOffXch + 2 * kPtXch * 4;
constexpr size_t kPtOffCnt = kPtOffList + kPtRing * kPtList * 4;
constexpr size_t kPtOffRInfo = kPtOffCnt + kPtRing * kPtRmax * 4;
constexpr size_t kPtOffTInfo = kPtOffRInfo + kPtRing * 8 * 4;
constexpr size_t kPtOffAbort = kPtOffTInfo + 2 * 4 * 4;
constexpr size_t kPtOffBars = kPtOffAbort + 8;
// full, tmem_empty (2 each), list_full, list_empty (ring), key_full, key_free (key buffers)
constexpr int kPtNumBars = 2 + 2 + 2 * kPtRing + 2 * kPtMaxKeyBufs;
constexpr size_t kPtOffSlot = kPtOffBars + kPtNumBars * 8;
constexpr size_t kPtTail = kPtOffSlot + 16;
static_assert(kPtOffBars % 8 == 0, "mbarriers need 8-byte alignment");
constexpr size_t kPtSmemMax = 232448;                  // 227 KB of opt-in shared memory per CTA

__host__ __device__ inline size_t lloyd_pt_planes(int rp) { return size_t(rp) * 512; }
// key buffers that fit beside the planes of rp centres (>= 2 for rp <= 256)
inline int lloyd_pt_key_bufs(int rp) {
  const size_t room = kPtSmemMax - 1024 - kPtTail - lloyd_pt_planes(rp);
  return int(std::min<size_t>(kPtMaxKeyBufs, room / kPtKeys));
}
inline size_t lloyd_pt_smem(int rp) {
  return 1024 + lloyd_pt_planes(rp) + size_t(lloyd_pt_key_bufs(rp)) * kPtKeys + kPtTail;
}

// Instruction descriptor of kind::f16 for N = n (a multiple of 16, <= 256).
__device__ __forceinline__ uint32_t pt_idesc(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(n >> 3) << 17) | (uint32_t(kTile >> 4) << 24);
}

__device__ __forceinline__ void pt_mma(uint32_t tmem_d, uint64_t ad, uint64_t bd, uint32_t idesc,
                                       bool accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(ad), "l"(bd), "r"(idesc), "r"(accumulate ? 1 : 0));
}

// 16 consecutive fp32 columns of this thread's TMEM lane from column address ta
__device__ __forceinline__ void tc_ld16(uint32_t ta, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, "
      "%13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15])
      : "r"(ta));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// one 128-token key tile (both 64-dim halves, 128-byte swizzle) from row y
// of the layer's keys, completing on bar
__device__ __forceinline__ void tma_keys(uint32_t dst, const CUtensorMap* map, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::
          "r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(y), "r"(0), "r"(smem_u32(bar))
      : "memory");
}

// A shared-memory descriptor advanced by `bytes` (a multiple of 16): the start
// address sits in bits 0..13 as address / 16, and stays below 2^14 for the
// 227 KB of shared memory, so the low word takes the addition without carry.
__device__ __forceinline__ uint64_t desc_plus(uint64_t d, uint32_t bytes) {
  return d + uint64_t(bytes >> 4);
}

// a probe of phase `parity` of bar that never blocks
__device__ __forceinline__ bool mbar_test_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ void pt_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// named barrier `id` over `n` threads
__device__ __forceinline__ void pt_bar(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

// named barrier `id` over `n` threads, returning whether any of them passed true
__device__ __forceinline__ bool pt_bar_or(int id, int n, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 q, %1, 0;\n\t"
      "bar.red.or.pred p, %2, %3, q;\n\tselp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(r)
      : "r"(v ? 1u : 0u), "r"(id), "r"(n)
      : "memory");
  return r != 0u;
}

// Wait for phase `parity` of bar; false after the bound or once the abort
// flag is up.
__device__ __forceinline__ bool pt_wait(uint64_t* bar, uint32_t parity, const volatile uint32_t* abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait(bar, parity)) {
    if (*abort != 0u || clock64() - t0 > kTcWaitCycles) return false;
  }
  return true;
}

__device__ __forceinline__ void pt_raise(volatile uint32_t* abort, uint32_t* status) {
  if (*abort == 0u) {
    *abort = 1u;
    report_status(status, kStatusWaitTimeout);
  }
}

// (x, jx) into a best-two list ordered by (distance, index) with the
// third-best distance alongside (the lists of different column sets meet here)
__device__ __forceinline__ void top3_insert_lex(float& d0, int& j0, float& d1, int& j1, float& d2,
                                                float x, int jx) {
  const bool c0 = x < d0 || (x == d0 && jx < j0);
  const bool c1 = x < d1 || (x == d1 && jx < j1);
  const bool c2 = x < d2;
  d2 = c1 ? d1 : (c2 ? x : d2);
  d1 = c0 ? d0 : (c1 ? x : d1);
  j1 = c0 ? j0 : (c1 ? jx : j1);
  d0 = c0 ? x : d0;
  j0 = c0 ? jx : j0;
}

// another list's best two and third-best distance into (d0, j0, d1, j1, d2)
__device__ __forceinline__ void top3_merge(float& d0, int& j0, float& d1, int& j1, float& d2,
                                           float e0, int k0, float e1, int k1, float e2) {
  top3_insert_lex(d0, j0, d1, j1, d2, e0, k0);
  top3_insert_lex(d0, j0, d1, j1, d2, e1, k1);
  d2 = fminf(d2, e2);
}

// A distance with the centre index in its 8 low significand bits (r <= 256):
// keys order like the distances up to |key - d| <= 2^-15 |d|, and distinct
// centres never tie, so three fminf / fmaxf pairs keep a token's best three.
__device__ __forceinline__ float pt_key(float d, int col) {
  return __int_as_float((__float_as_int(d) & ~0xFF) | col);
}
__device__ __forceinline__ int pt_key_index(float key) { return __float_as_int(key) & 0xFF; }

// pt_key by one byte permute: byte 0 from byte b of `cols`, which holds
// four consecutive centre indices (one per byte)
template <int b>
__device__ __forceinline__ float pt_key4(float d, uint32_t cols) {
  return __int_as_float(int(__byte_perm(uint32_t(__float_as_int(d)), cols, 0x3214u + b)));
}

// key into the ascending best three (x0, x1, x2)
__device__ __forceinline__ void pt_ins3(float& x0, float& x1, float& x2, float key) {
  const float t0 = fmaxf(x0, key);
  x0 = fminf(x0, key);
  const float t1 = fmaxf(x1, t0);
  x1 = fminf(x1, t0);
  x2 = fminf(x2, t1);
}

// fp32 ||k||^2 of every key row (a warp per row), for the certification
// bound: 128 products summed in any order stay within 130 u of the sum.
__global__ void k_key_norm2(const __nv_bfloat16* __restrict__ K, float* __restrict__ out, int64_t rows) {
  const int64_t row = int64_t(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (row >= rows) return;
  const int lane = threadIdx.x & 31;
  const uint2 w = *reinterpret_cast<const uint2*>(K + row * kHeadDim + 4 * lane);
  const float2 a = bf16x2_to_float2(w.x), b = bf16x2_to_float2(w.y);
  float s = fmaf(a.x, a.x, fmaf(a.y, a.y, fmaf(b.x, b.x, b.y * b.y)));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) out[row] = s;
}

// (unit, tile) of the flat tile order g = unit * ntiles + tile, stepped
// without divisions, skipping units with r = 0; r is read once per unit
struct PtCursor {
  int64_t g, g1;
  int u, tile, r;
  __device__ PtCursor(const LloydArgs& p, int64_t g0_, int64_t g1_) : g(g0_), g1(g1_) {
    u = int(g0_ / p.ntiles);
    tile = int(g0_ % p.ntiles);
    r = g < g1 ? p.r_unit[u] : 0;
    skip(p);
  }
  __device__ void skip(const LloydArgs& p) {
    while (g < g1 && r <= 0) {
      g += p.ntiles - tile;
      tile = 0;
      ++u;
      r = g < g1 ? p.r_unit[u] : 0;
    }
  }
  __device__ void next(const LloydArgs& p) {
    ++g;
    if (++tile == p.ntiles) {
      tile = 0;
      ++u;
      r = g < g1 ? p.r_unit[u] : 0;
    }
    skip(p);
  }
};

// Nearest centre of every evicted token of the tiles [g0, g1) of the flat
// (unit, tile) order, g = unit * ntiles + tile (assign: centre index, -1 for
// tokens outside E), and each tile's member count per centre (hist).  Units
// with r = 0 are skipped; every unit must have r <= 256; p.knorm2 holds the
// layer's key norms (k_key_norm2).
__global__ void __launch_bounds__(kPtThreads, 1)
    k_lloyd_assign_pt(LloydArgs p, int n_units, int rp_max, int nk, const __grid_constant__ CUtensorMap tmK) {
  extern __shared__ uint8_t pt_raw[];
  uint8_t* base = pt_raw + ((1024u - (smem_u32(pt_raw) & 1023u)) & 1023u);
  const uint32_t plane_half = uint32_t(rp_max) * 128u;           // one plane's 64-dim half, bytes
  uint8_t* tail = base + lloyd_pt_planes(rp_max) + size_t(nk) * kPtKeys;
  float* cn_s = reinterpret_cast<float*>(tail + kPtOffNorm);
  float* xch = reinterpret_cast<float*>(tail + kPtOffXch);        // [2][kPtXch]
  float* lists = reinterpret_cast<float*>(tail + kPtOffList);     // [kPtRing][kPtList]
  int* cnts = reinterpret_cast<int*>(tail + kPtOffCnt);           // [kPtRing][kPtRmax]
  int* rinfo = reinterpret_cast<int*>(tail + kPtOffRInfo);        // [kPtRing]: u, tile, r, max ||c||^2, keep
  int* tinfo = reinterpret_cast<int*>(tail + kPtOffTInfo);        // [2]: u, tile, r, max ||c||^2
  volatile uint32_t* abort_s = reinterpret_cast<volatile uint32_t*>(tail + kPtOffAbort);
  uint64_t* bars = reinterpret_cast<uint64_t*>(tail + kPtOffBars);
  uint64_t* full = bars;                                           // [2] MMA commit + producer lanes
  uint64_t* tmem_empty = bars + 2;                                 // [2] column threads
  uint64_t* list_full = bars + 4;                                  // [kPtRing] column half 0
  uint64_t* list_empty = bars + 4 + kPtRing;                       // [kPtRing] certifier threads
  uint64_t* key_full = bars + 4 + 2 * kPtRing;                     // [nk] the key tile's TMA bytes
  uint64_t* key_free = key_full + kPtMaxKeyBufs;                   // [nk] MMA commit: buffer read
  uint32_t* tslot = reinterpret_cast<uint32_t*>(tail + kPtOffSlot);
  const uint32_t planes_s = smem_u32(base), keys_s = planes_s + uint32_t(lloyd_pt_planes(rp_max));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t n_all = int64_t(n_units) * p.ntiles;
  const int64_t g0 = n_all * blockIdx.x / gridDim.x, g1 = n_all * (blockIdx.x + 1) / gridDim.x;

  for (int i = tid; i < kPtRing * kPtRmax; i += kPtThreads) cnts[i] = 0;
  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&full[i], 33);
      mbar_init(&tmem_empty[i], kPtColThreads);
    }
    for (int i = 0; i < kPtRing; ++i) {
      mbar_init(&list_full[i], kPtColThreads / 2);
      mbar_init(&list_empty[i], kPtCertThreads);
    }
    for (int i = 0; i < nk; ++i) {
      mbar_init(&key_full[i], 1);
      mbar_init(&key_free[i], 1);
    }
    *abort_s = 0u;
    fence_mbar_init();
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tslot)),
                 "r"(kPtCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;

  if (warp == kPtLoader) {
    // ---------------- loader ----------------
    // Key tiles by TMA into the ring of nk buffers, as far ahead of the MMAs
    // as the buffers allow (across unit changes too).
    int nl = 0;
    bool ok = true;
    for (PtCursor cl(p, g0, g1); cl.g < g1; cl.next(p), ++nl) {
      const int slot = nl % nk;
      if (nl >= nk) {                                // MMA(nl - nk) has read the buffer
        const bool w = pt_wait(&key_free[slot], uint32_t(((nl / nk) - 1) & 1), abort_s);
        if (__any_sync(0xffffffffu, !w)) {
          ok = false;
          break;
        }
      }
      if (lane == 0) {
        mbar_arrive_expect_tx(&key_full[slot], uint32_t(kPtKeys));
        tma_keys(keys_s + uint32_t(slot * kPtKeys), &tmK,
                 int(int64_t(cl.u) * p.s + int64_t(cl.tile) * kTile), &key_full[slot]);
      }
    }
    if (!ok && lane == 0) pt_raise(abort_s, p.status);
    // the copies in flight land before the CTA exits (the latest phase of
    // each buffer: no older one can alias it)
    const long long t0 = clock64();
    for (int i = nl > nk ? nl - nk : 0; i < nl; ++i)
      while (!mbar_try_wait(&key_full[i % nk], uint32_t((i / nk) & 1)) && clock64() - t0 < kTcWaitCycles) {
      }
  } else if (warp == kPtProducer) {
    // ---------------- MMA issue ----------------
    int nm = 0, cur_u = -1;
    float cmx = 0.f;                                 // max ||c||^2 of the staged unit
    bool ok = true;
    const uint64_t da0 = tc_desc(keys_s), db0 = tc_desc(planes_s);   // descriptors of the bases
    for (PtCursor cm(p, g0, g1); cm.g < g1; cm.next(p), ++nm) {
      const int u = cm.u, tile = cm.tile, r = cm.r;
      if (u != cur_u) {
        // the planes and norms of the old unit are in use until its last
        // tile's MMAs are done and the column warps have read that tile
        if (nm >= 1) {
          bool w = pt_wait(&full[(nm - 1) & 1], uint32_t(((nm - 1) >> 1) & 1), abort_s) &&
                   pt_wait(&tmem_empty[(nm - 1) & 1], uint32_t(((nm - 1) >> 1) & 1), abort_s);
          if (__any_sync(0xffffffffu, !w)) {
            ok = false;
            break;
          }
        }
        const int rpad = (r + 15) & ~15;
        const __nv_bfloat16* planes = p.cplanes + int64_t(u) * 2 * p.rmax * kHeadDim;
        for (int i = lane; i < 2 * rpad * 16; i += 32) {
          const int pl = i / (rpad * 16), rem = i - pl * (rpad * 16), row = rem >> 4, ch = rem & 15;
          const bool in = row < r;
          cp_async16(planes_s + uint32_t(pl * 2) * plane_half + uint32_t(ch >> 3) * plane_half + tc_sw128(row, ch & 7),
                     planes + (int64_t(pl) * p.rmax + (in ? row : 0)) * kHeadDim + 8 * ch, in ? 16u : 0u);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
        const float* cnorm = p.cnorm + int64_t(u) * p.rmax;
        cmx = 0.f;
        for (int i = lane; i < kPtRmax; i += 32) {
          const float c = i < r ? cnorm[i] : FLT_MAX;    // finite: padded keys stay ordered
          cn_s[i] = c;
          if (i < r) cmx = fmaxf(cmx, c);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) cmx = fmaxf(cmx, __shfl_xor_sync(0xffffffffu, cmx, o));
        asm volatile("cp.async.wait_group 0;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        cur_u = u;
      }
      // tile nm: its keys, a free TMEM buffer, then the MMA chain
      const int slot = nm % nk, bb = nm & 1;
      bool w = pt_wait(&key_full[slot], uint32_t((nm / nk) & 1), abort_s) &&
               (nm < 2 || pt_wait(&tmem_empty[bb], uint32_t(((nm - 2) >> 1) & 1), abort_s));
      if (__any_sync(0xffffffffu, !w)) {
        ok = false;
        break;
      }
      __syncwarp();
      if (lane == 0) {
        tinfo[4 * bb + 0] = u;
        tinfo[4 * bb + 1] = tile;
        tinfo[4 * bb + 2] = r;
        tinfo[4 * bb + 3] = __float_as_int(cmx);
        tc_fence_after();
        const uint32_t idesc = pt_idesc((r + 15) & ~15);
        const uint32_t d_tmem = tmem + uint32_t(bb) * kPtBufCols;
        const uint64_t da = desc_plus(da0, uint32_t(slot * kPtKeys));
#pragma unroll
        for (int pl = 0; pl < 2; ++pl)
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t half = uint32_t(k >> 2), kk = uint32_t(k & 3) * 32u;
            pt_mma(d_tmem, desc_plus(da, half * kTcHalf + kk),
                   desc_plus(db0, uint32_t(pl * 2 + half) * plane_half + kk), idesc, pl + k > 0);
          }
        tc_commit(&full[bb]);
        tc_commit(&key_free[slot]);
      }
      __syncwarp();
      pt_arrive(&full[bb]);
    }
    if (!ok && lane == 0) pt_raise(abort_s, p.status);
    // every issued MMA completes before TMEM is freed
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    if (nm >= 1) {
      const int lt = nm - 1;
      const long long t0 = clock64();
      while (!mbar_try_wait(&full[lt & 1], uint32_t((lt >> 1) & 1)) && clock64() - t0 < kTcWaitCycles) {
      }
    }
  } else if (warp < kPtColWarps) {
    // ---------------- column warps ----------------
    const int q = warp & 3, half = warp >> 2, tok = 32 * q + lane;
    int t = 0;
    for (PtCursor cc(p, g0, g1); cc.g < g1; cc.next(p)) {
      const int b = t & 1, slot = t % kPtRing;
      const bool ok = *abort_s == 0u && pt_wait(&full[b], uint32_t((t >> 1) & 1), abort_s);
      if (!ok) pt_raise(abort_s, p.status);
      if (pt_bar_or(1, kPtColThreads, !ok)) break;        // all column threads leave together
      tc_fence_after();
      const int r = tinfo[4 * b + 2], rpad = (r + 15) & ~15;
      const int tu = tinfo[4 * b + 0], ttile = tinfo[4 * b + 1], tcm = tinfo[4 * b + 3];
      // the token's rank and key norm, loaded now and used after the column loop
      const int64_t pos = int64_t(ttile) * kTile + tok;
      int rk = -1;
      float kn2 = 0.f;
      if (half == 0 && pos < p.s) {
        rk = p.rank_pos[int64_t(tu) * p.s + pos];
        kn2 = p.knorm2[int64_t(tu) * p.s + pos];
      }
      // token tok's distances over this half's chunks: lists A (even) and B (odd)
      float a0 = INFINITY, a1 = INFINITY, a2 = INFINITY, e0 = INFINITY, e1 = INFINITY, e2 = INFINITY;
      const uint32_t tb = tmem + (uint32_t(32 * q) << 16) + uint32_t(b) * kPtBufCols;
      for (int k = half; k < (rpad >> 4); k += 2) {
        float v[16];
        tc_ld16(tb + uint32_t(16 * k), v);
        const uint32_t c0 = uint32_t(16 * k) * 0x01010101u + 0x03020100u;   // columns 16k .. 16k + 3
#pragma unroll
        for (int m = 0; m < 4; ++m) {
          const uint32_t cols = c0 + uint32_t(4 * m) * 0x01010101u;
          const int col = 16 * k + 4 * m;
          pt_ins3(a0, a1, a2, pt_key4<0>(fmaf(-2.0f, v[4 * m], cn_s[col]), cols));
          pt_ins3(e0, e1, e2, pt_key4<1>(fmaf(-2.0f, v[4 * m + 1], cn_s[col + 1]), cols));
          pt_ins3(a0, a1, a2, pt_key4<2>(fmaf(-2.0f, v[4 * m + 2], cn_s[col + 2]), cols));
          pt_ins3(e0, e1, e2, pt_key4<3>(fmaf(-2.0f, v[4 * m + 3], cn_s[col + 3]), cols));
        }
      }
      pt_ins3(a0, a1, a2, e0);
      pt_ins3(a0, a1, a2, e1);
      pt_ins3(a0, a1, a2, e2);
      tc_fence_before();
      pt_arrive(&tmem_empty[b]);                          // TMEM buffer b and its tile info are free
      float* xb = xch + b * kPtXch + tok * 3;
      if (half == 1) {
        xb[0] = a0;
        xb[1] = a1;
        xb[2] = a2;
      }
      pt_bar(1, kPtColThreads);
      if (half == 0) {
        const bool ok2 = t < kPtRing ||
                         pt_wait(&list_empty[slot], uint32_t(((t / kPtRing) - 1) & 1), abort_s);
        if (!ok2) {
          pt_raise(abort_s, p.status);                    // the next tile's vote ends the loop
        } else {
          pt_ins3(a0, a1, a2, xb[0]);
          pt_ins3(a0, a1, a2, xb[1]);
          pt_ins3(a0, a1, a2, xb[2]);
          float* ls = lists + slot * kPtList + tok * 5;
          ls[0] = a0;
          ls[1] = a1;
          ls[2] = a2;
          ls[3] = __int_as_float(rk);
          ls[4] = kn2;
          if (tok == 0) {
            rinfo[8 * slot + 0] = tu;
            rinfo[8 * slot + 1] = ttile;
            rinfo[8 * slot + 2] = r;
            rinfo[8 * slot + 3] = tcm;
            // ranked main slots of the unit: evicted tokens rank at or past it
            rinfo[8 * slot + 4] = int(unit_budget(p.budgets, tu, p.budget)) - r - p.recent;
          }
          pt_arrive(&list_full[slot]);
        }
      }
      ++t;
    }
  } else {
    // ---------------- certifier warps ----------------
    const int ct = tid - kPtColThreads;                   // the token of the tile this thread certifies
    int t = 0;
    for (PtCursor cc(p, g0, g1); cc.g < g1; cc.next(p)) {
      const int slot = t % kPtRing;
      bool ok = *abort_s == 0u && pt_wait(&list_full[slot], uint32_t((t / kPtRing) & 1), abort_s);
      if (p.test_fault && blockIdx.x == 0 && t == 0) ok = false;   // a timed-out wait, injected
      if (!ok) pt_raise(abort_s, p.status);
      if (pt_bar_or(2, kPtCertThreads, !ok)) break;
      const int u = rinfo[8 * slot + 0], tile = rinfo[8 * slot + 1], r = rinfo[8 * slot + 2];
      const float cnmax = __int_as_float(rinfo[8 * slot + 3]);
      const int keep = rinfo[8 * slot + 4];
      const float* ls = lists + slot * kPtList + ct * 5;
      const float d0 = ls[0], d1 = ls[1], d2 = ls[2], s2 = ls[4];
      int j0 = pt_key_index(d0);
      const int j1 = pt_key_index(d1), rk = __float_as_int(ls[3]);
      int* cnt = cnts + slot * kPtRmax;
      const int64_t pos = int64_t(tile) * kTile + ct;
      const bool mine = pos < p.s;
      const bool ev = mine && rk >= 0 && rk >= keep;     // in E (in_evicted)
      bool amb = false, fullscan = false;
      if (ev) {
        // the bound of k_lloyd_assign_tc on the computed distances' error
        const float uu = 5.9604645e-8f, gam = 130.0f * uu, gam_tc = 2048.0f * uu;
        const float kn = sqrtf(s2) * (1.0f + gam), cm = sqrtf(cnmax);
        const float ee = 2.0f * (2.0f * gam_tc * cm * kn + 2.0f * gam * cm * cm + 4.0f * uu * kn * cm);
        // + the key packing: |key - d| <= 2^-15 |d|
        const float pk = 0x1p-15f;
        const float err0 = ee + (4.0f * uu + pk) * fabsf(d0);
        fullscan = d2 - d0 <= err0 + ee + (4.0f * uu + pk) * fabsf(d2);
        amb = fullscan || (j1 < r && d1 - d0 <= err0 + ee + (4.0f * uu + pk) * fabsf(d1));
        if (j0 >= r || !(d0 < INFINITY)) {                // only NaN or infinite distances get here
          report_status(p.status, kStatusBadIndex);
          j0 = 0;
          amb = false;
        }
      }
      if (amb) {
        // decided by k_lloyd_resolve in fp64; it also counts the token
        const int i = atomicAdd(p.amb_count, 1);
        p.amb[i] = make_int4(u, int(pos), j0 | (fullscan ? int(0x80000000u) : 0), j1);
      } else if (ev) {
        p.assign[int64_t(u) * p.s + pos] = j0;
        atomicAdd(&cnt[j0], 1);
      } else if (mine) {
        p.assign[int64_t(u) * p.s + pos] = -1;
      }
      pt_bar(2, kPtCertThreads);
      int32_t* h = p.hist + (int64_t(u) * p.ntiles + tile) * p.rmax;
      for (int i = ct; i < r; i += kPtCertThreads) {
        h[i] = cnt[i];
        cnt[i] = 0;
      }
      pt_arrive(&list_empty[slot]);
      ++t;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kPtCols));
  }
}

// The decision of the tokens k_lloyd_assign_pt left ambiguous, a warp per
// token (lane l holds dims 4l..4l+3).  Candidates: the two kept centres, or
// every centre when the third best was within the tensor-core bound.
//
// First their distances are taken directly in fp32, d32_j = sum_i (k_i -
// c32_i)^2 against the fp32 centres: no cancellation, so the error is small
// relative to the distance itself.  With u = 2^-24, |d32_j - D_j| <= b_j =
// 16 u d32_j + 3 u ||c_j|| (sqrt(d32_j) + u ||c_j||) bounds the difference to
// the exact distance D_j to the fp64 centre (12 u for the rounded differences,
// the 4-term chain and the 5 butterfly levels; 2 u ||c|| (2 sqrt(D) + u ||c||)
// for |c32 - c64| <= u ||c||; the rest is slack for using d32 in place of D).
// The fp32 best decides unless another candidate's interval
// [d32_j - b_j, d32_j + b_j] reaches the best's; those few are re-evaluated in
// fp64 as the streaming kernel does, ties to the lower index.  Writes assign
// and adds the token to its tile's member count.
constexpr int kResWarps = 8;

__global__ void __launch_bounds__(kResWarps * 32) k_lloyd_resolve(LloydArgs p) {
  __shared__ float dsm[kResWarps][kPtRmax];       // candidate distances (fp32)
  __shared__ int jsm[kResWarps][kPtRmax];         // centres left for fp64
  const int lane = threadIdx.x & 31, wb = threadIdx.x >> 5;
  float* dl = dsm[wb];
  int* jl = jsm[wb];
  const int n = *p.amb_count;
  const int nw = int((int64_t(gridDim.x) * blockDim.x) >> 5);
  const float uu = 5.9604645e-8f;
  for (int i = int((int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5); i < n; i += nw) {
    const int4 e = p.amb[i];
    const int u = e.x, r = p.r_unit[u];
    const int64_t pos = e.y;
    const bool fs = e.z < 0;
    const int js0 = e.z & 0x7fffffff, js1 = e.w;
    const int nc = fs ? r : 2;
    auto cand = [&](int k) { return fs ? k : (k == 0 ? js0 : js1); };
    const uint2 kw = *reinterpret_cast<const uint2*>(p.K + (int64_t(u) * p.s + pos) * kHeadDim + 4 * lane);
    const float2 k01 = bf16x2_to_float2(kw.x), k23 = bf16x2_to_float2(kw.y);
    const float* c32 = p.centers32 + int64_t(u) * p.rmax * kHeadDim + 4 * lane;
    const float* cnu = p.cnorm + int64_t(u) * p.rmax;
    // fp32 distances, eight centres at a time: a 4-term chain per lane, then
    // a transposed butterfly (9 shuffles) that leaves centre 4 b4 + 2 b3 + b2
    // (b_i: bit i of the lane) summed over all lanes -- five levels of adds,
    // as the bound assumes
    const int b4 = (lane >> 4) & 1, b3 = (lane >> 3) & 1, b2 = (lane >> 2) & 1;
    for (int k0 = 0; k0 < nc; k0 += 8) {
      float a[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int k = k0 + q < nc ? k0 + q : k0;
        const float4 c = *reinterpret_cast<const float4*>(c32 + int64_t(cand(k)) * kHeadDim);
        const float x0 = k01.x - c.x, x1 = k01.y - c.y, x2 = k23.x - c.z, x3 = k23.y - c.w;
        a[q] = fmaf(x3, x3, fmaf(x2, x2, fmaf(x1, x1, x0 * x0)));
      }
      float bq[4], cq[2];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float send = b4 ? a[i] : a[i + 4];
        bq[i] = (b4 ? a[i + 4] : a[i]) + __shfl_xor_sync(0xffffffffu, send, 16);
      }
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const float send = b3 ? bq[i] : bq[i + 2];
        cq[i] = (b3 ? bq[i + 2] : bq[i]) + __shfl_xor_sync(0xffffffffu, send, 8);
      }
      float dq = (b2 ? cq[1] : cq[0]) + __shfl_xor_sync(0xffffffffu, b2 ? cq[0] : cq[1], 4);
      dq += __shfl_xor_sync(0xffffffffu, dq, 2);
      dq += __shfl_xor_sync(0xffffffffu, dq, 1);
      const int v = 4 * b4 + 2 * b3 + b2;
      if ((lane & 3) == 0 && k0 + v < nc) dl[k0 + v] = dq;
    }
    __syncwarp();
    // the fp32 best (distance, index)
    float bd = INFINITY;
    int bj = INT_MAX;
    for (int k = lane; k < nc; k += 32) {
      const float d = dl[k];
      const int j = cand(k);
      if (d < bd || (d == bd && j < bj)) {
        bd = d;
        bj = j;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float od = __shfl_xor_sync(0xffffffffu, bd, o);
      const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
      if (od < bd || (od == bd && oj < bj)) {
        bd = od;
        bj = oj;
      }
    }
    auto bound = [&](float d, int j) {
      const float cn = sqrtf(cnu[j]) * 1.001f;
      return 16.0f * uu * d + 3.0f * uu * cn * (sqrtf(d) + uu * cn);
    };
    int res = bj;
    if (bj < r) {
      // centres whose interval reaches the best's: fp64 decides among them
      const float hi = bd + bound(bd, bj);
      int na = 0;
      for (int k0 = 0; k0 < nc; k0 += 32) {
        const int k = k0 + lane;
        bool m = false;
        if (k < nc) {
          const float d = dl[k];
          const int j = cand(k);
          m = j != bj && !(d - bound(d, j) > hi);
        }
        const unsigned bal = __ballot_sync(0xffffffffu, m);
        if (m) jl[na + __popc(bal & ((1u << lane) - 1u))] = cand(k);
        na += __popc(bal);
      }
      __syncwarp();
      if (na > 0) {
        const double kx[4] = {k01.x, k01.y, k23.x, k23.y};
        const double* c64 = p.centers64 + int64_t(u) * p.rmax * kHeadDim + 4 * lane;
        double bd64 = INFINITY;
        int bj64 = INT_MAX;
        // the best first, then the others, four at a time
        for (int k0 = -1; k0 < na; k0 += 4) {
          int jq[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) jq[q] = k0 + q < 0 ? bj : (k0 + q < na ? jl[k0 + q] : -1);
          double a[4];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const double4_32a c =
                *reinterpret_cast<const double4_32a*>(c64 + int64_t(jq[q] < 0 ? 0 : jq[q]) * kHeadDim);
            double tt = (kx[0] - c.x) * (kx[0] - c.x);
            tt = fma(kx[1] - c.y, kx[1] - c.y, tt);
            tt = fma(kx[2] - c.z, kx[2] - c.z, tt);
            a[q] = fma(kx[3] - c.w, kx[3] - c.w, tt);
          }
#pragma unroll
          for (int o = 16; o > 0; o >>= 1)
#pragma unroll
            for (int q = 0; q < 4; ++q) a[q] += __shfl_xor_sync(0xffffffffu, a[q], o);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const double dd = __shfl_sync(0xffffffffu, a[q], 0);
            if (jq[q] >= 0 && (dd < bd64 || (dd == bd64 && jq[q] < bj64))) {
              bd64 = dd;
              bj64 = jq[q];
            }
          }
        }
        res = bj64;
      }
    }
    if (lane == 0) {
      if (res >= r) {                                   // only NaN distances get here
        report_status(p.status, kStatusBadIndex);
        res = 0;
      }
      p.assign[int64_t(u) * p.s + pos] = res;
      atomicAdd(&p.hist[(int64_t(u) * p.ntiles + pos / kTile) * p.rmax + res], 1);
    }
    __syncwarp();                                       // dl / jl are reused by the next token
  }
}

}  // namespace build
}  // namespace reskv
