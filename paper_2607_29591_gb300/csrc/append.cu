// Decode-time growth of the cache (Sec. 3.1: each decode step appends the new
// token's key and value): one exact K row and V row per (batch, KV head) unit
// goes after the unit's main and residual slots and counts as a main-cache
// token from then on.
//
// The A slots after the residual entries hold the unit's appended tokens as a
// ring: token t (counted from the first append) sits at ring index t mod A.
// While fewer than A tokens were appended the new one takes the next free
// slot.  Once the ring is full the oldest token (index n_total mod A) leaves
// the exact window before the new token takes its slot; the append policy
// decides what becomes of it:
//   RESKV_APPEND_RING_DROP: it leaves the cache;
//   RESKV_APPEND_RING_FOLD: it becomes a member of its nearest residual entry
//     (Eq. residual_partition's nearest-centre rule on the stored keys, ties
//     to the lower entry), whose stored means and count are updated as a
//     running mean (Eq. summary): k_bar <- (c k_bar + k) / (c + 1) in fp64,
//     rounded to bf16, likewise v_bar, c <- c + 1, log-count beta log(c + 1).
//     A unit without residual entries drops the token.  This is the residual
//     refresh during generation that the paper leaves to future work (App. E).
//
// The nearest entry is decided exactly.  With every bf16 value written as
// M 2^e (integer M < 2^8), ||k - k_bar_j||^2 - ||k||^2 = sum_i (k_bar_ji^2 -
// 2 k_i k_bar_ji) is a signed sum of terms m 2^t with integer m < 2^17.  One
// warp per unit, entries spread over the lanes: within the unit's exponent
// window the terms are integers of a common scale that a signed 128-bit sum
// holds; a unit whose values span more than that window is decided by one
// lane with a 576-bit accumulator of 32-bit digits.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>

#include "device_utils.cuh"
#include "internal.h"

namespace reskv {
namespace {

using i128 = __int128;

struct AppendArgs {
  const __nv_bfloat16* K_new;   // [n, d]
  const __nv_bfloat16* V_new;
  __nv_bfloat16* kslots;
  __nv_bfloat16* vslots;
  float* logc;
  int32_t* slot_pos;
  int32_t* counts;
  const int32_t* n_main;
  const int32_t* n_res;
  int32_t* n_app;               // appended tokens in the cache, min(n_total, A)
  int32_t* n_total;             // tokens appended since construction
  const int32_t* offsets;       // [U+1] unit starts, or NULL (uniform stride)
  int64_t unit0;
  int32_t stride;
  int32_t capacity;             // A
  int32_t policy;               // RESKV_APPEND_*
  float beta;
  int64_t seq_len;
  uint32_t* status;
};

// A bf16 value as sign, integer M (< 2^8) and exponent e: value = +-M 2^e.
struct Bf {
  uint32_t m;
  int e;
  uint32_t neg;
};

__device__ __forceinline__ Bf bf_split(uint16_t b) {
  const uint32_t ef = (b >> 7) & 0xffu, mf = b & 0x7fu;
  return Bf{ef ? 128u + mf : mf, int(ef ? ef : 1u) - 134, uint32_t(b >> 15)};
}

__device__ __forceinline__ bool bf_finite(uint16_t b) { return ((b >> 7) & 0xffu) != 0xffu; }

// ---- the 576-bit accumulator of the wide case (one thread) ----------------
// Digit q holds bits 32q..32q+31 of the sum scaled by 2^266 (t >= -266).
constexpr int kDigits = 18;

__device__ void wide_add(int64_t* dig, uint32_t m, int t, bool negative) {
  const int q = t + 266;
  const uint64_t v = uint64_t(m) << (q & 31);
  const int64_t lo = int64_t(v & 0xffffffffu), hi = int64_t(v >> 32);
  dig[q >> 5] += negative ? -lo : lo;
  dig[(q >> 5) + 1] += negative ? -hi : hi;
}

// Carries into the upper digits; afterwards every digit but the top one is in
// [0, 2^32) and the top digit carries the sign.
__device__ void wide_normalise(int64_t* dig) {
  for (int q = 0; q < kDigits - 1; ++q) {
    const int64_t carry = dig[q] >> 32;          // arithmetic shift: floor division
    dig[q] -= carry * (int64_t(1) << 32);
    dig[q + 1] += carry;
  }
}

// -1, 0, 1 as a < b, a == b, a > b (both normalised).
__device__ int wide_cmp(const int64_t* a, const int64_t* b) {
  for (int q = kDigits - 1; q >= 0; --q)
    if (a[q] != b[q]) return a[q] < b[q] ? -1 : 1;
  return 0;
}

// The entry of [0, nr) nearest to key k (rows kb), exactly, by one thread.
__device__ int nearest_wide(const uint16_t* k, const uint16_t* kb, int nr) {
  int64_t best[kDigits], cur[kDigits];
  int bj = 0;
  for (int j = 0; j < nr; ++j) {
    for (int q = 0; q < kDigits; ++q) cur[q] = 0;
    for (int i = 0; i < kHeadDim; ++i) {
      const Bf b = bf_split(kb[size_t(j) * kHeadDim + i]);
      if (!b.m) continue;
      wide_add(cur, b.m * b.m, 2 * b.e, false);
      const Bf a = bf_split(k[i]);
      if (a.m) wide_add(cur, 2u * a.m * b.m, a.e + b.e, a.neg == b.neg);
    }
    wide_normalise(cur);
    if (j == 0 || wide_cmp(cur, best) < 0) {
      bj = j;
      for (int q = 0; q < kDigits; ++q) best[q] = cur[q];
    }
  }
  return bj;
}

// One warp per unit of the call.
__global__ void __launch_bounds__(32) k_append(AppendArgs a) {
  const int64_t i = blockIdx.x, u = a.unit0 + i;
  const int lane = threadIdx.x;
  const int total = a.n_total[u];
  const int64_t ubase = a.offsets ? int64_t(a.offsets[u]) : u * a.stride;
  const int nm = a.n_main[u], nr = a.n_res[u];
  const int64_t ring0 = ubase + nm + nr;            // first appended slot
  const bool full = total >= a.capacity;
  if (full && (a.policy == RESKV_APPEND_FAIL || a.capacity == 0)) {   // the host checks first
    if (lane == 0) report_status(a.status, kStatusBadIndex);
    return;
  }
  const int64_t row = ring0 + (a.capacity > 0 ? total % a.capacity : 0);
  if (full && a.policy == RESKV_APPEND_RING_FOLD && nr > 0) {
    // the oldest appended token, k and v of slot `row`, joins its nearest entry
    const uint16_t* k = reinterpret_cast<const uint16_t*>(a.kslots + row * kHeadDim);
    const uint16_t* kb = reinterpret_cast<const uint16_t*>(a.kslots + (ubase + nm) * kHeadDim);
    // the unit's exponent window: the largest exponent of any value involved
    bool finite = true;
    int emax = INT_MIN;
    for (int x = lane; x < (nr + 1) * kHeadDim; x += 32) {
      const uint16_t bits = x < kHeadDim ? k[x] : kb[x - kHeadDim];
      finite &= bf_finite(bits);
      const Bf b = bf_split(bits);
      if (b.m) emax = max(emax, b.e);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) emax = max(emax, __shfl_xor_sync(0xffffffffu, emax, o));
    finite = __all_sync(0xffffffffu, finite);
    int best = 0;
    if (!finite) {
      // distances undefined: the token is dropped instead
      if (lane == 0) report_status(a.status, kStatusBadIndex);
      best = -1;
    } else if (emax != INT_MIN) {
      // terms m 2^t (m < 2^17) as integers of scale 2^base; every |term| <
      // 2^(2 emax + 17) and 2 * 128 terms sum below 2^(2 emax + 25) < 2^(base + 127)
      const int base = 2 * emax - 102;
      bool wide = false;
      i128 dbest = 0;
      int jbest = INT_MAX;
      for (int j = lane; j < nr; j += 32) {
        i128 acc = 0;
        for (int d = 0; d < kHeadDim; ++d) {
          const Bf b = bf_split(kb[size_t(j) * kHeadDim + d]);
          if (!b.m) continue;
          const int t2 = 2 * b.e - base;
          if (t2 < 0) wide = true;
          else acc += i128(b.m * b.m) << t2;
          const Bf c = bf_split(k[d]);
          if (!c.m) continue;
          const int t1 = c.e + b.e - base;
          if (t1 < 0) {
            wide = true;
            continue;
          }
          const i128 pr = i128(2u * c.m * b.m) << t1;
          acc += c.neg == b.neg ? -pr : pr;
        }
        if (jbest == INT_MAX || acc < dbest) {
          dbest = acc;
          jbest = j;
        }
      }
      if (__any_sync(0xffffffffu, wide)) {
        best = lane == 0 ? nearest_wide(k, kb, nr) : 0;
        best = __shfl_sync(0xffffffffu, best, 0);
      } else {
        // warp argmin, ties to the lower entry (lanes without an entry hold INT_MAX)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          const uint64_t hi = __shfl_xor_sync(0xffffffffu, uint64_t((unsigned __int128)(dbest) >> 64), o);
          const uint64_t lo = __shfl_xor_sync(0xffffffffu, uint64_t(dbest), o);
          const int jo = __shfl_xor_sync(0xffffffffu, jbest, o);
          const i128 d_o = i128((unsigned __int128)(hi) << 64 | lo);
          if (jo != INT_MAX && (jbest == INT_MAX || d_o < dbest || (d_o == dbest && jo < jbest))) {
            dbest = d_o;
            jbest = jo;
          }
        }
        best = jbest;
      }
    }
    if (best >= 0) {
      // running mean of the stored summary and the token, 4 dims per lane
      const int64_t erow = ubase + nm + best;
      const int c = a.counts[erow];
      const double cd = double(c);
      __syncwarp();                                  // every lane has read the count
      for (int d = lane; d < kHeadDim; d += 32) {
        const double ko = double(__bfloat162float(a.kslots[row * kHeadDim + d]));
        const double vo = double(__bfloat162float(a.vslots[row * kHeadDim + d]));
        const double ke = double(__bfloat162float(a.kslots[erow * kHeadDim + d]));
        const double ve = double(__bfloat162float(a.vslots[erow * kHeadDim + d]));
        a.kslots[erow * kHeadDim + d] = __double2bfloat16(__ddiv_rn(__dadd_rn(__dmul_rn(cd, ke), ko), cd + 1.0));
        a.vslots[erow * kHeadDim + d] = __double2bfloat16(__ddiv_rn(__dadd_rn(__dmul_rn(cd, ve), vo), cd + 1.0));
      }
      if (lane == 0) {
        a.counts[erow] = c + 1;
        a.logc[erow] = a.beta * logf(float(c + 1));
      }
    }
    __syncwarp();
  }
  // the new token into slot `row`
  if (lane < 16) {
    reinterpret_cast<uint4*>(a.kslots + row * kHeadDim)[lane] =
        reinterpret_cast<const uint4*>(a.K_new + i * kHeadDim)[lane];
  } else {
    reinterpret_cast<uint4*>(a.vslots + row * kHeadDim)[lane - 16] =
        reinterpret_cast<const uint4*>(a.V_new + i * kHeadDim)[lane - 16];
  }
  if (lane == 0) {
    a.slot_pos[row] = int32_t(a.seq_len + total);    // position of the token in the sequence
    a.counts[row] = 0;
    a.logc[row] = 0.f;
    a.n_total[u] = total + 1;
    a.n_app[u] = total + 1 < a.capacity ? total + 1 : a.capacity;
  }
  // The rows are visible device-wide before this grid completes: decode
  // kernels launched after it read the cache before their own grid
  // dependency wait.
  __threadfence();
}

}  // namespace

cudaError_t launch_append(reskv_cache* c, int64_t unit0, int64_t n, const __nv_bfloat16* K_new,
                          const __nv_bfloat16* V_new, cudaStream_t stream) {
  AppendArgs a{K_new, V_new, c->kslots, c->vslots, c->logc, c->slot_pos, c->counts,
               c->n_main, c->n_res, c->n_app, c->n_total, c->ragged ? c->offsets : nullptr,
               unit0, c->stride, c->append_capacity, c->cfg.append_policy, c->cfg.beta,
               c->cfg.seq_len, c->status};
  k_append<<<unsigned(n), 32, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace reskv
