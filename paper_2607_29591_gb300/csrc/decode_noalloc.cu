// Decode entry point that allocates no device memory.
//
// Some callers cannot allocate GPU memory themselves at decode time: code
// embedded in a host application whose memory manager owns every device
// allocation (inference servers and frameworks that hand out memory only
// from their own pool), or latency-critical paths that must not pay for
// cudaMalloc, which can block and synchronise the device.  Such callers keep
// the compressed cache in memory they already own and pass it here as plain
// device pointers; the few kilobytes to megabytes of per-call scratch that the
// split decode needs (partial results of units cut between warps, their
// arrival tickets, a status word) come from one fixed array compiled into this
// library instead of from an allocation.
//
// The array is file-scope device memory: every GPU on which the library's
// code is loaded holds its 16 MiB until the process exits.  Host code cannot
// use the array's name as a device address (on the host it names a stand-in
// object), so every call looks the address up with cudaGetSymbolAddress, with
// the caller's device current, and hands it to the kernel.  The lookup
// allocates nothing; looking it up per call (rather than caching it) keeps it
// right after a cudaDeviceReset, which reloads the module at a new address.
//
// The kernels' status word (a bounded wait that gave up, an index out of
// range) is a separate device word that calls only OR into; it is read and
// cleared by reskv_noalloc_check_status, so a fault of any call since the
// last check is reported, not overwritten by the next call.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <string>

#include "internal.h"
#include "reskv.h"

namespace reskv {
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;   // 16 MiB

// Shared by every call of reskv_decode_attn_noalloc in the process; keeps the
// contents of the last call.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Kernel status of every call since the last reskv_noalloc_check_status on
// this device (codes ORed together).
static __device__ uint32_t g_noalloc_status;

// The kernel the last successful call on this thread launched
// (RESKV_DECODE_MMA or RESKV_DECODE_FMA; 0 before the first call).
thread_local int32_t g_last_kernel = 0;

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

reskv_status fail(reskv_status st, const std::string& msg) {
  set_error(msg);
  return st;
}

// Device addresses of the scratch array and the status word and the SM count
// of the current device `dev`.
reskv_status setup_device(int dev, void** addr, uint32_t** status, int* num_sms) {
  void* p = nullptr;
  cudaError_t err = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (err != cudaSuccess || !p)
    return fail(RESKV_ERR_CUDA, std::string("cudaGetSymbolAddress of the static scratch: ") +
                                    cudaGetErrorString(err));
  void* w = nullptr;
  err = cudaGetSymbolAddress(&w, g_noalloc_status);
  if (err != cudaSuccess || !w)
    return fail(RESKV_ERR_CUDA, std::string("cudaGetSymbolAddress of the status word: ") +
                                    cudaGetErrorString(err));
  int sms = 0;
  err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (err != cudaSuccess || sms < 1)
    return fail(RESKV_ERR_CUDA, std::string("reading the SM count: ") + cudaGetErrorString(err));
  *addr = p;
  *status = static_cast<uint32_t*>(w);
  *num_sms = sms;
  return RESKV_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace reskv

using namespace reskv;

extern "C" reskv_status reskv_decode_attn_noalloc(const reskv_device_cache* c, const void* Q,
                                                  void* O, void* stream) {
  if (!c || !Q || !O || !c->kslots || !c->vslots || !c->logc || !c->n_main || !c->n_res)
    return fail(RESKV_ERR_INVALID_ARG, "NULL argument");
  if (c->n_units < 1 || c->budget < 1 || c->n_kv_heads < 1 || c->n_units % c->n_kv_heads != 0)
    return fail(RESKV_ERR_INVALID_ARG,
                "need n_units >= 1, budget >= 1 and n_units a multiple of n_kv_heads");
  if (c->group != 1 && c->group != 2 && c->group != 4)
    return fail(RESKV_ERR_UNSUPPORTED, "group must be 1, 2 or 4");
  if (c->gate_mode != RESKV_GATE_DYNAMIC && c->gate_mode != RESKV_GATE_FIXED)
    return fail(RESKV_ERR_INVALID_ARG, "unknown gate_mode");
  if (!std::isfinite(c->tau) || !std::isfinite(c->alpha) || !(c->g_min >= 0.f) ||
      !(c->g_min <= 1.f) || !(c->g_fixed >= 0.f) || !(c->g_fixed <= 1.f))
    return fail(RESKV_ERR_INVALID_ARG, "gate parameters out of range (g_min, g_fixed in [0,1])");
  if (!aligned16(c->kslots) || !aligned16(c->vslots) || !aligned16(Q) || !aligned16(O))
    return fail(RESKV_ERR_INVALID_ARG, "kslots, vslots, Q and O must be 16-byte aligned");
  if (c->n_units >= (int64_t(1) << 31) || double(c->n_units) * c->budget >= double(int64_t(1) << 40))
    return fail(RESKV_ERR_INVALID_ARG, "cache too large");

  int dev = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err != cudaSuccess) return fail(RESKV_ERR_CUDA, cudaGetErrorString(err));

  reskv_status st = RESKV_OK;
  void* scratch = nullptr;
  uint32_t* status = nullptr;
  int num_sms = 0;
  st = setup_device(dev, &scratch, &status, &num_sms);
  if (st != RESKV_OK) return st;
  const int64_t total = c->n_units * int64_t(c->budget);
  // The tensor-core stream-K kernel of reskv_decode_attn when its 16-slot
  // copies stay inside the caller's arrays (budget a multiple of 16, so the
  // cache ends on a chunk boundary; log-counts 16-byte aligned for their
  // bulk copies) and slot indices fit in 32 bits; else the CUDA-core kernel,
  // which reads slot by slot.
  const bool mma = c->budget % kDecodeChunk == 0 && aligned16(c->logc) && total + 16 < (int64_t(1) << 31);
  CUtensorMap tk, tv;
  int kv_rank = 2;
  MmaPlan mp;
  int64_t W = 0;
  if (mma) {
    kv_rank = 3;                        // one copy per chunk, else two
    if (!encode_rows(&tk, c->kslots, uint64_t(total), 3) ||
        !encode_rows(&tv, c->vslots, uint64_t(total), 3))
      kv_rank = 2;
    if (kv_rank == 2 && (!encode_rows(&tk, c->kslots, uint64_t(total), 2) ||
                         !encode_rows(&tv, c->vslots, uint64_t(total), 2)))
      return fail(RESKV_ERR_CUDA, "cuTensorMapEncodeTiled refused the cache arrays");
    mp = plan_mma_shape(num_sms, int64_t(num_sms) * kDecodeWarpsPerCta, 0, c->budget, false,
                        c->n_units, total);
    W = mp.W;
  } else {
    W = total / 32;
    if (W > int64_t(num_sms) * kDecodeWarpsPerCta) W = int64_t(num_sms) * kDecodeWarpsPerCta;
    if (W < 1) W = 1;
  }

  // scratch layout: [tickets: n_units int32][partial records]
  const size_t ticket_bytes = align256(size_t(c->n_units) * 4);
  const size_t part_bytes = (mma ? decode_mma_partials_floats(c->n_units, int(W), c->group)
                                 : decode_partials_floats(c->n_units, int(W), c->group)) * 4;
  const size_t need = ticket_bytes + part_bytes;
  if (need > kNoAllocScratchBytes)
    return fail(RESKV_ERR_UNSUPPORTED,
                "this call needs " + std::to_string(need) + " bytes of scratch but the static "
                "buffer holds " + std::to_string(kNoAllocScratchBytes) +
                " (16 MiB); decode fewer units per call");

  unsigned char* base = static_cast<unsigned char*>(scratch);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the tickets must start at zero; the partial records are overwritten
  err = cudaMemsetAsync(base, 0, ticket_bytes, s);
  if (err != cudaSuccess) return fail(RESKV_ERR_CUDA, cudaGetErrorString(err));

  DecodeParams p{};
  p.kslots = static_cast<const __nv_bfloat16*>(c->kslots);
  p.vslots = static_cast<const __nv_bfloat16*>(c->vslots);
  p.logc = c->logc;
  p.n_main = c->n_main;
  p.n_res = c->n_res;
  p.Q = static_cast<const __nv_bfloat16*>(Q);
  p.O = static_cast<float*>(O);
  p.tickets = reinterpret_cast<int32_t*>(base);
  p.status = status;
  p.partials = reinterpret_cast<float*>(base + ticket_bytes);
  p.test_fault = take_test_wait_fault() ? 1 : 0;
  p.unit0 = 0;
  p.n_units = int32_t(c->n_units);
  p.stride = c->budget;                 // no appended rows: the stride is the budget
  p.tail_unused = 0;
  p.n_app = nullptr;
  p.offsets = nullptr;
  p.kv_rank = kv_rank;
  p.n_kv_heads = c->n_kv_heads;
  p.total_slots = total;
  p.n_warps = int32_t(W);
  p.gate_mode = c->gate_mode;
  p.softmax_mode = RESKV_SOFTMAX_SHARED;
  p.tau = c->tau;
  p.alpha = c->alpha;
  p.g_min = c->g_min;
  p.g_fixed = c->g_fixed;
  if (mma) {
    p.units_per_warp = mp.k;
    p.n_stages = mp.stages;
    err = launch_decode_mma(p, tk, tv, c->group, int((W + mp.wpc - 1) / mp.wpc), mp.wpc, s);
  } else {
    err = launch_decode(p, c->group, int((W + kDecodeWarpsPerCta - 1) / kDecodeWarpsPerCta), s);
  }
  if (err != cudaSuccess) return fail(RESKV_ERR_CUDA, std::string("decode launch: ") +
                                                          cudaGetErrorString(err));
  g_last_kernel = mma ? RESKV_DECODE_MMA : RESKV_DECODE_FMA;
  return RESKV_OK;
}

extern "C" reskv_status reskv_noalloc_check_status(void* stream, int32_t* last_kernel) {
  if (last_kernel) *last_kernel = g_last_kernel;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  uint32_t word = 0;
  cudaError_t err = cudaStreamSynchronize(s);
  if (err == cudaSuccess) err = cudaMemcpyFromSymbolAsync(&word, g_noalloc_status, 4, 0,
                                                          cudaMemcpyDeviceToHost, s);
  if (err == cudaSuccess) err = cudaStreamSynchronize(s);
  if (err != cudaSuccess)
    return fail(RESKV_ERR_CUDA, std::string("reading the status word: ") + cudaGetErrorString(err));
  if (word == 0) return RESKV_OK;
  const uint32_t zero = 0;
  err = cudaMemcpyToSymbolAsync(g_noalloc_status, &zero, 4, 0, cudaMemcpyHostToDevice, s);
  if (err == cudaSuccess) err = cudaStreamSynchronize(s);
  if (err != cudaSuccess)
    return fail(RESKV_ERR_CUDA, std::string("clearing the status word: ") + cudaGetErrorString(err));
  return fail(RESKV_ERR_DEVICE_STATUS, "no-allocation decode status word " + std::to_string(word) +
                                           " (1 = bounded wait timed out, 2 = index out of range)");
}
