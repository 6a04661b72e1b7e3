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
// object), so the address is looked up with cudaGetSymbolAddress once per
// device, with that device current, and handed to the kernel.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <mutex>
#include <string>

#include "internal.h"
#include "reskv.h"

namespace reskv {
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;   // 16 MiB
constexpr int kMaxDevices = 64;

// Shared by every call of reskv_decode_attn_noalloc in the process; keeps the
// contents of the last call.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_setup_mutex;
void* g_scratch_addr[kMaxDevices] = {};
int g_num_sms[kMaxDevices] = {};

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

reskv_status fail(reskv_status st, const std::string& msg) {
  set_error(msg);
  return st;
}

// Device address of the scratch array and the SM count of device `dev`
// (current), looked up on the first call on that device.
reskv_status setup_device(int dev, void** addr, int* num_sms) {
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    cudaError_t err = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (err != cudaSuccess || !p)
      return fail(RESKV_ERR_CUDA, std::string("cudaGetSymbolAddress of the static scratch: ") +
                                      cudaGetErrorString(err));
    int sms = 0;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess || sms < 1)
      return fail(RESKV_ERR_CUDA, std::string("reading the SM count: ") + cudaGetErrorString(err));
    g_num_sms[dev] = sms;
    g_scratch_addr[dev] = p;
  }
  *addr = g_scratch_addr[dev];
  *num_sms = g_num_sms[dev];
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
  if (dev < 0 || dev >= kMaxDevices) return fail(RESKV_ERR_UNSUPPORTED, "device ordinal >= 64");

  reskv_status st = RESKV_OK;
  void* scratch = nullptr;
  int num_sms = 0;
  st = setup_device(dev, &scratch, &num_sms);
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

  // scratch layout: [tickets: n_units int32][status word][partial records]
  const size_t ticket_bytes = align256(size_t(c->n_units) * 4);
  const size_t status_bytes = 256;
  const size_t part_bytes = (mma ? decode_mma_partials_floats(c->n_units, int(W), c->group)
                                 : decode_partials_floats(c->n_units, int(W), c->group)) * 4;
  const size_t need = ticket_bytes + status_bytes + part_bytes;
  if (need > kNoAllocScratchBytes)
    return fail(RESKV_ERR_UNSUPPORTED,
                "this call needs " + std::to_string(need) + " bytes of scratch but the static "
                "buffer holds " + std::to_string(kNoAllocScratchBytes) +
                " (16 MiB); decode fewer units per call");

  unsigned char* base = static_cast<unsigned char*>(scratch);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // tickets and the status word must start at zero; the rest is overwritten
  err = cudaMemsetAsync(base, 0, ticket_bytes + status_bytes, s);
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
  p.status = reinterpret_cast<uint32_t*>(base + ticket_bytes);
  p.partials = reinterpret_cast<float*>(base + ticket_bytes + status_bytes);
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
  return RESKV_OK;
}
