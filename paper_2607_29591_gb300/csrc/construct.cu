// Construction (Alg. 1) -- kernels follow.
#include <cuda_runtime.h>

#include "internal.h"

namespace reskv {

reskv_status build_all_layers(reskv_cache** out, const reskv_config& cfg,
                              const int32_t* override_host, const void* const* K,
                              const void* const* V, const void* const* Qobs,
                              cudaStream_t stream) {
  (void)out; (void)cfg; (void)override_host; (void)K; (void)V; (void)Qobs; (void)stream;
  set_error("construction not built yet");
  return RESKV_ERR_UNSUPPORTED;
}

}  // namespace reskv
