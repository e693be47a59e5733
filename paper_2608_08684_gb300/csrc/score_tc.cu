// Observation-window scoring on the tcgen05 tensor cores (bf16, d = 128):
// not built yet; every shape uses the fp32 SIMT path.
#include "common.cuh"
#include "kernels.cuh"

namespace ripple {

bool score_tc_supported(const LayerGeom &) { return false; }

cudaError_t launch_score_tc(const LayerGeom &, const void *, const void *, const CompressWs &,
                            float *, int32_t *, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace ripple
