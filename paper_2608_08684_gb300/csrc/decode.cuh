// Parameters of one decode step, shared by the decode kernels (SIMT and
// tensor-core) and their host-side set-up.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "ripple.h"

namespace ripple {

struct DecParams {
  int L, B, Hq, Hkv, G;
  float scale2;
  const void *q, *k_new, *v_new;
  int32_t *lens;
  float *out;
  float *ws_o;      // [items][G][D] unnormalised partial outputs
  float2 *ws_ml;    // [items][G] (max, sum) of each partial
  int *ctrl;        // [0] item counter, [1] exit counter, [2 + group] items done
  int32_t *status;
  const void *kc[RIPPLE_MAX_LAYERS];
  const void *vc[RIPPLE_MAX_LAYERS];
  int cap[RIPPLE_MAX_LAYERS];
  int order[RIPPLE_MAX_LAYERS];  // layers by decreasing capacity
};

// Tensor-core decode (bf16, d = 128, up to kTcMaxLayers layers per call).
constexpr int kTcMaxLayers = 80;
constexpr int kTcItemRows = 4096;  // cache rows per work item (32 tiles of 128)
bool decode_tc_supported(const ripple_decode_desc *d);
// Clears the counter block itself unless the previous tensor-core call on
// this device left this block at zero.
cudaError_t launch_decode_tc(const DecParams &p, size_t ctrl_bytes, cudaStream_t st);
// The counter block at `ctrl` is no longer known to be zero (another kernel
// used it).
void decode_tc_forget_ctrl(const void *ctrl);

}  // namespace ripple
