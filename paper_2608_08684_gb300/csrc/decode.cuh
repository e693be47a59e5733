// Parameters of one decode step, shared by the decode kernel and its
// host-side set-up.
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

constexpr int kItemRows = 4096;  // cache rows per work item

}  // namespace ripple
