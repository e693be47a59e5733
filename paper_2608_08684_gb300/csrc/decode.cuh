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
  int *ctrl;        // counters of the step (kCtrl* below)
  int32_t *status;
  int epoch;        // nonzero tag of this call: the init flag's value once the
                    // counters are zeroed
  long long wait_cycles;  // bound of the in-kernel waits
  int item_rows;          // cache rows per work item
  long long ws_items;     // work items the partials (ws_o, ws_ml) have room for
  int n_ctrl;             // words of the control block
  const void *kc[RIPPLE_MAX_LAYERS];
  const void *vc[RIPPLE_MAX_LAYERS];
  int cap[RIPPLE_MAX_LAYERS];
  int order[RIPPLE_MAX_LAYERS];  // layers by decreasing capacity
};

// Cache rows per work item: kMaxItemRows, or for steps with fewer such items
// than SMs (a single layer's step, short caches) smaller items, down to
// kMinItemRows, as long as they fit in one wave.
constexpr int kMaxItemRows = 4096;
constexpr int kMinItemRows = 256;

// Control block of a step in the workspace (int32 words). The init flag has a
// 128-byte line to itself; CTA 0 zeroes the counters at the start of every
// call and then sets the flag to the call's epoch, and the other CTAs use no
// counter before they have seen it. The last CTA to leave sets the flag back
// to 0, so that a replay of the same launch (same epoch) waits for CTA 0
// again.
constexpr int kCtrlFlag = 0;    // init flag
constexpr int kCtrlItem = 32;   // work-item counter
constexpr int kCtrlExit = 33;   // CTAs that have left
constexpr int kCtrlGroup = 34;  // + group: items of the group finished

}  // namespace ripple
