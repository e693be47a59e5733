// Host-side launchers shared between the translation units of libripple.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "ripple.h"

namespace ripple {

// Host-side count of kernel launches (ripple_kernel_launches).
void count_launches(int n);

// Bound, in SM clock cycles, that kernels launched now give their in-kernel
// waits (ripple_set_wait_limit_cycles; kDefaultWaitCycles unless changed).
long long wait_limit_cycles();

// Geometry of one layer's compression, derived from ripple_layer_desc.
struct LayerGeom {
  int B, Hq, Hkv, G, D, T, W, P, R;  // R = G * W window rows per unit
  int units;                          // B * Hkv
  int dtype;
  int pool_kernel, pool_type;
  float scale2;                       // logit scale * log2(e)
};

// Layers one multi-layer compression call covers.
constexpr int kCompressMaxLayers = RIPPLE_COMPRESS_MAX_LAYERS;

constexpr int kScoreChunk = 128;      // keys per scoring work item
constexpr int kSelectThreads = 1024;  // threads of the selection CTA
constexpr int kSelectSmemKeys = 48 * 1024;  // prefix lengths up to this keep keys in smem

// Workspace carve-up of one compression call.
struct CompressWs {
  float2 *row_partial;  // [units][n_chunks][2][R] (max, sum) in the log2 domain
  float *row_lognorm;   // [units][R] max + log2(sum), log2 domain
  float *votes;         // [units][P] unpooled votes (when scores_out is NULL)
  uint32_t *keys;       // [units][P] pooled-score sort keys (long prefixes only)
  int32_t *counters;    // small control block
  float *o_part;        // with the window rows' output: [units][items][G*w][d] partials
  int32_t *o_count;     // with the window rows' output: [units] items written
  size_t bytes;
};
CompressWs carve_compress_ws(const LayerGeom &g, void *base);

// Scoring, SIMT fp32 path (any dtype).
cudaError_t launch_score_simt(const LayerGeom &g, const void *q_win, const void *k,
                              const CompressWs &ws, float *votes, int32_t *status,
                              cudaStream_t st);
// Scoring, tcgen05 tensor-core path (bf16, d = 128).
bool score_tc_supported(const LayerGeom &g);
cudaError_t launch_score_tc(const LayerGeom &g, const void *q_win, const void *k,
                            const CompressWs &ws, float *votes, int32_t *status,
                            cudaStream_t st);
// The same for n_scored layers of one shape in one launch: scored layer i
// (q_win[i], k[i]) writes the votes of layer slots[i] of votes
// [n_slots][g.units][P]; ws is carved for n_scored * g.units units or more.
cudaError_t launch_score_tc(const LayerGeom &g, int n_slots, const int *slots, int n_scored,
                            const void *const *q_win, const void *const *k, const CompressWs &ws,
                            float *votes, int32_t *status, cudaStream_t st);
// Scoring on the tensor cores for G * w = 128 window rows (bf16, d = 128),
// for n_layers layers of the same shape in one launch; ws is carved for
// n_layers * g.units units and votes is [n_layers][g.units][P]. With v (the
// values of every layer) the same pass also gives the window rows' attention
// output o_win[l] [B][Hq][w][d] fp32 (ws carved with its partials).
bool score_tc1_supported(const LayerGeom &g);
cudaError_t launch_score_tc1(const LayerGeom &g, int n_layers, const void *const *q_win,
                             const void *const *k, const CompressWs &ws, float *votes,
                             int32_t *status, cudaStream_t st, const void *const *v = nullptr,
                             float *const *o_win = nullptr);
// Items per unit of launch_score_tc1 at most (sizes the output partials).
int score_tc1_max_items(const LayerGeom &g);
// The gather's inputs and outputs per layer (launch_gather's arguments).
struct GatherArgs {
  const void *const *k;
  const void *const *v;
  void *const *k_out;
  void *const *v_out;
  const int *cap;
};
// Pooling + exact top-k per unit of n_layers layers (votes [n_layers][units][P]);
// writes idx[l] [units][n_keep[l]]. With gather and gathered given, the
// kernel may also gather the kept rows (as launch_gather would); *gathered
// says whether it did.
cudaError_t launch_select(const LayerGeom &g, int n_layers, const float *votes,
                          const CompressWs &ws, const int *n_keep, int32_t *const *idx,
                          int32_t *status, cudaStream_t st, const GatherArgs *gather = nullptr,
                          bool *gathered = nullptr);
// idx = 0..T-1 for every unit (keep-all case).
cudaError_t launch_iota(const LayerGeom &g, int32_t *idx, cudaStream_t st);
// Gather kept K and V rows of n_layers layers into [units][cap[l]][d].
cudaError_t launch_gather(const LayerGeom &g, int n_layers, const void *const *k,
                          const void *const *v, const int32_t *const *idx, const int *n_keep,
                          void *const *k_out, void *const *v_out, const int *cap,
                          int32_t *status, cudaStream_t st);

}  // namespace ripple
