// ripple_compress_layer: the per-layer compression chain (Sec. 4.1 Eq. 4 and
// Sec. 4.4 last paragraph: RippleKV keeps the base method's scoring and
// selection and changes only the number of tokens each layer keeps).
//   scoring   -> votes [units][P]     (tcgen05 for bf16 d=128, fp32 SIMT otherwise)
//   selection -> idx   [units][n]     (pooling + exact top-k, window appended)
//   gather    -> k_out, v_out [units][cap][d]
// Everything is enqueued on the caller's stream; nothing synchronises.
#include <math.h>

#include <atomic>

#include "common.cuh"
#include "kernels.cuh"

namespace ripple {

static size_t round_up(size_t x) { return (x + 255) & ~(size_t)255; }

static std::atomic<uint64_t> g_launches{0};
void count_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }

static std::atomic<long long> g_wait_limit{kDefaultWaitCycles};
long long wait_limit_cycles() { return g_wait_limit.load(std::memory_order_relaxed); }

CompressWs carve_compress_ws(const LayerGeom &g, void *base) {
  CompressWs w{};
  uint8_t *p = (uint8_t *)base;
  size_t off = 0;
  const size_t n_chunks = (g.T + kScoreChunk - 1) / kScoreChunk;
  auto take = [&](size_t bytes) {
    uint8_t *r = p ? p + off : nullptr;
    off += round_up(bytes);
    return r;
  };
  // two partials per chunk: the tensor-core path keeps one per epilogue warpgroup
  w.row_partial = (float2 *)take(sizeof(float2) * g.units * n_chunks * 2 * g.R);
  w.row_lognorm = (float *)take(sizeof(float) * g.units * g.R);
  w.votes = (float *)take(sizeof(float) * g.units * (size_t)g.P);
  w.keys = (uint32_t *)take(g.P > kSelectSmemKeys ? sizeof(uint32_t) * g.units * (size_t)g.P : 0);
  w.counters = (int32_t *)take(sizeof(int32_t) * (128 + 2 * (size_t)g.units));
  w.bytes = off;
  return w;
}

static bool make_geom(const ripple_layer_desc *d, LayerGeom *g) {
  if (d == nullptr) return false;
  if (d->batch < 1 || d->n_q_heads < 1 || d->n_kv_heads < 1) return false;
  if (d->n_q_heads % d->n_kv_heads != 0) return false;
  if (d->head_dim != 64 && d->head_dim != 128) return false;
  if (d->seq_len < 1 || d->window < 1 || d->window > d->seq_len || d->window > 64) return false;
  if (d->pool_kernel < 1 || d->pool_kernel > 31 || (d->pool_kernel & 1) == 0) return false;
  if (d->pool_type != RIPPLE_POOL_MAX && d->pool_type != RIPPLE_POOL_AVG &&
      d->pool_type != RIPPLE_POOL_NONE)
    return false;
  if (d->dtype != RIPPLE_F32 && d->dtype != RIPPLE_BF16) return false;
  if (!(d->scale >= 0.f) || isinf(d->scale)) return false;
  const int G = d->n_q_heads / d->n_kv_heads;
  if (G * d->window > 256) return false;
  if ((int64_t)d->batch * d->n_kv_heads > 65535) return false;
  g->B = d->batch;
  g->Hq = d->n_q_heads;
  g->Hkv = d->n_kv_heads;
  g->G = G;
  g->D = d->head_dim;
  g->T = d->seq_len;
  g->W = d->window;
  g->P = d->seq_len - d->window;
  g->R = G * d->window;
  g->units = d->batch * d->n_kv_heads;
  g->dtype = d->dtype;
  g->pool_kernel = d->pool_kernel;
  g->pool_type = d->pool_type;
  const float scale = d->scale > 0.f ? d->scale : 1.0f / sqrtf((float)d->head_dim);
  g->scale2 = scale * kLog2e;
  return true;
}

}  // namespace ripple

using namespace ripple;

extern "C" uint64_t ripple_kernel_launches(void) { return g_launches.load(); }

extern "C" int64_t ripple_set_wait_limit_cycles(int64_t cycles) {
  const long long v = cycles > 0 ? (long long)cycles : kDefaultWaitCycles;
  return (int64_t)g_wait_limit.exchange(v);
}

extern "C" ripple_status ripple_compress_workspace_bytes(const ripple_layer_desc *desc,
                                                         size_t *bytes_host) {
  LayerGeom g;
  if (!make_geom(desc, &g) || bytes_host == nullptr) return RIPPLE_EINVAL;
  *bytes_host = carve_compress_ws(g, nullptr).bytes;
  return RIPPLE_OK;
}

extern "C" ripple_status ripple_compress_layer(const ripple_layer_desc *desc, int64_t budget,
                                               const void *q_win, const void *k, const void *v,
                                               void *k_out, void *v_out, int32_t cap,
                                               int32_t *idx_out, float *scores_out,
                                               int32_t *n_keep_host, void *workspace,
                                               size_t workspace_bytes, int32_t *dev_status,
                                               void *stream) {
  LayerGeom g;
  if (!make_geom(desc, &g)) return RIPPLE_EINVAL;
  if (budget < 0 || !q_win || !k || !v || !k_out || !v_out || !idx_out || !n_keep_host ||
      !workspace)
    return RIPPLE_EINVAL;
  auto aligned = [](const void *p) { return ((uintptr_t)p & 15u) == 0; };
  if (!aligned(q_win) || !aligned(k) || !aligned(v) || !aligned(k_out) || !aligned(v_out) ||
      !aligned(idx_out) || (scores_out && !aligned(scores_out)) || ((uintptr_t)workspace & 255u))
    return RIPPLE_EINVAL;
  const int n = ripple_keep_count(budget, g.T, g.W);
  if (n < 0 || cap < n) return RIPPLE_EINVAL;
  const CompressWs ws = carve_compress_ws(g, workspace);
  if (workspace_bytes < ws.bytes) return RIPPLE_EWORKSPACE;
  cudaStream_t st = (cudaStream_t)stream;

  const bool keep_all = (n == g.T);
  float *votes = scores_out ? scores_out : ws.votes;
  if (g.P > 0 && (!keep_all || scores_out)) {
    cudaError_t e = score_tc1_supported(g)  ? launch_score_tc1(g, 1, &q_win, &k, ws, votes, dev_status, st)
                    : score_tc_supported(g) ? launch_score_tc(g, q_win, k, ws, votes, dev_status, st)
                                            : launch_score_simt(g, q_win, k, ws, votes, dev_status, st);
    RIPPLE_CUDA_TRY(e);
  }
  if (keep_all) {
    RIPPLE_CUDA_TRY(launch_iota(g, idx_out, st));
  } else {
    RIPPLE_CUDA_TRY(launch_select(g, 1, votes, ws, &n, &idx_out, dev_status, st));
  }
  RIPPLE_CUDA_TRY(launch_gather(g, 1, &k, &v, &idx_out, &n, &k_out, &v_out, &cap, dev_status, st));
  *n_keep_host = n;
  return RIPPLE_OK;
}

extern "C" ripple_status ripple_select_layer(const ripple_layer_desc *desc, int64_t budget,
                                             const float *votes, const void *k, const void *v,
                                             void *k_out, void *v_out, int32_t cap,
                                             int32_t *idx_out, int32_t *n_keep_host,
                                             void *workspace, size_t workspace_bytes,
                                             int32_t *dev_status, void *stream) {
  LayerGeom g;
  if (!make_geom(desc, &g)) return RIPPLE_EINVAL;
  if (budget < 0 || !votes || !k || !v || !k_out || !v_out || !idx_out || !n_keep_host ||
      !workspace)
    return RIPPLE_EINVAL;
  auto aligned = [](const void *p) { return ((uintptr_t)p & 15u) == 0; };
  if (!aligned(votes) || !aligned(k) || !aligned(v) || !aligned(k_out) || !aligned(v_out) ||
      !aligned(idx_out) || ((uintptr_t)workspace & 255u))
    return RIPPLE_EINVAL;
  const int n = ripple_keep_count(budget, g.T, g.W);
  if (n < 0 || cap < n) return RIPPLE_EINVAL;
  const CompressWs ws = carve_compress_ws(g, workspace);
  if (workspace_bytes < ws.bytes) return RIPPLE_EWORKSPACE;
  cudaStream_t st = (cudaStream_t)stream;
  if (n == g.T) {
    RIPPLE_CUDA_TRY(launch_iota(g, idx_out, st));
  } else {
    RIPPLE_CUDA_TRY(launch_select(g, 1, votes, ws, &n, &idx_out, dev_status, st));
  }
  RIPPLE_CUDA_TRY(launch_gather(g, 1, &k, &v, &idx_out, &n, &k_out, &v_out, &cap, dev_status, st));
  *n_keep_host = n;
  return RIPPLE_OK;
}

// Workspace of a multi-layer call: the single-layer carve-up for all layers'
// units at once (votes [n_layers][units][P] contiguous).
static CompressWs carve_layers_ws(const LayerGeom &g, int n_layers, void *base) {
  LayerGeom all = g;
  all.units = g.units * n_layers;
  return carve_compress_ws(all, base);
}

// The multi-layer workspace with the window rows' output partials after it.
static CompressWs carve_layers_attn_ws(const LayerGeom &g, int n_layers, void *base) {
  CompressWs w = carve_layers_ws(g, n_layers, base);
  uint8_t *p = (uint8_t *)base;
  size_t off = w.bytes;
  const size_t units = (size_t)g.units * n_layers;
  w.o_part = p ? (float *)(p + off) : nullptr;
  off += round_up(sizeof(float) * units * score_tc1_max_items(g) * g.R * g.D);
  w.o_count = p ? (int32_t *)(p + off) : nullptr;
  off += round_up(sizeof(int32_t) * units);
  w.bytes = off;
  return w;
}

static bool layers_geom(const ripple_layer_desc *desc, int32_t n_layers, LayerGeom *g) {
  return make_geom(desc, g) && n_layers >= 1 && n_layers <= RIPPLE_COMPRESS_MAX_LAYERS &&
         (int64_t)g->units * n_layers <= 65535;
}

extern "C" ripple_status ripple_compress_layers_workspace_bytes(const ripple_layer_desc *desc,
                                                                int32_t n_layers,
                                                                size_t *bytes_host) {
  LayerGeom g;
  if (!layers_geom(desc, n_layers, &g) || bytes_host == nullptr) return RIPPLE_EINVAL;
  *bytes_host = carve_layers_ws(g, n_layers, nullptr).bytes;
  return RIPPLE_OK;
}

extern "C" ripple_status ripple_compress_layers_attn_workspace_bytes(const ripple_layer_desc *desc,
                                                                     int32_t n_layers,
                                                                     size_t *bytes_host) {
  LayerGeom g;
  if (!layers_geom(desc, n_layers, &g) || bytes_host == nullptr || !score_tc1_supported(g))
    return RIPPLE_EINVAL;
  *bytes_host = carve_layers_attn_ws(g, n_layers, nullptr).bytes;
  return RIPPLE_OK;
}

// Both multi-layer entry points; with o_win_host (non-NULL) the scoring pass
// also gives the window rows' attention output of every layer.
static ripple_status compress_layers_impl(
    const ripple_layer_desc *desc, int32_t n_layers, const int64_t *budgets_host,
    const void *const *q_win_host, const void *const *k_host, const void *const *v_host,
    void *const *k_out_host, void *const *v_out_host, const int32_t *caps_host,
    int32_t *const *idx_out_host, int32_t *n_keep_host, float *const *o_win_host,
    void *workspace, size_t workspace_bytes, int32_t *dev_status, void *stream) {
  LayerGeom g;
  if (!layers_geom(desc, n_layers, &g)) return RIPPLE_EINVAL;
  if (!budgets_host || !q_win_host || !k_host || !v_host || !k_out_host || !v_out_host ||
      !caps_host || !idx_out_host || !n_keep_host || !workspace || ((uintptr_t)workspace & 255u))
    return RIPPLE_EINVAL;
  auto aligned = [](const void *p) { return p != nullptr && ((uintptr_t)p & 15u) == 0; };
  int n[RIPPLE_COMPRESS_MAX_LAYERS];
  int cap[RIPPLE_COMPRESS_MAX_LAYERS];
  for (int l = 0; l < n_layers; ++l) {
    if (budgets_host[l] < 0 || !aligned(q_win_host[l]) || !aligned(k_host[l]) ||
        !aligned(v_host[l]) || !aligned(k_out_host[l]) || !aligned(v_out_host[l]) ||
        !aligned(idx_out_host[l]) || (o_win_host != nullptr && !aligned(o_win_host[l])))
      return RIPPLE_EINVAL;
    n[l] = ripple_keep_count(budgets_host[l], g.T, g.W);
    cap[l] = caps_host[l];
    if (n[l] < 0 || cap[l] < n[l]) return RIPPLE_EINVAL;
  }
  if (o_win_host != nullptr && !score_tc1_supported(g)) return RIPPLE_EINVAL;
  const CompressWs ws = o_win_host ? carve_layers_attn_ws(g, n_layers, workspace)
                                   : carve_layers_ws(g, n_layers, workspace);
  if (workspace_bytes < ws.bytes) return RIPPLE_EWORKSPACE;
  cudaStream_t st = (cudaStream_t)stream;
  // selection and gather in one launch where the selection kernel takes both
  const GatherArgs ga{k_host, v_host, k_out_host, v_out_host, cap};
  bool gathered = false;
  if (g.P > 0 && score_tc1_supported(g)) {
    // All layers in two or three launches: scoring, selection (+ gather).
    RIPPLE_CUDA_TRY(launch_score_tc1(g, n_layers, q_win_host, k_host, ws, ws.votes, dev_status,
                                     st, o_win_host ? v_host : nullptr, o_win_host));
    RIPPLE_CUDA_TRY(launch_select(g, n_layers, ws.votes, ws, n, idx_out_host, dev_status, st,
                                  &ga, &gathered));
    if (!gathered)
      RIPPLE_CUDA_TRY(launch_gather(g, n_layers, k_host, v_host,
                                    (const int32_t *const *)idx_out_host, n, k_out_host,
                                    v_out_host, cap, dev_status, st));
  } else {
    // Other shapes: the 256-row tensor-core scoring of every layer that needs
    // votes in one launch, or the CUDA-core scoring layer by layer (each
    // layer's votes in its part of the vote array, the scratch of the
    // multi-layer workspace reused); then one selection and one gather launch
    // for all layers. A layer that keeps every token needs no votes (the
    // selection writes 0..T-1 for it).
    if (g.P > 0 && score_tc_supported(g)) {
      // the layers that need votes, all in one tensor-core launch
      int slots[RIPPLE_COMPRESS_MAX_LAYERS];
      const void *qs[RIPPLE_COMPRESS_MAX_LAYERS];
      const void *ks[RIPPLE_COMPRESS_MAX_LAYERS];
      int n_scored = 0;
      for (int l = 0; l < n_layers; ++l) {
        if (n[l] == g.T) continue;
        slots[n_scored] = l;
        qs[n_scored] = q_win_host[l];
        ks[n_scored] = k_host[l];
        ++n_scored;
      }
      if (n_scored > 0)
        RIPPLE_CUDA_TRY(launch_score_tc(g, n_layers, slots, n_scored, qs, ks, ws, ws.votes,
                                        dev_status, st));
    } else {
      for (int l = 0; l < n_layers; ++l) {
        if (g.P == 0 || n[l] == g.T) continue;
        float *votes_l = ws.votes + (size_t)l * g.units * g.P;
        RIPPLE_CUDA_TRY(launch_score_simt(g, q_win_host[l], k_host[l], ws, votes_l, dev_status,
                                          st));
      }
    }
    RIPPLE_CUDA_TRY(launch_select(g, n_layers, ws.votes, ws, n, idx_out_host, dev_status, st,
                                  &ga, &gathered));
    if (!gathered)
      RIPPLE_CUDA_TRY(launch_gather(g, n_layers, k_host, v_host,
                                    (const int32_t *const *)idx_out_host, n, k_out_host,
                                    v_out_host, cap, dev_status, st));
  }
  for (int l = 0; l < n_layers; ++l) n_keep_host[l] = n[l];
  return RIPPLE_OK;
}

extern "C" ripple_status ripple_compress_layers(
    const ripple_layer_desc *desc, int32_t n_layers, const int64_t *budgets_host,
    const void *const *q_win_host, const void *const *k_host, const void *const *v_host,
    void *const *k_out_host, void *const *v_out_host, const int32_t *caps_host,
    int32_t *const *idx_out_host, int32_t *n_keep_host, void *workspace, size_t workspace_bytes,
    int32_t *dev_status, void *stream) {
  return compress_layers_impl(desc, n_layers, budgets_host, q_win_host, k_host, v_host,
                              k_out_host, v_out_host, caps_host, idx_out_host, n_keep_host,
                              nullptr, workspace, workspace_bytes, dev_status, stream);
}

extern "C" ripple_status ripple_compress_layers_attn(
    const ripple_layer_desc *desc, int32_t n_layers, const int64_t *budgets_host,
    const void *const *q_win_host, const void *const *k_host, const void *const *v_host,
    void *const *k_out_host, void *const *v_out_host, const int32_t *caps_host,
    int32_t *const *idx_out_host, int32_t *n_keep_host, float *const *o_win_host,
    void *workspace, size_t workspace_bytes, int32_t *dev_status, void *stream) {
  if (o_win_host == nullptr) return RIPPLE_EINVAL;
  return compress_layers_impl(desc, n_layers, budgets_host, q_win_host, k_host, v_host,
                              k_out_host, v_out_host, caps_host, idx_out_host, n_keep_host,
                              o_win_host, workspace, workspace_bytes, dev_status, stream);
}
