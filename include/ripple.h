/*
 * ripple.h -- C ABI of the RippleKV serving hot path on GB300 (sm_103a).
 *
 * RippleKV (arxiv 2608.08684) gives each layer l of a decoder a KV-cache
 * budget b_l from a per-layer sensitivity profile, keeps only b_l cached
 * positions of that layer (chosen by the base method's token scoring, SnapKV's
 * observation window), and decodes against the compressed caches. This library
 * implements that path: a host budget allocator (Sec. 4.4, Eqs. 9-12), a
 * per-layer compression chain on the GPU (scoring, pooling, top-k selection,
 * gather into a compact cache; Sec. 4.1 Eq. 4 and Sec. 4.4 last paragraph) and
 * GQA decode attention over the ragged compressed caches (Sec. 4.1); and, for
 * the offline profile the allocator takes, the Value perturbation and the
 * window KL divergence on the GPU and the calibration average (Sec. 4.3,
 * Eqs. 6-8).
 *
 * Conventions for every entry point:
 *   - Pointers named *_host are host memory; every other data pointer is CUDA
 *     device memory owned by the caller. The library never allocates, frees or
 *     keeps a reference to caller memory after a call returns.
 *   - `stream` is a cudaStream_t passed as void*; NULL means the legacy default
 *     stream. GPU work is enqueued on it in order; no call synchronises the
 *     host with the device.
 *   - Argument errors are detected on the host before anything is enqueued and
 *     returned as a ripple_status; outputs are then untouched. Errors found by
 *     the kernels (a full cache, a bounded wait that ran out, an index out of
 *     range) are written to *dev_status (a device int32 the caller zeroes and
 *     reads after synchronising the stream; the first error code written wins).
 *     dev_status may be NULL, in which case device-side errors are not reported.
 *   - dtype RIPPLE_BF16 means bfloat16 K/V/Q storage; RIPPLE_F32 means fp32.
 *     Arithmetic is fp32 (tensor cores take bf16 operands with fp32
 *     accumulation for the window-query/key contraction).
 *   - All tensors are dense, row-major, with the innermost dimension the head
 *     dimension d, and 16-byte aligned.
 */
#ifndef RIPPLE_H
#define RIPPLE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  RIPPLE_OK = 0,
  RIPPLE_EINVAL = 1,     /* invalid argument (shape, value, alignment, NULL) */
  RIPPLE_EWORKSPACE = 2, /* workspace smaller than the *_workspace_bytes query */
  RIPPLE_EFULL = 3,      /* decode: a layer's cache had no free row to append */
  RIPPLE_ECUDA = 4,      /* a CUDA runtime call failed (launch, attribute, ...) */
  RIPPLE_ETIMEOUT = 5,   /* a bounded in-kernel wait ran out (device status) */
  RIPPLE_EBOUNDS = 6,    /* a kernel met an out-of-range index (device status) */
  RIPPLE_ENOMEM = 7      /* a host-side allocation failed */
} ripple_status;

typedef enum { RIPPLE_F32 = 0, RIPPLE_BF16 = 1 } ripple_dtype;

typedef enum {
  RIPPLE_POOL_MAX = 0, /* max over the clipped window (default) */
  RIPPLE_POOL_AVG = 1, /* mean over the clipped window, summed in index order */
  RIPPLE_POOL_NONE = 2 /* votes used as they are */
} ripple_pool;

/* Largest number of layers one ripple_decode_attn call may cover. */
#define RIPPLE_MAX_LAYERS 128

/* ------------------------------------------------------------------------ */
/* Budget allocation (host only).                                            */
/* ------------------------------------------------------------------------ */

/*
 * ripple_alloc_budgets -- per-layer cache budgets from a sensitivity profile.
 *
 * Sec. 4.4 and Algorithm 1 "Budget Allocation":
 *   Eq. 9   s_hat_l = (s_l - s_min) / (s_max - s_min); all s_l equal -> s_hat = 0
 *   Eq. 10  w~_l = exp(log(ratio) * s_hat_l)
 *   Eq. 11  w = ClipNormalize(w~, gamma): clip to [1/gamma, gamma], then rescale
 *           to mean one over the layers
 *   Eq. 12  b_l = round(global_budget / n_layers * w_l), made to satisfy Eq. 5
 *           (sum_l b_l = global_budget) by taking floor(quota_l) and giving one
 *           more token to each of the global_budget - sum(floor) layers with
 *           the largest fractional parts, ties to the lower layer index.
 * The +epsilon of Algorithm 1's normalisation is not applied (Eq. 9 handles the
 * identical case explicitly). Computed in IEEE double with libm exp/log, in
 * layer order, without fused multiply-add: results are bit-reproducible.
 *
 * sens_host      [n_layers] sensitivity s_l (finite).
 * n_layers       |A| >= 1.
 * ratio          r >= 1, finite (r = 1 gives uniform budgets).
 * gamma          clip bound >= 1; gamma <= 0 or +infinity disables clipping.
 * global_budget  B >= 0, tokens summed over layers (per sequence and KV head).
 * budgets_host   [n_layers] output b_l.
 * Returns RIPPLE_EINVAL for NULL pointers, n_layers < 1, ratio < 1 or not
 * finite, 0 < gamma < 1, NaN gamma, a non-finite s_l or global_budget < 0;
 * RIPPLE_ENOMEM if its host scratch (16 bytes per layer) cannot be allocated.
 * Pure, reentrant, no CUDA calls.
 */
ripple_status ripple_alloc_budgets(const double *sens_host, int32_t n_layers, double ratio,
                                   double gamma, int64_t global_budget,
                                   int64_t *budgets_host);

/*
 * ripple_keep_count -- tokens one (batch, kv head) of a layer keeps:
 * n = min(seq_len, max(budget, window)). The budget counts the observation
 * window (SnapKV keeps the window; the paper's b_l = |S_l|, Eq. 4). Returns -1
 * for seq_len < 1, window < 1, window > seq_len or budget < 0.
 */
int32_t ripple_keep_count(int64_t budget, int32_t seq_len, int32_t window);

/* ------------------------------------------------------------------------ */
/* Per-layer compression (prefill time).                                     */
/* ------------------------------------------------------------------------ */

typedef struct {
  int32_t batch;       /* B >= 1 */
  int32_t n_q_heads;   /* Hq, a multiple of n_kv_heads */
  int32_t n_kv_heads;  /* Hkv >= 1; GQA group G = Hq / Hkv, G * window <= 256 */
  int32_t head_dim;    /* d: 64 or 128 */
  int32_t seq_len;     /* T >= 1, prompt tokens cached */
  int32_t window;      /* w, 1 <= w <= min(T, 64): observation window (last w prompt queries) */
  int32_t pool_kernel; /* odd, 1..31: 1-D pooling width over the prefix votes */
  int32_t pool_type;   /* ripple_pool */
  int32_t dtype;       /* ripple_dtype of q_win, k, v, k_out, v_out */
  float scale;         /* logit scale; 0 means 1/sqrt(head_dim) */
} ripple_layer_desc;

/* Device workspace bytes ripple_compress_layer needs for this shape. */
ripple_status ripple_compress_workspace_bytes(const ripple_layer_desc *desc, size_t *bytes_host);

/*
 * ripple_compress_layer -- compress one layer's KV cache to its budget.
 *
 * For every unit (b, h) (batch row, KV head), with P = T - w:
 *  1. scores every cached token from the observation window (SnapKV rule kept
 *     by RippleKV, Sec. 4.4 last paragraph): the G*w rows r = (query head
 *     h*G + g, window position i) of q_win, at positions P + i, give logits
 *     x[r][t] = scale * q_r . k_t for the keys t <= P + i they can see; each row
 *     is softmax-normalised over its keys, and the vote of key t is the sum of
 *     its probabilities over all G*w rows;
 *  2. pools the prefix votes (t < P) with a stride-1 window of pool_kernel,
 *     clipped to the prefix;
 *  3. keeps the n - w prefix tokens with the largest pooled score (ties: lower
 *     index), plus the w window tokens, n = ripple_keep_count(budget, T, w);
 *  4. copies the kept K and V rows, in ascending token order, to rows 0..n-1 of
 *     k_out / v_out (Eq. 4: compression only removes positions).
 * If n == T every token is kept (no scoring needed) and k_out/v_out are copies.
 *
 * q_win      [B][Hq][w][d]   the last w prompt queries of this layer
 * k, v       [B][Hkv][T][d]  this layer's prefill cache
 * k_out,v_out[B][Hkv][cap][d] compressed caches; rows >= n are left untouched
 * cap        rows per (b, h) of k_out/v_out, >= n (room for decode appends)
 * idx_out    int32 [B][Hkv][n] kept token positions, ascending (device)
 * scores_out fp32 [B][Hkv][P] unpooled votes of the prefix tokens, or NULL. When
 *            n == T and scores_out is not NULL the votes are still computed.
 * n_keep_host  receives n (host).
 * workspace  device scratch of at least ripple_compress_workspace_bytes bytes,
 *            256-byte aligned; its contents need no initialisation and are
 *            meaningless after the call. Calls that share a workspace must be
 *            ordered on the GPU (same stream, or events).
 * Errors: RIPPLE_EINVAL (bad desc, budget < 0, cap < n, NULL or misaligned
 * pointers), RIPPLE_EWORKSPACE, RIPPLE_ECUDA. Device status: RIPPLE_ETIMEOUT.
 */
ripple_status ripple_compress_layer(const ripple_layer_desc *desc, int64_t budget,
                                    const void *q_win, const void *k, const void *v,
                                    void *k_out, void *v_out, int32_t cap,
                                    int32_t *idx_out, float *scores_out,
                                    int32_t *n_keep_host, void *workspace,
                                    size_t workspace_bytes, int32_t *dev_status,
                                    void *stream);

/* Layers one ripple_compress_layers call may cover. */
#define RIPPLE_COMPRESS_MAX_LAYERS 80

/* Device workspace bytes ripple_compress_layers needs for n_layers layers of
 * this shape. */
ripple_status ripple_compress_layers_workspace_bytes(const ripple_layer_desc *desc,
                                                     int32_t n_layers, size_t *bytes_host);

/*
 * ripple_compress_layers -- ripple_compress_layer for n_layers layers of the
 * same shape (same desc) in one call, each with its own budget (the budgets
 * b_l of Eqs. 9-12). Layer l's result is exactly that of ripple_compress_layer
 * with budgets_host[l] and layer l's buffers; the layers are processed
 * together (bf16, d = 128, G * w = 128: two launches for all layers, scoring
 * and selection with the gather, so the GPU is not idle between layers),
 * otherwise one after another.
 *
 * n_layers     1..RIPPLE_COMPRESS_MAX_LAYERS, and n_layers * B * Hkv <= 65535
 * budgets_host host [n_layers]
 * q_win_host, k_host, v_host, k_out_host, v_out_host, idx_out_host
 *              host arrays of n_layers device pointers with the layouts of
 *              ripple_compress_layer (idx_out_host[l]: [B][Hkv][n_l] int32)
 * caps_host    host [n_layers]: rows per (b, h) of each layer's outputs
 * n_keep_host  host [n_layers], out: n_l of every layer
 * workspace    device scratch of at least
 *              ripple_compress_layers_workspace_bytes(desc, n_layers) bytes,
 *              256-byte aligned, no initialisation needed
 * Errors: RIPPLE_EINVAL (as ripple_compress_layer, for any layer),
 * RIPPLE_EWORKSPACE, RIPPLE_ECUDA. Device status as ripple_compress_layer.
 * The call may be captured in a CUDA graph (no host synchronisation, no
 * allocation).
 */
ripple_status ripple_compress_layers(const ripple_layer_desc *desc, int32_t n_layers,
                                     const int64_t *budgets_host, const void *const *q_win_host,
                                     const void *const *k_host, const void *const *v_host,
                                     void *const *k_out_host, void *const *v_out_host,
                                     const int32_t *caps_host, int32_t *const *idx_out_host,
                                     int32_t *n_keep_host, void *workspace,
                                     size_t workspace_bytes, int32_t *dev_status, void *stream);

/* Device workspace bytes ripple_compress_layers_attn needs for n_layers layers
 * of this shape (RIPPLE_EINVAL for shapes it does not take). */
ripple_status ripple_compress_layers_attn_workspace_bytes(const ripple_layer_desc *desc,
                                                          int32_t n_layers, size_t *bytes_host);

/*
 * ripple_compress_layers_attn -- ripple_compress_layers whose scoring pass also
 * gives the prefill attention output of the observation-window rows: the
 * SnapKV scoring that RippleKV keeps (Sec. 4.4, last paragraph; Sec. 2) fused
 * into the prefill attention of those rows, so that a real prefill reads each
 * layer's keys once for both (the rows' logits and normalisers are the same
 * quantities; no paper counterpart beyond that identity).
 *
 * For every layer l, batch b, query head q (KV head q / G) and window position
 * i (token P + i, P = T - w), with the causal mask of the window:
 *   o_win[l][b][q][i] = sum over t <= P + i of
 *                       softmax_t(scale * q_win[b][q][i] . k[b][q/G][t]) * v[b][q/G][t]
 * computed from the same logits and row normalisers as the votes.
 *
 * Shapes: bf16, head_dim 128, G * w = 128 window rows (the tensor-core path);
 * others return RIPPLE_EINVAL.
 * o_win_host  host array of n_layers device pointers, each fp32
 *             [B][Hq][w][head_dim], 16-byte aligned, written
 * workspace   at least ripple_compress_layers_attn_workspace_bytes bytes,
 *             256-byte aligned, no initialisation needed
 * Other arguments, outputs and errors as ripple_compress_layers, with the same
 * kept counts. The two calls split a unit's keys into different items (this
 * one takes up to 32768 keys a unit as one), so the row normalisers, merged
 * from the items' partial statistics, can differ in their last bits, and a
 * token whose pooled vote ties the selection threshold to within that
 * rounding can be kept by one call and not the other; units of at most 1152
 * keys are one item in both, and then the indices and gathered rows are
 * equal bit for bit. o_win is accumulated in fp32 from bf16 probabilities
 * (the tensor cores' operand type) in a fixed order: the same on every run.
 * The call may be captured in a CUDA graph.
 */
ripple_status ripple_compress_layers_attn(const ripple_layer_desc *desc, int32_t n_layers,
                                          const int64_t *budgets_host,
                                          const void *const *q_win_host,
                                          const void *const *k_host, const void *const *v_host,
                                          void *const *k_out_host, void *const *v_out_host,
                                          const int32_t *caps_host, int32_t *const *idx_out_host,
                                          int32_t *n_keep_host, float *const *o_win_host,
                                          void *workspace, size_t workspace_bytes,
                                          int32_t *dev_status, void *stream);

/*
 * ripple_select_layer -- steps 2-4 of ripple_compress_layer (pooling, top-k
 * selection with the window appended, gather) from caller-provided votes
 * instead of the window scoring. For scorers that produce the SnapKV votes
 * elsewhere (for instance inside a fused prefill attention), and for checking
 * the selection on chosen scores.
 *
 * votes      fp32 [B][Hkv][P] prefix votes (P = T - w), finite and >= 0.
 * Other arguments as in ripple_compress_layer (q_win is not needed).
 */
ripple_status ripple_select_layer(const ripple_layer_desc *desc, int64_t budget,
                                  const float *votes, const void *k, const void *v,
                                  void *k_out, void *v_out, int32_t cap, int32_t *idx_out,
                                  int32_t *n_keep_host, void *workspace, size_t workspace_bytes,
                                  int32_t *dev_status, void *stream);

/* ------------------------------------------------------------------------ */
/* Decoding against the ragged compressed caches.                            */
/* ------------------------------------------------------------------------ */

typedef struct {
  int32_t n_layers;   /* layers covered by this call, 1..RIPPLE_MAX_LAYERS */
  int32_t batch;      /* B */
  int32_t n_q_heads;  /* Hq, a multiple of n_kv_heads, G = Hq/Hkv <= 8 */
  int32_t n_kv_heads; /* Hkv */
  int32_t head_dim;   /* d: 64 or 128 */
  int32_t dtype;      /* ripple_dtype of q, k_new, v_new and the caches */
  float scale;        /* logit scale; 0 means 1/sqrt(head_dim) */
} ripple_decode_desc;

/* Device workspace bytes ripple_decode_attn needs for these layers' capacities. */
ripple_status ripple_decode_workspace_bytes(const ripple_decode_desc *desc,
                                            const int32_t *caps_host, size_t *bytes_host);

/*
 * ripple_decode_attn -- one decode step over several layers in one launch.
 *
 * Sec. 4.1: during decoding each new query attends to the cached states. For
 * every layer l, batch row b and KV head h, with len = lens[l]:
 *   1. appends the new key/value rows k_new[l][b][h], v_new[l][b][h] at row len
 *      of that layer's caches;
 *   2. for each of the G query heads of the group, attends over rows 0..len
 *      (the retained tokens, earlier appended tokens and the new token):
 *      out = sum_j softmax_j(scale * q . k_j) v_j, fp32 accumulation;
 *   3. after all layers are done, lens[l] = len + 1.
 * The query positions are not rotated (keys are stored post-rotation).
 *
 * q            [L][B][Hq][d]
 * k_new, v_new [L][B][Hkv][d]
 * k_caches_host, v_caches_host  host arrays of L device pointers; layer l's
 *              caches are [B][Hkv][caps_host[l]][d]
 * caps_host    host [L], rows per (b, h) of each layer's caches
 * lens         device int32 [L]: rows in use per layer (same for every b, h);
 *              read, then incremented by one per layer
 * out          device fp32 [L][B][Hq][d]
 * workspace    device scratch of at least ripple_decode_workspace_bytes bytes,
 *              256-byte aligned. Its contents need no initialisation and may
 *              be anything between calls (memory freed and handed out again
 *              by an allocator included): the kernel's first thread block
 *              zeroes the step's work counters at the start of every call
 *              and the other blocks touch no counter before it has done so.
 *              Calls that share a workspace must be ordered on the GPU (same
 *              stream, or events).
 * Consecutive calls on one stream may overlap: a call's thread blocks may
 * start while the previous call's last blocks finish; they read nothing the
 * previous call writes before it has completed.
 * After a call that reported RIPPLE_ETIMEOUT its outputs, appended rows and
 * lengths are unspecified; later calls are unaffected (a CUDA graph holding
 * that call should be captured again, since its replays reuse the call's
 * counter tag).
 * The call may be captured in a CUDA graph (no host synchronisation, no
 * allocation); capture was tested after one call outside the capture.
 * A layer with lens[l] >= caps_host[l] (or lens[l] < 0) is not appended to,
 * its output rows are zero, its length is unchanged, and RIPPLE_EFULL is
 * written to *dev_status.
 * Errors: RIPPLE_EINVAL, RIPPLE_EWORKSPACE, RIPPLE_ECUDA.
 */
ripple_status ripple_decode_attn(const ripple_decode_desc *desc, const void *q,
                                 const void *k_new, const void *v_new,
                                 void *const *k_caches_host, void *const *v_caches_host,
                                 const int32_t *caps_host, int32_t *lens, float *out,
                                 void *workspace, size_t workspace_bytes,
                                 int32_t *dev_status, void *stream);

/*
 * ripple_decode_attn_noalloc -- ripple_decode_attn for callers that cannot
 * allocate device memory. The paper has no counterpart; this is a deployment
 * variant.
 *
 * Some callers have no way to obtain scratch memory on the device where they
 * call a decode step: a plugin inside a host program that owns all device
 * memory through its own pool and only hands over the input and output
 * tensors, or a fixed-footprint server that reserves every byte at start-up.
 * This entry point takes no workspace: the split-K partials of the step live
 * in a library-owned array of RIPPLE_DECODE_NOALLOC_SCRATCH_BYTES bytes in
 * device global memory, which every GPU that loads the library keeps until the
 * process exits. The caller still passes all inputs and outputs, with the
 * meaning, layout and errors of ripple_decode_attn.
 *
 * - Allocates nothing: no cudaMalloc/cudaFree or allocating library call.
 * - The first call on a device looks up the array's device address on that
 *   device (once per device, with it current); make that first call before
 *   any stream capture begins.
 * - Returns RIPPLE_EWORKSPACE, before enqueuing anything, when the step needs
 *   more scratch than the array holds (ripple_decode_workspace_bytes(desc,
 *   caps) > RIPPLE_DECODE_NOALLOC_SCRATCH_BYTES).
 * - Every call on a device shares the one array. Each call zeroes the
 *   counters it uses before using them, and every partial a call reads it
 *   has written itself, so nothing carries over from the previous call (not
 *   even from one that reported RIPPLE_ETIMEOUT). Calls that may overlap on
 *   the GPU (different streams without ordering) race on it; order them,
 *   e.g. by issuing them on one stream.
 */
#define RIPPLE_DECODE_NOALLOC_SCRATCH_BYTES (8u << 20)
ripple_status ripple_decode_attn_noalloc(const ripple_decode_desc *desc, const void *q,
                                         const void *k_new, const void *v_new,
                                         void *const *k_caches_host, void *const *v_caches_host,
                                         const int32_t *caps_host, int32_t *lens, float *out,
                                         int32_t *dev_status, void *stream);

/* ------------------------------------------------------------------------ */
/* Sensitivity profiling (offline; Sec. 4.3, Algorithm 1 "Sensitivity        */
/* Profiling"). The model forwards that turn a perturbed cache into output    */
/* logits belong to the caller; these calls cover the perturbation (Eq. 6),   */
/* the window divergence (Eq. 7) and the calibration average (Eq. 8).         */
/* ------------------------------------------------------------------------ */

typedef struct {
  int32_t batch;      /* B >= 1 */
  int32_t n_kv_heads; /* Hkv >= 1 */
  int32_t seq_len;    /* T >= 1, cached positions per (batch, kv head) */
  int32_t head_dim;   /* d: 64 or 128 */
  int32_t dtype;      /* ripple_dtype of v and v_out */
} ripple_cache_desc;

/*
 * ripple_perturb_values -- norm-adaptive perturbation of one layer's Value
 * cache (Sec. 4.3, Eq. 6).
 *
 * For every batch row b, KV head h and eligible position u in
 * [pos_begin, pos_end):
 *   v~_u = v_u + alpha * ||v_u||_2 * eps_u,   eps_u ~ N(0, I) (given),
 * the norm taken over the d channels of the stored row. The positions the
 * base compression method protects are excluded by the range (SnapKV protects
 * its observation window, the last w cached positions: pos_end = T - w). Keys
 * and other layers are not touched by the method, and not by this call.
 *
 * v          [B][Hkv][T][d] the layer's Value cache
 * eps        fp32 [B][Hkv][pos_end - pos_begin][d] standard normal draws; row
 *            u - pos_begin belongs to position u. May be NULL when the range
 *            is empty.
 * alpha      perturbation strength, finite, >= 0
 * pos_begin, pos_end  0 <= pos_begin <= pos_end <= T
 * v_out      [B][Hkv][T][d]: the eligible rows receive v~ rounded to nearest
 *            (even) in dtype, the other rows a copy of v. v_out == v perturbs
 *            in place and writes only the eligible rows; any other overlap of
 *            v_out with v or eps is invalid.
 * Arithmetic is fp32. The call may be captured in a CUDA graph.
 * Errors: RIPPLE_EINVAL (bad desc or range, alpha < 0 or not finite, NULL or
 * not 16-byte aligned pointers), RIPPLE_ECUDA.
 */
ripple_status ripple_perturb_values(const ripple_cache_desc *desc, const void *v,
                                    const float *eps, float alpha, int32_t pos_begin,
                                    int32_t pos_end, void *v_out, void *stream);

/* Device workspace bytes ripple_window_kl needs for this shape. */
ripple_status ripple_window_kl_workspace_bytes(int32_t n_sets, int32_t n_pos, int32_t vocab,
                                               size_t *bytes_host);

/*
 * ripple_window_kl -- output divergence averaged over the evaluation window
 * (Sec. 4.3, Eq. 7), for n_sets perturbed runs against one reference run
 * (set s is typically the run with layer s perturbed).
 *
 * For every set s and window position t < n_pos, with P_t = softmax over the
 * vocabulary of p_logits[t] and Q_{s,t} = softmax of q_logits[s][t]:
 *   KL_{s,t} = sum_v P_t(v) (log P_t(v) - log Q_{s,t}(v))
 *   d_s      = (1 / n_pos) sum_t KL_{s,t}
 *
 * p_logits   [n_pos][vocab] reference logits (intact cache), finite
 * q_logits   [n_sets][n_pos][vocab] logits after the perturbation, finite
 * vocab      >= 1, a multiple of 8 (rows start on 16-byte boundaries)
 * dtype      ripple_dtype of both logit arrays
 * kl_out     fp32 [n_sets][n_pos] per-position divergences, or NULL
 * d_out      fp32 [n_sets] window averages
 * workspace  device scratch of at least ripple_window_kl_workspace_bytes
 *            bytes, 256-byte aligned; its contents need no initialisation
 *            (the call zeroes the counters it keeps there); calls that share
 *            a workspace must be ordered (one stream)
 * Arithmetic: with delta = q - p, KL = log E_P[exp(delta)] - E_P[delta].
 * Each row is cut into fixed slices of 8192 logits and each slice into fixed
 * shares of 512; a share is reduced in fp32 to the sums, over its logits, of
 * w = exp(p - max p), w x and w (exp(x) - 1 - x) with x = delta - c (c = delta
 * at the share's first largest p; the last sum by its Taylor polynomial where
 * |x| <= 1/2 across the share), or of exp(q - r) for a reference r where some
 * |x| is larger. The shares of a row are merged in double in a fixed order,
 * KL = log1p(E_P[x] + E_P[exp(x) - 1 - x]) - E_P[x] (so a small divergence
 * is not the difference of two large terms), and the window mean is summed
 * in double: results do not depend on the GPU or on the run. Identical p and
 * q rows give exactly 0. Two kernel launches. The call may be captured in a
 * CUDA graph; after RIPPLE_ETIMEOUT the outputs are unspecified and a graph
 * holding the call should be re-captured.
 * Errors: RIPPLE_EINVAL (n_sets < 1, n_pos < 1, bad vocab or dtype, NULL or
 * misaligned pointers), RIPPLE_EWORKSPACE, RIPPLE_ECUDA. Device status:
 * RIPPLE_ETIMEOUT (a bounded in-kernel wait ran out).
 */
ripple_status ripple_window_kl(const void *p_logits, const void *q_logits, int32_t n_sets,
                               int32_t n_pos, int32_t vocab, int32_t dtype, float *kl_out,
                               float *d_out, void *workspace, size_t workspace_bytes,
                               int32_t *dev_status, void *stream);

/*
 * ripple_sensitivity_profile -- calibration average (Sec. 4.3, Eq. 8), host:
 *   s_l = (1 / N) sum_i d_{i,l},
 * summed in example order in double. The result feeds ripple_alloc_budgets.
 *
 * d_host     [n_examples][n_layers] window divergences d_{i,l} (Eq. 7), finite
 * s_host     [n_layers] output
 * Returns RIPPLE_EINVAL for NULL pointers, n_examples < 1, n_layers < 1 or a
 * non-finite d. Pure, reentrant, no CUDA calls.
 */
ripple_status ripple_sensitivity_profile(const double *d_host, int32_t n_examples,
                                         int32_t n_layers, double *s_host);

/* Number of kernels this library has launched in this process so far
 * (host-side count of launch calls; for benchmarks and launch accounting). */
uint64_t ripple_kernel_launches(void);

/*
 * ripple_set_wait_limit_cycles -- bound of the in-kernel waits of kernels
 * launched from now on, in SM clock cycles (process-wide; returns the
 * previous value). cycles <= 0 restores the default, 4e9 cycles (about two
 * seconds). Every wait of a thread block on another role, on another thread
 * block or on its own bulk copies gives up after this many cycles, reports
 * RIPPLE_ETIMEOUT in *dev_status and lets the kernel leave; the waits that
 * then hold a block until the copies it issued have landed keep the default
 * bound. A diagnostic and test hook (a small limit makes the waits give up
 * on purpose); the paper has no counterpart. Launches already enqueued keep
 * the limit they were given.
 */
int64_t ripple_set_wait_limit_cycles(int64_t cycles);

/* Human-readable name of a status code (static string). */
const char *ripple_status_string(int32_t status);

#ifdef __cplusplus
}
#endif

#endif /* RIPPLE_H */
