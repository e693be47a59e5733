// GQA decode attention over the ragged compressed caches (Sec. 4.1: each new
// query attends to the cached states), with the append of the new token.
//
// Split-K over retained tokens: work item = (layer, batch row, KV head,
// chunk of kChunk cache rows). One 128-thread CTA per item computes, for the
// G query heads of the group, the chunk's (max, sum, unnormalised output) with
// warp-shuffle max/sum reductions; a second kernel combines the chunk
// partials in a fixed order (deterministic) and advances the lengths.
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "kernels.cuh"

namespace ripple {
namespace {

constexpr int kThreads = 128;
constexpr int kChunk = 128;

struct DecodeParams {
  int L, B, Hq, Hkv, G, D;
  float scale2;
  const void *q, *k_new, *v_new;
  int32_t *lens;
  float *out;
  float *ws_m, *ws_l, *ws_o;
  int32_t *status;
  int total_items;
  const void *kc[RIPPLE_MAX_LAYERS];
  const void *vc[RIPPLE_MAX_LAYERS];
  int cap[RIPPLE_MAX_LAYERS];
  int nch[RIPPLE_MAX_LAYERS];
  int item_base[RIPPLE_MAX_LAYERS + 1];
};

__device__ __forceinline__ int find_layer(const DecodeParams &p, int item) {
  int lo = 0, hi = p.L - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.item_base[mid] <= item) lo = mid; else hi = mid - 1;
  }
  return lo;
}

template <typename Tin, int D, int G>
__global__ void __launch_bounds__(kThreads) decode_partial(const __grid_constant__ DecodeParams p) {
  __shared__ float qs[G][D];
  __shared__ float ps[G][kChunk];
  __shared__ float red[kThreads / 32][G];
  __shared__ float mx[G], den[G];
  const int item = blockIdx.x;
  const int l = find_layer(p, item);
  const int nch = p.nch[l];
  const int local = item - p.item_base[l];
  const int unit = local / nch, c = local % nch;
  const int b = unit / p.Hkv, h = unit % p.Hkv;
  const int len = p.lens[l], cap = p.cap[l];
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  float *pm = p.ws_m + (size_t)item * G;
  float *pl = p.ws_l + (size_t)item * G;
  float *po = p.ws_o + (size_t)item * G * D;

  const int r0 = c * kChunk;
  const bool full = len < 0 || len >= cap;
  const int rows = full ? 0 : min(kChunk, len + 1 - r0);
  if (full && c == 0 && unit == 0 && tid == 0) report(p.status, RIPPLE_EFULL);
  if (rows <= 0) {
    if (tid < G) {
      pm[tid] = -INFINITY;
      pl[tid] = 0.f;
    }
    for (int e = tid; e < G * D; e += kThreads) po[e] = 0.f;
    return;
  }

  const Tin *qg = (const Tin *)p.q + (((size_t)l * p.B + b) * p.Hq + (size_t)h * G) * D;
  for (int e = tid; e < G * D; e += kThreads) qs[e / D][e % D] = to_f32(qg[e]) * p.scale2;
  const size_t unit_off = (size_t)unit * cap * D;
  const Tin *kc = (const Tin *)p.kc[l] + unit_off;
  const Tin *vc = (const Tin *)p.vc[l] + unit_off;
  const size_t new_off = (((size_t)l * p.B + b) * p.Hkv + h) * D;
  const Tin *k_new = (const Tin *)p.k_new + new_off;
  const Tin *v_new = (const Tin *)p.v_new + new_off;
  __syncthreads();

  // Scores of this chunk's rows, one row per thread.
  float s[G];
  const int j = tid, t = r0 + j;
#pragma unroll
  for (int g = 0; g < G; ++g) s[g] = -INFINITY;
  if (j < rows) {
    const Tin *krow = (t == len) ? k_new : kc + (size_t)t * D;
#pragma unroll
    for (int g = 0; g < G; ++g) s[g] = 0.f;
#pragma unroll 4
    for (int piece = 0; piece < D / 8; ++piece) {
      float kv[8];
      load8(krow + piece * 8, kv);
#pragma unroll
      for (int g = 0; g < G; ++g)
#pragma unroll
        for (int i = 0; i < 8; ++i) s[g] = fmaf(qs[g][piece * 8 + i], kv[i], s[g]);
    }
    if (t == len) {  // append the new token's rows to the cache
      Tin *kd = (Tin *)p.kc[l] + unit_off + (size_t)len * D;
      Tin *vd = (Tin *)p.vc[l] + unit_off + (size_t)len * D;
      for (int e = 0; e < D; ++e) {
        kd[e] = k_new[e];
        vd[e] = v_new[e];
      }
    }
  }
  // Chunk max per head.
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const float m = warp_max(s[g]);
    if (lane == 0) red[wid][g] = m;
  }
  __syncthreads();
  if (tid < G) {
    float m = red[0][tid];
    for (int w = 1; w < kThreads / 32; ++w) m = fmaxf(m, red[w][tid]);
    mx[tid] = m;
  }
  __syncthreads();
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const float e = (j < rows) ? exp2f(s[g] - mx[g]) : 0.f;
    ps[g][j] = e;
    const float sum = warp_sum(e);
    if (lane == 0) red[wid][g] = sum;
  }
  __syncthreads();
  if (tid < G) {
    float sum = 0.f;
    for (int w = 0; w < kThreads / 32; ++w) sum += red[w][tid];
    den[tid] = sum;
  }
  // Unnormalised output: thread -> one dimension, a subset of the heads.
  constexpr int kHeadStride = kThreads / D;  // 1 for d = 128, 2 for d = 64
  const int dim = tid % D, g0 = tid / D;
  float acc[G];
#pragma unroll
  for (int g = 0; g < G; ++g) acc[g] = 0.f;
  for (int jj = 0; jj < rows; ++jj) {
    const Tin *vrow = (r0 + jj == len) ? v_new : vc + (size_t)(r0 + jj) * D;
    const float v = to_f32(vrow[dim]);
#pragma unroll
    for (int g = 0; g < G; ++g)
      if (g % kHeadStride == g0) acc[g] = fmaf(ps[g][jj], v, acc[g]);
  }
#pragma unroll
  for (int g = 0; g < G; ++g)
    if (g % kHeadStride == g0) po[(size_t)g * D + dim] = acc[g];
  __syncthreads();
  if (tid < G) {
    pm[tid] = mx[tid];
    pl[tid] = den[tid];
  }
}

template <int D>
__global__ void decode_combine(const __grid_constant__ DecodeParams p) {
  const int bid = blockIdx.x;  // over L * B * Hq
  const int hq = bid % p.Hq, b = (bid / p.Hq) % p.B, l = bid / (p.Hq * p.B);
  const int h = hq / p.G, g = hq % p.G;
  const int nch = p.nch[l];
  const int item0 = p.item_base[l] + (b * p.Hkv + h) * nch;
  float M = -INFINITY;
  for (int c = 0; c < nch; ++c) M = fmaxf(M, p.ws_m[(size_t)(item0 + c) * p.G + g]);
  float num = 0.f, den = 0.f;
  if (M != -INFINITY) {
    for (int c = 0; c < nch; ++c) {
      const size_t ig = (size_t)(item0 + c) * p.G + g;
      const float wgt = exp2f(p.ws_m[ig] - M);
      den += wgt * p.ws_l[ig];
      num += wgt * p.ws_o[ig * D + threadIdx.x];
    }
  }
  p.out[(size_t)bid * D + threadIdx.x] = den > 0.f ? num / den : 0.f;
  if (b == 0 && hq == 0 && threadIdx.x == 0) {
    const int len = p.lens[l];
    if (len >= 0 && len < p.cap[l]) p.lens[l] = len + 1;
  }
}

template <typename Tin, int D>
cudaError_t launch_d(const DecodeParams &p, cudaStream_t st) {
  switch (p.G) {
    case 1: decode_partial<Tin, D, 1><<<p.total_items, kThreads, 0, st>>>(p); break;
    case 2: decode_partial<Tin, D, 2><<<p.total_items, kThreads, 0, st>>>(p); break;
    case 4: decode_partial<Tin, D, 4><<<p.total_items, kThreads, 0, st>>>(p); break;
    case 8: decode_partial<Tin, D, 8><<<p.total_items, kThreads, 0, st>>>(p); break;
    default: return cudaErrorInvalidValue;
  }
  decode_combine<D><<<p.L * p.B * p.Hq, D, 0, st>>>(p);
  count_launches(2);
  return cudaGetLastError();
}

// Items and workspace floats for the given capacities.
static bool plan(const ripple_decode_desc *d, const int32_t *caps, DecodeParams *p,
                 size_t *ws_floats) {
  const int G = d->n_q_heads / d->n_kv_heads;
  size_t items = 0;
  for (int l = 0; l < d->n_layers; ++l) {
    if (caps[l] < 1) return false;
    const int nch = (caps[l] + kChunk - 1) / kChunk;
    if (p) {
      p->cap[l] = caps[l];
      p->nch[l] = nch;
      p->item_base[l] = (int)items;
    }
    items += (size_t)d->batch * d->n_kv_heads * nch;
  }
  if (items > (size_t)0x7fffffff) return false;
  if (p) {
    p->item_base[d->n_layers] = (int)items;
    p->total_items = (int)items;
  }
  *ws_floats = items * G * (2 + (size_t)d->head_dim);
  return true;
}

static bool desc_ok(const ripple_decode_desc *d) {
  if (d == nullptr) return false;
  if (d->n_layers < 1 || d->n_layers > RIPPLE_MAX_LAYERS) return false;
  if (d->batch < 1 || d->n_kv_heads < 1 || d->n_q_heads < 1) return false;
  if (d->n_q_heads % d->n_kv_heads != 0) return false;
  const int G = d->n_q_heads / d->n_kv_heads;
  if (G != 1 && G != 2 && G != 4 && G != 8) return false;
  if (d->head_dim != 64 && d->head_dim != 128) return false;
  if (d->dtype != RIPPLE_F32 && d->dtype != RIPPLE_BF16) return false;
  if (!(d->scale >= 0.f) || isinf(d->scale)) return false;
  return true;
}

static size_t round_up(size_t x) { return (x + 255) & ~(size_t)255; }

}  // namespace
}  // namespace ripple

using namespace ripple;

extern "C" ripple_status ripple_decode_workspace_bytes(const ripple_decode_desc *desc,
                                                       const int32_t *caps_host,
                                                       size_t *bytes_host) {
  if (!desc_ok(desc) || caps_host == nullptr || bytes_host == nullptr) return RIPPLE_EINVAL;
  size_t f;
  if (!plan(desc, caps_host, nullptr, &f)) return RIPPLE_EINVAL;
  *bytes_host = round_up(f * sizeof(float)) + 256;
  return RIPPLE_OK;
}

extern "C" ripple_status ripple_decode_attn(const ripple_decode_desc *desc, const void *q,
                                            const void *k_new, const void *v_new,
                                            void *const *k_caches_host,
                                            void *const *v_caches_host,
                                            const int32_t *caps_host, int32_t *lens, float *out,
                                            void *workspace, size_t workspace_bytes,
                                            int32_t *dev_status, void *stream) {
  if (!desc_ok(desc)) return RIPPLE_EINVAL;
  if (!q || !k_new || !v_new || !k_caches_host || !v_caches_host || !caps_host || !lens || !out ||
      !workspace)
    return RIPPLE_EINVAL;
  const int L = desc->n_layers;
  auto aligned = [](const void *ptr) { return ((uintptr_t)ptr & 15u) == 0; };
  if (!aligned(q) || !aligned(k_new) || !aligned(v_new) || !aligned(out) ||
      ((uintptr_t)workspace & 255u))
    return RIPPLE_EINVAL;
  DecodeParams p;
  for (int l = 0; l < L; ++l) {
    if (!k_caches_host[l] || !v_caches_host[l]) return RIPPLE_EINVAL;
    if (!aligned(k_caches_host[l]) || !aligned(v_caches_host[l])) return RIPPLE_EINVAL;
    p.kc[l] = k_caches_host[l];
    p.vc[l] = v_caches_host[l];
  }
  size_t f;
  if (!plan(desc, caps_host, &p, &f)) return RIPPLE_EINVAL;
  if (workspace_bytes < round_up(f * sizeof(float)) + 256) return RIPPLE_EWORKSPACE;
  p.L = L;
  p.B = desc->batch;
  p.Hq = desc->n_q_heads;
  p.Hkv = desc->n_kv_heads;
  p.G = p.Hq / p.Hkv;
  p.D = desc->head_dim;
  const float scale = desc->scale > 0.f ? desc->scale : 1.0f / sqrtf((float)p.D);
  p.scale2 = scale * kLog2e;
  p.q = q;
  p.k_new = k_new;
  p.v_new = v_new;
  p.lens = lens;
  p.out = out;
  p.status = dev_status;
  const size_t per = (size_t)p.total_items * p.G;
  p.ws_m = (float *)workspace;
  p.ws_l = p.ws_m + per;
  p.ws_o = p.ws_l + per;
  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e;
  if (desc->dtype == RIPPLE_F32)
    e = p.D == 64 ? launch_d<float, 64>(p, st) : launch_d<float, 128>(p, st);
  else
    e = p.D == 64 ? launch_d<__nv_bfloat16, 64>(p, st) : launch_d<__nv_bfloat16, 128>(p, st);
  return e == cudaSuccess ? RIPPLE_OK : RIPPLE_ECUDA;
}

// ---------------------------------------------------------------------------
// Decode for callers that cannot allocate device memory (no paper counterpart).
//
// A plugin inside a host program that owns all device memory through its own
// pool, or a fixed-footprint server that reserves every byte at start-up, may
// have no way to hand this library a scratch buffer. For those callers the
// split-K partials of a step live in the file-scope device array below
// instead of a caller workspace. Every GPU that loads the library keeps it
// until the process exits; all calls on a device share it and overwrite what
// the previous call left (the partials are fully rewritten by every step, so
// nothing needs clearing); calls that overlap on the GPU race on it.

static __device__ __align__(256) float
    g_decode_scratch[RIPPLE_DECODE_NOALLOC_SCRATCH_BYTES / sizeof(float)];

namespace {

constexpr int kMaxDevices = 256;
std::mutex g_scratch_mutex;
float *g_scratch_addr[kMaxDevices] = {};

// Device address of g_decode_scratch on the current device. In host code the
// array's name is only a host-side handle, so the address is looked up once
// per device (with that device current) and cached.
ripple_status scratch_on_current_device(float **out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return RIPPLE_ECUDA;
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (g_scratch_addr[dev] == nullptr) {
    void *ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_decode_scratch) != cudaSuccess || ptr == nullptr)
      return RIPPLE_ECUDA;
    g_scratch_addr[dev] = (float *)ptr;
  }
  *out = g_scratch_addr[dev];
  return RIPPLE_OK;
}

}  // namespace

extern "C" ripple_status ripple_decode_attn_noalloc(const ripple_decode_desc *desc, const void *q,
                                                    const void *k_new, const void *v_new,
                                                    void *const *k_caches_host,
                                                    void *const *v_caches_host,
                                                    const int32_t *caps_host, int32_t *lens,
                                                    float *out, int32_t *dev_status,
                                                    void *stream) {
  if (!desc_ok(desc)) return RIPPLE_EINVAL;
  if (!q || !k_new || !v_new || !k_caches_host || !v_caches_host || !caps_host || !lens || !out)
    return RIPPLE_EINVAL;
  const int L = desc->n_layers;
  auto aligned = [](const void *ptr) { return ((uintptr_t)ptr & 15u) == 0; };
  if (!aligned(q) || !aligned(k_new) || !aligned(v_new) || !aligned(out)) return RIPPLE_EINVAL;
  DecodeParams p;
  for (int l = 0; l < L; ++l) {
    if (!k_caches_host[l] || !v_caches_host[l]) return RIPPLE_EINVAL;
    if (!aligned(k_caches_host[l]) || !aligned(v_caches_host[l])) return RIPPLE_EINVAL;
    p.kc[l] = k_caches_host[l];
    p.vc[l] = v_caches_host[l];
  }
  size_t f;
  if (!plan(desc, caps_host, &p, &f)) return RIPPLE_EINVAL;
  if (f * sizeof(float) > RIPPLE_DECODE_NOALLOC_SCRATCH_BYTES) return RIPPLE_EWORKSPACE;
  float *scratch = nullptr;
  const ripple_status s = scratch_on_current_device(&scratch);
  if (s != RIPPLE_OK) return s;
  p.L = L;
  p.B = desc->batch;
  p.Hq = desc->n_q_heads;
  p.Hkv = desc->n_kv_heads;
  p.G = p.Hq / p.Hkv;
  p.D = desc->head_dim;
  const float scale = desc->scale > 0.f ? desc->scale : 1.0f / sqrtf((float)p.D);
  p.scale2 = scale * kLog2e;
  p.q = q;
  p.k_new = k_new;
  p.v_new = v_new;
  p.lens = lens;
  p.out = out;
  p.status = dev_status;
  const size_t per = (size_t)p.total_items * p.G;
  p.ws_m = scratch;
  p.ws_l = p.ws_m + per;
  p.ws_o = p.ws_l + per;
  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e;
  if (desc->dtype == RIPPLE_F32)
    e = p.D == 64 ? launch_d<float, 64>(p, st) : launch_d<float, 128>(p, st);
  else
    e = p.D == 64 ? launch_d<__nv_bfloat16, 64>(p, st) : launch_d<__nv_bfloat16, 128>(p, st);
  return e == cudaSuccess ? RIPPLE_OK : RIPPLE_ECUDA;
}
