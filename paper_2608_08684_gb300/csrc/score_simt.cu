// Observation-window token scoring on the fp32 pipes (SnapKV rule kept by
// RippleKV, Sec. 4.4 last paragraph). Used for fp32 caches, where running the
// contraction on tf32 tensor cores would spend the score tolerance.
//
// Two passes over each unit's keys, both in key chunks of kScoreChunk:
//   pass 1: per window row, (max, sum of exp) over the chunk's visible keys;
//   merge : per row, combine the chunk partials into max + log2(sum);
//   pass 2: per prefix key, sum over rows of exp2(x - lognorm_row).
// All arithmetic in the log2 domain: x = scale * log2(e) * q.k.
#include <math.h>

#include "common.cuh"
#include "kernels.cuh"

namespace ripple {
namespace {

constexpr int kThreads = 256;
constexpr int kRowsPerGroup = 32;  // window rows per inner iteration
constexpr int kKeysPerThread = kScoreChunk / 8;

// Loads the chunk's keys (fp32, padded rows) and returns the number loaded.
template <typename Tin, int D>
__device__ void load_keys(const Tin *k_unit, int T, int key0, float *Ks) {
  constexpr int kPieces = D / 8;
  for (int e = threadIdx.x; e < kScoreChunk * kPieces; e += kThreads) {
    const int row = e / kPieces, piece = e % kPieces;
    float v[8];
    if (key0 + row < T) {
      load8(k_unit + (size_t)(key0 + row) * D + piece * 8, v);
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = 0.f;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) Ks[row * (D + 1) + piece * 8 + i] = v[i];
  }
}

template <typename Tin, int D>
__device__ void load_rows(const Tin *q_unit, int R, int row0, float *Qs) {
  constexpr int kPieces = D / 8;
  for (int e = threadIdx.x; e < kRowsPerGroup * kPieces; e += kThreads) {
    const int row = e / kPieces, piece = e % kPieces;
    float v[8];
    if (row0 + row < R) {
      load8(q_unit + (size_t)(row0 + row) * D + piece * 8, v);
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = 0.f;
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) Qs[row * (D + 1) + piece * 8 + i] = v[i];
  }
}

// acc[m] = q_row . k_{tk + 8m} for the thread's row and keys.
template <int D>
__device__ __forceinline__ void dot_block(const float *Qs, const float *Ks, int tr, int tk,
                                          float (&acc)[kKeysPerThread]) {
#pragma unroll
  for (int m = 0; m < kKeysPerThread; ++m) acc[m] = 0.f;
#pragma unroll 4
  for (int c = 0; c < D; ++c) {
    const float qv = Qs[tr * (D + 1) + c];
#pragma unroll
    for (int m = 0; m < kKeysPerThread; ++m) acc[m] = fmaf(qv, Ks[(tk + 8 * m) * (D + 1) + c], acc[m]);
  }
}

__device__ __forceinline__ void combine(float &m, float &l, float m2, float l2) {
  const float mm = fmaxf(m, m2);
  if (mm == -INFINITY) return;
  l = l * exp2f(m - mm) + l2 * exp2f(m2 - mm);
  m = mm;
}

template <typename Tin, int D>
__global__ void __launch_bounds__(kThreads) score_pass1_simt(LayerGeom g, const Tin *q_win,
                                                             const Tin *k, float2 *partial,
                                                             int32_t *status) {
  extern __shared__ float smem[];
  float *Ks = smem;
  float *Qs = smem + kScoreChunk * (D + 1);
  const int unit = blockIdx.y, chunk = blockIdx.x, n_chunks = gridDim.x;
  const int b = unit / g.Hkv, h = unit % g.Hkv;
  const Tin *k_unit = k + (size_t)unit * g.T * D;
  const Tin *q_unit = q_win + ((size_t)b * g.Hq + (size_t)h * g.G) * g.W * D;
  const int key0 = chunk * kScoreChunk;
  load_keys<Tin, D>(k_unit, g.T, key0, Ks);
  const int tr = threadIdx.x >> 3, tk = threadIdx.x & 7;
  for (int row0 = 0; row0 < g.R; row0 += kRowsPerGroup) {
    __syncthreads();
    load_rows<Tin, D>(q_unit, g.R, row0, Qs);
    __syncthreads();
    float acc[kKeysPerThread];
    dot_block<D>(Qs, Ks, tr, tk, acc);
    const int r = row0 + tr;
    const int last_visible = g.P + (r % g.W);  // causal inside the window
    float m = -INFINITY;
#pragma unroll
    for (int j = 0; j < kKeysPerThread; ++j) {
      const int t = key0 + tk + 8 * j;
      acc[j] *= g.scale2;
      if (t < g.T && t <= last_visible) m = fmaxf(m, acc[j]);
    }
    float l = 0.f;
    if (m != -INFINITY) {
#pragma unroll
      for (int j = 0; j < kKeysPerThread; ++j) {
        const int t = key0 + tk + 8 * j;
        if (t < g.T && t <= last_visible) l += exp2f(acc[j] - m);
      }
    }
#pragma unroll
    for (int o = 1; o < 8; o <<= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
      const float l2 = __shfl_xor_sync(0xffffffffu, l, o);
      combine(m, l, m2, l2);
    }
    if (tk == 0 && r < g.R)
      partial[guard(((long long)unit * n_chunks + chunk) * g.R + r, 1,
                    (long long)g.units * n_chunks * g.R, status)] = make_float2(m, l);
  }
}

__global__ void merge_row_stats(LayerGeom g, int n_chunks, const float2 *partial, float *lognorm,
                                int32_t *status) {
  const int unit = blockIdx.x;
  for (int r = threadIdx.x; r < g.R; r += blockDim.x) {
    float m = -INFINITY, l = 0.f;
    for (int c = 0; c < n_chunks; ++c) {
      const float2 p = partial[((size_t)unit * n_chunks + c) * g.R + r];
      combine(m, l, p.x, p.y);
    }
    lognorm[guard((long long)unit * g.R + r, 1, (long long)g.units * g.R, status)] = m + log2f(l);
  }
}

template <typename Tin, int D>
__global__ void __launch_bounds__(kThreads) score_pass2_simt(LayerGeom g, const Tin *q_win,
                                                             const Tin *k, const float *lognorm,
                                                             float *votes, int32_t *status) {
  extern __shared__ float smem[];
  float *Ks = smem;
  float *Qs = smem + kScoreChunk * (D + 1);
  float *red = Qs + kRowsPerGroup * (D + 1);  // [32][kScoreChunk + 1]
  const int unit = blockIdx.y, chunk = blockIdx.x;
  const int b = unit / g.Hkv, h = unit % g.Hkv;
  const Tin *k_unit = k + (size_t)unit * g.T * D;
  const Tin *q_unit = q_win + ((size_t)b * g.Hq + (size_t)h * g.G) * g.W * D;
  const float *ln = lognorm + (size_t)unit * g.R;
  const int key0 = chunk * kScoreChunk;
  load_keys<Tin, D>(k_unit, g.T, key0, Ks);
  const int tr = threadIdx.x >> 3, tk = threadIdx.x & 7;
  float vote[kKeysPerThread];
#pragma unroll
  for (int j = 0; j < kKeysPerThread; ++j) vote[j] = 0.f;
  for (int row0 = 0; row0 < g.R; row0 += kRowsPerGroup) {
    __syncthreads();
    load_rows<Tin, D>(q_unit, g.R, row0, Qs);
    __syncthreads();
    float acc[kKeysPerThread];
    dot_block<D>(Qs, Ks, tr, tk, acc);
    const int r = row0 + tr;
    if (r < g.R) {
      const float off = ln[r];
#pragma unroll
      for (int j = 0; j < kKeysPerThread; ++j) vote[j] += exp2f(fmaf(acc[j], g.scale2, -off));
    }
  }
  // Sum over the 32 row slots of each key in a fixed order.
#pragma unroll
  for (int j = 0; j < kKeysPerThread; ++j) red[tr * (kScoreChunk + 1) + tk + 8 * j] = vote[j];
  __syncthreads();
  if (threadIdx.x < kScoreChunk) {
    const int t = key0 + threadIdx.x;
    float s = 0.f;
    for (int i = 0; i < kRowsPerGroup; ++i) s += red[i * (kScoreChunk + 1) + threadIdx.x];
    if (t < g.P) votes[guard((long long)unit * g.P + t, 1, (long long)g.units * g.P, status)] = s;
  }
}

template <typename Tin, int D>
cudaError_t launch_typed(const LayerGeom &g, const void *q_win, const void *k,
                         const CompressWs &ws, float *votes, int32_t *status, cudaStream_t st) {
  const size_t smem1 = sizeof(float) * (kScoreChunk + kRowsPerGroup) * (D + 1);
  const size_t smem2 = smem1 + sizeof(float) * kRowsPerGroup * (kScoreChunk + 1);
  cudaError_t e;
  e = cudaFuncSetAttribute(score_pass1_simt<Tin, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem1);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(score_pass2_simt<Tin, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem2);
  if (e != cudaSuccess) return e;
  const int n_chunks = (g.T + kScoreChunk - 1) / kScoreChunk;
  score_pass1_simt<Tin, D><<<dim3(n_chunks, g.units), kThreads, smem1, st>>>(
      g, (const Tin *)q_win, (const Tin *)k, ws.row_partial, status);
  merge_row_stats<<<g.units, 256, 0, st>>>(g, n_chunks, ws.row_partial, ws.row_lognorm, status);
  const int n_chunks2 = (g.P + kScoreChunk - 1) / kScoreChunk;
  if (n_chunks2 > 0)
    score_pass2_simt<Tin, D><<<dim3(n_chunks2, g.units), kThreads, smem2, st>>>(
        g, (const Tin *)q_win, (const Tin *)k, ws.row_lognorm, votes, status);
  count_launches(n_chunks2 > 0 ? 3 : 2);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_score_simt(const LayerGeom &g, const void *q_win, const void *k,
                              const CompressWs &ws, float *votes, int32_t *status,
                              cudaStream_t st) {
  if (g.dtype == RIPPLE_F32) {
    if (g.D == 64) return launch_typed<float, 64>(g, q_win, k, ws, votes, status, st);
    return launch_typed<float, 128>(g, q_win, k, ws, votes, status, st);
  }
  if (g.D == 64) return launch_typed<__nv_bfloat16, 64>(g, q_win, k, ws, votes, status, st);
  return launch_typed<__nv_bfloat16, 128>(g, q_win, k, ws, votes, status, st);
}

}  // namespace ripple
