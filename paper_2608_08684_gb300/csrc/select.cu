// Pooling of the prefix votes and exact top-k selection per unit (SnapKV's
// selection rule kept by RippleKV; retained set S_l of Eq. 4).
//
// One 1024-thread CTA per unit (b, h):
//   1. pooled score of every prefix token (max or mean over the clipped
//      window), mapped to an order-preserving uint32 key, kept in shared
//      memory when the prefix fits (global scratch otherwise);
//   2. radix select over the keys, 11 + 11 + 10 bits from the top, finds the
//      K-th largest key tau and how many keys equal to tau are kept;
//   3. an ordered compaction writes every token with key > tau and the first
//      tokens with key == tau (lower index wins ties) in ascending order,
//      followed by the w window positions P..T-1.
// The result is bit-exact and deterministic for a given vote array.
#include <math.h>

#include "common.cuh"
#include "kernels.cuh"

namespace ripple {
namespace {

constexpr int kThreads = kSelectThreads;
constexpr int kWarps = kThreads / 32;
constexpr int kBins = 2048;

// Order-preserving map float -> uint32 (larger float, larger key); -0 folds to +0.
__device__ __forceinline__ uint32_t order_key(float x) {
  const uint32_t b = __float_as_uint(x + 0.0f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

__device__ __forceinline__ float pooled_score(const float *v, int P, int t, int half, int type) {
  const int lo = max(0, t - half), hi = min(P - 1, t + half);
  if (type == RIPPLE_POOL_MAX) {
    float m = v[lo];
    for (int j = lo + 1; j <= hi; ++j) m = fmaxf(m, v[j]);
    return m;
  }
  if (type == RIPPLE_POOL_AVG) {
    float s = 0.f;
    for (int j = lo; j <= hi; ++j) s = __fadd_rn(s, v[j]);
    return __fdiv_rn(s, (float)(hi - lo + 1));
  }
  return v[t];
}

// Exclusive block-wide prefix sum of one int per thread; *total gets the sum.
__device__ __forceinline__ int block_exclusive_scan(int x, int *warp_tot, int *total) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  int incl = x;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) warp_tot[wid] = incl;
  __syncthreads();
  if (wid == 0) {
    int t = warp_tot[lane];
    int ti = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, ti, o);
      if (lane >= o) ti += y;
    }
    warp_tot[lane] = ti - t;  // exclusive warp offsets
    if (lane == 31) warp_tot[32] = ti;
  }
  __syncthreads();
  const int res = warp_tot[wid] + incl - x;
  *total = warp_tot[32];
  __syncthreads();
  return res;
}

__global__ void __launch_bounds__(kThreads) select_kernel(LayerGeom g, const float *votes,
                                                          uint32_t *keys_global, int n_keep,
                                                          int in_smem, int32_t *idx) {
  extern __shared__ uint32_t sm[];
  uint32_t *hist = sm;                              // [kBins]
  int *warp_tot = (int *)(sm + kBins);              // [33]
  int *ctrl = warp_tot + 40;                        // [8] control words
  uint32_t *keys = in_smem ? sm + kBins + 48 : keys_global + (size_t)blockIdx.x * g.P;

  const int unit = blockIdx.x;
  const int P = g.P, K = n_keep - g.W;
  const float *v = votes + (size_t)unit * P;
  int32_t *out = idx + (size_t)unit * n_keep;
  const int tid = threadIdx.x;

  for (int j = tid; j < g.W; j += kThreads) out[K + j] = P + j;
  if (K <= 0) return;
  if (K >= P) {
    for (int t = tid; t < P; t += kThreads) out[t] = t;
    return;
  }

  const int half = g.pool_kernel / 2;
  for (int t = tid; t < P; t += kThreads) keys[t] = order_key(pooled_score(v, P, t, half, g.pool_type));
  __syncthreads();

  // Radix select of the K-th largest key.
  uint32_t prefix = 0, mask = 0;
  int remaining = K;
  const int shifts[3] = {21, 10, 0};
  const int widths[3] = {11, 11, 10};
  for (int round = 0; round < 3; ++round) {
    const int shift = shifts[round];
    const uint32_t dmask = (1u << widths[round]) - 1u;
    for (int i = tid; i < kBins; i += kThreads) hist[i] = 0;
    __syncthreads();
    // Scores cluster in few bins: lanes with the same bin add once per warp.
    for (int base = 0; base < P; base += kThreads) {
      const int t = base + tid;
      const uint32_t u = t < P ? keys[t] : 0u;
      const bool hit = t < P && (u & mask) == prefix;
      const uint32_t bin = hit ? (u >> shift) & dmask : 0xffffffffu;
      const uint32_t peers = __match_any_sync(0xffffffffu, bin);
      if (hit && (threadIdx.x & 31) == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
    }
    __syncthreads();
    // Thread j owns digits 2047-2j and 2046-2j (descending).
    const int d0 = kBins - 1 - 2 * tid, d1 = d0 - 1;
    const int c0 = (int)hist[d0], c1 = (int)hist[d1];
    int total;
    const int above0 = block_exclusive_scan(c0 + c1, warp_tot, &total);
    const int above1 = above0 + c0;
    if (above0 < remaining && remaining <= above0 + c0) {
      ctrl[0] = d0;
      ctrl[1] = remaining - above0;
    } else if (above1 < remaining && remaining <= above1 + c1) {
      ctrl[0] = d1;
      ctrl[1] = remaining - above1;
    }
    __syncthreads();
    prefix |= (uint32_t)ctrl[0] << shift;
    mask |= dmask << shift;
    remaining = ctrl[1];
    __syncthreads();
  }
  const uint32_t tau = prefix;
  const int take_eq = remaining;  // keys equal to tau that are kept (>= 1)

  // Ordered compaction: all keys > tau, plus the first take_eq keys == tau.
  int carry_gt = 0, carry_eq = 0;
  for (int base = 0; base < P; base += kThreads) {
    const int t = base + tid;
    int gt = 0, eq = 0;
    if (t < P) {
      const uint32_t u = keys[t];
      gt = u > tau;
      eq = u == tau;
    }
    int total;
    const int before = block_exclusive_scan(gt | (eq << 16), warp_tot, &total);
    const int gt_before = before & 0xffff, eq_before = before >> 16;
    const int eq_rank = carry_eq + eq_before;
    if (gt || (eq && eq_rank < take_eq)) out[carry_gt + gt_before + min(eq_rank, take_eq)] = t;
    carry_gt += total & 0xffff;
    carry_eq += total >> 16;
    if (carry_gt + min(carry_eq, take_eq) >= K) break;
  }
}

}  // namespace

cudaError_t launch_select(const LayerGeom &g, const float *votes, const CompressWs &ws,
                          int n_keep, int32_t *idx, cudaStream_t st) {
  const int in_smem = g.P <= kSelectSmemKeys;
  const size_t smem = sizeof(uint32_t) * (kBins + 48 + (in_smem ? g.P : 0));
  cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  select_kernel<<<g.units, kThreads, smem, st>>>(g, votes, ws.keys, n_keep, in_smem, idx);
  count_launches(1);
  return cudaGetLastError();
}

__global__ void iota_kernel(int T, int32_t *idx) {
  for (int t = blockIdx.x * blockDim.x + threadIdx.x; t < T; t += gridDim.x * blockDim.x)
    idx[(size_t)blockIdx.y * T + t] = t;
}

cudaError_t launch_iota(const LayerGeom &g, int32_t *idx, cudaStream_t st) {
  iota_kernel<<<dim3((g.T + 255) / 256, g.units), 256, 0, st>>>(g.T, idx);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace ripple
