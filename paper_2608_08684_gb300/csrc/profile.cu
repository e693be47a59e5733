// Offline sensitivity profiling on the GPU (Sec. 4.3): the norm-adaptive Value
// perturbation of one layer (Eq. 6), a single streaming pass over HBM (the
// window divergence of Eq. 7 is in window_kl.cu).
//
// perturb_kernel: a cache row of d channels is spread over d/4 lanes (four
//   channels each: 8-byte bf16 or 16-byte fp32 loads, plus 16 bytes of draws);
//   the squared norm is summed by shuffles among the row's lanes. Each warp
//   issues the loads of kPerturbUnroll row groups before any arithmetic.
#include <math.h>

#include "common.cuh"
#include "kernels.cuh"

namespace ripple {
namespace {

constexpr int kPerturbThreads = 256;
constexpr int kPerturbUnroll = 4;

__device__ __forceinline__ void load4(const float *p, float (&x)[4]) {
  const float4 a = *reinterpret_cast<const float4 *>(p);
  x[0] = a.x;
  x[1] = a.y;
  x[2] = a.z;
  x[3] = a.w;
}
__device__ __forceinline__ void load4(const __nv_bfloat16 *p, float (&x)[4]) {
  const uint2 u = *reinterpret_cast<const uint2 *>(p);
  const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&u.x));
  const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&u.y));
  x[0] = a.x;
  x[1] = a.y;
  x[2] = b.x;
  x[3] = b.y;
}
__device__ __forceinline__ void store4(float *p, const float (&x)[4]) {
  *reinterpret_cast<float4 *>(p) = make_float4(x[0], x[1], x[2], x[3]);
}
__device__ __forceinline__ void store4(__nv_bfloat16 *p, const float (&x)[4]) {
  __nv_bfloat162 a = __floats2bfloat162_rn(x[0], x[1]);
  __nv_bfloat162 b = __floats2bfloat162_rn(x[2], x[3]);
  uint2 u;
  u.x = *reinterpret_cast<uint32_t *>(&a);
  u.y = *reinterpret_cast<uint32_t *>(&b);
  *reinterpret_cast<uint2 *>(p) = u;
}

// Eq. 6 over the rows (unit, u) of a cache, unit = b * Hkv + h. With
// all_rows every row of the cache is visited (out of place: rows outside
// [pos_begin, pos_begin + n_range) are copied); otherwise only the eligible
// rows are (in place). n_rows < 2^31.
template <typename Tv, int D>
__global__ void __launch_bounds__(kPerturbThreads) perturb_kernel(
    const Tv *__restrict__ v, const float *__restrict__ eps, Tv *v_out, float alpha, int T,
    int pos_begin, int n_range, int n_rows, int all_rows) {
  constexpr int kLanes = D / 4;  // lanes per row
  constexpr int kRowsPerWarp = 32 / kLanes;
  const int lane = threadIdx.x & 31;
  const int sub = lane / kLanes, c0 = (lane % kLanes) * 4;
  const int n_groups = (n_rows + kRowsPerWarp - 1) / kRowsPerWarp;
  const int warp = (int)((blockIdx.x * (unsigned)kPerturbThreads + threadIdx.x) >> 5);
  const int n_warps = (int)((gridDim.x * (unsigned)kPerturbThreads) >> 5);
  for (long long g0 = warp; g0 < n_groups; g0 += (long long)n_warps * kPerturbUnroll) {
    float x[kPerturbUnroll][4], e[kPerturbUnroll][4];
    size_t off[kPerturbUnroll];
    bool live[kPerturbUnroll], pert[kPerturbUnroll];
#pragma unroll
    for (int k = 0; k < kPerturbUnroll; ++k) {
      const long long g = g0 + (long long)k * n_warps;
      const long long r64 = g * kRowsPerWarp + sub;
      live[k] = r64 < n_rows;
      const unsigned r = live[k] ? (unsigned)r64 : 0u;
      unsigned unit, u, erow;
      bool in_range;
      if (all_rows) {
        unit = r / (unsigned)T;
        u = r - unit * (unsigned)T;
        in_range = u >= (unsigned)pos_begin && u < (unsigned)(pos_begin + n_range);
        erow = in_range ? unit * (unsigned)n_range + (u - (unsigned)pos_begin) : 0u;
      } else {
        unit = r / (unsigned)n_range;
        u = (unsigned)pos_begin + (r - unit * (unsigned)n_range);
        in_range = true;
        erow = r;
      }
      pert[k] = live[k] && in_range;
      off[k] = ((size_t)unit * T + u) * D + c0;
#pragma unroll
      for (int i = 0; i < 4; ++i) x[k][i] = e[k][i] = 0.f;
      if (live[k]) load4(v + off[k], x[k]);
      if (pert[k]) load4(eps + (size_t)erow * D + c0, e[k]);
    }
#pragma unroll
    for (int k = 0; k < kPerturbUnroll; ++k) {
      float ss = x[k][0] * x[k][0];
      ss += x[k][1] * x[k][1];
      ss += x[k][2] * x[k][2];
      ss += x[k][3] * x[k][3];
#pragma unroll
      for (int o = kLanes / 2; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
      if (pert[k]) {
        const float s = alpha * sqrtf(ss);  // alpha * ||v_u||_2
        float y[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) y[i] = x[k][i] + s * e[k][i];
        store4(v_out + off[k], y);
      } else if (live[k]) {
        store4(v_out + off[k], x[k]);
      }
    }
  }
}

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

// Resident CTAs of `kernel` over the whole device (SMs x CTAs per SM).
template <typename K>
cudaError_t device_slots(K kernel, int threads, int *slots) {
  int dev = 0, sms = 0, per_sm = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, 0);
  *slots = sms * (per_sm > 0 ? per_sm : 1);
  return e;
}

template <typename Tv, int D>
cudaError_t launch_perturb(const void *v, const float *eps, void *v_out, float alpha, int T,
                           int pos_begin, int n_range, int n_rows, int all_rows,
                           cudaStream_t st) {
  auto kernel = perturb_kernel<Tv, D>;
  int slots = 0;
  cudaError_t e = device_slots(kernel, kPerturbThreads, &slots);
  if (e != cudaSuccess) return e;
  constexpr int kRowsPerBlock = (kPerturbThreads / 32) * (128 / D);
  const long long want = ((long long)n_rows + kRowsPerBlock - 1) / kRowsPerBlock;
  const int grid = (int)(want < slots ? want : slots);
  kernel<<<grid, kPerturbThreads, 0, st>>>((const Tv *)v, eps, (Tv *)v_out, alpha, T, pos_begin,
                                          n_range, n_rows, all_rows);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace
}  // namespace ripple

using namespace ripple;

extern "C" ripple_status ripple_perturb_values(const ripple_cache_desc *desc, const void *v,
                                               const float *eps, float alpha,
                                               int32_t pos_begin, int32_t pos_end,
                                               void *v_out, void *stream) {
  if (desc == nullptr || v == nullptr || v_out == nullptr) return RIPPLE_EINVAL;
  const ripple_cache_desc d = *desc;
  if (d.batch < 1 || d.n_kv_heads < 1 || d.seq_len < 1) return RIPPLE_EINVAL;
  if (d.head_dim != 64 && d.head_dim != 128) return RIPPLE_EINVAL;
  if (d.dtype != RIPPLE_F32 && d.dtype != RIPPLE_BF16) return RIPPLE_EINVAL;
  if (pos_begin < 0 || pos_end < pos_begin || pos_end > d.seq_len) return RIPPLE_EINVAL;
  if (!(alpha >= 0.f) || isinf(alpha)) return RIPPLE_EINVAL;
  const long long units = (long long)d.batch * d.n_kv_heads;
  const long long all = units * d.seq_len;
  if (all > 0x7fffffffLL) return RIPPLE_EINVAL;
  const int n_range = pos_end - pos_begin;
  if (n_range > 0 && eps == nullptr) return RIPPLE_EINVAL;
  if (!aligned16(v) || !aligned16(v_out) || (eps != nullptr && !aligned16(eps)))
    return RIPPLE_EINVAL;
  const bool in_place = (v == v_out);
  const int n_rows = in_place ? (int)(units * n_range) : (int)all;
  if (n_rows == 0) return RIPPLE_OK;
  const int all_rows = in_place ? 0 : 1;
  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e;
  if (d.dtype == RIPPLE_BF16)
    e = d.head_dim == 128
            ? launch_perturb<__nv_bfloat16, 128>(v, eps, v_out, alpha, d.seq_len, pos_begin,
                                                 n_range, n_rows, all_rows, st)
            : launch_perturb<__nv_bfloat16, 64>(v, eps, v_out, alpha, d.seq_len, pos_begin,
                                                n_range, n_rows, all_rows, st);
  else
    e = d.head_dim == 128 ? launch_perturb<float, 128>(v, eps, v_out, alpha, d.seq_len,
                                                       pos_begin, n_range, n_rows, all_rows, st)
                          : launch_perturb<float, 64>(v, eps, v_out, alpha, d.seq_len,
                                                      pos_begin, n_range, n_rows, all_rows, st);
  RIPPLE_CUDA_TRY(e);
  return RIPPLE_OK;
}
