// Offline sensitivity profiling on the GPU (Sec. 4.3): the norm-adaptive Value
// perturbation of one layer (Eq. 6) and the KL divergence of the output
// distribution averaged over the evaluation window (Eq. 7). Both are single
// streaming passes over HBM.
//
// perturb_kernel: a cache row of d channels is spread over d/4 lanes (four
//   channels each: 8-byte bf16 or 16-byte fp32 loads, plus 16 bytes of draws);
//   the squared norm is summed by shuffles among the row's lanes. Each warp
//   issues the loads of kPerturbUnroll row groups before any arithmetic.
// kl_stream_kernel: every logits row is cut into slices of kKlSlice entries;
//   each consumer warp reduces its share of every (set, position, slice) item
//   to the softmax statistics of p, (max, sum of exp, P-weighted p - q), and
//   of q, (max, sum of exp). One CTA per SM takes a contiguous run of items
//   ordered with the set innermost: a producer lane streams the q slices
//   through a ring of bulk async (TMA) copies into shared memory, and the
//   consumer warps keep the shared reference slice p and exp(p - max) in
//   registers across the sets, so p is read from HBM about once and its
//   exponentials computed once.
//   Each warp writes its own partial per item (no CTA-wide barrier).
// kl_combine_kernel: one CTA per set, a warp per window position merges the
//   position's partials, and a fixed-order sum gives the window mean.
// Every reduction has a fixed order: results do not depend on scheduling.
#include <math.h>

#include "common.cuh"
#include "kernels.cuh"

namespace ripple {
namespace {

constexpr int kPerturbThreads = 256;
constexpr int kPerturbUnroll = 4;
constexpr int kKlConsumerWarps = 8;
constexpr int kKlThreads = (kKlConsumerWarps + 1) * 32;  // + one producer warp
constexpr int kKlSlice = 8192;                           // logits per work item
constexpr int kKlStageBytes = kKlSlice * 4;              // a fp32 slice
constexpr int kKlStages = 4;                             // q ring: 128 KB in flight
constexpr int kKlCombineThreads = 1024;

// A consumer thread's share of a slice: CH chunks of V16 logits (16 bytes).
template <typename Tl>
struct KlCfg {
  static constexpr int V16 = 16 / (int)sizeof(Tl);
  static constexpr int CH = kKlSlice / (kKlConsumerWarps * 32 * V16);
  static constexpr int E = CH * V16;  // 32 logits
};

// Softmax statistics of one consumer warp's share of a slice (1024 logits),
// relative to that share's maxima.
struct KlPart {
  float mp, zp, ap;  // max p, sum exp(p - mp), sum exp(p - mp) * (p - q)
  float mq, zq;      // max q, sum exp(q - mq)
  float pad[3];
};

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

// Merge of two (max, sum, weighted sum) triples; an empty side has max -inf.
// Explicit roundings (no contraction into fused multiply-adds): the p and q
// statistics go through the same operations, so identical rows give
// identical sums; and the merge is symmetric, so a butterfly leaves the same
// result in every lane.
__device__ __forceinline__ void merge_stats(float &m, float &z, float &a, float m2, float z2,
                                            float a2) {
  const float nm = fmaxf(m, m2);
  if (nm == -INFINITY) return;
  const float f1 = fast_exp2(__fmul_rn(__fsub_rn(m, nm), kLog2e));
  const float f2 = fast_exp2(__fmul_rn(__fsub_rn(m2, nm), kLog2e));
  z = __fadd_rn(__fmul_rn(z, f1), __fmul_rn(z2, f2));
  a = __fadd_rn(__fmul_rn(a, f1), __fmul_rn(a2, f2));
  m = nm;
}

// Butterflies over the 32 lanes (every lane ends with the same value: max
// and a rounded add are symmetric in their operands).
__device__ __forceinline__ float warp_max_all(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum_rn(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Bounded mbarrier wait; gives up when another role has given up, or after
// `limit` cycles (then raises the abort flag and reports RIPPLE_ETIMEOUT).
__device__ __forceinline__ bool kl_wait(uint64_t *bar, uint32_t parity, int *abort_flag,
                                        int32_t *status, long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*(volatile int *)abort_flag) return false;
    if (clock64() - t0 > limit) {
      *(volatile int *)abort_flag = 1;
      report(status, RIPPLE_ETIMEOUT);
      return false;
    }
  }
}

struct KlSmem {
  alignas(128) uint8_t q[kKlStages][kKlStageBytes];
  alignas(128) uint8_t p[2][kKlStageBytes];
  uint64_t q_full[kKlStages], q_empty[kKlStages], p_full[2], p_empty[2];
  int abort_flag;
};

// This thread's share of a slice staged in shared memory: chunk c holds the
// V16 logits from (c * 256 + ctid) * V16 (16-byte reads, no bank conflicts).
// ok[c] is false for chunks past the slice's length (a multiple of 8, so a
// chunk is wholly in or out); their values are not read.
template <typename Tl>
__device__ __forceinline__ void read_share(const uint8_t *stage, int ctid, int len,
                                           float (&x)[KlCfg<Tl>::E], bool (&ok)[KlCfg<Tl>::CH]) {
  using C = KlCfg<Tl>;
  const Tl *src = reinterpret_cast<const Tl *>(stage);
#pragma unroll
  for (int c = 0; c < C::CH; ++c) {
    const int i = (c * kKlConsumerWarps * 32 + ctid) * C::V16;
    ok[c] = i < len;
#pragma unroll
    for (int j = 0; j < C::V16; ++j) x[c * C::V16 + j] = 0.f;
    if (ok[c]) {
      if constexpr (C::V16 == 8) {
        float t[8];
        load8(src + i, t);
#pragma unroll
        for (int j = 0; j < 8; ++j) x[c * 8 + j] = t[j];
      } else {
        const float4 t = *reinterpret_cast<const float4 *>(src + i);
        x[c * 4 + 0] = t.x;
        x[c * 4 + 1] = t.y;
        x[c * 4 + 2] = t.z;
        x[c * 4 + 3] = t.w;
      }
    }
  }
}

// Softmax statistics of the warp's share of a slice: m = the warp's maximum,
// z = sum over the valid logits of exp(x - m) (four accumulators per lane,
// then a butterfly); with kStore the exponentials are kept in ex. The p and q
// shares go through exactly these operations, so identical rows give
// identical statistics.
template <typename Tl, bool kStore>
__device__ __forceinline__ void share_stats(const float (&x)[KlCfg<Tl>::E],
                                            const bool (&ok)[KlCfg<Tl>::CH], float &m, float &z,
                                            float (&ex)[KlCfg<Tl>::E]) {
  using C = KlCfg<Tl>;
  float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
  for (int c = 0; c < C::CH; ++c)
    if (ok[c])
#pragma unroll
      for (int j = 0; j < C::V16; ++j) m4[j & 3] = fmaxf(m4[j & 3], x[c * C::V16 + j]);
  m = warp_max_all(fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])));
  float z4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int c = 0; c < C::CH; ++c)
#pragma unroll
    for (int j = 0; j < C::V16; ++j) {
      const int e = c * C::V16 + j;
      // x - m is exact near the maximum, where the terms matter
      const float t = ok[c] ? fast_exp2(__fmul_rn(__fsub_rn(x[e], m), kLog2e)) : 0.f;
      if (kStore) ex[e] = t;
      if (ok[c]) z4[j & 3] = __fadd_rn(z4[j & 3], t);
    }
  z = warp_sum_rn(__fadd_rn(__fadd_rn(z4[0], z4[1]), __fadd_rn(z4[2], z4[3])));
}

// Eq. 7, first stage, streamed. Work items are (pos, slice, set) with the set
// innermost; CTA b takes a contiguous range of items, so the items that share
// a reference slice p[pos][slice] follow one another and the consumers keep
// that slice and exp(p - max) in registers across the sets. One lane of warp
// 8 streams the q slices through a kKlStages ring of bulk async copies, and
// the p slices through two slots. part: [n_sets][n_pos][n_slices][8] per-warp
// statistics.
template <typename Tl>
__global__ void __launch_bounds__(kKlThreads, 1)
    kl_stream_kernel(const Tl *__restrict__ p, const Tl *__restrict__ q, int n_sets, int n_pos,
                     int vocab, int n_slices, long long n_items, KlPart *part, int32_t *status,
                     long long wait_cycles) {
  using C = KlCfg<Tl>;
  extern __shared__ __align__(128) uint8_t smem_raw[];
  KlSmem &s = *reinterpret_cast<KlSmem *>(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long i0 = n_items * blockIdx.x / gridDim.x;
  const long long i1 = n_items * (blockIdx.x + 1) / gridDim.x;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kKlStages; ++i) {
      mbar_init(&s.q_full[i], 1);
      mbar_init(&s.q_empty[i], kKlConsumerWarps);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.p_full[i], 1);
      mbar_init(&s.p_empty[i], kKlConsumerWarps);
    }
    s.abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();

  if (warp == kKlConsumerWarps) {
    // ------------------------------------------------------------- producer
    if (lane != 0) return;
    uint32_t qc = 0, pc = 0;
    for (long long item = i0; item < i1; ++item) {
      const long long g = item / n_sets;
      const int set = (int)(item - g * n_sets);
      const int pos = (int)(g / n_slices), slice = (int)(g - (long long)pos * n_slices);
      const int begin = slice * kKlSlice;
      const uint32_t bytes = (uint32_t)(min(kKlSlice, vocab - begin) * (int)sizeof(Tl));
      if (item == i0 || set == 0) {
        const int ps = pc & 1;
        if (!kl_wait(&s.p_empty[ps], ((pc >> 1) & 1) ^ 1, &s.abort_flag, status, wait_cycles)) break;
        mbar_arrive_expect_tx(&s.p_full[ps], bytes);
        bulk_g2s(s.p[ps], p + (size_t)pos * vocab + begin, bytes, &s.p_full[ps]);
        ++pc;
      }
      const int st = qc % kKlStages;
      if (!kl_wait(&s.q_empty[st], ((qc / kKlStages) & 1) ^ 1, &s.abort_flag, status, wait_cycles)) break;
      mbar_arrive_expect_tx(&s.q_full[st], bytes);
      bulk_g2s(s.q[st], q + ((size_t)set * n_pos + pos) * vocab + begin, bytes, &s.q_full[st]);
      ++qc;
    }
    // Copies still in flight must land before the CTA exits (after an abort;
    // otherwise the consumers have already seen every phase complete).
    for (uint32_t j = qc > (uint32_t)kKlStages ? qc - kKlStages : 0; j < qc; ++j) {
      int never = 0;
      kl_wait(&s.q_full[j % kKlStages], (j / kKlStages) & 1, &never, status, kDefaultWaitCycles);
    }
    for (uint32_t j = pc > 2u ? pc - 2 : 0; j < pc; ++j) {
      int never = 0;
      kl_wait(&s.p_full[j & 1], (j >> 1) & 1, &never, status, kDefaultWaitCycles);
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  // Each warp reduces its share (1024 logits) of every item on its own, with
  // exponentials relative to the warp's maximum, and writes one partial per
  // item: no CTA-wide barrier in this loop.
  const int ctid = threadIdx.x;
  float pv[C::E], ep[C::E];
  bool pok[C::CH];
  float MPw = -INFINITY, ZPw = 0.f;  // the warp's share of the reference slice
  uint32_t qc = 0, pc = 0;
  for (long long item = i0; item < i1; ++item) {
    const long long g = item / n_sets;
    const int set = (int)(item - g * n_sets);
    const int pos = (int)(g / n_slices), slice = (int)(g - (long long)pos * n_slices);
    const int len = min(kKlSlice, vocab - slice * kKlSlice);
    if (item == i0 || set == 0) {
      const int ps = pc & 1;
      if (!__all_sync(0xffffffffu, kl_wait(&s.p_full[ps], (pc >> 1) & 1, &s.abort_flag, status, wait_cycles)))
        break;
      read_share<Tl>(s.p[ps], ctid, len, pv, pok);
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.p_empty[ps]);
      ++pc;
      share_stats<Tl, true>(pv, pok, MPw, ZPw, ep);
    }
    const int st = qc % kKlStages;
    if (!__all_sync(0xffffffffu,
                    kl_wait(&s.q_full[st], (qc / kKlStages) & 1, &s.abort_flag, status, wait_cycles)))
      break;
    float qv[C::E];
    bool qok[C::CH];
    read_share<Tl>(s.q[st], ctid, len, qv, qok);
    __syncwarp();
    if (lane == 0) mbar_arrive(&s.q_empty[st]);
    ++qc;
    float MQw, ZQw, unused[C::E];
    share_stats<Tl, false>(qv, qok, MQw, ZQw, unused);
    float a4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int c = 0; c < C::CH; ++c)
      if (qok[c])
#pragma unroll
        for (int j = 0; j < C::V16; ++j) {
          const int e = c * C::V16 + j;
          a4[j & 3] = fmaf(ep[e], pv[e] - qv[e], a4[j & 3]);
        }
    const float APw = warp_sum_rn(__fadd_rn(__fadd_rn(a4[0], a4[1]), __fadd_rn(a4[2], a4[3])));
    if (lane == 0) {
      KlPart r;
      r.mp = MPw;
      r.zp = ZPw;
      r.ap = APw;
      r.mq = MQw;
      r.zq = ZQw;
      r.pad[0] = r.pad[1] = r.pad[2] = 0.f;
      part[(((size_t)set * n_pos + pos) * n_slices + slice) * kKlConsumerWarps + warp] = r;
    }
  }
}

// Eq. 7, second stage: per set (one CTA), a warp per window position merges
// the position's partials (one per slice and consumer warp; lane i takes
// partials i, i + 32, ...; then a butterfly), and the window mean is summed
// over the warps in a fixed order.
//   KL = E_P[p - q] - lse(p) + lse(q) = ap / zp + (mq - mp) + log(zq / zp)
// All in fp32 (the three terms are formed from sums with relative errors
// near 1e-6 already); the window mean is accumulated in double.
__global__ void __launch_bounds__(kKlCombineThreads) kl_combine_kernel(const KlPart *part,
                                                                       int n_pos, int n_parts,
                                                                       float *kl_out,
                                                                       float *d_out) {
  __shared__ double red[kKlCombineThreads / 32];
  const int set = blockIdx.x, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  double acc = 0.0;
  for (int pos = warp; pos < n_pos; pos += kKlCombineThreads / 32) {
    const long long row = (long long)set * n_pos + pos;
    float mp = -INFINITY, zp = 0.f, ap = 0.f, mq = -INFINITY, zq = 0.f;
    for (int j = lane; j < n_parts; j += 32) {
      const KlPart x = part[row * n_parts + j];
      merge_stats(mp, zp, ap, x.mp, x.zp, x.ap);
      float unused = 0.f;
      merge_stats(mq, zq, unused, x.mq, x.zq, 0.f);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, mp, o);
      const float z2 = __shfl_xor_sync(0xffffffffu, zp, o);
      const float a2 = __shfl_xor_sync(0xffffffffu, ap, o);
      const float mq2 = __shfl_xor_sync(0xffffffffu, mq, o);
      const float zq2 = __shfl_xor_sync(0xffffffffu, zq, o);
      merge_stats(mp, zp, ap, m2, z2, a2);
      float unused = 0.f;
      merge_stats(mq, zq, unused, mq2, zq2, 0.f);
    }
    const float kl = __fadd_rn(__fadd_rn(__fdiv_rn(ap, zp), __fsub_rn(mq, mp)),
                               logf(__fdiv_rn(zq, zp)));
    if (lane == 0 && kl_out != nullptr) kl_out[row] = kl;
    acc += (double)kl;
  }
  if (lane == 0) red[warp] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < kKlCombineThreads / 32; ++w) t += red[w];
    d_out[set] = (float)(t / (double)n_pos);
  }
}

int kl_slices(int vocab) { return (vocab + kKlSlice - 1) / kKlSlice; }

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

template <typename Tl>
cudaError_t launch_kl(const void *p, const void *q, int n_sets, int n_pos, int vocab,
                      float *kl_out, float *d_out, KlPart *part, int32_t *status,
                      cudaStream_t st) {
  const int n_slices = kl_slices(vocab);
  const long long n_items = (long long)n_sets * n_pos * n_slices;
  auto kernel = kl_stream_kernel<Tl>;
  const int smem = (int)sizeof(KlSmem);
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0;
  e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const int grid = (int)(n_items < sms ? n_items : sms);  // one CTA per SM
  kernel<<<grid, kKlThreads, smem, st>>>((const Tl *)p, (const Tl *)q, n_sets, n_pos, vocab,
                                         n_slices, n_items, part, status, wait_limit_cycles());
  kl_combine_kernel<<<n_sets, kKlCombineThreads, 0, st>>>(part, n_pos,
                                                          n_slices * kKlConsumerWarps, kl_out,
                                                          d_out);
  count_launches(2);
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

extern "C" ripple_status ripple_window_kl_workspace_bytes(int32_t n_sets, int32_t n_pos,
                                                          int32_t vocab, size_t *bytes_host) {
  if (bytes_host == nullptr || n_sets < 1 || n_pos < 1 || vocab < 1 || vocab % 8 != 0)
    return RIPPLE_EINVAL;
  const size_t b = sizeof(KlPart) * (size_t)n_sets * (size_t)n_pos * (size_t)kl_slices(vocab) *
                   kKlConsumerWarps;
  *bytes_host = (b + 255) & ~(size_t)255;
  return RIPPLE_OK;
}

extern "C" ripple_status ripple_window_kl(const void *p_logits, const void *q_logits,
                                          int32_t n_sets, int32_t n_pos, int32_t vocab,
                                          int32_t dtype, float *kl_out, float *d_out,
                                          void *workspace, size_t workspace_bytes,
                                          int32_t *dev_status, void *stream) {
  size_t need = 0;
  if (ripple_window_kl_workspace_bytes(n_sets, n_pos, vocab, &need) != RIPPLE_OK)
    return RIPPLE_EINVAL;
  if (dtype != RIPPLE_F32 && dtype != RIPPLE_BF16) return RIPPLE_EINVAL;
  if (p_logits == nullptr || q_logits == nullptr || d_out == nullptr || workspace == nullptr)
    return RIPPLE_EINVAL;
  if (!aligned16(p_logits) || !aligned16(q_logits) || ((uintptr_t)workspace & 255u) ||
      ((uintptr_t)d_out & 3u) || ((uintptr_t)kl_out & 3u))
    return RIPPLE_EINVAL;
  if ((long long)n_sets * n_pos > 0x7fffffffLL) return RIPPLE_EINVAL;
  if (workspace_bytes < need) return RIPPLE_EWORKSPACE;
  cudaStream_t st = (cudaStream_t)stream;
  KlPart *part = (KlPart *)workspace;
  const cudaError_t e =
      dtype == RIPPLE_BF16
          ? launch_kl<__nv_bfloat16>(p_logits, q_logits, n_sets, n_pos, vocab, kl_out, d_out,
                                     part, dev_status, st)
          : launch_kl<float>(p_logits, q_logits, n_sets, n_pos, vocab, kl_out, d_out, part,
                             dev_status, st);
  RIPPLE_CUDA_TRY(e);
  return RIPPLE_OK;
}
