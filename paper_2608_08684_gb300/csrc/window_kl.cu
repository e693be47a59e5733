// Output divergence averaged over the evaluation window (Sec. 4.3, Eq. 7),
// one streaming pass over the perturbed runs' logits.
//
// For a reference row p (intact cache) and a perturbed row q over the
// vocabulary, with P = softmax(p), Q = softmax(q) and delta = q - p,
//   KL(P || Q) = log E_P[exp(delta)] - E_P[delta].
// Both terms are of the order of the perturbation while their difference is
// of its square, so the kernel does not subtract two log-partition functions.
// With a shift c and x = delta - c it forms, per logit, the positive series
// g(x) = exp(x) - 1 - x, and
//   E_P[exp(delta)] = exp(c) (1 + E_P[x] + E_P[g(x)]),
//   KL = log1p(E_P[x] + E_P[g(x)]) - E_P[x],
// so a small divergence keeps its relative precision.
//
// Work: every row is cut into slices of kKlSlice logits and every slice into
// kKlConsumerWarps shares, one per consumer warp (16 logits a lane). A share
// is reduced in fp32 to a KlPart: the largest p (mp), the sum of the weights
// w = exp(p - mp), c = delta at the first largest p, and the sums of w x and
// of w g(x) -- g by its Taylor polynomial when |x| <= kKlPolyBound across the
// share -- or, otherwise, of exp(q - r) for a reference r (kind 1).
// Work items are (position, slice, set) with the set innermost; one CTA per
// SM takes a contiguous run of items, so the items that share a reference
// slice follow one another: its logits and weights stay in the consumers'
// registers across the sets and p is read from HBM about once. A producer
// lane streams the q slices through a ring of bulk async (TMA) copies into
// shared memory. Consumer warps never wait on one another: each writes its
// partial to the workspace and goes on.
// kl_merge_kernel, a programmatic dependent launch of the stream kernel
// (its CTAs take SMs as the stream kernel's leave and wait until it has
// completed): one warp per row merges the row's partials in double, and the
// warp that completes a set's rows (atomic count; the stream kernel's CTA 0
// zeroes the counts) sums the window mean in double.
// Every wait is bounded (RIPPLE_ETIMEOUT). Every reduction has a fixed order:
// results do not depend on scheduling.
#include <float.h>
#include <limits.h>
#include <math.h>

#include "common.cuh"
#include "kernels.cuh"

namespace ripple {
namespace {

constexpr int kKlConsumerWarps = 16;
constexpr int kKlThreads = (kKlConsumerWarps + 1) * 32;  // + one producer warp
constexpr int kKlShareThreads = kKlConsumerWarps * 32;
constexpr int kKlSlice = 8192;               // logits per work item
constexpr int kKlStageBytes = kKlSlice * 4;  // a fp32 slice
constexpr int kKlStages = 4;                 // q ring: 128 KB in flight
constexpr float kKlPolyBound = 0.5f;         // |x| bound of the Taylor form of g
constexpr int kKlMergeWarps = 4;             // rows per merge CTA

// A consumer thread's part of a share: CH chunks of V16 logits (16 bytes);
// chunk k of thread t starts at logit (k * kKlShareThreads + t) * V16 of the
// slice (16-byte shared-memory reads without bank conflicts).
template <typename Tl>
struct KlCfg {
  static constexpr int V16 = 16 / (int)sizeof(Tl);
  static constexpr int CH = kKlSlice / (kKlShareThreads * V16);
  static constexpr int E = CH * V16;  // 16 logits
};

// One consumer warp's share of a slice of a row (see the file comment).
struct KlPart {
  float mp;  // largest p of the share; -inf when the share holds no logit
  float zp;  // sum of w = exp(p - mp)
  float c;   // delta at the share's first largest p
  float a;   // sum of w x, x = delta - c
  float b;   // kind 0: sum of w g(x); kind 1: sum of exp(q - r)
  float r;   // kind 1: the reference r
  int kind;  // 0: every |x| <= kKlPolyBound; 1: otherwise
  int pad;
};
static_assert(sizeof(KlPart) == 32, "two 16-byte stores");

struct KlParams {
  const void *p;      // [n_pos][vocab]
  const void *q;      // [n_sets][n_pos][vocab]
  int n_sets, n_pos, vocab, n_slices;
  long long n_items;  // n_sets * n_pos * n_slices
  KlPart *part;       // [n_sets * n_pos][n_slices * kKlConsumerWarps]
  double *row_kl;     // [n_sets * n_pos]
  int *set_count;     // [n_sets] rows merged per set
  float *kl_out;      // [n_sets][n_pos] or NULL
  float *d_out;       // [n_sets]
  int32_t *status;
  long long wait_cycles;
};

struct KlSmem {
  alignas(128) uint8_t q[kKlStages][kKlStageBytes];
  alignas(128) uint8_t p[2][kKlStageBytes];
  uint64_t q_full[kKlStages], q_empty[kKlStages], p_full[2], p_empty[2];
  int abort_flag;
};

// Butterflies over the 32 lanes: every lane ends with the same value (max and
// rounded adds are symmetric in their operands).
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
__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = __dadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
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

// g(x) / x^2 = 1/2 + x/6 + ... + x^6/8! (Horner); the first omitted term is
// below 5e-8 of g for |x| <= 1/2.
__device__ __forceinline__ float2 g_over_x2(float2 x) {
  float2 h = __ffma2_rn(x, make_float2(1.f / 40320.f, 1.f / 40320.f),
                        make_float2(1.f / 5040.f, 1.f / 5040.f));
  h = __ffma2_rn(x, h, make_float2(1.f / 720.f, 1.f / 720.f));
  h = __ffma2_rn(x, h, make_float2(1.f / 120.f, 1.f / 120.f));
  h = __ffma2_rn(x, h, make_float2(1.f / 24.f, 1.f / 24.f));
  h = __ffma2_rn(x, h, make_float2(1.f / 6.f, 1.f / 6.f));
  return __ffma2_rn(x, h, make_float2(0.5f, 0.5f));
}

// log1p(t) - t without cancellation: with s = t / (2 + t), log1p(t) =
// 2 atanh(s) and 2 s - t = -t s, so
//   log1p(t) - t = -t s + 2 s^3 (1/3 + s^2/5 + s^4/7 + ... + s^10/13);
// for |t| <= 1/2 (|s| <= 1/3) the first omitted term is below 1e-7 of the
// result. Larger |t| directly.
__device__ __forceinline__ float log1p_minus_t(float t) {
  if (!(fabsf(t) <= 0.5f)) return __fsub_rn(log1pf(t), t);
  const float s = __fdiv_rn(t, __fadd_rn(2.f, t));
  const float s2 = __fmul_rn(s, s);
  float h = __fmaf_rn(s2, 1.f / 13.f, 1.f / 11.f);
  h = __fmaf_rn(s2, h, 1.f / 9.f);
  h = __fmaf_rn(s2, h, 1.f / 7.f);
  h = __fmaf_rn(s2, h, 1.f / 5.f);
  h = __fmaf_rn(s2, h, 1.f / 3.f);
  return __fmaf_rn(__fmul_rn(__fmul_rn(2.f, s), s2), h, -__fmul_rn(t, s));
}

// This thread's part of a share staged in shared memory. Chunks past the
// slice's length (a multiple of 8, so a chunk is wholly in or out) read as 0
// and are flagged in the returned mask (bit k: chunk k holds logits).
template <typename Tl, bool kFull>
__device__ __forceinline__ uint32_t read_share(const uint8_t *stage, int ctid, int len,
                                               float (&x)[KlCfg<Tl>::E]) {
  using C = KlCfg<Tl>;
  const Tl *src = reinterpret_cast<const Tl *>(stage);
  uint32_t ok = 0;
#pragma unroll
  for (int k = 0; k < C::CH; ++k) {
    const int i = (k * kKlShareThreads + ctid) * C::V16;
    const bool in = kFull || i < len;
    ok |= (in ? 1u : 0u) << k;
    if (in) {
      if constexpr (C::V16 == 8) {
        float t[8];
        load8(src + i, t);
#pragma unroll
        for (int j = 0; j < 8; ++j) x[k * 8 + j] = t[j];
      } else {
        const float4 t = *reinterpret_cast<const float4 *>(src + i);
        x[k * 4 + 0] = t.x;
        x[k * 4 + 1] = t.y;
        x[k * 4 + 2] = t.z;
        x[k * 4 + 3] = t.w;
      }
    } else {
#pragma unroll
      for (int j = 0; j < C::V16; ++j) x[k * C::V16 + j] = 0.f;
    }
  }
  return ok;
}

// Reference share of a slice: logits pv, weights w = exp(p - mp) (0 outside
// the slice), the warp's largest p mp and weight sum zp, and the slice
// offset of the first largest p (-1 when the share holds no logit).
template <typename Tl, bool kFull>
__device__ __forceinline__ void p_share(const uint8_t *stage, int ctid, int len,
                                        float (&pv)[KlCfg<Tl>::E], float (&w)[KlCfg<Tl>::E],
                                        float &mp, float &zp, int &istar) {
  using C = KlCfg<Tl>;
  const uint32_t ok = read_share<Tl, kFull>(stage, ctid, len, pv);
  float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
  for (int k = 0; k < C::CH; ++k)
    if (kFull || (ok >> k & 1u))
#pragma unroll
      for (int j = 0; j < C::V16; ++j) m4[j & 3] = fmaxf(m4[j & 3], pv[k * C::V16 + j]);
  mp = warp_max_all(fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])));
  float z4[4] = {0.f, 0.f, 0.f, 0.f};
  int first = INT_MAX;
  // descending offsets, so that `first` ends at the lane's lowest one
#pragma unroll
  for (int k = C::CH - 1; k >= 0; --k)
#pragma unroll
    for (int j = C::V16 - 1; j >= 0; --j) {
      const int e = k * C::V16 + j;
      const bool in = kFull || (ok >> k & 1u);
      w[e] = in ? fast_exp2(__fmul_rn(__fsub_rn(pv[e], mp), kLog2e)) : 0.f;
      z4[j & 3] = __fadd_rn(z4[j & 3], w[e]);
      if (in && pv[e] == mp) first = (k * kKlShareThreads + ctid) * C::V16 + j;
    }
  zp = warp_sum_rn(__fadd_rn(__fadd_rn(z4[0], z4[1]), __fadd_rn(z4[2], z4[3])));
  const int f = __reduce_min_sync(0xffffffffu, first);
  istar = f == INT_MAX ? -1 : f;
}

// Sum over the thread's logits in the slice of exp(q - r), then over the warp.
template <typename Tl, bool kFull>
__device__ __forceinline__ float q_exp_sum(const float (&qv)[KlCfg<Tl>::E], uint32_t ok, float r) {
  using C = KlCfg<Tl>;
  float2 y2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
  for (int e = 0; e < C::E; e += 2) {
    const bool in = kFull || (ok >> (e / C::V16) & 1u);
    const float2 t = __fmul2_rn(__fadd2_rn(make_float2(qv[e], qv[e + 1]), make_float2(-r, -r)),
                                make_float2(kLog2e, kLog2e));
    const float2 u = in ? make_float2(fast_exp2(t.x), fast_exp2(t.y)) : make_float2(0.f, 0.f);
    y2[(e >> 1) & 1] = __fadd2_rn(y2[(e >> 1) & 1], u);
  }
  return warp_sum_rn(__fadd_rn(__fadd_rn(y2[0].x, y2[0].y), __fadd_rn(y2[1].x, y2[1].y)));
}

// One work item: the warp's share of a q slice against the reference share
// held in registers. The ring stage is released as soon as the share and q
// at the largest p are in registers. Every lane returns the same partial.
template <typename Tl, bool kFull>
__device__ __forceinline__ KlPart q_share(const uint8_t *stage, uint64_t *empty, int ctid,
                                          int lane, int len, const float (&pv)[KlCfg<Tl>::E],
                                          const float (&w)[KlCfg<Tl>::E], float mp, float zp,
                                          int istar) {
  using C = KlCfg<Tl>;
  constexpr int E = C::E;
  float qv[E];
  const uint32_t ok = read_share<Tl, kFull>(stage, ctid, len, qv);
  const float qs = istar >= 0 ? to_f32(reinterpret_cast<const Tl *>(stage)[istar]) : 0.f;
  __syncwarp();
  if (lane == 0) mbar_arrive(empty);

  KlPart r;
  r.mp = mp;
  r.zp = zp;
  r.pad = 0;
  const float c = istar >= 0 ? __fsub_rn(qs, mp) : 0.f;  // p at istar is mp
  r.c = c;
  // x = (q - p) - c; q - p rounded once (a fused multiply-add by -1)
  float x[E];
  float mx4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int e = 0; e < E; e += 2) {
    const bool in = kFull || (ok >> (e / C::V16) & 1u);
    float2 t = __ffma2_rn(make_float2(pv[e], pv[e + 1]), make_float2(-1.f, -1.f),
                          make_float2(qv[e], qv[e + 1]));
    t = __fadd2_rn(t, make_float2(-c, -c));
    x[e] = in ? t.x : 0.f;
    x[e + 1] = in ? t.y : 0.f;
    mx4[(e >> 1) & 3] = fmaxf(mx4[(e >> 1) & 3], fmaxf(fabsf(x[e]), fabsf(x[e + 1])));
  }
  const float mabs = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3]));
  float2 a2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
  if (__all_sync(0xffffffffu, mabs <= kKlPolyBound)) {
    float2 b2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
    for (int e = 0; e < E; e += 2) {
      const float2 x2 = make_float2(x[e], x[e + 1]), w2 = make_float2(w[e], w[e + 1]);
      a2[(e >> 1) & 1] = __ffma2_rn(w2, x2, a2[(e >> 1) & 1]);
      const float2 g = __fmul2_rn(__fmul2_rn(x2, x2), g_over_x2(x2));
      b2[(e >> 1) & 1] = __ffma2_rn(w2, g, b2[(e >> 1) & 1]);
    }
    r.kind = 0;
    r.r = 0.f;
    r.b = warp_sum_rn(__fadd_rn(__fadd_rn(b2[0].x, b2[0].y), __fadd_rn(b2[1].x, b2[1].y)));
  } else {
    // Some |x| above the bound (so istar >= 0): the sum of exp(q - r) with
    // r = q at the largest p (its own term is 1), or, where that sum
    // overflows, r = the largest q.
#pragma unroll
    for (int e = 0; e < E; e += 2)
      a2[(e >> 1) & 1] = __ffma2_rn(make_float2(w[e], w[e + 1]), make_float2(x[e], x[e + 1]),
                                    a2[(e >> 1) & 1]);
    float ref = qs;
    float y = q_exp_sum<Tl, kFull>(qv, ok, ref);
    if (!(y <= FLT_MAX)) {
      float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
      for (int e = 0; e < E; ++e)
        if (kFull || (ok >> (e / C::V16) & 1u)) m4[e & 3] = fmaxf(m4[e & 3], qv[e]);
      ref = warp_max_all(fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])));
      y = q_exp_sum<Tl, kFull>(qv, ok, ref);
    }
    r.kind = 1;
    r.r = ref;
    r.b = y;
  }
  r.a = warp_sum_rn(__fadd_rn(__fadd_rn(a2[0].x, a2[0].y), __fadd_rn(a2[1].x, a2[1].y)));
  return r;
}

// KL(P || Q) of one row from its n partials (read from L2); every lane
// returns the same value. With M the largest mp, C the c of its first
// partial and, per partial, f = exp(mp - M), dc = c - C, e = exp(dc) - 1:
//   Zp = sum f zp                                   (the row's weight sum),
//   U  = sum f (a + dc zp)                          (Zp E_P[delta - C]),
//   V  = sum f ((e - dc) zp + e (a + b) + b)        (Zp E_P[g(delta - C)]),
// every term of V of the order of the perturbation's square; with u = U / Zp,
// v = V / Zp and t = u + v:
//   KL = log1p(t) - u = v + (log1p(t) - t),
// which holds while every partial is of kind 0 and every |dc| <= kKlPolyBound.
// Otherwise E_P[exp(delta - C)] is summed from the partials' masses in the
// log2 domain (relative to the largest, so nothing overflows). Sums per lane
// in fp32, over the lanes in double; the final scalar, free of cancellation,
// in fp32.
// Partial k of a row as two float4: (mp, zp, c, a) and (b, r, kind, -).
struct KlRaw {
  float4 x, y;
};
__device__ __forceinline__ KlRaw load_part(const KlPart *rp, int k, int n) {
  KlRaw r;
  if (k < n) {
    r.x = __ldcg(reinterpret_cast<const float4 *>(rp + k));
    r.y = __ldcg(reinterpret_cast<const float4 *>(rp + k) + 1);
  } else {
    r.x = make_float4(-INFINITY, 0.f, 0.f, 0.f);  // empty
    r.y = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  return r;
}

// Rows of up to kKlMergeCached * 32 partials (vocabularies up to 16 slices,
// 131072 logits) are read once into registers; longer rows are read per pass.
constexpr int kKlMergeCached = 8;

template <bool kCached>
__device__ __forceinline__ double merge_row(const KlPart *rp, int n, int lane) {
  constexpr int kSpan = kCached ? kKlMergeCached * 32 : 0x7fffffff;  // one pass when cached
  KlRaw c[kKlMergeCached];
  if constexpr (kCached) {
#pragma unroll
    for (int r = 0; r < kKlMergeCached; ++r) c[r] = load_part(rp, r * 32 + lane, n);
  }
  float mloc = -INFINITY, cloc = 0.f;
  int kloc = INT_MAX, kinds = 0;
  for (int base = 0; base < n && base < kSpan; base += kKlMergeCached * 32)
#pragma unroll
    for (int r = 0; r < kKlMergeCached; ++r) {
      const KlRaw q = (kCached ? c[r] : load_part(rp, base + r * 32 + lane, n));
      if (q.x.x > mloc) {  // ascending k: the lane's first largest
        mloc = q.x.x;
        kloc = base + r * 32 + lane;
        cloc = q.x.z;
      }
      kinds |= __float_as_int(q.y.z);
    }
  const float M = warp_max_all(mloc);
  const int kc = __reduce_min_sync(0xffffffffu, mloc == M ? kloc : INT_MAX);
  const float C = __shfl_sync(0xffffffffu, cloc, kc & 31);  // c of partial kc
  float zp = 0.f, uu = 0.f, vv = 0.f;
  bool far = kinds != 0;
  for (int base = 0; base < n && base < kSpan; base += kKlMergeCached * 32)
#pragma unroll
    for (int r = 0; r < kKlMergeCached; ++r) {
      const KlRaw q = (kCached ? c[r] : load_part(rp, base + r * 32 + lane, n));
      if (q.x.x == -INFINITY) continue;
      const float f = fast_exp2(__fmul_rn(__fsub_rn(q.x.x, M), kLog2e));
      const float dc = __fsub_rn(q.x.z, C);
      zp = __fmaf_rn(f, q.x.y, zp);
      uu = __fmaf_rn(f, __fmaf_rn(dc, q.x.y, q.x.w), uu);
      if (fabsf(dc) <= kKlPolyBound) {
        const float g = __fmul_rn(__fmul_rn(dc, dc), g_over_x2(make_float2(dc, dc)).x);
        const float e = __fadd_rn(dc, g);
        vv = __fmaf_rn(f, __fmaf_rn(g, q.x.y, __fmaf_rn(e, __fadd_rn(q.x.w, q.y.x), q.y.x)), vv);
      } else {
        far = true;
      }
    }
  const double Zp = warp_sum_d((double)zp);
  const double U = warp_sum_d((double)uu);
  const float zpf = (float)Zp;
  if (!__any_sync(0xffffffffu, far)) {
    const double V = warp_sum_d((double)vv);
    const float v = __fdiv_rn((float)V, zpf), t = __fdiv_rn((float)(U + V), zpf);
    return (double)__fadd_rn(v, log1p_minus_t(t));
  }

  // log2 of each partial's mass sum_i w_i exp(delta_i - C) times f; a running
  // maximum per lane, then one over the warp
  float lm = -INFINITY, s = 0.f;
  for (int base = 0; base < n && base < kSpan; base += kKlMergeCached * 32)
#pragma unroll
    for (int r = 0; r < kKlMergeCached; ++r) {
      const KlRaw q = (kCached ? c[r] : load_part(rp, base + r * 32 + lane, n));
      if (q.x.x == -INFINITY) continue;
      float l;
      if (__float_as_int(q.y.z) == 0) {
        const float m = __fadd_rn(__fadd_rn(q.x.y, q.x.w), q.y.x);  // zp + a + b
        if (!(m > 0.f)) continue;
        l = __fmaf_rn(__fadd_rn(__fsub_rn(q.x.x, M), __fsub_rn(q.x.z, C)), kLog2e, log2f(m));
      } else {
        l = __fmaf_rn(__fsub_rn(__fsub_rn(q.y.y, M), C), kLog2e, log2f(q.y.x));
      }
      if (l > lm) {
        s = lm == -INFINITY ? 0.f : __fmul_rn(s, fast_exp2(__fsub_rn(lm, l)));
        lm = l;
      }
      s = __fadd_rn(s, fast_exp2(__fsub_rn(l, lm)));
    }
  const float LM = warp_max_all(lm);
  const double S = warp_sum_d(lm == -INFINITY ? 0.0 : (double)s * (double)fast_exp2(lm - LM));
  // log(S 2^LM / Zp) - U / Zp; S >= 1 and Zp >= 1 (the largest terms are 1)
  const float l2 = __fadd_rn(__fsub_rn(LM, log2f(zpf)), log2f((float)S));
  return (double)__fsub_rn(__fmul_rn(l2, 0.69314718f), __fdiv_rn((float)U, zpf));
}

// Item i = ((pos * n_slices) + slice) * n_sets + set.
struct KlItem {
  int set, pos, slice;
  __device__ __forceinline__ KlItem(const KlParams &P, long long i) {
    const long long g = i / P.n_sets;
    set = (int)(i - g * P.n_sets);
    pos = (int)(g / P.n_slices);
    slice = (int)(g - (long long)pos * P.n_slices);
  }
  __device__ __forceinline__ void next(const KlParams &P) {
    if (++set == P.n_sets) {
      set = 0;
      if (++slice == P.n_slices) {
        slice = 0;
        ++pos;
      }
    }
  }
};

// Producer lane: the p slice when the run of sets starts, then the q slice of
// every item, through bulk async copies.
template <typename Tl>
__device__ __forceinline__ void kl_produce(const KlParams &P, KlSmem &s, long long i0,
                                           long long i1) {
  const Tl *p = (const Tl *)P.p, *q = (const Tl *)P.q;
  uint32_t qc = 0, pc = 0;
  KlItem it(P, i0);
  for (long long item = i0; item < i1; ++item, it.next(P)) {
    const int begin = it.slice * kKlSlice;
    const uint32_t bytes = (uint32_t)(min(kKlSlice, P.vocab - begin) * (int)sizeof(Tl));
    if (item == i0 || it.set == 0) {
      const int ps = pc & 1;
      if (!kl_wait(&s.p_empty[ps], ((pc >> 1) & 1) ^ 1, &s.abort_flag, P.status, P.wait_cycles))
        break;
      mbar_arrive_expect_tx(&s.p_full[ps], bytes);
      const long long po = guard((long long)it.pos * P.vocab + begin, bytes / sizeof(Tl),
                                 (long long)P.n_pos * P.vocab, P.status);
      bulk_g2s(s.p[ps], p + po, bytes, &s.p_full[ps]);
      ++pc;
    }
    const int st = qc % kKlStages;
    if (!kl_wait(&s.q_empty[st], ((qc / kKlStages) & 1) ^ 1, &s.abort_flag, P.status,
                 P.wait_cycles))
      break;
    mbar_arrive_expect_tx(&s.q_full[st], bytes);
    const long long qo = guard(((long long)it.set * P.n_pos + it.pos) * P.vocab + begin,
                               bytes / sizeof(Tl), (long long)P.n_sets * P.n_pos * P.vocab,
                               P.status);
    bulk_g2s(s.q[st], q + qo, bytes, &s.q_full[st]);
    ++qc;
  }
  // Copies still in flight must land before the CTA exits (after an abort;
  // otherwise the consumers have already seen every phase complete).
  for (uint32_t j = qc > (uint32_t)kKlStages ? qc - kKlStages : 0; j < qc; ++j) {
    int never = 0;
    kl_wait(&s.q_full[j % kKlStages], (j / kKlStages) & 1, &never, P.status, kDefaultWaitCycles);
  }
  for (uint32_t j = pc > 2u ? pc - 2 : 0; j < pc; ++j) {
    int never = 0;
    kl_wait(&s.p_full[j & 1], (j >> 1) & 1, &never, P.status, kDefaultWaitCycles);
  }
}

// Consumer warp: its share of every item of the CTA's run.
template <typename Tl>
__device__ __forceinline__ void kl_consume(const KlParams &P, KlSmem &s, int warp, int lane,
                                           long long i0, long long i1) {
  using C = KlCfg<Tl>;
  const int ctid = warp * 32 + lane;
  const int n_parts = P.n_slices * kKlConsumerWarps;
  float pv[C::E], w[C::E];
  float mp = -INFINITY, zp = 0.f;
  int istar = -1;
  uint32_t qc = 0, pc = 0;
  KlItem it(P, i0);
  for (long long item = i0; item < i1; ++item, it.next(P)) {
    const int len = min(kKlSlice, P.vocab - it.slice * kKlSlice);
    if (item == i0 || it.set == 0) {
      const int ps = pc & 1;
      if (!__all_sync(0xffffffffu, kl_wait(&s.p_full[ps], (pc >> 1) & 1, &s.abort_flag,
                                            P.status, P.wait_cycles)))
        break;
      if (len == kKlSlice)
        p_share<Tl, true>(s.p[ps], ctid, len, pv, w, mp, zp, istar);
      else
        p_share<Tl, false>(s.p[ps], ctid, len, pv, w, mp, zp, istar);
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.p_empty[ps]);
      ++pc;
    }
    const int st = qc % kKlStages;
    if (!__all_sync(0xffffffffu, kl_wait(&s.q_full[st], (qc / kKlStages) & 1, &s.abort_flag,
                                          P.status, P.wait_cycles)))
      break;
    const KlPart r =
        len == kKlSlice
            ? q_share<Tl, true>(s.q[st], &s.q_empty[st], ctid, lane, len, pv, w, mp, zp, istar)
            : q_share<Tl, false>(s.q[st], &s.q_empty[st], ctid, lane, len, pv, w, mp, zp,
                                 istar);
    ++qc;
    if (lane == 0) {
      float4 *dst = reinterpret_cast<float4 *>(
          P.part + guard(((long long)it.set * P.n_pos + it.pos) * n_parts +
                             it.slice * kKlConsumerWarps + warp,
                         1, (long long)P.n_sets * P.n_pos * n_parts, P.status));
      dst[0] = make_float4(r.mp, r.zp, r.c, r.a);
      dst[1] = make_float4(r.b, r.r, __int_as_float(r.kind), 0.f);
    }
  }
}

template <typename Tl>
__global__ void __launch_bounds__(kKlThreads, 1)
    kl_window_kernel(const __grid_constant__ KlParams P) {
  extern __shared__ __align__(128) uint8_t smem_raw[];
  KlSmem &s = *reinterpret_cast<KlSmem *>(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long i0 = P.n_items * blockIdx.x / gridDim.x;
  const long long i1 = P.n_items * (blockIdx.x + 1) / gridDim.x;
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
    if (lane == 0) {
      kl_produce<Tl>(P, s, i0, i1);
    } else if (blockIdx.x == 0) {
      // the other producer lanes of CTA 0 zero the merge kernel's counts
      for (int i = lane - 1; i < P.n_sets; i += 31) P.set_count[i] = 0;
    }
  } else {
    kl_consume<Tl>(P, s, warp, lane, i0, i1);
  }
}

// One warp per row: KL of the row from its partials, then, for the warp that
// completes its set's rows, the window mean. Launched as a programmatic
// dependent of the stream kernel: griddepcontrol.wait returns once that grid
// has completed and its writes (partials, zeroed counts) are visible.
// kCached: the row's partials fit kKlMergeCached per lane.
template <bool kCached>
__global__ void __launch_bounds__(kKlMergeWarps * 32)
    kl_merge_kernel(const __grid_constant__ KlParams P) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * kKlMergeWarps + (threadIdx.x >> 5);
  if (row >= P.n_sets * P.n_pos) return;
  const int set = row / P.n_pos;
  const int n_parts = P.n_slices * kKlConsumerWarps;
  const long long rows = (long long)P.n_sets * P.n_pos;
  const double kl = merge_row<kCached>(
      P.part + guard((long long)row * n_parts, n_parts, rows * n_parts, P.status), n_parts, lane);
  int old = 0;
  if (lane == 0) {
    P.row_kl[guard(row, 1, rows, P.status)] = kl;
    if (P.kl_out != nullptr) P.kl_out[guard(row, 1, rows, P.status)] = (float)kl;
    __threadfence();
    old = atomicAdd(&P.set_count[guard(set, 1, P.n_sets, P.status)], 1);
  }
  if (__shfl_sync(0xffffffffu, old, 0) != P.n_pos - 1) return;
  __threadfence();
  double s = 0.0;
  const long long r0 = guard((long long)set * P.n_pos, P.n_pos, rows, P.status);
  for (int t = lane; t < P.n_pos; t += 32) s += __ldcg(&P.row_kl[r0 + t]);
  s = warp_sum_d(s);
  if (lane == 0) P.d_out[guard(set, 1, P.n_sets, P.status)] = (float)(s / (double)P.n_pos);
}

// ------------------------------------------------------------ host side

int kl_slices(int vocab) { return (vocab + kKlSlice - 1) / kKlSlice; }

size_t round256(size_t x) { return (x + 255) & ~(size_t)255; }

// Workspace carve-up: set counts, row divergences, partials.
size_t carve_kl(int n_sets, int n_pos, int vocab, void *base, KlParams *P) {
  const size_t rows = (size_t)n_sets * n_pos;
  uint8_t *b = (uint8_t *)base;
  size_t off = 0;
  if (P) P->set_count = (int *)(b + off);
  off += round256((size_t)n_sets * sizeof(int));
  if (P) P->row_kl = (double *)(b + off);
  off += round256(rows * sizeof(double));
  if (P) P->part = (KlPart *)(b + off);
  off += round256(rows * (size_t)kl_slices(vocab) * kKlConsumerWarps * sizeof(KlPart));
  return off;
}

template <typename Tl>
cudaError_t launch_kl(const KlParams &P, cudaStream_t st) {
  auto kernel = kl_window_kernel<Tl>;
  const int smem = (int)sizeof(KlSmem);
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0;
  e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  const int grid = (int)(P.n_items < sms ? P.n_items : sms);  // one CTA per SM
  kernel<<<grid, kKlThreads, smem, st>>>(P);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const long long rows = (long long)P.n_sets * P.n_pos;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((rows + kKlMergeWarps - 1) / kKlMergeWarps));
  cfg.blockDim = dim3(kKlMergeWarps * 32);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 0;
  e = P.n_slices * kKlConsumerWarps <= kKlMergeCached * 32
          ? cudaLaunchKernelEx(&cfg, kl_merge_kernel<true>, P)
          : cudaLaunchKernelEx(&cfg, kl_merge_kernel<false>, P);
  count_launches(2);
  return e;
}

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

}  // namespace
}  // namespace ripple

using namespace ripple;

extern "C" ripple_status ripple_window_kl_workspace_bytes(int32_t n_sets, int32_t n_pos,
                                                          int32_t vocab, size_t *bytes_host) {
  if (bytes_host == nullptr || n_sets < 1 || n_pos < 1 || vocab < 1 || vocab % 8 != 0)
    return RIPPLE_EINVAL;
  if ((long long)n_sets * n_pos > 0x7fffffffLL) return RIPPLE_EINVAL;
  *bytes_host = carve_kl(n_sets, n_pos, vocab, nullptr, nullptr);
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
  if (workspace_bytes < need) return RIPPLE_EWORKSPACE;
  KlParams P{};
  P.p = p_logits;
  P.q = q_logits;
  P.n_sets = n_sets;
  P.n_pos = n_pos;
  P.vocab = vocab;
  P.n_slices = kl_slices(vocab);
  P.n_items = (long long)n_sets * n_pos * P.n_slices;
  carve_kl(n_sets, n_pos, vocab, workspace, &P);
  P.kl_out = kl_out;
  P.d_out = d_out;
  P.status = dev_status;
  P.wait_cycles = wait_limit_cycles();
  cudaStream_t st = (cudaStream_t)stream;
  const cudaError_t e =
      dtype == RIPPLE_BF16 ? launch_kl<__nv_bfloat16>(P, st) : launch_kl<float>(P, st);
  RIPPLE_CUDA_TRY(e);
  return RIPPLE_OK;
}
