// GQA decode attention over the ragged compressed caches (Sec. 4.1: each new
// query attends to the cached states), with the append of the new token.
//
// One persistent launch per step covers every layer; one CTA per SM with 16
// compute warps and one producer warp. Work item = up to kItemSub sub-chunks
// of one (layer, batch row, KV head) group's cache rows; items are fetched
// with an atomic counter, layers with the longest caches first (longest-
// processing-time order). The producer warp stages each sub-chunk's K and V
// rows in shared memory with bulk-async (TMA engine) copies, two stages
// deep plus an L2 prefetch further ahead, and writes the new token's rows into
// the stage (and appends them to the cache). Every compute warp owns CR/16
// rows of each sub-chunk and keeps its
// own online-softmax state, so no block-wide barrier is needed per sub-chunk
// (stages are released through mbarriers):
//   scores  q_g . k_row * scale * log2(e): S lanes per row, the query slice in
//           registers, packed fp32x2 FMAs, a reduce-scatter over the S lanes
//           that leaves each lane with one head's full dot product;
//   softmax per head over the warp's rows (running max / sum per warp);
//   output  lanes over head dims, probabilities broadcast from shared memory.
// At an item's end the 16 warps' states are merged; an item covering its
// whole group writes the output, otherwise its unnormalised partial is stored
// and the group's last finishing item (atomic count) combines the partials in
// item order (deterministic). The last CTA to exit advances the lengths.
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "decode.cuh"
#include "kernels.cuh"

namespace ripple {
namespace {

constexpr int kWarps = 16;                    // compute warps
constexpr int kThreads = (kWarps + 1) * 32;   // + one producer warp
constexpr int kStageBytes = 32768;            // K (or V) bytes of one sub-chunk
constexpr int kStages = 2;
constexpr int kItemSub = 16;                  // sub-chunks per work item (merges are costly)
constexpr int kItemSlots = 4;
constexpr int kPrefetchAhead = 2;             // sub-chunks prefetched into L2 past the stages

template <typename Tin, int D, int G>
struct DecCfg {
  static constexpr int ROW_BYTES = D * (int)sizeof(Tin);
  static constexpr int CR = kStageBytes / ROW_BYTES;     // rows per sub-chunk
  static constexpr int ITEM_ROWS = CR * kItemSub;
  static constexpr int RPW = CR / kWarps;                // rows per warp per sub-chunk
  static constexpr int S = G <= 2 ? 8 : (G == 4 ? 16 : 32);  // lanes per row in the scores
  static constexpr int PB0 = ROW_BYTES / S;
  static constexpr int PB = PB0 < 16 ? PB0 : 16;         // bytes per piece
  static constexpr int PIECES = ROW_BYTES / PB;          // pieces per row
  static constexpr int PE = PB / (int)sizeof(Tin);       // elements per piece
  static constexpr int PPL = PIECES / S;                 // pieces per lane
  static constexpr int NPIECE = ROW_BYTES / 16;          // 16-byte units per row
  static constexpr int DL = PPL * PE;                    // dims per lane in the scores
  static constexpr int RPI = 32 / S;                     // rows per warp step
  static constexpr int NIT = RPW / RPI;                  // warp steps per sub-chunk
  static constexpr int HL = S / G;                       // lanes per head after reduce-scatter
  static constexpr int DV = D / 32;                      // dims per lane in the output
  static_assert(NIT >= 1 && RPW % RPI == 0, "rows per warp");
  static_assert(PPL * S == PIECES && HL >= 1, "lanes per row");
  static_assert(DL % 2 == 0 && DV % 2 == 0, "fp32x2 pairs");
};

template <typename Tin, int D, int G>
struct DecSmem {
  using C = DecCfg<Tin, D, G>;
  alignas(128) uint8_t kv[kStages][2][kStageBytes];  // [stage][K, V]
  alignas(16) float red_o[kWarps][G * D];             // per-warp outputs at an item's end
  alignas(16) float pw[kWarps][C::RPW][G];            // per-warp probabilities
  alignas(16) float aw[kWarps][G];                    // per-warp rescale factors
  float red_m[kWarps][G], red_l[kWarps][G];
  uint64_t full[kStages], empty[kStages], item_full[kItemSlots], item_empty[kItemSlots];
  int item_id[kItemSlots];
  int len[RIPPLE_MAX_LAYERS];    // by work-order position; -1 = full layer
  int nch[RIPPLE_MAX_LAYERS];    // items per group, by work-order position
  int base[RIPPLE_MAX_LAYERS + 1];
  int last;
};

struct ItemInfo {
  int pos, layer, group, b, h, chunk, nch, len, r0, rows, full;
};

template <typename Tin, int D, int G>
__device__ __forceinline__ ItemInfo item_info(const DecParams &p, const DecSmem<Tin, D, G> &s,
                                              int it) {
  using C = DecCfg<Tin, D, G>;
  int lo = 0, hi = p.L - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s.base[mid] <= it) lo = mid; else hi = mid - 1;
  }
  ItemInfo f;
  f.pos = lo;
  f.layer = p.order[lo];
  f.nch = s.nch[lo];
  const int local = it - s.base[lo];
  const int unit = local / f.nch;
  f.chunk = local % f.nch;
  f.b = unit / p.Hkv;
  f.h = unit % p.Hkv;
  f.group = (f.layer * p.B + f.b) * p.Hkv + f.h;
  f.len = s.len[lo];
  f.full = f.len < 0;
  f.r0 = f.chunk * C::ITEM_ROWS;
  f.rows = f.full ? 0 : min(C::ITEM_ROWS, f.len + 1 - f.r0);
  return f;
}

// 2*NP consecutive elements (one aligned load of 4 * NP bytes for bf16, or
// 8 * NP bytes for fp32) as fp32 pairs; bf16 widens by placing its 16 bits in
// the upper half of an fp32.
__device__ __forceinline__ float2 bf16x2_pair(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}
template <int NP>
__device__ __forceinline__ void load_pairs(const __nv_bfloat16 *p, float2 (&o)[NP]) {
  if constexpr (NP == 4) {
    const uint4 u = *reinterpret_cast<const uint4 *>(p);
    o[0] = bf16x2_pair(u.x); o[1] = bf16x2_pair(u.y);
    o[2] = bf16x2_pair(u.z); o[3] = bf16x2_pair(u.w);
  } else if constexpr (NP == 2) {
    const uint2 u = *reinterpret_cast<const uint2 *>(p);
    o[0] = bf16x2_pair(u.x); o[1] = bf16x2_pair(u.y);
  } else {
    static_assert(NP == 1, "pairs");
    o[0] = bf16x2_pair(*reinterpret_cast<const uint32_t *>(p));
  }
}
template <int NP>
__device__ __forceinline__ void load_pairs(const float *p, float2 (&o)[NP]) {
  if constexpr (NP == 2) {
    const float4 u = *reinterpret_cast<const float4 *>(p);
    o[0] = make_float2(u.x, u.y);
    o[1] = make_float2(u.z, u.w);
  } else {
    static_assert(NP == 1, "pairs");
    o[0] = *reinterpret_cast<const float2 *>(p);
  }
}

// L2 prefetch of one sub-chunk's cache rows (K and V, rows before the new
// token); `sub` may run past the item's end into the following item.
template <typename Tin, int D, int G>
__device__ __forceinline__ void prefetch_sub(const DecParams &p, const DecSmem<Tin, D, G> &s,
                                             int total, int it, int nxt, int sub) {
  using C = DecCfg<Tin, D, G>;
  if (it >= total) return;
  ItemInfo f = item_info(p, s, it);
  int nsub = f.full ? 0 : (f.rows + C::CR - 1) / C::CR;
  if (sub >= nsub) {
    sub -= nsub;
    if (nxt >= total) return;
    f = item_info(p, s, nxt);
    nsub = f.full ? 0 : (f.rows + C::CR - 1) / C::CR;
    if (sub >= nsub) return;
  }
  const int rs = f.r0 + sub * C::CR;
  const int re = min(rs + C::CR, f.len);
  if (re <= rs) return;
  const size_t off = ((size_t)(f.b * p.Hkv + f.h) * p.cap[f.layer] + rs) * C::ROW_BYTES;
  const uint32_t bytes = (uint32_t)(re - rs) * C::ROW_BYTES;
  bulk_prefetch_l2((const uint8_t *)p.kc[f.layer] + off, bytes);
  bulk_prefetch_l2((const uint8_t *)p.vc[f.layer] + off, bytes);
}

template <int G>
__device__ __forceinline__ void load_probs(const float *src, float (&pr)[G]) {
  if constexpr (G % 4 == 0) {
#pragma unroll
    for (int i = 0; i < G; i += 4) {
      const float4 x = *reinterpret_cast<const float4 *>(src + i);
      pr[i] = x.x; pr[i + 1] = x.y; pr[i + 2] = x.z; pr[i + 3] = x.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < G; ++i) pr[i] = src[i];
  }
}

template <typename Tin, int D, int G>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(const __grid_constant__ DecParams p) {
  using C = DecCfg<Tin, D, G>;
  extern __shared__ __align__(128) uint8_t smem_raw[];
  DecSmem<Tin, D, G> &s = *reinterpret_cast<DecSmem<Tin, D, G> *>(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int units = p.B * p.Hkv;

  // Work list of this step from the current lengths (read once, before any
  // CTA can advance them: that happens after every CTA has exited).
  if (tid < p.L) {
    const int l = p.order[tid];
    const int len = p.lens[l];
    const bool full = len < 0 || len >= p.cap[l];
    s.len[tid] = full ? -1 : len;
    s.nch[tid] = full ? 1 : (len + 1 + C::ITEM_ROWS - 1) / C::ITEM_ROWS;
    if (full && blockIdx.x == 0) report(p.status, RIPPLE_EFULL);
  }
  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], kWarps);
    }
    for (int i = 0; i < kItemSlots; ++i) {
      mbar_init(&s.item_full[i], 1);
      mbar_init(&s.item_empty[i], kWarps);
    }
    fence_mbar_init();
  }
  __syncthreads();
  if (tid == 0) {
    int acc = 0;
    for (int t = 0; t < p.L; ++t) {
      s.base[t] = acc;
      acc += units * s.nch[t];
    }
    s.base[p.L] = acc;
  }
  __syncthreads();
  const int total = s.base[p.L];

  if (warp == kWarps) {
    // ------------------------------------------------ producer warp
    int icount = 0;
    uint32_t j = 0;
    int it = lane == 0 ? atomicAdd(&p.ctrl[0], 1) : 0;
    int nxt = lane == 0 ? atomicAdd(&p.ctrl[0], 1) : 0;
    it = __shfl_sync(0xffffffffu, it, 0);
    nxt = __shfl_sync(0xffffffffu, nxt, 0);
    for (;;) {
      const int slot = icount % kItemSlots;
      mbar_wait(&s.item_empty[slot], ((icount / kItemSlots) & 1) ^ 1, p.status);
      __syncwarp();
      if (lane == 0) {
        s.item_id[slot] = it;
        mbar_arrive(&s.item_full[slot]);
      }
      ++icount;
      if (it >= total) break;
      // The first sub-chunks of the very first item get an L2 prefetch too.
      if (lane == 0 && icount == 1)
        for (int k = 0; k < kPrefetchAhead; ++k) prefetch_sub(p, s, total, it, nxt, k);
      int nxt2 = lane == 0 ? atomicAdd(&p.ctrl[0], 1) : 0;
      const ItemInfo f = item_info(p, s, it);
      if (!f.full) {
        const int nsub = (f.rows + C::CR - 1) / C::CR;
        const size_t gbase = (size_t)(f.b * p.Hkv + f.h) * p.cap[f.layer];
        for (int sub = 0; sub < nsub; ++sub, ++j) {
          const int stage = j % kStages;
          mbar_wait(&s.empty[stage], ((j / kStages) & 1) ^ 1, p.status);
          __syncwarp();
          const int rs = f.r0 + sub * C::CR;
          const int re = min(rs + C::CR, f.len);  // rows >= len are not in the cache yet
          const int nk = re > rs ? re - rs : 0;
          if (f.len >= rs && f.len < rs + C::CR) {
            // The new token: into the stage and appended to the cache.
            const size_t nb = ((size_t)f.layer * units + f.b * p.Hkv + f.h) * C::ROW_BYTES;
            for (int e = lane; e < 2 * C::NPIECE; e += 32) {
              const int v = e >= C::NPIECE, pc = e % C::NPIECE;
              const uint4 val = reinterpret_cast<const uint4 *>(
                  (const uint8_t *)(v ? p.v_new : p.k_new) + nb)[pc];
              reinterpret_cast<uint4 *>(s.kv[stage][v] + (size_t)(f.len - rs) * C::ROW_BYTES)[pc] =
                  val;
              reinterpret_cast<uint4 *>((uint8_t *)(v ? p.vc[f.layer] : p.kc[f.layer]) +
                                        (gbase + f.len) * C::ROW_BYTES)[pc] = val;
            }
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            if (nk > 0) {
              const size_t off = (gbase + rs) * C::ROW_BYTES;
              mbar_arrive_expect_tx(&s.full[stage], 2u * nk * C::ROW_BYTES);
              bulk_g2s(s.kv[stage][0], (const uint8_t *)p.kc[f.layer] + off, nk * C::ROW_BYTES,
                       &s.full[stage]);
              bulk_g2s(s.kv[stage][1], (const uint8_t *)p.vc[f.layer] + off, nk * C::ROW_BYTES,
                       &s.full[stage]);
            } else {
              mbar_arrive(&s.full[stage]);
            }
            // Keep kPrefetchAhead more sub-chunks on their way into L2.
            prefetch_sub(p, s, total, it, nxt, sub + kPrefetchAhead);
          }
        }
      }
      it = nxt;
      nxt = __shfl_sync(0xffffffffu, nxt2, 0);
    }
  } else {
    // ------------------------------------------------ compute warps
    const int slot_l = lane % C::S;            // lane within its row
    const int hq = slot_l / C::HL;             // head this lane holds after the reduce-scatter
    const int rw0 = warp * C::RPW;             // this warp's first row in a sub-chunk
    int icount = 0;
    uint32_t j = 0;
    for (;;) {
      const int slot = icount % kItemSlots;
      mbar_wait(&s.item_full[slot], (icount / kItemSlots) & 1, p.status);
      __syncwarp();
      const int it = s.item_id[slot];
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.item_empty[slot]);
      ++icount;
      if (it >= total) break;
      const ItemInfo f = item_info(p, s, it);
      const size_t qrow = ((size_t)f.layer * p.B + f.b) * p.Hq + (size_t)f.h * G;
      if (f.full) {
        for (int e = tid; e < G * D; e += kWarps * 32) p.out[qrow * D + e] = 0.f;
        continue;
      }
      // Query slice (the lane's pieces of each head), pre-scaled to log2 units.
      float2 q2[G][C::DL / 2];
      {
        const Tin *qg = (const Tin *)p.q + qrow * D;
#pragma unroll
        for (int g = 0; g < G; ++g)
#pragma unroll
          for (int k = 0; k < C::PPL; ++k) {
            float2 t[C::PE / 2];
            load_pairs<C::PE / 2>(qg + g * D + (slot_l + k * C::S) * C::PE, t);
#pragma unroll
            for (int e = 0; e < C::PE / 2; ++e)
              q2[g][k * C::PE / 2 + e] = make_float2(t[e].x * p.scale2, t[e].y * p.scale2);
          }
      }
      float2 acc[G][C::DV / 2];
#pragma unroll
      for (int g = 0; g < G; ++g)
#pragma unroll
        for (int e = 0; e < C::DV / 2; ++e) acc[g][e] = make_float2(0.f, 0.f);
      float m_run = -INFINITY, l_run = 0.f;  // of head hq, over this warp's rows
      const int nsub = (f.rows + C::CR - 1) / C::CR;

      for (int sub = 0; sub < nsub; ++sub, ++j) {
        const int stage = j % kStages;
        mbar_wait(&s.full[stage], (j / kStages) & 1, p.status);
        __syncwarp();
        const int nrows = min(C::CR, f.r0 + f.rows - (f.r0 + sub * C::CR));
        const Tin *ks = (const Tin *)s.kv[stage][0];
        const Tin *vs = (const Tin *)s.kv[stage][1];

        // Scores of this warp's rows.
        float sc[C::NIT];
#pragma unroll
        for (int t = 0; t < C::NIT; ++t) {
          const int row = rw0 + t * C::RPI + lane / C::S;
          float2 d2[G];
#pragma unroll
          for (int g = 0; g < G; ++g) d2[g] = make_float2(0.f, 0.f);
          if (row < nrows) {
#pragma unroll
            for (int k = 0; k < C::PPL; ++k) {
              float2 kp[C::PE / 2];
              load_pairs<C::PE / 2>(ks + (size_t)row * D + (slot_l + k * C::S) * C::PE, kp);
#pragma unroll
              for (int g = 0; g < G; ++g)
#pragma unroll
                for (int e = 0; e < C::PE / 2; ++e)
                  d2[g] = __ffma2_rn(q2[g][k * C::PE / 2 + e], kp[e], d2[g]);
            }
          }
          float v[G];
#pragma unroll
          for (int g = 0; g < G; ++g) v[g] = d2[g].x + d2[g].y;
          // Reduce-scatter over the S lanes of the row: afterwards every lane
          // holds the full dot product of head hq.
          int nv = G;
#pragma unroll
          for (int o = C::S / 2; o >= 1; o >>= 1) {
            if (nv > 1) {
              const bool upper = (lane & o) != 0;
              const int half = nv / 2;
#pragma unroll
              for (int i = 0; i < G / 2; ++i) {
                if (i < half) {
                  const float send = upper ? v[i] : v[i + half];
                  const float keep = upper ? v[i + half] : v[i];
                  v[i] = keep + __shfl_xor_sync(0xffffffffu, send, o);
                }
              }
              nv = half;
            } else {
              v[0] += __shfl_xor_sync(0xffffffffu, v[0], o);
            }
          }
          sc[t] = row < nrows ? v[0] : -INFINITY;
        }

        // Online softmax of head hq over this warp's rows.
        float mloc = sc[0];
#pragma unroll
        for (int t = 1; t < C::NIT; ++t) mloc = fmaxf(mloc, sc[t]);
#pragma unroll
        for (int o = C::S; o < 32; o <<= 1) mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, o));
        const float mnew = fmaxf(m_run, mloc);
        const bool any = mnew != -INFINITY;
        const float alpha = any ? fast_exp2(m_run - mnew) : 1.f;
        float lsum = 0.f;
#pragma unroll
        for (int t = 0; t < C::NIT; ++t) {
          const float e = any ? fast_exp2(sc[t] - mnew) : 0.f;
          sc[t] = e;
          lsum += e;
        }
#pragma unroll
        for (int o = C::S; o < 32; o <<= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
        l_run = l_run * alpha + lsum;
        m_run = mnew;
        if (slot_l % C::HL == 0) {
#pragma unroll
          for (int t = 0; t < C::NIT; ++t) s.pw[warp][t * C::RPI + lane / C::S][hq] = sc[t];
          if (lane < C::S) s.aw[warp][hq] = alpha;
        }
        __syncwarp();

        // Output rows of this warp.
        {
          float a[G];
          load_probs<G>(s.aw[warp], a);
#pragma unroll
          for (int g = 0; g < G; ++g)
#pragma unroll
            for (int e = 0; e < C::DV / 2; ++e) {
              acc[g][e].x *= a[g];
              acc[g][e].y *= a[g];
            }
          const int rmax = min(C::RPW, nrows - rw0);
#pragma unroll
          for (int r = 0; r < C::RPW; ++r) {
            if (r >= rmax) break;
            float pr[G];
            load_probs<G>(s.pw[warp][r], pr);
            float2 vp[C::DV / 2];
            load_pairs<C::DV / 2>(vs + (size_t)(rw0 + r) * D + lane * C::DV, vp);
#pragma unroll
            for (int g = 0; g < G; ++g)
#pragma unroll
              for (int e = 0; e < C::DV / 2; ++e)
                acc[g][e] = __ffma2_rn(make_float2(pr[g], pr[g]), vp[e], acc[g][e]);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&s.empty[stage]);
      }

      // Item end: merge the 16 warps' states.
      if (slot_l % C::HL == 0 && lane < C::S) {
        s.red_m[warp][hq] = m_run;
        s.red_l[warp][hq] = l_run;
      }
#pragma unroll
      for (int g = 0; g < G; ++g)
#pragma unroll
        for (int e = 0; e < C::DV / 2; ++e)
          *reinterpret_cast<float2 *>(&s.red_o[warp][g * D + lane * C::DV + 2 * e]) = acc[g][e];
      named_bar_sync(1, kWarps * 32);
      const bool single = f.nch == 1;
      const int item_base = s.base[f.pos] + (f.b * p.Hkv + f.h) * f.nch;
      const int item = item_base + f.chunk;
      for (int e = tid; e < G * D; e += kWarps * 32) {
        const int g = e / D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) M = fmaxf(M, s.red_m[w][g]);
        float num = 0.f, den = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
          const float wgt = fast_exp2(s.red_m[w][g] - M);
          num += wgt * s.red_o[w][e];
          den += wgt * s.red_l[w][g];
        }
        if (single) {
          p.out[qrow * D + e] = num / den;
        } else {
          p.ws_o[(size_t)item * G * D + e] = num;
          if (e % D == 0) p.ws_ml[(size_t)item * G + g] = make_float2(M, den);
        }
      }
      if (!single) {
        __threadfence();
        named_bar_sync(1, kWarps * 32);
        if (tid == 0) s.last = atomicAdd(&p.ctrl[2 + f.group], 1) == f.nch - 1;
        named_bar_sync(1, kWarps * 32);
        if (s.last) {
          __threadfence();
          for (int e = tid; e < G * D; e += kWarps * 32) {
            const int g = e / D;
            float M = -INFINITY;
            for (int c = 0; c < f.nch; ++c)
              M = fmaxf(M, __ldcg(&p.ws_ml[(size_t)(item_base + c) * G + g]).x);
            float num = 0.f, den = 0.f;
            for (int c = 0; c < f.nch; ++c) {
              const float2 ml = __ldcg(&p.ws_ml[(size_t)(item_base + c) * G + g]);
              const float wgt = fast_exp2(ml.x - M);
              den += wgt * ml.y;
              num += wgt * __ldcg(&p.ws_o[(size_t)(item_base + c) * G * D + e]);
            }
            p.out[qrow * D + e] = num / den;
          }
        }
      }
      named_bar_sync(1, kWarps * 32);  // red_* free for the next item
    }
  }

  // The last CTA to leave advances the lengths of the layers it could append to.
  __syncwarp();
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    if (atomicAdd(&p.ctrl[1], 1) == (int)gridDim.x - 1) {
      for (int t = 0; t < p.L; ++t)
        if (s.len[t] >= 0) p.lens[p.order[t]] = s.len[t] + 1;
    }
  }
}

int sm_count_cached() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

template <typename Tin, int D, int G>
cudaError_t launch_g(const DecParams &p, cudaStream_t st) {
  const int smem = (int)sizeof(DecSmem<Tin, D, G>);
  cudaError_t e = cudaFuncSetAttribute(decode_kernel<Tin, D, G>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  decode_kernel<Tin, D, G><<<sm_count_cached(), kThreads, smem, st>>>(p);
  count_launches(1);
  return cudaGetLastError();
}

template <typename Tin, int D>
cudaError_t launch_d(const DecParams &p, cudaStream_t st) {
  switch (p.G) {
    case 1: return launch_g<Tin, D, 1>(p, st);
    case 2: return launch_g<Tin, D, 2>(p, st);
    case 4: return launch_g<Tin, D, 4>(p, st);
    case 8: return launch_g<Tin, D, 8>(p, st);
    default: return cudaErrorInvalidValue;
  }
}

// Cache rows per work item of the kernel that serves this descriptor.
int item_rows(const ripple_decode_desc *d) {
  if (decode_tc_supported(d)) return kTcItemRows;
  const int row_bytes = d->head_dim * (d->dtype == RIPPLE_F32 ? 4 : 2);
  return (kStageBytes / row_bytes) * kItemSub;
}

static size_t round_up(size_t x) { return (x + 255) & ~(size_t)255; }

// Workspace layout for these capacities: control block, partial (max, sum),
// partial outputs. Returns the total bytes; fills p's pointers if given.
size_t plan(const ripple_decode_desc *d, const int32_t *caps, void *ws, DecParams *p) {
  const int G = d->n_q_heads / d->n_kv_heads;
  const int rows = item_rows(d);
  size_t items = 0;
  for (int l = 0; l < d->n_layers; ++l)
    items += (size_t)d->batch * d->n_kv_heads * ((caps[l] + rows - 1) / rows);
  const size_t groups = (size_t)d->n_layers * d->batch * d->n_kv_heads;
  const size_t ctrl = round_up(sizeof(int) * (2 + groups));
  const size_t ml = round_up(sizeof(float2) * items * G);
  const size_t o = round_up(sizeof(float) * items * G * d->head_dim);
  if (p != nullptr) {
    uint8_t *base = (uint8_t *)ws;
    p->ctrl = (int *)base;
    p->ws_ml = (float2 *)(base + ctrl);
    p->ws_o = (float *)(base + ctrl + ml);
  }
  return ctrl + ml + o;
}

size_t ctrl_bytes(const ripple_decode_desc *d) {
  return sizeof(int) * (2 + (size_t)d->n_layers * d->batch * d->n_kv_heads);
}

bool desc_ok(const ripple_decode_desc *d) {
  if (d == nullptr) return false;
  if (d->n_layers < 1 || d->n_layers > RIPPLE_MAX_LAYERS) return false;
  if (d->batch < 1 || d->n_kv_heads < 1 || d->n_q_heads < 1) return false;
  if (d->n_q_heads % d->n_kv_heads != 0) return false;
  const int G = d->n_q_heads / d->n_kv_heads;
  if (G != 1 && G != 2 && G != 4 && G != 8) return false;
  if (d->head_dim != 64 && d->head_dim != 128) return false;
  if (d->dtype != RIPPLE_F32 && d->dtype != RIPPLE_BF16) return false;
  if (!(d->scale >= 0.f) || isinf(d->scale)) return false;
  if ((int64_t)d->n_layers * d->batch * d->n_kv_heads > (1 << 24)) return false;
  return true;
}

// Shared argument checks and parameter set-up of both decode entry points.
ripple_status prepare(const ripple_decode_desc *desc, const void *q, const void *k_new,
                      const void *v_new, void *const *k_caches_host, void *const *v_caches_host,
                      const int32_t *caps_host, int32_t *lens, float *out, int32_t *dev_status,
                      DecParams *p) {
  if (!desc_ok(desc)) return RIPPLE_EINVAL;
  if (!q || !k_new || !v_new || !k_caches_host || !v_caches_host || !caps_host || !lens || !out)
    return RIPPLE_EINVAL;
  auto aligned = [](const void *ptr) { return ((uintptr_t)ptr & 15u) == 0; };
  if (!aligned(q) || !aligned(k_new) || !aligned(v_new) || !aligned(out)) return RIPPLE_EINVAL;
  const int L = desc->n_layers;
  for (int l = 0; l < L; ++l) {
    if (!k_caches_host[l] || !v_caches_host[l] || caps_host[l] < 1) return RIPPLE_EINVAL;
    if (!aligned(k_caches_host[l]) || !aligned(v_caches_host[l])) return RIPPLE_EINVAL;
    p->kc[l] = k_caches_host[l];
    p->vc[l] = v_caches_host[l];
    p->cap[l] = caps_host[l];
    p->order[l] = l;
  }
  // longest caches first (stable insertion sort, L <= 128)
  for (int i = 1; i < L; ++i) {
    const int v = p->order[i];
    int k = i - 1;
    while (k >= 0 && p->cap[p->order[k]] < p->cap[v]) {
      p->order[k + 1] = p->order[k];
      --k;
    }
    p->order[k + 1] = v;
  }
  p->L = L;
  p->B = desc->batch;
  p->Hq = desc->n_q_heads;
  p->Hkv = desc->n_kv_heads;
  p->G = p->Hq / p->Hkv;
  const float scale = desc->scale > 0.f ? desc->scale : 1.0f / sqrtf((float)desc->head_dim);
  p->scale2 = scale * kLog2e;
  p->q = q;
  p->k_new = k_new;
  p->v_new = v_new;
  p->lens = lens;
  p->out = out;
  p->status = dev_status;
  return RIPPLE_OK;
}

ripple_status run(const ripple_decode_desc *desc, const DecParams &p, void *stream) {
  cudaStream_t st = (cudaStream_t)stream;
  if (decode_tc_supported(desc))
    return launch_decode_tc(p, ctrl_bytes(desc), st) == cudaSuccess ? RIPPLE_OK : RIPPLE_ECUDA;
  decode_tc_forget_ctrl(p.ctrl);
  if (cudaMemsetAsync(p.ctrl, 0, ctrl_bytes(desc), st) != cudaSuccess) return RIPPLE_ECUDA;
  cudaError_t e;
  if (desc->dtype == RIPPLE_F32)
    e = desc->head_dim == 64 ? launch_d<float, 64>(p, st) : launch_d<float, 128>(p, st);
  else
    e = desc->head_dim == 64 ? launch_d<__nv_bfloat16, 64>(p, st)
                             : launch_d<__nv_bfloat16, 128>(p, st);
  return e == cudaSuccess ? RIPPLE_OK : RIPPLE_ECUDA;
}

}  // namespace
}  // namespace ripple

using namespace ripple;

extern "C" ripple_status ripple_decode_workspace_bytes(const ripple_decode_desc *desc,
                                                       const int32_t *caps_host,
                                                       size_t *bytes_host) {
  if (!desc_ok(desc) || caps_host == nullptr || bytes_host == nullptr) return RIPPLE_EINVAL;
  for (int l = 0; l < desc->n_layers; ++l)
    if (caps_host[l] < 1) return RIPPLE_EINVAL;
  *bytes_host = plan(desc, caps_host, nullptr, nullptr);
  return RIPPLE_OK;
}

extern "C" ripple_status ripple_decode_attn(const ripple_decode_desc *desc, const void *q,
                                            const void *k_new, const void *v_new,
                                            void *const *k_caches_host,
                                            void *const *v_caches_host,
                                            const int32_t *caps_host, int32_t *lens, float *out,
                                            void *workspace, size_t workspace_bytes,
                                            int32_t *dev_status, void *stream) {
  DecParams p;
  const ripple_status s = prepare(desc, q, k_new, v_new, k_caches_host, v_caches_host,
                                  caps_host, lens, out, dev_status, &p);
  if (s != RIPPLE_OK) return s;
  if (workspace == nullptr || ((uintptr_t)workspace & 255u)) return RIPPLE_EINVAL;
  if (workspace_bytes < plan(desc, caps_host, workspace, &p)) return RIPPLE_EWORKSPACE;
  return run(desc, p, stream);
}

// ---------------------------------------------------------------------------
// Decode for callers that cannot allocate device memory (no paper counterpart).
//
// A plugin inside a host program that owns all device memory through its own
// pool, or a fixed-footprint server that reserves every byte at start-up, may
// have no way to hand this library a scratch buffer. For those callers the
// step's control counters and split-K partials live in the file-scope device
// array below instead of a caller workspace. Every GPU that loads the library
// keeps it until the process exits; all calls on a device share it. Its
// counters start at zero (zero-initialised at load) and every call leaves them
// at zero (the tensor-core kernel resets them as it exits, the other kernels
// are preceded by a memset on the stream); every partial a call reads it has
// rewritten, so no state carries over from the previous call. Calls that
// overlap on the GPU race on it.

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
  DecParams p;
  const ripple_status s = prepare(desc, q, k_new, v_new, k_caches_host, v_caches_host,
                                  caps_host, lens, out, dev_status, &p);
  if (s != RIPPLE_OK) return s;
  if (plan(desc, caps_host, nullptr, nullptr) > RIPPLE_DECODE_NOALLOC_SCRATCH_BYTES)
    return RIPPLE_EWORKSPACE;
  float *scratch = nullptr;
  const ripple_status a = scratch_on_current_device(&scratch);
  if (a != RIPPLE_OK) return a;
  plan(desc, caps_host, scratch, &p);
  return run(desc, p, stream);
}
