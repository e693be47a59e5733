// GQA decode attention over the ragged compressed caches on the tensor cores
// (Sec. 4.1: each new query attends to the cached states), with the append of
// the new token. bf16 caches, d = 128, G = Hq / Hkv query heads per KV head.
//
// One persistent launch per step covers every layer; one CTA per SM. Work
// item = up to 16 tiles (2048 rows) of one (layer, batch row, KV head)
// group's cache, fetched with an atomic counter, longest layers first.
// Per tile of 128 cache rows:
//   S = K_tile . Q^T       tcgen05.mma, M = 128 rows, N = 16 (G heads, rest
//                          zero), K = d; A = key tile (TMA, 128-byte swizzle),
//                          B = the group's queries; fp32 scores in TMEM;
//   softmax                one thread per row: mask rows >= len, scale, per
//                          warp (32 rows) max and sum per head; P (bf16) to
//                          shared memory;
//   O_q = V_q^T . P_q      tcgen05.mma per warp's 32 rows, M = 128 dims,
//                          N = 16, K = 32 rows; A = value tile read MN-major;
//                          fp32 in TMEM;
//   combine                one thread per dim folds the four warps' O_q into
//                          its running (max, sum, output) per head.
// The new token (not yet in the cache) is scored on the CUDA cores and folded
// in at the end of its group's last item; it is appended to the cache there.
// An item covering its whole group writes the output; otherwise it stores its
// unnormalised partial and the group's last item combines them in item order.
//
// Warp roles (224 threads): warp 0 = tile producer (work items, key / value
// tiles), warp 1 = MMA issuer and TMEM owner, warps 2-5 = epilogue (TMEM lane
// quarter = warp % 4), warp 6 = per-item set-up (queries, new token). Every wait is bounded; on timeout the CTA raises
// RIPPLE_ETIMEOUT, every role leaves its loop and TMEM is released.
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "decode.cuh"
#include "kernels.cuh"
#include "tc_ptx.cuh"

namespace ripple {
namespace {

constexpr int kTile = 128;                  // cache rows per tile
constexpr int kTileBytes = kTile * 256;     // 32 KB of bf16 rows, d = 128
constexpr int kHalf = kTileBytes / 2;       // one TMA box: 64 dims of 128 rows
constexpr int kRing = 6;                    // K / V tile slots
constexpr int kNS = 4;                      // score accumulators (16 TMEM columns each)
constexpr int kStatSlots = 3;
constexpr int kItemSlots = 4;
constexpr int kThreads = 224;
constexpr int kOpBytes = 4096;              // a 16 x 128 bf16 operand (queries or P)
constexpr uint32_t kSCol = 0;               // TMEM: scores  [kNS][16]
constexpr uint32_t kOCol = 64;              //       outputs [2][4 warps][16]
constexpr long long kWaitCycles = 4000000000LL;

struct TcDecParams {
  DecParams p;
  CUtensorMap kmap[kTcMaxLayers];
  CUtensorMap vmap[kTcMaxLayers];
};

struct Misc {
  uint64_t kv_full[kRing], kv_empty[kRing];
  uint64_t q_full[2], q_empty[2];
  uint64_t s_full[kNS], s_empty[kNS];
  uint64_t p_full[2], o_full[2], o_empty[2];
  uint64_t item_full[kItemSlots], item_empty[kItemSlots], new_full[kItemSlots];
  uint64_t mma_done;
  int item_id[kItemSlots];
  float s_new[kItemSlots][8];          // new token's scaled scores per head
  float2 stats[kStatSlots][4][8];      // per tile and warp: (max, sum) per head
  int len[RIPPLE_MAX_LAYERS];          // by work-order position; -1 = full layer
  int nch[RIPPLE_MAX_LAYERS];
  int base[RIPPLE_MAX_LAYERS + 1];
  uint32_t tmem_base;
  int abort_flag;
  int last;
};

constexpr int kOffRing = 0;
constexpr int kOffQ = kOffRing + kRing * kTileBytes;
constexpr int kOffP = kOffQ + 2 * kOpBytes;
constexpr int kOffMisc = kOffP + 2 * kOpBytes;
constexpr int kSmemBytes = kOffMisc + (int)sizeof(Misc) + 1024;  // + alignment slack
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");

__device__ __forceinline__ bool wait_bar(uint64_t *bar, uint32_t parity, Misc *ms,
                                         int32_t *status) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*(volatile int *)&ms->abort_flag) return false;
    if (clock64() - t0 > kWaitCycles) {
      *(volatile int *)&ms->abort_flag = 1;
      report(status, RIPPLE_ETIMEOUT);
      return false;
    }
  }
}

// All lanes wait; the warp agrees on the outcome and is converged afterwards.
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, Misc *ms,
                                          int32_t *status) {
  const bool ok = wait_bar(bar, parity, ms, status);
  return __all_sync(0xffffffffu, ok);
}

struct Item {
  int layer, pos, group, b, h, chunk, nch, len, r0, rows, tiles, full;
};

__device__ __forceinline__ Item item_of(const DecParams &p, const Misc *ms, int it) {
  int lo = 0, hi = p.L - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (ms->base[mid] <= it) lo = mid; else hi = mid - 1;
  }
  Item f;
  f.pos = lo;
  f.layer = p.order[lo];
  f.nch = ms->nch[lo];
  const int local = it - ms->base[lo];
  const int unit = local / f.nch;
  f.chunk = local % f.nch;
  f.b = unit / p.Hkv;
  f.h = unit % p.Hkv;
  f.group = (f.layer * p.B + f.b) * p.Hkv + f.h;
  f.len = ms->len[lo];
  f.full = f.len < 0;
  f.r0 = f.chunk * kTcItemRows;
  f.rows = f.full ? 0 : max(0, min(kTcItemRows, f.len - f.r0));
  f.tiles = (f.rows + kTile - 1) / kTile;
  return f;
}

// Byte offset of element (row n, column k) of a 16 x 128 bf16 K-major operand
// with 128-byte swizzle: two 64-column atoms of 16 rows x 128 bytes.
__device__ __forceinline__ uint32_t op_offset(int n, int k) {
  return (uint32_t)((k >> 6) * 2048 + n * 128 + ((((k & 63) >> 3) ^ (n & 7)) << 4) + (k & 7) * 2);
}

__device__ __forceinline__ float bf16_round(float x) {
  return __bfloat162float(__float2bfloat16_rn(x));
}

template <int G>
__global__ void __launch_bounds__(kThreads, 1)
    decode_tc_kernel(const __grid_constant__ TcDecParams tp) {
  const DecParams &p = tp.p;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t *ring = smem + kOffRing;
  uint8_t *qbuf = smem + kOffQ;
  uint8_t *pbuf = smem + kOffP;
  Misc *ms = (Misc *)(smem + kOffMisc);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int units = p.B * p.Hkv;

  // Launched as a programmatic dependent of the previous step: let the next
  // step's CTAs take SMs as this grid's CTAs leave, and wait here until the
  // previous grid has finished and its writes (lengths, appended rows,
  // counters) are visible.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // Work list of this step from the current lengths (read once, before any
  // CTA can advance them: that happens after every CTA has exited).
  if (tid < p.L) {
    const int l = p.order[tid];
    const int len = p.lens[l];
    const bool full = len < 0 || len >= p.cap[l];
    ms->len[tid] = full ? -1 : len;
    ms->nch[tid] = full ? 1 : max(1, (len + kTcItemRows - 1) / kTcItemRows);
    if (full && blockIdx.x == 0) report(p.status, RIPPLE_EFULL);
  }
  // Query and P operands: rows >= G stay zero.
  for (int i = tid; i < 4 * kOpBytes / 16; i += kThreads)
    reinterpret_cast<uint4 *>(qbuf)[i] = make_uint4(0, 0, 0, 0);
  if (tid == 0) {
    for (int i = 0; i < kRing; ++i) {
      mbar_init(&ms->kv_full[i], 1);
      mbar_init(&ms->kv_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&ms->q_full[i], 1);
      mbar_init(&ms->q_empty[i], 1);
      mbar_init(&ms->p_full[i], 1);
      mbar_init(&ms->o_full[i], 1);
      mbar_init(&ms->o_empty[i], 4);
    }
    for (int i = 0; i < kNS; ++i) {
      mbar_init(&ms->s_full[i], 1);
      mbar_init(&ms->s_empty[i], 4);
    }
    for (int i = 0; i < kItemSlots; ++i) {
      mbar_init(&ms->item_full[i], 1);
      mbar_init(&ms->item_empty[i], 6);  // MMA, set-up and 4 epilogue warps
      mbar_init(&ms->new_full[i], 1);
    }
    mbar_init(&ms->mma_done, 1);
    ms->abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&ms->tmem_base, 256);
    tmem_relinquish();
  }
  fence_proxy_async_smem();  // zeroed operands, seen by the tensor cores
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (tid == 0) {
    int acc = 0;
    for (int t = 0; t < p.L; ++t) {
      ms->base[t] = acc;
      acc += units * ms->nch[t];
    }
    ms->base[p.L] = acc;
  }
  __syncthreads();
  const int total = ms->base[p.L];
  const uint32_t tmem = ms->tmem_base;

  if (warp == 0) {
    // ------------------------------------------------ tile producer (one lane)
    // Work items are fetched one ahead; an item is published to the other
    // roles and its key / value tiles are issued at once, so the ring keeps
    // streaming across item boundaries.
    if (lane == 0) {
      int lcount = 0;
      int it = atomicAdd(&p.ctrl[0], 1);
      for (int icount = 0;; ++icount) {
        const int slot = icount % kItemSlots;
        const int nxt = it < total ? atomicAdd(&p.ctrl[0], 1) : total;
        if (!wait_bar(&ms->item_empty[slot], ((icount / kItemSlots) & 1) ^ 1, ms, p.status)) break;
        ms->item_id[slot] = min(it, total);
        mbar_arrive(&ms->item_full[slot]);
        if (it >= total) break;
        const Item f = item_of(p, ms, it);
        bool ok = true;
        if (f.tiles > 0) {
          const CUtensorMap *km = &tp.kmap[f.pos];
          const CUtensorMap *vm = &tp.vmap[f.pos];
          const int unit = f.b * p.Hkv + f.h;
          const uint64_t pol = policy_evict_first();  // every cache row is read once
          for (int j = 0; j < f.tiles && ok; ++j) {
            const int y = f.r0 + j * kTile;
            for (int kv = 0; kv < 2; ++kv, ++lcount) {
              const int rs = lcount % kRing;
              if (!wait_bar(&ms->kv_empty[rs], ((lcount / kRing) & 1) ^ 1, ms, p.status)) {
                ok = false;
                break;
              }
              mbar_arrive_expect_tx(&ms->kv_full[rs], kTileBytes);
              uint8_t *dst = ring + rs * kTileBytes;
              const CUtensorMap *m = kv ? vm : km;
              tma_load_3d(dst, m, 0, y, unit, &ms->kv_full[rs], pol);
              tma_load_3d(dst + kHalf, m, 64, y, unit, &ms->kv_full[rs], pol);
            }
          }
        }
        if (!ok) break;
        it = nxt;
      }
      // Let issued copies land before the CTA can exit (after an abort).
      for (int j = max(0, lcount - kRing); j < lcount; ++j)
        mbar_wait(&ms->kv_full[j % kRing], (j / kRing) & 1, nullptr, kWaitCycles / 4);
    }
  } else if (warp == 6) {
    // ------------------------------------------------ per-item set-up warp
    // Stages each item's queries as the score product's operand, and for a
    // group's last item scores the new token and appends it to the cache.
    int qcount = 0;
    for (int icount = 0;; ++icount) {
      const int slot = icount % kItemSlots;
      if (!warp_wait(&ms->item_full[slot], (icount / kItemSlots) & 1, ms, p.status)) break;
      const int it = ms->item_id[slot];
      if (it >= total) break;
      const Item f = item_of(p, ms, it);
      if (!f.full) {
        const size_t qrow = ((size_t)f.layer * p.B + f.b) * p.Hq + (size_t)f.h * G;
        if (f.tiles > 0) {
          const int qs = qcount & 1;
          const bool ok = warp_wait(&ms->q_empty[qs], ((qcount >> 1) & 1) ^ 1, ms, p.status);
          ++qcount;
          if (ok) {
            // the group's G query rows into the operand (16-byte pieces)
            const uint8_t *qg = (const uint8_t *)p.q + qrow * 256;
            uint8_t *qb = qbuf + qs * kOpBytes;
            for (int c = lane; c < G * 16; c += 32) {
              const int g = c >> 4, k = (c & 15) * 8;
              *reinterpret_cast<uint4 *>(qb + op_offset(g, k)) =
                  *reinterpret_cast<const uint4 *>(qg + (size_t)g * 256 + k * 2);
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&ms->q_full[qs]);
          }
        }
        if (f.chunk == f.nch - 1) {
          // The new token: its scores, and its append to the cache.
          const size_t nb = ((size_t)f.layer * units + f.b * p.Hkv + f.h) * 256;
          const uint2 kn = reinterpret_cast<const uint2 *>((const uint8_t *)p.k_new + nb)[lane];
          const float2 k01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&kn.x));
          const float2 k23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&kn.y));
#pragma unroll
          for (int g = 0; g < G; ++g) {
            const uint2 qv =
                reinterpret_cast<const uint2 *>((const uint8_t *)p.q + (qrow + g) * 256)[lane];
            const float2 q01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&qv.x));
            const float2 q23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&qv.y));
            float s = fmaf(q01.x, k01.x, fmaf(q01.y, k01.y, fmaf(q23.x, k23.x, q23.y * k23.y)));
            s = warp_sum(s);
            if (lane == 0) ms->s_new[slot][g] = s * p.scale2;
          }
          const size_t row = ((size_t)(f.b * p.Hkv + f.h) * p.cap[f.layer] + f.len) * 256;
          const int v = lane >> 4, pc = lane & 15;
          const uint4 val =
              reinterpret_cast<const uint4 *>((const uint8_t *)(v ? p.v_new : p.k_new) + nb)[pc];
          reinterpret_cast<uint4 *>((uint8_t *)(v ? p.vc[f.layer] : p.kc[f.layer]) + row)[pc] =
              val;
        }
      }
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&ms->new_full[slot]);
        mbar_arrive(&ms->item_empty[slot]);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t id_s = idesc_bf16(128, 16);
      constexpr uint32_t id_o = idesc_bf16_amn(128, 16);
      const uint32_t ring_a = smem_u32(ring), q_a = smem_u32(qbuf), p_a = smem_u32(pbuf);
      int lcount = 0, u = 0, qcount = 0;
      bool ok = true;
      // P.V of tile t (its value tile is load `vload`) into output slot t % 2.
      auto pv = [&](int t, int vload) -> bool {
        const int vs = vload % kRing, os = t & 1;
        if (!wait_bar(&ms->kv_full[vs], (vload / kRing) & 1, ms, p.status) ||
            !wait_bar(&ms->p_full[os], (t >> 1) & 1, ms, p.status) ||
            !wait_bar(&ms->o_empty[os], ((t >> 1) & 1) ^ 1, ms, p.status))
          return false;
        tc_fence_after();
        const uint32_t va = ring_a + vs * kTileBytes, pa = p_a + os * kOpBytes;
#pragma unroll
        for (int q = 0; q < 4; ++q)
#pragma unroll
          for (int k2 = 0; k2 < 2; ++k2) {
            const int kk = 2 * q + k2;  // rows 16 kk .. 16 kk + 15
            mma_bf16(tmem + kOCol + os * 64 + q * 16, sw128_desc_mn(va + kk * 2048, kHalf, 1024),
                     sw128_desc(pa + (kk >> 2) * 2048 + (kk & 3) * 32), id_o, k2);
          }
        mma_commit(&ms->kv_empty[vs]);
        mma_commit(&ms->o_full[os]);
        return true;
      };
      // S of tile u+1 is issued before P.V of tile u, also across items, so
      // the softmax of one tile overlaps the score product of the next and
      // an item's end does not stall the key stream. An item without tiles
      // (empty or full cache) flushes the pending P.V first: the epilogue
      // finishes items in order.
      int pend = -1, pend_v = 0;  // tile waiting for its P.V, its value load
      for (int icount = 0; ok; ++icount) {
        const int slot = icount % kItemSlots;
        if (!wait_bar(&ms->item_full[slot], (icount / kItemSlots) & 1, ms, p.status)) break;
        const int it = ms->item_id[slot];
        mbar_arrive(&ms->item_empty[slot]);
        if (it >= total) break;
        const Item f = item_of(p, ms, it);
        if (f.tiles == 0) {
          if (pend >= 0 && !pv(pend, pend_v)) break;
          pend = -1;
          continue;
        }
        const int qs = qcount & 1;
        if (!wait_bar(&ms->q_full[qs], (qcount >> 1) & 1, ms, p.status)) break;
        ++qcount;
        for (int j = 0; j < f.tiles; ++j, ++u) {
          const int ks = lcount % kRing, ss = u % kNS;
          if (!wait_bar(&ms->kv_full[ks], (lcount / kRing) & 1, ms, p.status) ||
              !wait_bar(&ms->s_empty[ss], ((u / kNS) & 1) ^ 1, ms, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t ka = ring_a + ks * kTileBytes, qa = q_a + qs * kOpBytes;
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t off_k = (kk >> 2) * kHalf + (kk & 3) * 32;
            const uint32_t off_q = (kk >> 2) * 2048 + (kk & 3) * 32;
            mma_bf16(tmem + kSCol + ss * 16, sw128_desc(ka + off_k), sw128_desc(qa + off_q), id_s,
                     kk > 0);
          }
          mma_commit(&ms->kv_empty[ks]);
          mma_commit(&ms->s_full[ss]);
          lcount += 2;  // this tile's K and V loads
          if (pend >= 0 && !pv(pend, pend_v)) {
            ok = false;
            break;
          }
          pend = u;
          pend_v = lcount - 1;
        }
        if (!ok) break;
        mma_commit(&ms->q_empty[qs]);  // the item's queries are no longer read
      }
      if (ok && pend >= 0) pv(pend, pend_v);
      mma_commit(&ms->mma_done);
      mbar_wait(&ms->mma_done, 0, nullptr, kWaitCycles / 4);
    }
  } else {
    // ------------------------------------------------ epilogue (4 warps)
    const int quarter = warp & 3;
    const int i = quarter * 32 + lane;  // score row in a tile, output dim
    const uint32_t lane_addr = (uint32_t)(quarter * 32) << 16;
    int u = 0;
    for (int icount = 0;; ++icount) {
      const int slot = icount % kItemSlots;
      if (!warp_wait(&ms->item_full[slot], (icount / kItemSlots) & 1, ms, p.status)) break;
      const int it = ms->item_id[slot];
      if (it >= total) break;
      const Item f = item_of(p, ms, it);
      const size_t qrow = ((size_t)f.layer * p.B + f.b) * p.Hq + (size_t)f.h * G;
      if (f.full) {
#pragma unroll
        for (int g = 0; g < G; ++g) p.out[(qrow + g) * 128 + i] = 0.f;
        __syncwarp();
        if (lane == 0) mbar_arrive(&ms->item_empty[slot]);
        continue;
      }
      float M[G], L[G], acc[G];
#pragma unroll
      for (int g = 0; g < G; ++g) {
        M[g] = -INFINITY;
        L[g] = 0.f;
        acc[g] = 0.f;
      }
      // Folds tile t's four warp outputs into the running state.
      auto combine = [&](int t) {
        const int os = t & 1;
        warp_wait(&ms->o_full[os], (t >> 1) & 1, ms, p.status);
        tc_fence_after();
        uint32_t o[4][G];
#pragma unroll
        for (int q = 0; q < 4; ++q) tmem_ld_cols<G>(tmem + lane_addr + kOCol + os * 64 + q * 16, o[q]);
        tmem_wait_ld();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&ms->o_empty[os]);
        const float2(*st)[8] = ms->stats[t % kStatSlots];
#pragma unroll
        for (int g = 0; g < G; ++g) {
          float mn = M[g];
#pragma unroll
          for (int q = 0; q < 4; ++q) mn = fmaxf(mn, st[q][g].x);
          if (mn == -INFINITY) continue;
          const float a0 = M[g] == -INFINITY ? 0.f : fast_exp2(M[g] - mn);
          float a = acc[g] * a0, l = L[g] * a0;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float2 ml = st[q][g];
            if (ml.x == -INFINITY) continue;
            const float c = fast_exp2(ml.x - mn);
            a = fmaf(__uint_as_float(o[q][g]), c, a);
            l = fmaf(ml.y, c, l);
          }
          acc[g] = a;
          L[g] = l;
          M[g] = mn;
        }
      };
      for (int j = 0; j < f.tiles; ++j, ++u) {
        // ---- scores of tile u -> P
        const int ss = u % kNS;
        warp_wait(&ms->s_full[ss], (u / kNS) & 1, ms, p.status);
        tc_fence_after();
        uint32_t x[G];
        tmem_ld_cols<G>(tmem + lane_addr + kSCol + ss * 16, x);
        tmem_wait_ld();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&ms->s_empty[ss]);
        const int row = f.r0 + j * kTile + i;
        const bool valid = row < f.len;
        uint8_t *pb = pbuf + (u & 1) * kOpBytes;
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const float s = valid ? __uint_as_float(x[g]) * p.scale2 : -INFINITY;
          const float m = warp_max(s);
          const float e = m == -INFINITY ? 0.f : bf16_round(fast_exp2(s - m));
          const float l = warp_sum(e);
          *reinterpret_cast<__nv_bfloat16 *>(pb + op_offset(g, i)) = __float2bfloat16_rn(e);
          if (lane == 0) ms->stats[u % kStatSlots][quarter][g] = make_float2(m, l);
        }
        if (!valid) {
          // Rows past the cache length may hold anything: zero the value row
          // so that 0 * garbage cannot reach the product.
          const int vload = 2 * u + 1;  // loads are K, V per tile in order
          if (wait_bar(&ms->kv_full[vload % kRing], (vload / kRing) & 1, ms, p.status)) {
            uint8_t *vt = ring + (vload % kRing) * kTileBytes;
#pragma unroll
            for (int c = 0; c < 8; ++c) {
              reinterpret_cast<uint4 *>(vt + i * 128)[c] = make_uint4(0, 0, 0, 0);
              reinterpret_cast<uint4 *>(vt + kHalf + i * 128)[c] = make_uint4(0, 0, 0, 0);
            }
          }
        }
        fence_proxy_async_smem();
        named_bar_sync(1, 128);
        if (i == 0) mbar_arrive(&ms->p_full[u & 1]);
        // ---- outputs of the previous tile
        if (j > 0) combine(u - 1);
      }
      if (f.tiles > 0) combine(u - 1);
      // The new token, after the group's cache rows.
      warp_wait(&ms->new_full[slot], (icount / kItemSlots) & 1, ms, p.status);
      if (f.chunk == f.nch - 1) {
        const size_t nb = ((size_t)f.layer * units + f.b * p.Hkv + f.h) * 128;
        const float vn = __bfloat162float(((const __nv_bfloat16 *)p.v_new)[nb + i]);
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const float sn = ms->s_new[slot][g];
          const float mn = fmaxf(M[g], sn);
          const float a0 = M[g] == -INFINITY ? 0.f : fast_exp2(M[g] - mn);
          const float c = fast_exp2(sn - mn);
          acc[g] = fmaf(vn, c, acc[g] * a0);
          L[g] = fmaf(L[g], a0, c);
          M[g] = mn;
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&ms->item_empty[slot]);
      if (f.nch == 1) {
#pragma unroll
        for (int g = 0; g < G; ++g) p.out[(qrow + g) * 128 + i] = acc[g] / L[g];
        continue;
      }
      // Split group: store the partial; the group's last item combines.
      const int item_base = ms->base[f.pos] + (f.b * p.Hkv + f.h) * f.nch;
      const int item = item_base + f.chunk;
#pragma unroll
      for (int g = 0; g < G; ++g) {
        p.ws_o[((size_t)item * G + g) * 128 + i] = acc[g];
        if (i == 0) p.ws_ml[(size_t)item * G + g] = make_float2(M[g], L[g]);
      }
      __threadfence();
      named_bar_sync(1, 128);
      if (i == 0) ms->last = atomicAdd(&p.ctrl[2 + f.group], 1) == f.nch - 1;
      named_bar_sync(1, 128);
      const bool last = ms->last;
      named_bar_sync(1, 128);  // `last` read by all before it is written again
      if (last) {
        __threadfence();
        if (i == 0) p.ctrl[2 + f.group] = 0;  // left at zero for the next call
#pragma unroll
        for (int g = 0; g < G; ++g) {
          float mx = -INFINITY;
          for (int c = 0; c < f.nch; ++c)
            mx = fmaxf(mx, __ldcg(&p.ws_ml[(size_t)(item_base + c) * G + g]).x);
          float num = 0.f, den = 0.f;
          for (int c = 0; c < f.nch; ++c) {
            const float2 ml = __ldcg(&p.ws_ml[(size_t)(item_base + c) * G + g]);
            const float w = ml.x == -INFINITY ? 0.f : fast_exp2(ml.x - mx);
            den = fmaf(w, ml.y, den);
            num = fmaf(w, __ldcg(&p.ws_o[((size_t)(item_base + c) * G + g) * 128 + i]), num);
          }
          p.out[(qrow + g) * 128 + i] = num / den;
        }
      }
    }
  }

  tc_fence_before();
  __syncwarp();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
  // The last CTA to leave advances the lengths of the layers it appended to
  // and leaves the item and exit counters at zero for the next call.
  if (tid == 0) {
    __threadfence();
    if (atomicAdd(&p.ctrl[1], 1) == (int)gridDim.x - 1) {
      for (int t = 0; t < p.L; ++t)
        if (ms->len[t] >= 0) p.lens[p.order[t]] = ms->len[t] + 1;
      p.ctrl[0] = 0;
      p.ctrl[1] = 0;
    }
  }
}

// ------------------------------------------------------------ host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (EncodeTiledFn)ptr;
  });
  return fn;
}

// Cache [units][cap][128] bf16 as a 3-D tensor map with 64 x 128 boxes.
bool encode_cache(EncodeTiledFn enc, CUtensorMap *m, const void *base, int cap, int units) {
  cuuint64_t dims[3] = {128, (cuuint64_t)cap, (cuuint64_t)units};
  cuuint64_t strides[2] = {256, (cuuint64_t)cap * 256};
  cuuint32_t box[3] = {64, (cuuint32_t)kTile, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box,
             es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

constexpr int kMaxDevices = 64;

int sm_count(int dev) {
  static int n[kMaxDevices] = {};
  if (dev < 0 || dev >= kMaxDevices) return 1;
  if (n[dev] == 0) {
    int v = 0;
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
    n[dev] = v > 0 ? v : 1;
  }
  return n[dev];
}

template <int G>
cudaError_t launch_g(const TcDecParams &tp, int dev, cudaStream_t st) {
  static bool attr_set[kMaxDevices] = {};
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  if (!attr_set[dev]) {
    const cudaError_t e = cudaFuncSetAttribute(
        decode_tc_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(sm_count(dev));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, decode_tc_kernel<G>, tp);
  count_launches(1);
  return e;
}

// True when the tensor maps in `tp` already describe p's caches.
bool same_caches(const TcDecParams &tp, int tp_dev, const DecParams &p, int dev) {
  if (tp_dev != dev || tp.p.L != p.L || tp.p.B != p.B || tp.p.Hkv != p.Hkv) return false;
  for (int t = 0; t < p.L; ++t) {
    const int l = p.order[t];
    if (tp.p.order[t] != l || tp.p.kc[l] != p.kc[l] || tp.p.vc[l] != p.vc[l] ||
        tp.p.cap[l] != p.cap[l])
      return false;
  }
  return true;
}

// Counter blocks this path left at zero, per device: the kernel resets its
// counters on exit, so a workspace used by the previous call on the device
// needs no clearing.
struct CleanCtrl {
  const void *ptr = nullptr;
  size_t bytes = 0;
};
CleanCtrl g_clean[kMaxDevices];
std::mutex g_clean_mu;

cudaError_t clear_ctrl_if_needed(int dev, int *ctrl, size_t bytes, cudaStream_t st) {
  std::lock_guard<std::mutex> lock(g_clean_mu);
  CleanCtrl &c = g_clean[dev];
  if (c.ptr == ctrl && c.bytes >= bytes) return cudaSuccess;
  const cudaError_t e = cudaMemsetAsync(ctrl, 0, bytes, st);
  if (e == cudaSuccess) {
    c.ptr = ctrl;
    c.bytes = bytes;
  }
  return e;
}

}  // namespace

bool decode_tc_supported(const ripple_decode_desc *d) {
  const int G = d->n_q_heads / d->n_kv_heads;
  return d->dtype == RIPPLE_BF16 && d->head_dim == 128 && d->n_layers <= kTcMaxLayers &&
         (G == 1 || G == 2 || G == 4 || G == 8) && encode_fn() != nullptr;
}

void decode_tc_forget_ctrl(const void *ctrl) {
  std::lock_guard<std::mutex> lock(g_clean_mu);
  for (auto &c : g_clean)
    if (c.ptr == ctrl) c = CleanCtrl{};
}

cudaError_t launch_decode_tc(const DecParams &p, size_t ctrl_bytes, cudaStream_t st) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr || p.L > kTcMaxLayers) return cudaErrorNotSupported;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  e = clear_ctrl_if_needed(dev, p.ctrl, ctrl_bytes, st);
  if (e != cudaSuccess) return e;
  // Tensor maps by work-order position (the kernel indexes them that way);
  // re-encoded only when the caches change (serving loops reuse them).
  static TcDecParams tp;  // large: kept off the stack, filled under the lock
  static int tp_dev = -1;
  static std::mutex mu;
  std::lock_guard<std::mutex> lock(mu);
  if (!same_caches(tp, tp_dev, p, dev)) {
    tp_dev = -1;
    const int units = p.B * p.Hkv;
    for (int t = 0; t < p.L; ++t) {
      const int l = p.order[t];
      if (!encode_cache(enc, &tp.kmap[t], p.kc[l], p.cap[l], units) ||
          !encode_cache(enc, &tp.vmap[t], p.vc[l], p.cap[l], units))
        return cudaErrorInvalidValue;
    }
    tp_dev = dev;
  }
  tp.p = p;
  switch (p.G) {
    case 1: return launch_g<1>(tp, dev, st);
    case 2: return launch_g<2>(tp, dev, st);
    case 4: return launch_g<4>(tp, dev, st);
    case 8: return launch_g<8>(tp, dev, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace ripple
