// Observation-window token scoring on the 5th-generation tensor cores
// (tcgen05, accumulators in TMEM), bf16 keys and queries, d = 128, G*w = 128
// or 256 window rows. SnapKV's rule as RippleKV keeps it (Sec. 4.4, last
// paragraph): logits x = scale * q.k of the window rows against every key,
// causal inside the window, softmax per row over all visible keys, vote of a
// prefix key = sum over rows of its probability.
//
// One launch for all the layers of a call (a unit is a (layer, b, h); each
// layer's keys and queries come through its own tensor maps and its votes go
// to its slot of the vote array), one persistent CTA per SM, co-resident
// (cooperative launch). A unit is cut into items of `tpi` key tiles; item i belongs
// to CTA i mod grid, so every unit is spread over many CTAs that work on it at
// the same time. Each CTA runs its items in the order
//     P1(a0) P1(a1) P2(a0) P1(a2) P2(a1) ...
//   pass 1 of an item: per window row, (max, sum of exp) over the item's key
//     tiles -> partial[unit][item][row] (the publisher warp combines the two
//     epilogue warpgroups' statistics); it counts the unit's finished items
//     and the last one merges them into
//     lognorm[unit][row] = max + log2(sum) and raises ready[unit];
//   pass 2 of an item: per prefix key, vote = sum over rows of
//     exp2(x * scale * log2e - lognorm[row]), once ready[unit] is up.
// An item's keys are read again one item later, so the second read is served
// from L2 (about two items per SM are in flight). A pass-2 wait only depends
// on first passes of strictly earlier units as long as a unit has at most
// twice as many items as there are CTAs, so with every CTA resident the
// schedule cannot deadlock.
//
// Warp roles (352 threads): warp 0 = TMA producers (keys, queries), warp 1 = MMA issuer and
// TMEM owner, warps 2-9 = two epilogue warpgroups taking alternate key tiles,
// warp 10 = publisher of pass-1 results. Pass 1 computes D[row][key]
// (A = window queries, B = key tile); pass 2 computes D[key][row] (A = key
// tile, B = window queries), so each epilogue thread owns one row (pass 1) or
// one key (pass 2) and every reduction is thread-local.
// Every wait is bounded: on timeout the CTA raises RIPPLE_ETIMEOUT, all roles
// leave their loops, and TMEM is released.
#include <cuda.h>
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "kernels.cuh"
#include "tc_ptx.cuh"

namespace ripple {
namespace {

constexpr int kTile = 128;                      // keys per tile
constexpr int kHalfBytes = kTile * 64 * 2;      // 64 bf16 columns of 128 rows: 16 KB
constexpr int kTileBytes = 2 * kHalfBytes;      // one 128 x 128 bf16 tile
constexpr int kThreads = 352;
constexpr int kPubSlots = 2;
// Items of at least 64 key tiles: with every layer of a call in one launch the
// pipeline's fill and drain no longer favour small items, and fewer items
// mean fewer partial statistics to publish and merge (80 layers of the 70B
// shape: 12.36 / 12.07 / 11.76 / 11.59 / 11.58 / 11.53 / 13.11 ms with items
// of 14 / 18 / 32 / 64 / 128 / 256 / 1024 tiles; one item per unit leaves the
// last wave of units short).
constexpr int kMinTilesPerItem = 64;


// ------------------------------------------------------------ work list

struct TcParams {
  int units, upl, T, P, W, Hq, Hkv, G;  // units of all scored layers, units per layer
  int n_tiles1, n_tiles2;  // key tiles of pass 1 (all keys) and pass 2 (prefix keys)
  int tpi, n_ch;           // key tiles per item, items per unit
  int total_items;
  float scale2;
  float2 *partial;  // [units][n_ch][R] (max, sum) per item and row, log2 domain
  float *lognorm;   // [units][R]
  float *votes;     // [n_layers][upl][P]: unit u's votes at layer_of[u / upl]
  int layer_of[kCompressMaxLayers];  // the layer (votes slot) of each scored layer
  int n_slots;                       // layers (votes slots) of the votes array
  int *ctrl;        // [u] items of unit u published; [units + u] row statistics ready
  int32_t *status;
  long long wait_cycles;  // bound of the in-kernel waits
};

struct ItemRef {
  int unit, chunk;
};

// The k-th item of this CTA.
__device__ __forceinline__ ItemRef item_of(const TcParams &p, int k) {
  const int i = (int)blockIdx.x + k * (int)gridDim.x;
  return {i / p.n_ch, i % p.n_ch};
}

__device__ __forceinline__ int items_of_cta(const TcParams &p) {
  const int b = (int)blockIdx.x;
  return b < p.total_items ? (p.total_items - 1 - b) / (int)gridDim.x + 1 : 0;
}

__device__ __forceinline__ void tiles_of(const TcParams &p, const ItemRef &it, int pass, int &t0,
                                         int &t1) {
  t0 = it.chunk * p.tpi;
  t1 = min(pass == 1 ? p.n_tiles1 : p.n_tiles2, t0 + p.tpi);
}

// ------------------------------------------------------------ shared memory

template <int NR>
struct Cfg {
  static constexpr int R = 128 * NR;             // window rows
  static constexpr int NK = NR == 1 ? 3 : 2;     // key-tile stages
  // Query buffers: two items are in flight (pass 1 of one, pass 2 of the
  // previous); a third lets the next item's queries load ahead.
  static constexpr int NQ = NR == 1 ? 3 : 2;
  static constexpr int NA = NR == 1 ? 4 : 2;     // TMEM accumulator stages
  static constexpr int ACC_COLS = 128 * NR;      // TMEM columns per stage
  static constexpr int QBYTES = R * 256;         // R rows x 128 bf16
  static constexpr int OFF_K = 0;
  static constexpr int OFF_Q = OFF_K + NK * kTileBytes;
  static constexpr int OFF_MISC = OFF_Q + NQ * QBYTES;
};

struct Misc {
  uint64_t k_full[4], k_empty[4], q_full[3], q_empty[3], acc_full[4], acc_empty[4], mma_done;
  uint64_t pub_full[kPubSlots], pub_empty[kPubSlots];
  uint32_t tmem_base;
  int abort_flag;
  long long wait_cycles;  // bound of the waits of this launch
  alignas(16) float off[2][256];  // per-warpgroup row log-normalisers of a pass-2 item
  float2 pstat[kPubSlots][2][256];  // pass-1 row statistics per slot and warpgroup
};

static_assert(offsetof(Misc, off) % 16 == 0, "float4-read shared arrays are 16-byte aligned");

template <int NR>
constexpr int smem_bytes() {
  return Cfg<NR>::OFF_MISC + (int)sizeof(Misc) + 1024;  // + 1024-byte alignment slack
}

// Bounded mbarrier wait that also gives up as soon as another role aborted.
__device__ __forceinline__ bool wait_bar(uint64_t *bar, uint32_t parity, Misc *ms,
                                         int32_t *status) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*(volatile int *)&ms->abort_flag) return false;
    if (clock64() - t0 > ms->wait_cycles) {
      *(volatile int *)&ms->abort_flag = 1;
      report(status, RIPPLE_ETIMEOUT);
      return false;
    }
  }
}

// Warp-uniform variant: all lanes wait, the warp then agrees on the outcome
// (and is converged for the .sync.aligned TMEM loads that follow).
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, Misc *ms,
                                          int32_t *status) {
  const bool ok = wait_bar(bar, parity, ms, status);
  return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ bool wait_ready(const int *flag, Misc *ms, int32_t *status) {
  if (ld_acquire(flag)) return true;
  const long long t0 = clock64();
  for (;;) {
    if (ld_acquire(flag)) return true;
    if (*(volatile int *)&ms->abort_flag) return false;
    if (clock64() - t0 > ms->wait_cycles) {
      *(volatile int *)&ms->abort_flag = 1;
      report(status, RIPPLE_ETIMEOUT);
      return false;
    }
    __nanosleep(64);
  }
}

__device__ __forceinline__ void combine(float &m, float &l, float m2, float l2) {
  const float mm = fmaxf(m, m2);
  if (mm == -INFINITY) return;
  l = l * fast_exp2(m - mm) + l2 * fast_exp2(m2 - mm);
  m = mm;
}

// ------------------------------------------------------------ kernel

// Kernel argument: the keys of every scored layer as 3-D tensor maps
// [unit][T][128], their window queries as 2-D maps [B * Hq * W][128], and the
// parameters.
struct TcLaunch {
  CUtensorMap kmap[kCompressMaxLayers];
  CUtensorMap qmap[kCompressMaxLayers];
  TcParams p;
};

template <int NR>
__global__ void __launch_bounds__(kThreads, 1)
    score_tc_kernel(const __grid_constant__ TcLaunch lp) {
  using C = Cfg<NR>;
  const TcParams &p = lp.p;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t *ktiles = smem + C::OFF_K;
  uint8_t *qbufs = smem + C::OFF_Q;
  Misc *ms = (Misc *)(smem + C::OFF_MISC);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = items_of_cta(p);

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::NK; ++i) {
      mbar_init(&ms->k_full[i], 1);
      mbar_init(&ms->k_empty[i], 1);
    }
    for (int i = 0; i < C::NQ; ++i) {
      mbar_init(&ms->q_full[i], 1);
      mbar_init(&ms->q_empty[i], 1);
    }
    for (int i = 0; i < C::NA; ++i) {
      mbar_init(&ms->acc_full[i], 1);
      mbar_init(&ms->acc_empty[i], 4);
    }
    for (int i = 0; i < kPubSlots; ++i) {
      mbar_init(&ms->pub_full[i], 8);
      mbar_init(&ms->pub_empty[i], 1);
    }
    mbar_init(&ms->mma_done, 1);
    ms->abort_flag = 0;
    ms->wait_cycles = p.wait_cycles;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&ms->tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ms->tmem_base;

  // Every role walks the same sequence: for k = 0..n, P1(item k) if k < n,
  // then P2(item k - 1) if k >= 1.
  if (warp == 0) {
    // ------------------------------------------------ TMA producers
    // Lane 0 streams key tiles through the ring; lane 1 loads each item's
    // window queries as soon as a query buffer is free, so that the key
    // stream never waits for a query load.
    if (lane == 0) {
      int kcount = 0;
      const uint64_t keep = policy_evict_last(), drop = policy_evict_first();
      bool ok = true;
      for (int k = 0; k <= n && ok; ++k) {
        for (int pass = 1; pass <= 2 && ok; ++pass) {
          if ((pass == 1 && k >= n) || (pass == 2 && k < 1)) continue;
          const ItemRef it = item_of(p, pass == 1 ? k : k - 1);
          int t0, t1;
          tiles_of(p, it, pass, t0, t1);
          for (int t = t0; t < t1; ++t) {
            const int ks = kcount % C::NK;
            if (!wait_bar(&ms->k_empty[ks], ((kcount / C::NK) & 1) ^ 1, ms, p.status)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&ms->k_full[ks], kTileBytes);
            uint8_t *kb = ktiles + ks * kTileBytes;
            const uint64_t pol = pass == 1 ? keep : drop;
            const CUtensorMap *km = &lp.kmap[it.unit / p.upl];
            const int local = it.unit % p.upl;
            tma_load_3d(kb, km, 0, t * kTile, local, &ms->k_full[ks], pol);
            tma_load_3d(kb + kHalfBytes, km, 64, t * kTile, local, &ms->k_full[ks], pol);
            ++kcount;
          }
        }
      }
      // Let every issued copy land before the CTA can exit (matters only after
      // an abort; in normal operation every stage was already consumed).
      for (int j = max(0, kcount - C::NK); j < kcount; ++j)
        mbar_wait(&ms->k_full[j % C::NK], (j / C::NK) & 1, nullptr);
    } else if (lane == 1) {
      int qcount = 0;
      for (int k = 0; k < n; ++k) {
        const ItemRef it = item_of(p, k);
        const int local = it.unit % p.upl;
        const int b = local / p.Hkv, h = local % p.Hkv;
        const int qrow0 = (b * p.Hq + h * p.G) * p.W;
        const CUtensorMap *qm = &lp.qmap[it.unit / p.upl];
        const int qs = k % C::NQ;
        if (!wait_bar(&ms->q_empty[qs], ((k / C::NQ) & 1) ^ 1, ms, p.status)) break;
        mbar_arrive_expect_tx(&ms->q_full[qs], C::QBYTES);
        uint8_t *qb = qbufs + qs * C::QBYTES;
        for (int half = 0; half < 2; ++half)
          for (int nr = 0; nr < NR; ++nr)
            tma_load_2d(qb + half * (NR * kHalfBytes) + nr * kHalfBytes, qm, half * 64,
                        qrow0 + nr * 128, &ms->q_full[qs]);
        ++qcount;
      }
      for (int k = max(0, qcount - C::NQ); k < qcount; ++k)
        mbar_wait(&ms->q_full[k % C::NQ], (k / C::NQ) & 1, nullptr);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      int kcount = 0, acount = 0;
      constexpr uint32_t id1 = idesc_bf16(128, 128);
      constexpr uint32_t id2 = idesc_bf16(128, 128 * NR);
      const uint32_t kbase = smem_u32(ktiles), qbase = smem_u32(qbufs);
      bool ok = true;
      for (int k = 0; k <= n && ok; ++k) {
        for (int pass = 1; pass <= 2 && ok; ++pass) {
          if ((pass == 1 && k >= n) || (pass == 2 && k < 1)) continue;
          const int item = pass == 1 ? k : k - 1;
          const ItemRef it = item_of(p, item);
          const int qs = item % C::NQ;
          if (pass == 1 && !wait_bar(&ms->q_full[qs], (item / C::NQ) & 1, ms, p.status)) {
            ok = false;
            break;
          }
          const uint32_t qa = qbase + qs * C::QBYTES;
          int t0, t1;
          tiles_of(p, it, pass, t0, t1);
          for (int t = t0; t < t1; ++t) {
            const int ks = kcount % C::NK, as = acount % C::NA;
            if (!wait_bar(&ms->k_full[ks], (kcount / C::NK) & 1, ms, p.status) ||
                !wait_bar(&ms->acc_empty[as], ((acount / C::NA) & 1) ^ 1, ms, p.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t d = tmem + as * C::ACC_COLS;
            const uint32_t ka = kbase + ks * kTileBytes;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              const uint32_t koff = (kk >> 2) * kHalfBytes + (kk & 3) * 32;
              const uint32_t qoff = (kk >> 2) * (NR * kHalfBytes) + (kk & 3) * 32;
              if (pass == 1) {
#pragma unroll
                for (int nr = 0; nr < NR; ++nr)
                  mma_bf16(d + nr * 128, sw128_desc(qa + qoff + nr * kHalfBytes),
                           sw128_desc(ka + koff), id1, kk > 0);
              } else {
                mma_bf16(d, sw128_desc(ka + koff), sw128_desc(qa + qoff), id2, kk > 0);
              }
            }
            mma_commit(&ms->k_empty[ks]);
            mma_commit(&ms->acc_full[as]);
            ++kcount;
            ++acount;
          }
          if (ok && pass == 2) mma_commit(&ms->q_empty[qs]);  // the item is done with its queries
        }
      }
      // All issued MMAs complete before TMEM is released.
      mma_commit(&ms->mma_done);
      mbar_wait(&ms->mma_done, 0, nullptr);
    }
  } else if (warp == 10) {
    // ------------------------------------------------ publisher of pass-1 results
    constexpr int RJ = C::R / 32;   // rows per lane
    constexpr int CB = 32 / RJ;     // items merged per batch: 32 loads in flight per lane
    for (int k = 0; k < n; ++k) {
      const int slot = k % kPubSlots;
      if (!warp_wait(&ms->pub_full[slot], (k / kPubSlots) & 1, ms, p.status)) break;
      const ItemRef it = item_of(p, k);
      // One partial per item: the two warpgroups' statistics combined here.
      float2 *mine = p.partial + guard((long long)it.unit * p.n_ch + it.chunk, 1,
                                       (long long)p.units * p.n_ch, p.status) *
                                     C::R;
#pragma unroll
      for (int j = 0; j < RJ; ++j) {
        const int r = lane + 32 * j;
        float2 a = ms->pstat[slot][0][r];
        const float2 b = ms->pstat[slot][1][r];
        combine(a.x, a.y, b.x, b.y);
        mine[r] = a;
      }
      __syncwarp();  // all lanes' rows are written (and the slot read) before lane 0 goes on
      int last = 0;
      if (lane == 0) {
        mbar_arrive(&ms->pub_empty[slot]);
        __threadfence();  // the item's partial becomes visible GPU-wide before it is counted
        last = atomicAdd(&p.ctrl[guard(it.unit, 1, p.units, p.status)], 1) == p.n_ch - 1;
      }
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        // Last item of the unit: merge its n_ch partials per row.
        __threadfence();
        const float2 *part =
            p.partial + guard((long long)it.unit * p.n_ch, p.n_ch, (long long)p.units * p.n_ch,
                              p.status) *
                            C::R;
        float mm[RJ], ll[RJ];
#pragma unroll
        for (int j = 0; j < RJ; ++j) {
          mm[j] = -INFINITY;
          ll[j] = 0.f;
        }
        for (int c0 = 0; c0 < p.n_ch; c0 += CB) {
          float2 q[CB][RJ];
#pragma unroll
          for (int c = 0; c < CB; ++c)
#pragma unroll
            for (int j = 0; j < RJ; ++j)
              q[c][j] = c0 + c < p.n_ch ? __ldcg(&part[(size_t)(c0 + c) * C::R + lane + 32 * j])
                                        : make_float2(-INFINITY, 0.f);
#pragma unroll
          for (int c = 0; c < CB; ++c)
#pragma unroll
            for (int j = 0; j < RJ; ++j) combine(mm[j], ll[j], q[c][j].x, q[c][j].y);
        }
#pragma unroll
        for (int j = 0; j < RJ; ++j)
          p.lognorm[guard(it.unit, 1, p.units, p.status) * C::R + lane + 32 * j] =
              mm[j] + __log2f(ll[j]);
        __threadfence();
        __syncwarp();
        if (lane == 0) st_release(&p.ctrl[guard(p.units + it.unit, 1, 2LL * p.units, p.status)], 1);
      }
    }
  } else {
    // ------------------------------------------------ epilogue warpgroups
    const int wg = (warp - 2) >> 2;
    const int quarter = warp & 3;              // TMEM lanes this warp may access
    const int lrow = quarter * 32 + lane;      // row (pass 1) or key (pass 2) in the tile
    const int wtid = threadIdx.x - 64 - wg * 128;  // 0..127 within the warpgroup
    const uint32_t lane_addr = (uint32_t)(quarter * 32) << 16;
    int tcount = 0;
    // Inside an item every warp follows the same control flow even if a wait
    // gives up (the tile is then skipped), so that the named barriers below
    // are always reached by all of their threads.
    for (int k = 0; k <= n; ++k) {
      if (k < n) {
        // ---------------- pass 1 of item k
        const ItemRef it = item_of(p, k);
        int t0, t1;
        tiles_of(p, it, 1, t0, t1);
        float m[NR], l[NR];
        int last_vis[NR];
#pragma unroll
        for (int nr = 0; nr < NR; ++nr) {
          m[nr] = -INFINITY;
          l[nr] = 0.f;
          last_vis[nr] = p.P + (lrow + nr * 128) % p.W;
        }
        for (int t = t0; t < t1; ++t, ++tcount) {
          if ((tcount & 1) != wg) continue;
          const int as = tcount % C::NA;
          if (!warp_wait(&ms->acc_full[as], (tcount / C::NA) & 1, ms, p.status)) continue;
          tc_fence_after();
          const bool masked = (t + 1) * kTile - 1 >= p.P;
#pragma unroll
          for (int nr = 0; nr < NR; ++nr) {
            uint32_t x[4][32];
            const uint32_t base = tmem + lane_addr + as * C::ACC_COLS + nr * 128;
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_ld32(base + c * 32, x[c]);
            tmem_wait_ld();
            if (nr == NR - 1) {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(&ms->acc_empty[as]);
            }
            if (masked) {  // keys this row cannot see (causal window, past T) -> -inf
#pragma unroll
              for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int j = 0; j < 32; ++j)
                  if (t * kTile + c * 32 + j > last_vis[nr]) x[c][j] = 0xff800000u;
            }
            // Eight independent chains keep the max and the sum off one long
            // dependency chain.
            float mx[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) mx[i] = -INFINITY;
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
              for (int j = 0; j < 32; ++j) mx[j & 7] = fmaxf(mx[j & 7], __uint_as_float(x[c][j]));
            const float tmax = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                                     fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
            if (tmax == -INFINITY) continue;
            const float mnew = fmaxf(m[nr], tmax * p.scale2);
            // fp32x2: logits scaled and shifted two at a time, sums in pairs
            float2 sv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) sv[i] = make_float2(0.f, 0.f);
            const float2 s2 = make_float2(p.scale2, p.scale2), mn2 = make_float2(-mnew, -mnew);
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
              for (int j = 0; j < 32; j += 2) {
                const float2 y = __ffma2_rn(
                    make_float2(__uint_as_float(x[c][j]), __uint_as_float(x[c][j + 1])), s2, mn2);
                sv[(j >> 1) & 3] =
                    __fadd2_rn(sv[(j >> 1) & 3], make_float2(fast_exp2(y.x), fast_exp2(y.y)));
              }
            const float s = ((sv[0].x + sv[0].y) + (sv[1].x + sv[1].y)) +
                            ((sv[2].x + sv[2].y) + (sv[3].x + sv[3].y));
            l[nr] = l[nr] * fast_exp2(m[nr] - mnew) + s;
            m[nr] = mnew;
          }
        }
        // This warpgroup's row statistics of the item go to the publisher warp
        // through a shared-memory slot.
        const int slot = k % kPubSlots;
        warp_wait(&ms->pub_empty[slot], ((k / kPubSlots) & 1) ^ 1, ms, p.status);
#pragma unroll
        for (int nr = 0; nr < NR; ++nr) ms->pstat[slot][wg][nr * 128 + lrow] = make_float2(m[nr], l[nr]);
        __syncwarp();  // every lane's rows are written before lane 0 arrives
        if (lane == 0) mbar_arrive(&ms->pub_full[slot]);
      }
      if (k >= 1) {
        // ---------------- pass 2 of item k - 1
        const ItemRef it = item_of(p, k - 1);
        int t0, t1;
        tiles_of(p, it, 2, t0, t1);
        if (t1 > t0) {
          if (wtid == 0)
            wait_ready(&p.ctrl[guard(p.units + it.unit, 1, 2LL * p.units, p.status)], ms, p.status);
          named_bar_sync(3 + wg, 128);
          for (int r = wtid; r < C::R; r += 128)
            ms->off[wg][r] = __ldcg(&p.lognorm[guard(it.unit, 1, p.units, p.status) * C::R + r]);
          named_bar_sync(3 + wg, 128);
        }
        const float4 *off4 = (const float4 *)ms->off[wg];
        // the unit's votes slot: its layer's in the vote array
        const int vunit = p.layer_of[it.unit / p.upl] * p.upl + it.unit % p.upl;
        for (int t = t0; t < t1; ++t, ++tcount) {
          if ((tcount & 1) != wg) continue;
          const int as = tcount % C::NA;
          if (!warp_wait(&ms->acc_full[as], (tcount / C::NA) & 1, ms, p.status)) continue;
          tc_fence_after();
          // fp32x2: logits scaled and shifted two at a time, sums in pairs
          float2 vs[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) vs[i] = make_float2(0.f, 0.f);
          const float2 s2 = make_float2(p.scale2, p.scale2);
          const uint32_t base = tmem + lane_addr + as * C::ACC_COLS;
#pragma unroll
          for (int c4 = 0; c4 < NR; ++c4) {
            uint32_t x[4][32];
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_ld32(base + c4 * 128 + c * 32, x[c]);
            tmem_wait_ld();
            if (c4 == NR - 1) {
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(&ms->acc_empty[as]);
            }
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
              for (int j = 0; j < 32; j += 4) {
                const float4 o = off4[(c4 * 128 + c * 32 + j) >> 2];
                const int h = (j >> 1) & 2;  // two pair chains per 4 columns: 4 in flight
                const float2 y0 = __ffma2_rn(
                    make_float2(__uint_as_float(x[c][j]), __uint_as_float(x[c][j + 1])), s2,
                    make_float2(-o.x, -o.y));
                const float2 y1 = __ffma2_rn(
                    make_float2(__uint_as_float(x[c][j + 2]), __uint_as_float(x[c][j + 3])), s2,
                    make_float2(-o.z, -o.w));
                vs[h] = __fadd2_rn(vs[h], make_float2(fast_exp2(y0.x), fast_exp2(y0.y)));
                vs[h + 1] = __fadd2_rn(vs[h + 1], make_float2(fast_exp2(y1.x), fast_exp2(y1.y)));
              }
          }
          const float vote = ((vs[0].x + vs[0].y) + (vs[1].x + vs[1].y)) +
                             ((vs[2].x + vs[2].y) + (vs[3].x + vs[3].y));
          const int key = t * kTile + lrow;
          if (key < p.P)
            p.votes[guard((long long)vunit * p.P + key, 1, (long long)p.n_slots * p.upl * p.P,
                          p.status)] = vote;
        }
      }
    }
  }

  tc_fence_before();
  __syncwarp();  // idle lanes of the single-thread roles wait for their lane 0 here
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ------------------------------------------------------------ host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (fn == nullptr) {
    void *ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (EncodeTiledFn)ptr;
  }
  return fn;
}

int sm_count() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

template <int NR>
cudaError_t launch_nr(const LayerGeom &g, int n_slots, const int *slots, int n_scored,
                      const void *const *q_win, const void *const *k, const CompressWs &ws,
                      float *votes, int32_t *status, cudaStream_t st) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return cudaErrorNotSupported;
  if (n_scored < 1 || n_scored > kCompressMaxLayers || n_slots < 1) return cudaErrorInvalidValue;
  static TcLaunch lp;  // large: kept off the stack, filled under the lock
  static std::mutex mu;
  std::lock_guard<std::mutex> lock(mu);
  for (int l = 0; l < n_scored; ++l) {
    cuuint64_t dims[3] = {128, (cuuint64_t)g.T, (cuuint64_t)g.units};
    cuuint64_t strides[2] = {256, (cuuint64_t)g.T * 256};
    cuuint32_t box[3] = {64, 128, 1};
    cuuint32_t es[3] = {1, 1, 1};
    if (enc(&lp.kmap[l], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(k[l]), dims,
            strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
    cuuint64_t qdims[2] = {128, (cuuint64_t)g.B * g.Hq * g.W};
    cuuint64_t qstrides[1] = {256};
    cuuint32_t qbox[2] = {64, 128};
    cuuint32_t qes[2] = {1, 1};
    if (enc(&lp.qmap[l], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(q_win[l]), qdims,
            qstrides, qbox, qes, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  const int sms = sm_count();
  TcParams &p = lp.p;
  p.upl = g.units;
  p.units = g.units * n_scored;
  p.T = g.T;
  p.P = g.P;
  p.W = g.W;
  p.Hq = g.Hq;
  p.Hkv = g.Hkv;
  p.G = g.G;
  p.n_tiles1 = (g.T + kTile - 1) / kTile;
  p.n_tiles2 = (g.P + kTile - 1) / kTile;
  // Tiles per item: at least kMinTilesPerItem (hand-offs are per item), and
  // enough that a unit has no more items than there are SMs (deadlock-free
  // schedule, see the header comment).
  const int tpi_min = (p.n_tiles1 + sms - 1) / sms;
  p.tpi = tpi_min > kMinTilesPerItem ? tpi_min : kMinTilesPerItem;
  p.n_ch = (p.n_tiles1 + p.tpi - 1) / p.tpi;
  p.total_items = p.units * p.n_ch;
  p.scale2 = g.scale2;
  p.partial = ws.row_partial;
  p.lognorm = ws.row_lognorm;
  p.votes = votes;
  for (int l = 0; l < n_scored; ++l) {
    if (slots[l] < 0 || slots[l] >= n_slots) return cudaErrorInvalidValue;
    p.layer_of[l] = slots[l];
  }
  p.n_slots = n_slots;
  p.ctrl = ws.counters;
  p.status = status;
  p.wait_cycles = wait_limit_cycles();
  cudaError_t e = cudaMemsetAsync(ws.counters, 0, sizeof(int) * 2 * p.units, st);
  if (e != cudaSuccess) return e;
  constexpr int smem = smem_bytes<NR>();
  static_assert(smem <= 227 * 1024, "shared memory budget");
  e = cudaFuncSetAttribute(score_tc_kernel<NR>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int grid = p.total_items < sms ? p.total_items : sms;
  // Cooperative launch: every CTA resident at once, which the cross-CTA waits
  // of the schedule rely on.
  void *args[] = {(void *)&lp};
  e = cudaLaunchCooperativeKernel((const void *)score_tc_kernel<NR>, dim3(grid), dim3(kThreads),
                                  args, (size_t)smem, st);
  count_launches(1);
  return e;
}

}  // namespace

bool score_tc_supported(const LayerGeom &g) {
  return g.dtype == RIPPLE_BF16 && g.D == 128 && (g.R == 128 || g.R == 256) && g.P > 0 &&
         encode_fn() != nullptr;
}

cudaError_t launch_score_tc(const LayerGeom &g, int n_slots, const int *slots, int n_scored,
                            const void *const *q_win, const void *const *k, const CompressWs &ws,
                            float *votes, int32_t *status, cudaStream_t st) {
  if (g.R == 128)
    return launch_nr<1>(g, n_slots, slots, n_scored, q_win, k, ws, votes, status, st);
  return launch_nr<2>(g, n_slots, slots, n_scored, q_win, k, ws, votes, status, st);
}

cudaError_t launch_score_tc(const LayerGeom &g, const void *q_win, const void *k,
                            const CompressWs &ws, float *votes, int32_t *status,
                            cudaStream_t st) {
  const int slot = 0;
  return launch_score_tc(g, 1, &slot, 1, &q_win, &k, ws, votes, status, st);
}

}  // namespace ripple
