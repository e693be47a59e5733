// Observation-window token scoring for G * w = 128 window rows (SnapKV's rule
// as RippleKV keeps it, Sec. 4.4, last paragraph), bf16, d = 128, on the
// 5th-generation tensor cores.
//
// One persistent CTA per SM, item i on CTA i mod grid; in its step k a CTA
// runs P1(a_k) then P2(a_k-1), so that keys are re-read from L2 one item
// after their first read; a publisher warp merges pass-1 row statistics.
// Each pass takes the layout in which its reduction stays inside one thread:
//   pass 1  D[row][key] = Q . K_tile^T; a thread owns a row and folds its
//           keys into the row's running max and sum;
//   pass 2  D[key][row] = K_tile . Q^T; a thread owns a key and sums its 128
//           rows' probabilities, so a key's vote needs no shuffles and no
//           exchange between warps.
// Both passes take the queries from shared memory (a 32 KB buffer per pass,
// loaded by TMA once per item) and the key tile from a 4-stage TMA ring; TMEM
// holds four 128-column accumulators, so the MMA issuer can run two tiles
// ahead of each epilogue warpgroup.
//
// Warp roles (352 threads): warp 0 = key-tile and query producer, warp 1 =
// MMA issuer and TMEM owner, warps 2-9 = two epilogue warpgroups taking
// alternate tiles, warp 10 = publisher of pass-1 results. Every wait is
// bounded; on timeout the CTA raises RIPPLE_ETIMEOUT, every role leaves its
// loop and TMEM is released.
#include <cuda.h>
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "kernels.cuh"
#include "tc_ptx.cuh"

namespace ripple {
namespace {

constexpr int kTile = 128;                      // keys per tile
constexpr int kHalfBytes = kTile * 64 * 2;      // one TMA box: 64 dims of 128 keys
constexpr int kTileBytes = 2 * kHalfBytes;
constexpr int kThreads = 352;
constexpr int kNK = 4;                          // key-tile stages
constexpr int kLag = 1;                         // pass 2 of item k runs in step k + kLag
constexpr int kNA = 4;                          // accumulators in TMEM (128 columns each)
constexpr int kPubSlots = 2;
constexpr int kMinTilesPerItem = 9;
static_assert(kNA * 128 <= 512, "TMEM columns");

struct Tc1Params {
  int units, upl, T, P, W, Hq, Hkv, G;  // units of all layers, units per layer
  int n_tiles1, n_tiles2;  // key tiles of pass 1 (all keys) and pass 2 (prefix keys)
  int tpi, n_ch;           // key tiles per item, items per unit
  int total_items;
  float scale2;
  const uint8_t *q[kCompressMaxLayers];  // per layer: window queries [B][Hq][W][128] bf16
  float2 *partial;   // [units][n_ch][128] (max, sum) per item and row, log2 domain
  float *lognorm;    // [units][128]
  float *votes;      // [units][P], layer-major
  int *ctrl;         // [u] items of unit u published; [units + u] row statistics ready
  int32_t *status;
  long long wait_cycles;  // bound of the in-kernel waits
};

struct ItemRef {
  int unit, chunk;
};

__device__ __forceinline__ ItemRef item_of(const Tc1Params &p, int k) {
  const int i = (int)blockIdx.x + k * (int)gridDim.x;
  return {i / p.n_ch, i % p.n_ch};
}

__device__ __forceinline__ int items_of_cta(const Tc1Params &p) {
  const int b = (int)blockIdx.x;
  return b < p.total_items ? (p.total_items - 1 - b) / (int)gridDim.x + 1 : 0;
}

__device__ __forceinline__ void tiles_of(const Tc1Params &p, const ItemRef &it, int pass, int &t0,
                                         int &t1) {
  t0 = it.chunk * p.tpi;
  t1 = min(pass == 1 ? p.n_tiles1 : p.n_tiles2, t0 + p.tpi);
}

// Step k of a CTA's schedule: pass 1 of its item k (if k < n), then pass 2
// of its item k - kLag (if k >= kLag). With a lag of one item, an item's keys
// are re-read one item later, so about two items of keys per CTA (78 MB over
// the GPU) stay in L2 and the keys come from DRAM once; a lag of two leaves
// the other CTAs more time to publish the statistics pass 2 waits for, but
// its three items per CTA no longer fit in L2 (measured: 3% faster, 1.6x the
// DRAM reads).

struct Step {
  int u1, a0, n1;  // pass 1: unit, first tile, tiles
  int u2, b0, n2;  // pass 2
  int len;         // max(n1, n2)
};

__device__ __forceinline__ Step step_of(const Tc1Params &p, int k, int n) {
  Step s{0, 0, 0, 0, 0, 0, 0};
  int e;
  if (k < n) {
    const ItemRef it = item_of(p, k);
    tiles_of(p, it, 1, s.a0, e);
    s.u1 = it.unit;
    s.n1 = max(0, e - s.a0);
  }
  if (k >= kLag) {
    const ItemRef it = item_of(p, k - kLag);
    tiles_of(p, it, 2, s.b0, e);
    s.u2 = it.unit;
    s.n2 = max(0, e - s.b0);
  }
  s.len = s.n1 + s.n2;
  return s;
}

// The epilogue warpgroup that takes the CTA's tile number `tc`: alternate
// tiles, so that each warpgroup meets every phase of its accumulator slot.
__device__ __forceinline__ int wg_of(int tc) { return tc & 1; }

// Position j of step s's tile sequence: its pass-1 tiles, then its pass-2
// tiles.
__device__ __forceinline__ void seq_at(const Step &s, int j, int &pass, int &idx) {
  pass = j < s.n1 ? 1 : 2;
  idx = j < s.n1 ? j : j - s.n1;
}

struct Misc {
  uint64_t k_full[kNK], k_empty[kNK], q_full, q_empty, acc_full[kNA], acc_empty[kNA];
  uint64_t qs_full, qs_empty;           // pass-2 queries in shared memory
  uint64_t pub_full[kPubSlots], pub_empty[kPubSlots], mma_done;
  uint32_t tmem_base;
  int abort_flag;
  long long wait_cycles;  // bound of the waits of this launch
  float2 pstat[kPubSlots][2][128];      // pass-1 row statistics per slot and warpgroup
  alignas(16) float offs[2][128];       // per warpgroup: the pass-2 item's row log-normalisers
};

constexpr int kOffQs = kNK * kTileBytes;          // pass-2 queries: two 64-dim halves
constexpr int kOffQ1 = kOffQs + kTileBytes;       // pass-1 queries
constexpr int kOffMisc = kOffQ1 + kTileBytes;
constexpr int kSmemBytes = kOffMisc + (int)sizeof(Misc) + 1024;  // + alignment slack
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");

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

// Kernel argument: the keys of every layer as 3-D tensor maps [unit][T][128],
// the window queries of every layer as 2-D maps [B * Hq * W][128], and the
// parameters.
struct Tc1Launch {
  CUtensorMap kmap[kCompressMaxLayers];
  CUtensorMap qmap[kCompressMaxLayers];
  Tc1Params p;
};

__global__ void __launch_bounds__(kThreads, 1)
    score_tc1_kernel(const __grid_constant__ Tc1Launch lp) {
  const Tc1Params &p = lp.p;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t *ktiles = smem;
  uint8_t *qsm = smem + kOffQs;
  uint8_t *q1m = smem + kOffQ1;
  Misc *ms = (Misc *)(smem + kOffMisc);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = items_of_cta(p);

  if (threadIdx.x == 0) {
    for (int i = 0; i < kNK; ++i) {
      mbar_init(&ms->k_full[i], 1);
      mbar_init(&ms->k_empty[i], 1);
    }
    mbar_init(&ms->q_full, 1);
    mbar_init(&ms->q_empty, 1);
    for (int i = 0; i < kNA; ++i) {
      mbar_init(&ms->acc_full[i], 1);
      mbar_init(&ms->acc_empty[i], 4);
    }
    mbar_init(&ms->qs_full, 1);
    mbar_init(&ms->qs_empty, 1);
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

  // Every role walks the same sequence of steps k = 0 .. n + kLag - 1.
  if (warp == 0) {
    // ------------------------------------------------ key-tile producer
    if (lane == 0) {
      int kcount = 0, qcount = 0;
      const uint64_t keep = policy_evict_last(), drop = policy_evict_first();
      bool ok = true;
      for (int k = 0; k < n + kLag && ok; ++k) {
        const Step st = step_of(p, k, n);
        for (int j = 0; j < st.len && ok; ++j) {
          {
            int pass, s;
            seq_at(st, j, pass, s);
            if (pass == 1 && s == 0) {
              // item k's queries into the pass-1 buffer, once the previous
              // item's pass-1 MMAs have read it
              if (!wait_bar(&ms->q_empty, (k & 1) ^ 1, ms, p.status)) {
                ok = false;
                break;
              }
              const int layer = st.u1 / p.upl, local = st.u1 % p.upl;
              const int b = local / p.Hkv, h = local % p.Hkv;
              const int qrow0 = (b * p.Hq + h * p.G) * p.W;
              mbar_arrive_expect_tx(&ms->q_full, kTileBytes);
              tma_load_2d(q1m, &lp.qmap[layer], 0, qrow0, &ms->q_full);
              tma_load_2d(q1m + kHalfBytes, &lp.qmap[layer], 64, qrow0, &ms->q_full);
            }
            if (pass == 2 && s == 0) {
              // the pass-2 item's queries (rows of its unit) into shared memory
              if (!wait_bar(&ms->qs_empty, (qcount & 1) ^ 1, ms, p.status)) {
                ok = false;
                break;
              }
              const int layer = st.u2 / p.upl, local = st.u2 % p.upl;
              const int b = local / p.Hkv, h = local % p.Hkv;
              const int qrow0 = (b * p.Hq + h * p.G) * p.W;
              mbar_arrive_expect_tx(&ms->qs_full, kTileBytes);
              tma_load_2d(qsm, &lp.qmap[layer], 0, qrow0, &ms->qs_full);
              tma_load_2d(qsm + kHalfBytes, &lp.qmap[layer], 64, qrow0, &ms->qs_full);
              ++qcount;
            }
            const int unit = pass == 1 ? st.u1 : st.u2;
            const int tt = pass == 1 ? st.a0 + s : st.b0 + s;
            const int ks = kcount % kNK;
            if (!wait_bar(&ms->k_empty[ks], ((kcount / kNK) & 1) ^ 1, ms, p.status)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&ms->k_full[ks], kTileBytes);
            uint8_t *kb = ktiles + ks * kTileBytes;
            const uint64_t pol = pass == 1 ? keep : drop;
            const CUtensorMap *km = &lp.kmap[unit / p.upl];
            const int local = unit % p.upl;
            tma_load_3d(kb, km, 0, tt * kTile, local, &ms->k_full[ks], pol);
            tma_load_3d(kb + kHalfBytes, km, 64, tt * kTile, local, &ms->k_full[ks], pol);
            ++kcount;
          }
        }
      }
      for (int j = max(0, kcount - kNK); j < kcount; ++j)
        mbar_wait(&ms->k_full[j % kNK], (j / kNK) & 1, nullptr);
      if (qcount > 0) mbar_wait(&ms->qs_full, (qcount - 1) & 1, nullptr);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      int kcount = 0, acount = 0, qcount = 0;
      constexpr uint32_t id = idesc_bf16(128, 128);
      const uint32_t kbase = smem_u32(ktiles), qsbase = smem_u32(qsm), q1base = smem_u32(q1m);
      bool ok = true;
      for (int k = 0; k < n + kLag && ok; ++k) {
        const Step st = step_of(p, k, n);
        if (k < n && !wait_bar(&ms->q_full, k & 1, ms, p.status)) break;
        for (int j = 0; j < st.len && ok; ++j) {
          {
            int pass, s;
            seq_at(st, j, pass, s);
            if (pass == 2 && s == 0) {
              if (st.n1 > 0) mma_commit(&ms->q_empty);  // item k's pass-1 queries are free
              if (!wait_bar(&ms->qs_full, qcount & 1, ms, p.status)) {
                ok = false;
                break;
              }
            }
            const int ks = kcount % kNK, as = acount % kNA;
            if (!wait_bar(&ms->k_full[ks], (kcount / kNK) & 1, ms, p.status) ||
                !wait_bar(&ms->acc_empty[as], ((acount / kNA) & 1) ^ 1, ms, p.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t d = tmem + as * 128;
            const uint32_t ka = kbase + ks * kTileBytes;
            if (pass == 1) {
#pragma unroll
              for (int kk = 0; kk < 8; ++kk) {
                const uint32_t off = (kk >> 2) * kHalfBytes + (kk & 3) * 32;
                mma_bf16(d, sw128_desc(q1base + off), sw128_desc(ka + off), id, kk > 0);
              }
            } else {
#pragma unroll
              for (int kk = 0; kk < 8; ++kk) {
                const uint32_t off = (kk >> 2) * kHalfBytes + (kk & 3) * 32;
                mma_bf16(d, sw128_desc(ka + off), sw128_desc(qsbase + off), id, kk > 0);
              }
            }
            mma_commit(&ms->k_empty[ks]);
            mma_commit(&ms->acc_full[as]);
            ++kcount;
            ++acount;
          }
        }
        if (ok && st.n2 > 0) {
          mma_commit(&ms->qs_empty);  // the pass-2 queries are free
          ++qcount;
        } else if (ok && st.n1 > 0) {
          mma_commit(&ms->q_empty);  // no pass-2 tiles: item k's pass-1 queries are free
        }
      }
      mma_commit(&ms->mma_done);
      mbar_wait(&ms->mma_done, 0, nullptr);
    }
  } else if (warp == 10) {
    // ------------------------------------------------ publisher of pass-1 results
    for (int k = 0; k < n; ++k) {
      const int slot = k % kPubSlots;
      if (!warp_wait(&ms->pub_full[slot], (k / kPubSlots) & 1, ms, p.status)) break;
      const ItemRef it = item_of(p, k);
      float2 *mine = p.partial + guard((long long)it.unit * p.n_ch + it.chunk, 1,
                                       (long long)p.units * p.n_ch, p.status) *
                                     128;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int r = lane + 32 * j;
        float2 a = ms->pstat[slot][0][r];
        const float2 b = ms->pstat[slot][1][r];
        combine(a.x, a.y, b.x, b.y);
        mine[r] = a;
      }
      __syncwarp();
      int last = 0;
      if (lane == 0) {
        mbar_arrive(&ms->pub_empty[slot]);
        __threadfence();
        last = atomicAdd(&p.ctrl[guard(it.unit, 1, p.units, p.status)], 1) == p.n_ch - 1;
      }
      last = __shfl_sync(0xffffffffu, last, 0);
      if (last) {
        __threadfence();
        const float2 *part =
            p.partial + guard((long long)it.unit * p.n_ch, p.n_ch, (long long)p.units * p.n_ch,
                              p.status) *
                            128;
        float mm[4], ll[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          mm[j] = -INFINITY;
          ll[j] = 0.f;
        }
        for (int c0 = 0; c0 < p.n_ch; c0 += 8) {
          float2 q[8][4];
#pragma unroll
          for (int c = 0; c < 8; ++c)
#pragma unroll
            for (int j = 0; j < 4; ++j)
              q[c][j] = c0 + c < p.n_ch ? __ldcg(&part[(size_t)(c0 + c) * 128 + lane + 32 * j])
                                        : make_float2(-INFINITY, 0.f);
#pragma unroll
          for (int c = 0; c < 8; ++c)
#pragma unroll
            for (int j = 0; j < 4; ++j) combine(mm[j], ll[j], q[c][j].x, q[c][j].y);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j)
          p.lognorm[guard(it.unit, 1, p.units, p.status) * 128 + lane + 32 * j] =
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
    const int r = quarter * 32 + lane;         // window row of this thread
    const int wtid = threadIdx.x - 64 - wg * 128;
    const uint32_t lane_addr = (uint32_t)(quarter * 32) << 16;
    int tcount = 0;  // tiles seen

    // Inside an item every warp follows the same control flow even if a wait
    // gives up (the tile is then skipped), so that the named barriers below
    // are always reached by all of their threads.
    for (int k = 0; k < n + kLag; ++k) {
      const Step st = step_of(p, k, n);
      float m = -INFINITY, l = 0.f;    // pass 1 of item k: this row's max and sum
      const int last_vis = p.P + r % p.W;
      for (int j = 0; j < st.len; ++j) {
        int pass, s;
        seq_at(st, j, pass, s);
        if (pass == 1) {
          // ---------------- a pass-1 tile of item k
          const int t = st.a0 + s;
          const int mine = wg_of(tcount) == wg;
          const int as = tcount % kNA, ph = (tcount / kNA) & 1;
          ++tcount;
          if (mine && warp_wait(&ms->acc_full[as], ph, ms, p.status)) {
            tc_fence_after();
            uint32_t x[4][32];
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_ld32(tmem + lane_addr + as * 128 + c * 32, x[c]);
            tmem_wait_ld();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&ms->acc_empty[as]);
            if ((t + 1) * kTile - 1 >= p.P) {  // keys this row cannot see -> -inf
#pragma unroll
              for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int j = 0; j < 32; ++j)
                  if (t * kTile + c * 32 + j > last_vis) x[c][j] = 0xff800000u;
            }
            float mx[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) mx[i] = -INFINITY;
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
              for (int j = 0; j < 32; ++j) mx[j & 7] = fmaxf(mx[j & 7], __uint_as_float(x[c][j]));
            const float tmax = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                                     fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
            if (tmax != -INFINITY) {
              const float mnew = fmaxf(m, tmax * p.scale2);
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
              const float sum = ((sv[0].x + sv[0].y) + (sv[1].x + sv[1].y)) +
                                ((sv[2].x + sv[2].y) + (sv[3].x + sv[3].y));
              l = l * fast_exp2(m - mnew) + sum;
              m = mnew;
            }
          }
          if (s == st.n1 - 1) {
            // Item k's last pass-1 tile: this warpgroup's row statistics go to
            // the publisher now, ahead of the step's pass-2 tiles.
            const int slot = k % kPubSlots;
            warp_wait(&ms->pub_empty[slot], ((k / kPubSlots) & 1) ^ 1, ms, p.status);
            ms->pstat[slot][wg][r] = make_float2(m, l);
            __syncwarp();
            if (lane == 0) mbar_arrive(&ms->pub_full[slot]);
          }
        }
        if (pass == 2) {
          // ---------------- a pass-2 tile of item k - kLag: votes of its keys
          // (D[key][row]: this thread's TMEM lane is key t * 128 + r)
          if (s == 0) {
            if (wtid == 0)
              wait_ready(&p.ctrl[guard(p.units + st.u2, 1, 2LL * p.units, p.status)], ms,
                         p.status);
            named_bar_sync(3 + wg, 128);
            ms->offs[wg][wtid] =
                __ldcg(&p.lognorm[guard(st.u2, 1, p.units, p.status) * 128 + wtid]);
            named_bar_sync(3 + wg, 128);
          }
          const int t = st.b0 + s;
          const int mine = wg_of(tcount) == wg;
          const int as = tcount % kNA, ph = (tcount / kNA) & 1;
          ++tcount;
          if (mine && warp_wait(&ms->acc_full[as], ph, ms, p.status)) {
            tc_fence_after();
            uint32_t x[4][32];
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_ld32(tmem + lane_addr + as * 128 + c * 32, x[c]);
            tmem_wait_ld();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&ms->acc_empty[as]);
            // fp32x2: logits scaled and shifted two at a time, sums in pairs
            float2 sv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) sv[i] = make_float2(0.f, 0.f);
            const float2 s2 = make_float2(p.scale2, p.scale2);
            const float4 *o4 = reinterpret_cast<const float4 *>(ms->offs[wg]);
#pragma unroll
            for (int c = 0; c < 4; ++c)
#pragma unroll
              for (int j4 = 0; j4 < 8; ++j4) {
                const float4 o = o4[c * 8 + j4];
                const float2 y0 = __ffma2_rn(make_float2(__uint_as_float(x[c][4 * j4]),
                                                         __uint_as_float(x[c][4 * j4 + 1])),
                                             s2, make_float2(-o.x, -o.y));
                const float2 y1 = __ffma2_rn(make_float2(__uint_as_float(x[c][4 * j4 + 2]),
                                                         __uint_as_float(x[c][4 * j4 + 3])),
                                             s2, make_float2(-o.z, -o.w));
                sv[(2 * j4) & 3] =
                    __fadd2_rn(sv[(2 * j4) & 3], make_float2(fast_exp2(y0.x), fast_exp2(y0.y)));
                sv[(2 * j4 + 1) & 3] =
                    __fadd2_rn(sv[(2 * j4 + 1) & 3], make_float2(fast_exp2(y1.x), fast_exp2(y1.y)));
              }
            const float vote = ((sv[0].x + sv[0].y) + (sv[1].x + sv[1].y)) +
                               ((sv[2].x + sv[2].y) + (sv[3].x + sv[3].y));
            const int key = t * kTile + r;
            if (key < p.P)
              p.votes[guard((long long)st.u2 * p.P + key, 1, (long long)p.units * p.P, p.status)] =
                  vote;
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncwarp();
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

}  // namespace

bool score_tc1_supported(const LayerGeom &g) {
  return g.dtype == RIPPLE_BF16 && g.D == 128 && g.R == 128 && g.P > 0 && encode_fn() != nullptr;
}

cudaError_t launch_score_tc1(const LayerGeom &g, int n_layers, const void *const *q_win,
                             const void *const *k, const CompressWs &ws, float *votes,
                             int32_t *status, cudaStream_t st) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr || n_layers < 1 || n_layers > kCompressMaxLayers) return cudaErrorNotSupported;
  static Tc1Launch lp;  // large: kept off the stack, filled under the lock
  static std::mutex mu;
  std::lock_guard<std::mutex> lock(mu);
  for (int l = 0; l < n_layers; ++l) {
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
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (sms <= 0) sms = 1;
  Tc1Params &p = lp.p;
  p.upl = g.units;
  p.units = g.units * n_layers;
  p.T = g.T;
  p.P = g.P;
  p.W = g.W;
  p.Hq = g.Hq;
  p.Hkv = g.Hkv;
  p.G = g.G;
  p.n_tiles1 = (g.T + kTile - 1) / kTile;
  p.n_tiles2 = (g.P + kTile - 1) / kTile;
  // At least kMinTilesPerItem tiles per item, and no more items per unit than
  // SMs (the deadlock-free schedule needs <= 2x as many as CTAs).
  const int tpi_min = (p.n_tiles1 + sms - 1) / sms;
  p.tpi = tpi_min > kMinTilesPerItem ? tpi_min : kMinTilesPerItem;
  p.n_ch = (p.n_tiles1 + p.tpi - 1) / p.tpi;
  p.total_items = p.units * p.n_ch;
  p.scale2 = g.scale2;
  for (int l = 0; l < n_layers; ++l) p.q[l] = (const uint8_t *)q_win[l];
  p.partial = ws.row_partial;
  p.lognorm = ws.row_lognorm;
  p.votes = votes;
  p.ctrl = ws.counters;
  p.status = status;
  p.wait_cycles = wait_limit_cycles();
  cudaError_t e = cudaMemsetAsync(ws.counters, 0, sizeof(int) * 2 * p.units, st);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(score_tc1_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           kSmemBytes);
  if (e != cudaSuccess) return e;
  const int grid = p.total_items < sms ? p.total_items : sms;
  void *args[] = {(void *)&lp};
  e = cudaLaunchCooperativeKernel((const void *)score_tc1_kernel, dim3(grid), dim3(kThreads), args,
                                  (size_t)kSmemBytes, st);
  count_launches(1);
  return e;
}

}  // namespace ripple
