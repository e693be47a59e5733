// Observation-window token scoring on the 5th-generation tensor cores
// (tcgen05, accumulators in TMEM), bf16 keys and queries, d = 128, G*w = 128
// or 256 window rows. SnapKV's rule as RippleKV keeps it (Sec. 4.4, last
// paragraph): logits x = scale * q.k of the window rows against every key,
// causal inside the window, softmax per row over all visible keys, vote of a
// prefix key = sum over rows of its probability.
//
// One persistent launch per layer (grid = SM count, one CTA per SM) does both
// passes over every unit (b, h) of the layer:
//   pass 1 item (unit, chunk): per window row, (max, sum of exp) over the
//     chunk's key tiles -> partial[unit][chunk][row]; the CTA finishing the
//     unit's last chunk merges them into lognorm[unit][row] = max + log2(sum)
//     and raises ready[unit];
//   pass 2 item (unit, chunk): per prefix key of the chunk, vote = sum over
//     rows of exp2(x * scale * log2e - lognorm[row]), after ready[unit].
// Items are fetched dynamically in a list ordered group by group,
// P1(0) P1(1) P2(0) P1(2) P2(1) ..., with groups of units sized so that a
// unit's keys are still in L2 when pass 2 re-reads them.
//
// Warp roles (320 threads): warp 0 = TMA producer, warp 1 = MMA issuer and
// TMEM owner, warps 2-9 = two epilogue warpgroups taking alternate key tiles.
// Pass 1 computes D[row][key] (A = window queries, B = key tile, M = 128 per
// row block); pass 2 computes D[key][row] (A = key tile, B = window queries,
// N = G*w), so that each epilogue thread owns one row (pass 1) or one key
// (pass 2) and every reduction is thread-local.
// Every wait is bounded: on timeout the CTA raises RIPPLE_ETIMEOUT, all roles
// leave their loops, and TMEM is released.
#include <cuda.h>
#include <math.h>

#include "common.cuh"
#include "kernels.cuh"

namespace ripple {
namespace {

constexpr int kTile = 128;                      // keys per tile
constexpr int kHalfBytes = kTile * 64 * 2;      // 64 bf16 columns of 128 rows: 16 KB
constexpr int kTileBytes = 2 * kHalfBytes;      // one 128 x 128 bf16 tile
constexpr int kThreads = 320;
constexpr int kItemSlots = 4;
constexpr long long kWaitCycles = 4000000000LL;  // ~2 s at 2 GHz

// ------------------------------------------------------------ PTX wrappers

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, int x, int y,
                                            uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(smem_u32(dst)),
      "l"((uint64_t)map), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tma_load_3d(void *dst, const CUtensorMap *map, int x, int y, int z,
                                            uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(smem_u32(dst)),
      "l"((uint64_t)map), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t *dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(dst)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulation.
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on `bar` when every tcgen05.mma issued so far by this thread is done.
__device__ __forceinline__ void mma_commit(uint64_t *bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
          smem_u32(bar))
      : "memory");
}

// 32 TMEM columns of this warp's 32 lanes: thread i gets lane (base + i).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, "
      "%28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Named barrier; the warp is converged first (bar.sync is warp-aligned).
__device__ __forceinline__ void named_bar(int id, int threads) {
  __syncwarp();
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

__device__ __forceinline__ int ld_acquire(const int *p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(int *p, int v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, rows of
// 128 bytes, 8-row core groups 1024 bytes apart (tcgen05 descriptor format).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;             // leading-dimension offset (unused with this swizzle)
  d |= (uint64_t)(1024 >> 4) << 32;   // stride between 8-row groups
  d |= (uint64_t)1 << 46;             // descriptor version
  d |= (uint64_t)2 << 61;             // 128-byte swizzle
  return d;
}

// Instruction descriptor of kind::f16: bf16 A and B (K-major), fp32 D.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

// ------------------------------------------------------------ work list

struct TcParams {
  int units, T, P, W, Hq, Hkv, G;
  int n_tiles1, n_tiles2, chunk, n_ch1, n_ch2, group_units, n_groups, n_items;
  float scale2;
  float2 *partial;  // [units][n_ch1][R]
  float *lognorm;   // [units][R]
  float *votes;     // [units][P]
  int *ctrl;        // [0] item counter; [32 + u] pass-1 chunks done; [32 + units + u] ready
  int32_t *status;
};

struct Item {
  int pass, unit, chunk;  // pass 0 marks the end of the work
};

__device__ Item decode_item(const TcParams &p, int idx) {
  if (idx >= p.n_items) return {0, 0, 0};
  for (int k = 0; k < 2 * p.n_groups; ++k) {
    int pass, g;
    if (k == 0) {
      pass = 1; g = 0;
    } else if (k == 2 * p.n_groups - 1) {
      pass = 2; g = p.n_groups - 1;
    } else if (k & 1) {
      pass = 1; g = (k + 1) / 2;
    } else {
      pass = 2; g = k / 2 - 1;
    }
    const int u0 = g * p.group_units;
    const int ug = min(p.group_units, p.units - u0);
    const int nch = pass == 1 ? p.n_ch1 : p.n_ch2;
    const int sz = ug * nch;
    if (idx < sz) return {pass, u0 + idx / nch, idx % nch};
    idx -= sz;
  }
  return {0, 0, 0};
}

__device__ __forceinline__ void item_tiles(const TcParams &p, const Item &it, int &t0, int &t1) {
  const int n = it.pass == 1 ? p.n_tiles1 : p.n_tiles2;
  t0 = it.chunk * p.chunk;
  t1 = min(n, t0 + p.chunk);
}

// ------------------------------------------------------------ shared memory

template <int NR>
struct Cfg {
  static constexpr int R = 128 * NR;             // window rows
  static constexpr int NK = NR == 1 ? 4 : 2;     // key-tile stages
  static constexpr int NQ = 2;                   // query buffers
  static constexpr int NA = NR == 1 ? 4 : 2;     // TMEM accumulator stages
  static constexpr int ACC_COLS = 128 * NR;      // TMEM columns per stage
  static constexpr int QBYTES = R * 256;         // R rows x 128 bf16
  static constexpr int OFF_K = 0;
  static constexpr int OFF_Q = OFF_K + NK * kTileBytes;
  static constexpr int OFF_MISC = OFF_Q + NQ * QBYTES;
};

struct Misc {
  uint64_t k_full[4], k_empty[4], q_full[2], q_empty[2], acc_full[4], acc_empty[4], mma_done;
  uint64_t item_full[kItemSlots], item_empty[kItemSlots];
  Item items[kItemSlots];
  uint32_t tmem_base;
  int abort_flag;
  int last_flag;
  alignas(16) float off[2][256];  // per-warpgroup row offsets of a pass-2 item (read as float4)
  alignas(16) float2 xch[256];    // warpgroup 1 -> 0 exchange of pass-1 row stats
};

static_assert(offsetof(Misc, off) % 16 == 0 && offsetof(Misc, xch) % 16 == 0,
              "vector-accessed shared arrays must be 16-byte aligned");

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
    if (clock64() - t0 > kWaitCycles) {
      *(volatile int *)&ms->abort_flag = 1;
      report(status, RIPPLE_ETIMEOUT);
      return false;
    }
  }
}

// Warp-uniform variant for the epilogue warps: all lanes wait, the warp then
// agrees on the outcome (and is converged for the .sync.aligned TMEM loads).
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
    if (clock64() - t0 > kWaitCycles) {
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

template <int NR>
__global__ void __launch_bounds__(kThreads, 1)
    score_tc_kernel(const __grid_constant__ CUtensorMap kmap,
                    const __grid_constant__ CUtensorMap qmap, const __grid_constant__ TcParams p) {
  using C = Cfg<NR>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t *ktiles = smem + C::OFF_K;
  uint8_t *qbufs = smem + C::OFF_Q;
  Misc *ms = (Misc *)(smem + C::OFF_MISC);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

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
    for (int i = 0; i < kItemSlots; ++i) {
      mbar_init(&ms->item_full[i], 1);
      mbar_init(&ms->item_empty[i], 1 + 8);
    }
    mbar_init(&ms->mma_done, 1);
    ms->abort_flag = 0;
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

  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    if (lane == 0) {
      int kcount = 0, qcount = 0, icount = 0;
      int next = atomicAdd(&p.ctrl[0], 1);
      for (;;) {
        const Item it = decode_item(p, next);
        if (it.pass) next = atomicAdd(&p.ctrl[0], 1);
        const int slot = icount % kItemSlots;
        if (!wait_bar(&ms->item_empty[slot], ((icount / kItemSlots) & 1) ^ 1, ms, p.status)) break;
        ms->items[slot] = it;
        mbar_arrive(&ms->item_full[slot]);
        ++icount;
        if (!it.pass) break;
        const int b = it.unit / p.Hkv, h = it.unit % p.Hkv;
        const int qrow0 = (b * p.Hq + h * p.G) * p.W;
        const int qs = qcount % C::NQ;
        if (!wait_bar(&ms->q_empty[qs], ((qcount / C::NQ) & 1) ^ 1, ms, p.status)) break;
        mbar_arrive_expect_tx(&ms->q_full[qs], C::QBYTES);
        uint8_t *qb = qbufs + qs * C::QBYTES;
        for (int half = 0; half < 2; ++half)
          for (int nr = 0; nr < NR; ++nr)
            tma_load_2d(qb + half * (NR * kHalfBytes) + nr * kHalfBytes, &qmap, half * 64,
                        qrow0 + nr * 128, &ms->q_full[qs]);
        ++qcount;
        int t0, t1;
        item_tiles(p, it, t0, t1);
        bool ok = true;
        for (int t = t0; t < t1; ++t) {
          const int ks = kcount % C::NK;
          if (!wait_bar(&ms->k_empty[ks], ((kcount / C::NK) & 1) ^ 1, ms, p.status)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&ms->k_full[ks], kTileBytes);
          uint8_t *kb = ktiles + ks * kTileBytes;
          tma_load_3d(kb, &kmap, 0, t * kTile, it.unit, &ms->k_full[ks]);
          tma_load_3d(kb + kHalfBytes, &kmap, 64, t * kTile, it.unit, &ms->k_full[ks]);
          ++kcount;
        }
        if (!ok) break;
      }
      // Let every issued copy land before the CTA can exit (matters only after
      // an abort; in normal operation every stage was already consumed).
      for (int j = max(0, kcount - C::NK); j < kcount; ++j)
        mbar_wait(&ms->k_full[j % C::NK], (j / C::NK) & 1, nullptr, kWaitCycles / 4);
      for (int j = max(0, qcount - C::NQ); j < qcount; ++j)
        mbar_wait(&ms->q_full[j % C::NQ], (j / C::NQ) & 1, nullptr, kWaitCycles / 4);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      int kcount = 0, qcount = 0, icount = 0, acount = 0;
      constexpr uint32_t id1 = idesc_bf16(128, 128);
      constexpr uint32_t id2 = idesc_bf16(128, 128 * NR);
      const uint32_t kbase = smem_u32(ktiles), qbase = smem_u32(qbufs);
      for (;;) {
        const int slot = icount % kItemSlots;
        if (!wait_bar(&ms->item_full[slot], (icount / kItemSlots) & 1, ms, p.status)) break;
        const Item it = ms->items[slot];
        mbar_arrive(&ms->item_empty[slot]);
        ++icount;
        if (!it.pass) break;
        const int qs = qcount % C::NQ;
        if (!wait_bar(&ms->q_full[qs], (qcount / C::NQ) & 1, ms, p.status)) break;
        const uint32_t qa = qbase + qs * C::QBYTES;
        int t0, t1;
        item_tiles(p, it, t0, t1);
        bool ok = true;
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
          for (int k = 0; k < 8; ++k) {
            const uint32_t koff = (k >> 2) * kHalfBytes + (k & 3) * 32;
            const uint32_t qoff = (k >> 2) * (NR * kHalfBytes) + (k & 3) * 32;
            if (it.pass == 1) {
#pragma unroll
              for (int nr = 0; nr < NR; ++nr)
                mma_bf16(d + nr * 128, sw128_desc(qa + qoff + nr * kHalfBytes),
                         sw128_desc(ka + koff), id1, k > 0);
            } else {
              mma_bf16(d, sw128_desc(ka + koff), sw128_desc(qa + qoff), id2, k > 0);
            }
          }
          mma_commit(&ms->k_empty[ks]);
          mma_commit(&ms->acc_full[as]);
          ++kcount;
          ++acount;
        }
        if (!ok) break;
        mma_commit(&ms->q_empty[qs]);
        ++qcount;
      }
      // All issued MMAs complete before TMEM is released.
      mma_commit(&ms->mma_done);
      mbar_wait(&ms->mma_done, 0, nullptr, kWaitCycles / 4);
    }
  } else {
    // ------------------------------------------------ epilogue warpgroups
    const int wg = (warp - 2) >> 2;
    const int quarter = warp & 3;              // TMEM lanes this warp may access
    const int lrow = quarter * 32 + lane;      // row (pass 1) or key (pass 2) in the tile
    const int wtid = threadIdx.x - 64 - wg * 128;  // 0..127 within the warpgroup
    const uint32_t lane_addr = (uint32_t)(quarter * 32) << 16;
    int icount = 0, tcount = 0;
    for (;;) {
      const int slot = icount % kItemSlots;
      if (!warp_wait(&ms->item_full[slot], (icount / kItemSlots) & 1, ms, p.status)) break;
      const Item it = ms->items[slot];
      __syncwarp();
      if (lane == 0) mbar_arrive(&ms->item_empty[slot]);
      ++icount;
      if (!it.pass) break;
      int t0, t1;
      item_tiles(p, it, t0, t1);
      // Inside an item every warp follows the same control flow even if a wait
      // gives up (the tile is then skipped), so that the named barriers below
      // are always reached by all of their threads.
      if (it.pass == 1) {
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
            float tmax = -INFINITY;
            if (!masked) {
#pragma unroll
              for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int j = 0; j < 32; ++j) tmax = fmaxf(tmax, __uint_as_float(x[c][j]));
            } else {
#pragma unroll
              for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int j = 0; j < 32; ++j)
                  if (t * kTile + c * 32 + j <= last_vis[nr])
                    tmax = fmaxf(tmax, __uint_as_float(x[c][j]));
            }
            if (tmax == -INFINITY) continue;
            const float mnew = fmaxf(m[nr], tmax * p.scale2);
            float s = 0.f;
            if (!masked) {
#pragma unroll
              for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int j = 0; j < 32; ++j)
                  s += fast_exp2(fmaf(__uint_as_float(x[c][j]), p.scale2, -mnew));
            } else {
#pragma unroll
              for (int c = 0; c < 4; ++c)
#pragma unroll
                for (int j = 0; j < 32; ++j)
                  if (t * kTile + c * 32 + j <= last_vis[nr])
                    s += fast_exp2(fmaf(__uint_as_float(x[c][j]), p.scale2, -mnew));
            }
            l[nr] = l[nr] * fast_exp2(m[nr] - mnew) + s;
            m[nr] = mnew;
          }
        }
        // Combine the two warpgroups' row stats; warpgroup 0 publishes them.
        if (wg == 1) {
#pragma unroll
          for (int nr = 0; nr < NR; ++nr) ms->xch[nr * 128 + lrow] = make_float2(m[nr], l[nr]);
        }
        named_bar(1, 256);
        if (wg == 0) {
          const size_t prow = ((size_t)it.unit * p.n_ch1 + it.chunk) * C::R;
#pragma unroll
          for (int nr = 0; nr < NR; ++nr) {
            const float2 o = ms->xch[nr * 128 + lrow];
            combine(m[nr], l[nr], o.x, o.y);
            p.partial[prow + nr * 128 + lrow] = make_float2(m[nr], l[nr]);
          }
          __threadfence();
          named_bar(2, 128);
          if (wtid == 0) {
            const int done = atomicAdd(&p.ctrl[32 + it.unit], 1);
            ms->last_flag = (done == p.n_ch1 - 1);
          }
          named_bar(2, 128);
          if (ms->last_flag) {
            __threadfence();
#pragma unroll
            for (int nr = 0; nr < NR; ++nr) {
              const int r = nr * 128 + lrow;
              float mm = -INFINITY, ll = 0.f;
              for (int c = 0; c < p.n_ch1; ++c) {
                const float2 q = __ldcg(&p.partial[((size_t)it.unit * p.n_ch1 + c) * C::R + r]);
                combine(mm, ll, q.x, q.y);
              }
              p.lognorm[(size_t)it.unit * C::R + r] = mm + __log2f(ll);
            }
            __threadfence();
            named_bar(2, 128);
            if (wtid == 0) st_release(&p.ctrl[32 + p.units + it.unit], 1);
          }
        }
        named_bar(1, 256);
      } else {
        // pass 2: wait for the unit's row statistics, then vote per key
        if (wtid == 0) wait_ready(&p.ctrl[32 + p.units + it.unit], ms, p.status);
        named_bar(3 + wg, 128);
        for (int r = wtid; r < C::R; r += 128)
          ms->off[wg][r] = __ldcg(&p.lognorm[(size_t)it.unit * C::R + r]);
        named_bar(3 + wg, 128);
        const float4 *off4 = (const float4 *)ms->off[wg];
        for (int t = t0; t < t1; ++t, ++tcount) {
          if ((tcount & 1) != wg) continue;
          const int as = tcount % C::NA;
          if (!warp_wait(&ms->acc_full[as], (tcount / C::NA) & 1, ms, p.status)) continue;
          tc_fence_after();
          float vote = 0.f;
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
                vote += fast_exp2(fmaf(__uint_as_float(x[c][j + 0]), p.scale2, -o.x));
                vote += fast_exp2(fmaf(__uint_as_float(x[c][j + 1]), p.scale2, -o.y));
                vote += fast_exp2(fmaf(__uint_as_float(x[c][j + 2]), p.scale2, -o.z));
                vote += fast_exp2(fmaf(__uint_as_float(x[c][j + 3]), p.scale2, -o.w));
              }
          }
          const int key = t * kTile + lrow;
          if (key < p.P) p.votes[(size_t)it.unit * p.P + key] = vote;
        }
      }
    }
  }

  tc_fence_before();
  __syncwarp();  // lanes 1..31 of the producer and MMA warps wait for lane 0 here
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
cudaError_t launch_nr(const LayerGeom &g, const void *q_win, const void *k, const CompressWs &ws,
                      float *votes, int32_t *status, cudaStream_t st) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return cudaErrorNotSupported;
  CUtensorMap kmap, qmap;
  {
    cuuint64_t dims[3] = {128, (cuuint64_t)g.T, (cuuint64_t)g.units};
    cuuint64_t strides[2] = {256, (cuuint64_t)g.T * 256};
    cuuint32_t box[3] = {64, 128, 1};
    cuuint32_t es[3] = {1, 1, 1};
    if (enc(&kmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(k), dims, strides, box,
            es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  {
    cuuint64_t dims[2] = {128, (cuuint64_t)g.B * g.Hq * g.W};
    cuuint64_t strides[1] = {256};
    cuuint32_t box[2] = {64, 128};
    cuuint32_t es[2] = {1, 1};
    if (enc(&qmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(q_win), dims, strides,
            box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  const int sms = sm_count();
  TcParams p;
  p.units = g.units;
  p.T = g.T;
  p.P = g.P;
  p.W = g.W;
  p.Hq = g.Hq;
  p.Hkv = g.Hkv;
  p.G = g.G;
  p.n_tiles1 = (g.T + kTile - 1) / kTile;
  p.n_tiles2 = (g.P + kTile - 1) / kTile;
  // tiles per item: enough items to keep every SM busy, at most 8
  int chunk = (p.n_tiles1 * g.units) / (3 * sms);
  p.chunk = chunk < 1 ? 1 : (chunk > 8 ? 8 : chunk);
  p.n_ch1 = (p.n_tiles1 + p.chunk - 1) / p.chunk;
  p.n_ch2 = (p.n_tiles2 + p.chunk - 1) / p.chunk;
  // units per group: about 48 MB of keys, so that two groups stay in L2
  const long long unit_bytes = (long long)g.T * 256;
  int gu = (int)((48ll << 20) / unit_bytes);
  p.group_units = gu < 1 ? 1 : (gu > g.units ? g.units : gu);
  p.n_groups = (g.units + p.group_units - 1) / p.group_units;
  p.n_items = g.units * (p.n_ch1 + p.n_ch2);
  p.scale2 = g.scale2;
  p.partial = ws.row_partial;
  p.lognorm = ws.row_lognorm;
  p.votes = votes;
  p.ctrl = ws.counters;
  p.status = status;
  cudaError_t e = cudaMemsetAsync(ws.counters, 0, sizeof(int) * (32 + 2 * g.units), st);
  if (e != cudaSuccess) return e;
  constexpr int smem = smem_bytes<NR>();
  static_assert(smem <= 227 * 1024, "shared memory budget");
  e = cudaFuncSetAttribute(score_tc_kernel<NR>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int grid = p.n_items < sms ? p.n_items : sms;
  score_tc_kernel<NR><<<grid, kThreads, smem, st>>>(kmap, qmap, p);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace

bool score_tc_supported(const LayerGeom &g) {
  return g.dtype == RIPPLE_BF16 && g.D == 128 && (g.R == 128 || g.R == 256) && g.P > 0 &&
         encode_fn() != nullptr;
}

cudaError_t launch_score_tc(const LayerGeom &g, const void *q_win, const void *k,
                            const CompressWs &ws, float *votes, int32_t *status,
                            cudaStream_t st) {
  if (g.R == 128) return launch_nr<1>(g, q_win, k, ws, votes, status, st);
  return launch_nr<2>(g, q_win, k, ws, votes, status, st);
}

}  // namespace ripple
