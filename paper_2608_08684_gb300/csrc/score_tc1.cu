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
//
// With the window rows' attention output (kO; the scoring fused into the
// prefill attention of the window rows, so that a real prefill reads the keys
// for both in one pass): pass 2 covers every key, causal inside the window;
// the producer streams each value tile behind the next key tile through the
// same ring (three stages); both epilogue warpgroups take every pass-2 tile,
// each for 64 of its 128 window rows, and write those rows' probabilities as
// bf16 into a shared-memory tile (MN-major, the A operand; a key's vote is
// its two halves summed through shared memory), and the MMA warp
// accumulates O[row][dim] += P . V in the last 128 TMEM columns (V, MN-major,
// the B operand). The probabilities are final (pass 1 has fixed every row's
// normaliser), so O needs no rescaling. At an item's end both warpgroups
// write its partial O to the workspace and count it on its unit. kOReduceLag
// steps later the CTA that computed the item sums its slice of the unit's
// output rows (a 1/n_ch share) over the unit's partials in item order (the
// unit's other items are done by then; a bounded wait covers the rest), so
// the sum is deterministic and no CTA holds up the others with a whole
// unit's sum.
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
constexpr int kLag = 1;                         // pass 2 of item k runs in step k + kLag
constexpr int kPubSlots = 2;
constexpr int kMinTilesPerItem = 9;
// kO: a whole unit per item up to 32768 keys. An item's partial output, its
// row-slice sum and pass 2's wait on the unit's other items cost more than
// re-reading the keys from DRAM in pass 2 (an item's keys no longer stay in
// L2 until then): 32 layers of the 32k workload took 5.39 / 5.25 / 5.08 /
// 5.11 / 5.00 ms with items of 32 / 64 / 86 / 128 / 256 tiles.
constexpr int kMinTilesPerItemO = 256;
constexpr int kMaxStages = 4;
constexpr int kOReduceLag = 2;  // kO: a step's item rows are summed this many steps later

// With kO (the window rows' attention output as well as the votes) pass 2
// covers every key and also streams the value tiles, multiplies the
// probabilities by them on the tensor cores and accumulates O in TMEM; the
// probabilities go through a 32 KB shared-memory tile, so the ring has one
// stage less, and O takes the last 128 TMEM columns.
template <bool kO>
struct Tc1Cfg {
  static constexpr int NK = kO ? 3 : 4;   // ring stages (key tiles; value tiles with kO)
  static constexpr int NA = kO ? 3 : 4;   // S accumulators in TMEM (128 columns each)
  static constexpr uint32_t OCol = NA * 128;  // O accumulator (kO)
  static_assert(NA * 128 + (kO ? 128 : 0) <= 512, "TMEM columns");
  static_assert(NK <= kMaxStages && NA <= kMaxStages, "barrier arrays");
};

struct Tc1Params {
  int units, upl, T, P, W, Hq, Hkv, G;  // units of all layers, units per layer
  int n_tiles1, n_tiles2;  // key tiles of pass 1 (all keys) and pass 2 (prefix keys; all with kO)
  int tpi, n_ch;           // key tiles per item, items per unit
  int total_items;
  float scale2;
  float *o_win[kCompressMaxLayers];  // kO, per layer: window-row outputs [B][Hq][W][128] fp32
  float *o_part;     // kO: [units][n_ch][128][128] fp32 per-item partial outputs
  int *o_count;      // kO: [units] items of unit u whose partial is written
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
// its three items per CTA no longer fit in L2. Measured on 32 layers of the
// 32k-token workload: 2.80 ms with a lag of two against 2.57 ms with one;
// with a lag of two and each step's pass-1 and pass-2 tiles alternating,
// 2.90 / 2.95 / 3.13 / 3.84 ms with items of 9 / 7 / 6 / 5 tiles.

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
  uint64_t k_full[kMaxStages], k_empty[kMaxStages], q_full, q_empty;
  uint64_t acc_full[kMaxStages], acc_empty[kMaxStages];
  uint64_t qs_full, qs_empty;           // pass-2 queries in shared memory
  uint64_t pub_full[kPubSlots], pub_empty[kPubSlots], mma_done;
  // kO: the probability tile (all eight epilogue warps write each tile, the
  // P . V MMA releases it) and the O accumulator
  uint64_t p_full, p_empty, o_full, o_empty;
  float vhalf[2][128];  // kO: warpgroup 1's half of each key's vote, per tile parity
  uint32_t tmem_base;
  int abort_flag;
  long long wait_cycles;  // bound of the waits of this launch
  float2 pstat[kPubSlots][2][128];      // pass-1 row statistics per slot and warpgroup
  alignas(16) float offs[2][128];       // per warpgroup: the pass-2 item's row log-normalisers
};

// Shared memory: the ring, the pass-2 and pass-1 queries (two 64-dim halves
// each), with kO the probability tile, then the barriers and statistics.
template <bool kO>
struct Tc1Smem {
  static constexpr int OffQs = Tc1Cfg<kO>::NK * kTileBytes;
  static constexpr int OffQ1 = OffQs + kTileBytes;
  static constexpr int OffP = OffQ1 + kTileBytes;
  static constexpr int OffMisc = OffP + (kO ? kTileBytes : 0);
  static constexpr int Bytes = OffMisc + (int)sizeof(Misc) + 1024;  // + alignment slack
  static_assert(Bytes <= 227 * 1024, "shared memory budget");
};

// count arrivals on a barrier at once
__device__ __forceinline__ void mbar_arrive_cnt(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(count)
               : "memory");
}

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

// Kernel argument: the keys (and with kO the values) of every layer as 3-D
// tensor maps [unit][T][128], the window queries of every layer as 2-D maps
// [B * Hq * W][128], and the parameters.
struct Tc1Launch {
  CUtensorMap kmap[kCompressMaxLayers];
  CUtensorMap qmap[kCompressMaxLayers];
  CUtensorMap vmap[kCompressMaxLayers];
  Tc1Params p;
};

// With kO the producer and the MMA warp walk a step as: the pass-1 key tiles,
// then the pass-2 item's key tiles with value tile s - kPvLag after key tile
// s (the order the MMA warp consumes them in: it multiplies a tile's
// probabilities by its values after issuing the logits kPvLag tiles on, so
// that the warpgroup that has just written a tile's probabilities finds its
// next tile's logits done), then the last value tiles.
// kind 1: pass-1 key tile, 2: pass-2 key tile, 3: pass-2 value tile.
constexpr int kPvLag = 2;
__device__ __forceinline__ void oseq_at(const Step &s, int j, int &kind, int &idx) {
  if (j < s.n1) {
    kind = 1;
    idx = j;
    return;
  }
  const int q = j - s.n1;
  const int a = min(s.n2, kPvLag);           // leading key tiles
  const int pairs = max(0, s.n2 - kPvLag);   // (key s, value s - kPvLag)
  if (q < a) {
    kind = 2;
    idx = q;
  } else if (q - a < 2 * pairs) {
    const int t = (q - a) >> 1;
    kind = (q - a) & 1 ? 3 : 2;
    idx = (q - a) & 1 ? t : kPvLag + t;
  } else {
    kind = 3;
    idx = pairs + (q - a - 2 * pairs);
  }
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t *>(&b);
}

// Probabilities of this thread's key for 64 window rows (logit columns
// c0 * 32 .. c0 * 32 + 63 of a pass-2 tile, x = those columns) and their sum
// in a fixed order; with kP also as bf16 pairs (rows 2i, 2i + 1 of the 64 in
// pk[i]), zero for the rows a window key is hidden from (hidden_below: the
// rows of window position below it; -1 for a prefix key). A key's vote is
// the sum of its two halves, half 0 + half 1, in every mode.
template <bool kP>
__device__ __forceinline__ float half_probs(const uint32_t (&x)[2][32], const float4 *o4, int c0,
                                            float scale2, int hidden_below, int W,
                                            uint32_t (&pk)[32]) {
  // fp32x2: logits scaled and shifted two at a time, sums in pairs
  float2 sv[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) sv[i] = make_float2(0.f, 0.f);
  const float2 s2 = make_float2(scale2, scale2);
#pragma unroll
  for (int cc = 0; cc < 2; ++cc)
#pragma unroll
    for (int j4 = 0; j4 < 8; ++j4) {
      const int c = c0 + cc;
      const float4 o = o4[c * 8 + j4];
      const float2 y0 = __ffma2_rn(make_float2(__uint_as_float(x[cc][4 * j4]),
                                               __uint_as_float(x[cc][4 * j4 + 1])),
                                   s2, make_float2(-o.x, -o.y));
      const float2 y1 = __ffma2_rn(make_float2(__uint_as_float(x[cc][4 * j4 + 2]),
                                               __uint_as_float(x[cc][4 * j4 + 3])),
                                   s2, make_float2(-o.z, -o.w));
      float2 e0 = make_float2(fast_exp2(y0.x), fast_exp2(y0.y));
      float2 e1 = make_float2(fast_exp2(y1.x), fast_exp2(y1.y));
      if constexpr (kP) {
        if (hidden_below >= 0) {
          const int col = c * 32 + 4 * j4;  // window row of e0.x
          if ((col + 0) % W < hidden_below) e0.x = 0.f;
          if ((col + 1) % W < hidden_below) e0.y = 0.f;
          if ((col + 2) % W < hidden_below) e1.x = 0.f;
          if ((col + 3) % W < hidden_below) e1.y = 0.f;
        }
        pk[(cc * 32 + 4 * j4) >> 1] = pack_bf16x2(e0.x, e0.y);
        pk[((cc * 32 + 4 * j4) >> 1) + 1] = pack_bf16x2(e1.x, e1.y);
      }
      sv[(2 * j4) & 3] = __fadd2_rn(sv[(2 * j4) & 3], e0);
      sv[(2 * j4 + 1) & 3] = __fadd2_rn(sv[(2 * j4 + 1) & 3], e1);
    }
  return ((sv[0].x + sv[0].y) + (sv[1].x + sv[1].y)) + ((sv[2].x + sv[2].y) + (sv[3].x + sv[3].y));
}

// Half h (window rows 64h .. 64h + 63) of one key's probabilities (this
// thread's TMEM lane), as bf16 pairs (rows 2i and 2i + 1 of the half in
// pk[i]), into the shared-memory tile in the MN-major, 128-byte-swizzled
// layout the tensor core reads as the A operand of O = P . V: rows 0-63 and
// 64-127 in two 16 KB halves, in each the key's 128-byte line holds its 64
// rows, 16-byte chunk c at position c ^ (key mod 8).
__device__ __forceinline__ void store_p_half(uint8_t *ptile, int key, int h,
                                             const uint32_t (&pk)[32]) {
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const int w = c * 4;  // rows 8c .. 8c + 7 of the half
    uint8_t *dst = ptile + h * kHalfBytes + (key >> 3) * 1024 + (key & 7) * 128 +
                   ((c ^ (key & 7)) << 4);
    *reinterpret_cast<uint4 *>(dst) = make_uint4(pk[w], pk[w + 1], pk[w + 2], pk[w + 3]);
  }
}

// kO: the output rows of item `it`'s slice of its unit (rows chunk * 128 /
// n_ch up to the next chunk's), summed over the unit's item partials in item
// order, once every item of the unit has written its partial (bounded wait).
// Run by both epilogue warpgroups (256 threads, named barrier 5).
__device__ __forceinline__ void reduce_rows(const Tc1Params &p, Misc *ms, const ItemRef &it,
                                            int tid) {
  if (tid == 0) {
    const int *cnt = &p.o_count[guard(it.unit, 1, p.units, p.status)];
    const long long t0 = clock64();
    while (ld_acquire(cnt) < p.n_ch) {
      if (*(volatile int *)&ms->abort_flag) break;
      if (clock64() - t0 > ms->wait_cycles) {
        *(volatile int *)&ms->abort_flag = 1;
        report(p.status, RIPPLE_ETIMEOUT);
        break;
      }
      __nanosleep(64);
    }
  }
  named_bar_sync(5, 256);
  const int r0 = it.chunk * 128 / p.n_ch, r1 = (it.chunk + 1) * 128 / p.n_ch;
  const int layer = it.unit / p.upl, local = it.unit % p.upl;
  const int b = local / p.Hkv, h = local % p.Hkv;
  const long long orow0 = (long long)(b * p.Hq + h * p.G) * p.W;
  const size_t ubase = (size_t)it.unit * p.n_ch * 128;
  // 32 float4 per row; consecutive threads take consecutive float4
  for (int e = tid; e < (r1 - r0) * 32; e += 256) {
    const int row = r0 + (e >> 5), q4 = e & 31;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int c = 0; c < p.n_ch; ++c) {
      const float4 v4 = __ldcg(reinterpret_cast<const float4 *>(
                                   p.o_part + (ubase + (size_t)c * 128 + row) * 128) +
                               q4);
      acc.x += v4.x;
      acc.y += v4.y;
      acc.z += v4.z;
      acc.w += v4.w;
    }
    reinterpret_cast<float4 *>(
        p.o_win[layer] + guard((orow0 + row) * 128, 128,
                               (long long)p.upl / p.Hkv * p.Hq * p.W * 128, p.status))[q4] = acc;
  }
}

template <bool kO>
__global__ void __launch_bounds__(kThreads, 1)
    score_tc1_kernel(const __grid_constant__ Tc1Launch lp) {
  using C = Tc1Cfg<kO>;
  using SM = Tc1Smem<kO>;
  const Tc1Params &p = lp.p;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t *ktiles = smem;
  uint8_t *qsm = smem + SM::OffQs;
  uint8_t *q1m = smem + SM::OffQ1;
  uint8_t *ptile = smem + SM::OffP;
  Misc *ms = (Misc *)(smem + SM::OffMisc);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n = items_of_cta(p);

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::NK; ++i) {
      mbar_init(&ms->k_full[i], 1);
      mbar_init(&ms->k_empty[i], 1);
    }
    mbar_init(&ms->q_full, 1);
    mbar_init(&ms->q_empty, 1);
    for (int i = 0; i < C::NA; ++i) {
      mbar_init(&ms->acc_full[i], 1);
      // kO: pass-2 tiles are released by all eight epilogue warps, pass-1
      // tiles by the four of their warpgroup with two arrivals each
      mbar_init(&ms->acc_empty[i], kO ? 8 : 4);
    }
    mbar_init(&ms->qs_full, 1);
    mbar_init(&ms->qs_empty, 1);
    for (int i = 0; i < kPubSlots; ++i) {
      mbar_init(&ms->pub_full[i], 8);
      mbar_init(&ms->pub_empty[i], 1);
    }
    mbar_init(&ms->mma_done, 1);
    mbar_init(&ms->p_full, 8);
    mbar_init(&ms->p_empty, 1);
    mbar_init(&ms->o_full, 1);
    mbar_init(&ms->o_empty, 8);
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
        const int l1 = st.u1 / p.upl, loc1 = st.u1 - l1 * p.upl;
        const int l2 = st.u2 / p.upl, loc2 = st.u2 - l2 * p.upl;
        const int len = kO ? st.n1 + 2 * st.n2 : st.len;
        for (int j = 0; j < len && ok; ++j) {
          int pass, s, kind;
          if (kO) {
            oseq_at(st, j, kind, s);
            pass = kind == 1 ? 1 : 2;
          } else {
            seq_at(st, j, pass, s);
            kind = pass;
          }
          if (kind == 1 && s == 0) {
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
          if (kind == 2 && s == 0) {
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
          const int tt = pass == 1 ? st.a0 + s : st.b0 + s;
          const int ks = kcount % C::NK;
          if (!wait_bar(&ms->k_empty[ks], ((kcount / C::NK) & 1) ^ 1, ms, p.status)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&ms->k_full[ks], kTileBytes);
          uint8_t *kb = ktiles + ks * kTileBytes;
          const uint64_t pol = pass == 1 ? keep : drop;
          // the step's two units' layers and local indices (divisions hoisted
          // out of the tile loop)
          const int layer = pass == 1 ? l1 : l2, local = pass == 1 ? loc1 : loc2;
          const CUtensorMap *km = kind == 3 ? &lp.vmap[layer] : &lp.kmap[layer];
          tma_load_3d(kb, km, 0, tt * kTile, local, &ms->k_full[ks], pol);
          tma_load_3d(kb + kHalfBytes, km, 64, tt * kTile, local, &ms->k_full[ks], pol);
          ++kcount;
        }
      }
      for (int j = max(0, kcount - C::NK); j < kcount; ++j)
        mbar_wait(&ms->k_full[j % C::NK], (j / C::NK) & 1, nullptr);
      if (qcount > 0) mbar_wait(&ms->qs_full, (qcount - 1) & 1, nullptr);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0) {
      int kcount = 0, acount = 0, qcount = 0, ocount = 0;
      int pv_count = 0;  // kO: probability tiles multiplied
      constexpr uint32_t id = idesc_bf16(128, 128);
      // O = P . V: P (rows x keys) and V (keys x dims) both MN-major
      constexpr uint32_t id_pv = idesc_bf16(128, 128) | (1u << 15) | (1u << 16);
      const uint32_t kbase = smem_u32(ktiles), qsbase = smem_u32(qsm), q1base = smem_u32(q1m);
      const uint32_t pbase = smem_u32(ptile);
      const uint64_t q1d = sw128_desc(q1base), qsd = sw128_desc(qsbase);
      bool ok = true;
      for (int k = 0; k < n + kLag && ok; ++k) {
        const Step st = step_of(p, k, n);
        if (k < n && !wait_bar(&ms->q_full, k & 1, ms, p.status)) break;
        const int len = kO ? st.n1 + 2 * st.n2 : st.len;
        for (int j = 0; j < len && ok; ++j) {
          int pass, s, kind;
          if (kO) {
            oseq_at(st, j, kind, s);
            pass = kind == 1 ? 1 : 2;
          } else {
            seq_at(st, j, pass, s);
            kind = pass;
          }
          const int ks = kcount % C::NK;
          const uint32_t ka = kbase + ks * kTileBytes;
          if (kO && kind == 3) {
            // O (+)= P . V for pass-2 tile s, once the epilogue has written
            // its probabilities (and, for the item's first tile, has read
            // out the previous item's O)
            if ((s == 0 && !wait_bar(&ms->o_empty, (ocount & 1) ^ 1, ms, p.status)) ||
                !wait_bar(&ms->p_full, pv_count & 1, ms, p.status) ||
                !wait_bar(&ms->k_full[ks], (kcount / C::NK) & 1, ms, p.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            // K step kk: 16 keys further along both MN-major operands
            const uint64_t pd = sw128_desc_mn(pbase, kHalfBytes, 1024);
            const uint64_t vd = sw128_desc_mn(ka, kHalfBytes, 1024);
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              const uint64_t step = (uint64_t)(kk * 2048 >> 4);
              mma_bf16(tmem + C::OCol, pd + step, vd + step, id_pv, kk > 0 || s > 0);
            }
            mma_commit(&ms->k_empty[ks]);
            mma_commit(&ms->p_empty);
            ++kcount;
            ++pv_count;
            if (s == st.n2 - 1) {
              mma_commit(&ms->o_full);
              ++ocount;
            }
            continue;
          }
          if (pass == 2 && s == 0) {
            if (st.n1 > 0) mma_commit(&ms->q_empty);  // item k's pass-1 queries are free
            if (!wait_bar(&ms->qs_full, qcount & 1, ms, p.status)) {
              ok = false;
              break;
            }
          }
          const int as = acount % C::NA;
          if (!wait_bar(&ms->k_full[ks], (kcount / C::NK) & 1, ms, p.status) ||
              !wait_bar(&ms->acc_empty[as], ((acount / C::NA) & 1) ^ 1, ms, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + as * 128;
          {
            // descriptors of the tile's first K step; the others differ only
            // in their start-address field (16-byte units, no carry)
            const uint64_t kd = sw128_desc(ka);
            const uint64_t qd = pass == 1 ? q1d : qsd;
            const uint64_t ad = pass == 1 ? qd : kd, bd = pass == 1 ? kd : qd;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              const uint64_t off = (uint64_t)(((kk >> 2) * kHalfBytes + (kk & 3) * 32) >> 4);
              mma_bf16(d, ad + off, bd + off, id, kk > 0);
            }
          }
          mma_commit(&ms->k_empty[ks]);
          mma_commit(&ms->acc_full[as]);
          ++kcount;
          ++acount;
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
    int oc = 0;            // kO: pass-2 items seen
    int ptc = 0;           // kO: probability tiles written

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
          const int as = tcount % C::NA, ph = (tcount / C::NA) & 1;
          ++tcount;
          if (mine && warp_wait(&ms->acc_full[as], ph, ms, p.status)) {
            tc_fence_after();
            uint32_t x[4][32];
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_ld32(tmem + lane_addr + as * 128 + c * 32, x[c]);
            tmem_wait_ld();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cnt(&ms->acc_empty[as], kO ? 2 : 1);
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
          const int as = tcount % C::NA, ph = (tcount / C::NA) & 1;
          if constexpr (kO) {
            const int key = t * kTile + r;
            // both warpgroups take every pass-2 tile, each for 64 of its 128
            // window rows (logit columns 64 wg ..): its half of the key's
            // probabilities, half of the vote (summed over the warpgroups
            // through shared memory) and its half of the probability tile
            const bool got = warp_wait(&ms->acc_full[as], ph, ms, p.status);
            float half = 0.f;
            if (got) {
              tc_fence_after();
              uint32_t x[2][32];
              tmem_ld32(tmem + lane_addr + as * 128 + wg * 64, x[0]);
              tmem_ld32(tmem + lane_addr + as * 128 + wg * 64 + 32, x[1]);
              tmem_wait_ld();
              tc_fence_before();
              __syncwarp();
              if (lane == 0) mbar_arrive(&ms->acc_empty[as]);
              // a window key (or a key past the end) is seen only by the rows
              // at or after it (causal inside the window)
              uint32_t pk[32];
              half = half_probs<true>(x, reinterpret_cast<const float4 *>(ms->offs[wg]), 2 * wg,
                                      p.scale2, key >= p.P ? key - p.P : -1, p.W, pk);
              // into the tile once the previous tile's probabilities have
              // been multiplied
              if (ptc > 0) warp_wait(&ms->p_empty, (ptc - 1) & 1, ms, p.status);
              store_p_half(ptile, r, wg, pk);
              fence_proxy_async_smem();
              __syncwarp();
              if (lane == 0) mbar_arrive(&ms->p_full);
            }
            if (wg == 1) ms->vhalf[ptc & 1][r] = half;
            named_bar_sync(6, 256);
            if (wg == 0 && got && key < p.P)
              p.votes[guard((long long)st.u2 * p.P + key, 1, (long long)p.units * p.P, p.status)] =
                  half + ms->vhalf[ptc & 1][r];
            ++ptc;
          } else if (wg_of(tcount) == wg && warp_wait(&ms->acc_full[as], ph, ms, p.status)) {
            tc_fence_after();
            uint32_t x[4][32];
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_ld32(tmem + lane_addr + as * 128 + c * 32, x[c]);
            tmem_wait_ld();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&ms->acc_empty[as]);
            const float4 *o4 = reinterpret_cast<const float4 *>(ms->offs[wg]);
            // the two halves' sums as half_probs forms them, in one pass
            float2 sv[2][4];
#pragma unroll
            for (int i = 0; i < 8; ++i) sv[i >> 2][i & 3] = make_float2(0.f, 0.f);
            const float2 s2 = make_float2(p.scale2, p.scale2);
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
                float2 *h = sv[c >> 1];
                h[(2 * j4) & 3] =
                    __fadd2_rn(h[(2 * j4) & 3], make_float2(fast_exp2(y0.x), fast_exp2(y0.y)));
                h[(2 * j4 + 1) & 3] = __fadd2_rn(h[(2 * j4 + 1) & 3],
                                                 make_float2(fast_exp2(y1.x), fast_exp2(y1.y)));
              }
            const float h0 = ((sv[0][0].x + sv[0][0].y) + (sv[0][1].x + sv[0][1].y)) +
                             ((sv[0][2].x + sv[0][2].y) + (sv[0][3].x + sv[0][3].y));
            const float h1 = ((sv[1][0].x + sv[1][0].y) + (sv[1][1].x + sv[1][1].y)) +
                             ((sv[1][2].x + sv[1][2].y) + (sv[1][3].x + sv[1][3].y));
            const int key = t * kTile + r;
            if (key < p.P)
              p.votes[guard((long long)st.u2 * p.P + key, 1, (long long)p.units * p.P, p.status)] =
                  h0 + h1;
          }
          ++tcount;
        }
      }
      if (kO && st.n2 > 0) {
        // ---------------- kO: item k - kLag's partial O (both warpgroups:
        // this thread's row, warpgroup wg's 64 dims), and the unit's output
        // from its items' partials, summed in item order by the item that
        // completes the unit
        const ItemRef it = item_of(p, k - kLag);
        const size_t prow = ((size_t)it.unit * p.n_ch + it.chunk) * 128 + r;
        if (warp_wait(&ms->o_full, oc & 1, ms, p.status)) {
          tc_fence_after();
          uint32_t x[2][32];
          tmem_ld32(tmem + lane_addr + C::OCol + wg * 64, x[0]);
          tmem_ld32(tmem + lane_addr + C::OCol + wg * 64 + 32, x[1]);
          tmem_wait_ld();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&ms->o_empty);
          float4 *dst = reinterpret_cast<float4 *>(
              p.o_part + guard((long long)prow * 128 + wg * 64, 64,
                               (long long)p.units * p.n_ch * 128 * 128, p.status));
#pragma unroll
          for (int i = 0; i < 16; ++i)
            dst[i] = make_float4(__uint_as_float(x[i >> 3][(i & 7) * 4]),
                                 __uint_as_float(x[i >> 3][(i & 7) * 4 + 1]),
                                 __uint_as_float(x[i >> 3][(i & 7) * 4 + 2]),
                                 __uint_as_float(x[i >> 3][(i & 7) * 4 + 3]));
        }
        ++oc;
        // count the item once every row of its partial is written
        __threadfence();
        named_bar_sync(5, 256);
        if (wg == 0 && wtid == 0) atomicAdd(&p.o_count[guard(it.unit, 1, p.units, p.status)], 1);
      }
      // kO: this CTA's slice of the output rows of the unit of its pass-2
      // item of kOReduceLag steps ago (its other items are done by then)
      if (kO && k - kOReduceLag >= kLag) reduce_rows(p, ms, item_of(p, k - kOReduceLag - kLag), wg * 128 + wtid);
    }
    // kO: the slices whose steps would come after the last one
    if (kO)
      for (int kr = max(kLag, n + kLag - kOReduceLag); kr < n + kLag; ++kr)
        reduce_rows(p, ms, item_of(p, kr - kLag), wg * 128 + wtid);
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

int score_tc1_max_items(const LayerGeom &g) {
  const int n_tiles = (g.T + kTile - 1) / kTile;
  return (n_tiles + kMinTilesPerItemO - 1) / kMinTilesPerItemO;
}

bool score_tc1_supported(const LayerGeom &g) {
  return g.dtype == RIPPLE_BF16 && g.D == 128 && g.R == 128 && g.P > 0 && encode_fn() != nullptr;
}

cudaError_t launch_score_tc1(const LayerGeom &g, int n_layers, const void *const *q_win,
                             const void *const *k, const CompressWs &ws, float *votes,
                             int32_t *status, cudaStream_t st, const void *const *v,
                             float *const *o_win) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr || n_layers < 1 || n_layers > kCompressMaxLayers) return cudaErrorNotSupported;
  const bool with_o = v != nullptr;
  if (with_o && (o_win == nullptr || ws.o_part == nullptr || ws.o_count == nullptr))
    return cudaErrorInvalidValue;
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
    if (with_o &&
        enc(&lp.vmap[l], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(v[l]), dims,
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
  p.n_tiles2 = with_o ? p.n_tiles1 : (g.P + kTile - 1) / kTile;
  // At least kMinTilesPerItem tiles per item, and no more items per unit than
  // SMs (the deadlock-free schedule needs <= 2x as many as CTAs).
  const int tpi_min = (p.n_tiles1 + sms - 1) / sms;
  const int tpi_floor = with_o ? kMinTilesPerItemO : kMinTilesPerItem;
  p.tpi = tpi_min > tpi_floor ? tpi_min : tpi_floor;
  p.n_ch = (p.n_tiles1 + p.tpi - 1) / p.tpi;
  p.total_items = p.units * p.n_ch;
  p.scale2 = g.scale2;
  for (int l = 0; l < n_layers; ++l) p.o_win[l] = with_o ? o_win[l] : nullptr;
  p.o_part = with_o ? ws.o_part : nullptr;
  p.o_count = with_o ? ws.o_count : nullptr;
  p.partial = ws.row_partial;
  p.lognorm = ws.row_lognorm;
  p.votes = votes;
  p.ctrl = ws.counters;
  p.status = status;
  p.wait_cycles = wait_limit_cycles();
  cudaError_t e = cudaMemsetAsync(ws.counters, 0, sizeof(int) * 2 * p.units, st);
  if (e == cudaSuccess && with_o) e = cudaMemsetAsync(ws.o_count, 0, sizeof(int) * p.units, st);
  if (e != cudaSuccess) return e;
  const void *kernel = with_o ? (const void *)score_tc1_kernel<true>
                              : (const void *)score_tc1_kernel<false>;
  const int smem = with_o ? Tc1Smem<true>::Bytes : Tc1Smem<false>::Bytes;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const int grid = p.total_items < sms ? p.total_items : sms;
  void *args[] = {(void *)&lp};
  e = cudaLaunchCooperativeKernel(kernel, dim3(grid), dim3(kThreads), args, (size_t)smem, st);
  count_launches(1);
  return e;
}

}  // namespace ripple
