// Pooling of the prefix votes and exact top-k selection per unit (SnapKV's
// selection rule kept by RippleKV; retained set S_l of Eq. 4).
//
// Three kernels, one result (bit for bit): select_unit_kernel (one CTA per
// unit, launches with many units), select_cluster_kernel (8-CTA clusters per
// unit, few units) and select_kernel (very long prefixes). The steps, for
// one unit (b, h):
//   1. pooled score of every prefix token (max or mean over the clipped
//      window), mapped to an order-preserving uint32 key (in registers, in
//      shared memory, or in global scratch for very long prefixes);
//   2. radix select over the keys (4 x 8 bits, or 11 + 11 + 10 bits, from
//      the top) finds the K-th largest key tau and how many keys equal to
//      tau are kept;
//   3. an ordered compaction writes every token with key > tau and the first
//      tokens with key == tau (lower index wins ties) in ascending order,
//      followed by the w window positions P..T-1.
// The result is bit-exact and deterministic for a given vote array. In a
// multi-layer call select_unit_kernel also gathers its unit's kept K and V
// rows (as gather_kernel would), so selection and gather are one launch.
#include <math.h>

#include "common.cuh"
#include "kernels.cuh"

namespace ripple {
namespace {

constexpr int kThreads = kSelectThreads;
constexpr int kWarps = kThreads / 32;
constexpr int kBins = 2048;
// Shared words after the histogram: scan scratch [0, 33), control [40, 48),
// per-warp exclusive counts [0, 32) and [48, 80) during the compaction.
constexpr int kCtrlWords = 128;

// Order-preserving map float -> uint32 (larger float, larger key); -0 folds to +0.
__device__ __forceinline__ uint32_t order_key(float x) {
  const uint32_t b = __float_as_uint(x + 0.0f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
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
                                                          int in_smem, int32_t *idx,
                                                          int32_t *status) {
  extern __shared__ uint32_t sm[];
  uint32_t *hist = sm;                              // [kBins]
  int *warp_tot = (int *)(sm + kBins);              // [33]
  int *ctrl = warp_tot + 40;                        // [8] control words
  uint32_t *keys = in_smem ? sm + kBins + kCtrlWords : keys_global + (size_t)blockIdx.x * g.P;

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

  // Pooling: each warp step loads 32 consecutive votes (coalesced) and the
  // lanes away from the edges take their window through shuffles.
  const int half = g.pool_kernel / 2;
  const int lane = tid & 31, wid = tid >> 5;
  const int step = 32 - 2 * half;
  for (int seg = wid * step; seg < P; seg += kWarps * step) {
    const int src = seg - half + lane;
    const bool in = src >= 0 && src < P;
    const float x = in ? v[src] : 0.f;
    float r;
    if (g.pool_type == RIPPLE_POOL_MAX) {
      r = in ? x : -INFINITY;
      const float own = r;
      for (int d = 1; d <= half; ++d) {
        r = fmaxf(r, __shfl_up_sync(0xffffffffu, own, d));
        r = fmaxf(r, __shfl_down_sync(0xffffffffu, own, d));
      }
    } else if (g.pool_type == RIPPLE_POOL_AVG) {
      // ascending positions from zero, like the definition's sum
      float s = 0.f;
      int cnt = 0;
      for (int d = -half; d <= half; ++d) {
        const float xv = d < 0 ? __shfl_up_sync(0xffffffffu, x, -d)
                               : __shfl_down_sync(0xffffffffu, x, d);
        const int pos = src + d;
        if (pos >= 0 && pos < P) {
          s = __fadd_rn(s, d == 0 ? x : xv);
          ++cnt;
        }
      }
      r = __fdiv_rn(s, (float)cnt);
    } else {
      r = x;
    }
    if (lane >= half && lane < 32 - half && src < P) keys[src] = order_key(r);
  }
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
  // Each warp owns one contiguous index range: it counts, one block scan gives
  // every warp its output offsets, then it writes its range in order.
  const int per = ((P + kWarps - 1) / kWarps + 31) & ~31;
  const int r0 = min(P, wid * per), r1 = min(P, r0 + per);
  int cgt = 0, ceq = 0;
  for (int b = r0; b < r1; b += 32) {
    const int t = b + lane;
    const uint32_t u = t < r1 ? keys[t] : 0u;
    cgt += __popc(__ballot_sync(0xffffffffu, t < r1 && u > tau));
    ceq += __popc(__ballot_sync(0xffffffffu, t < r1 && u == tau));
  }
  int *wgt = warp_tot, *weq = warp_tot + 40 + 8;  // [32] each
  if (lane == 0) {
    wgt[wid] = cgt;
    weq[wid] = ceq;
  }
  __syncthreads();
  if (wid == 0) {
    int a = wgt[lane], e = weq[lane];
    int ia = a, ie = e;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int ya = __shfl_up_sync(0xffffffffu, ia, o), ye = __shfl_up_sync(0xffffffffu, ie, o);
      if (lane >= o) {
        ia += ya;
        ie += ye;
      }
    }
    wgt[lane] = ia - a;
    weq[lane] = ie - e;
  }
  __syncthreads();
  int gt_before = wgt[wid], eq_before = weq[wid];
  const uint32_t below = (1u << lane) - 1u;
  for (int b = r0; b < r1; b += 32) {
    const int t = b + lane;
    const uint32_t u = t < r1 ? keys[t] : 0u;
    const bool gt = t < r1 && u > tau, eq = t < r1 && u == tau;
    const uint32_t bg = __ballot_sync(0xffffffffu, gt), be = __ballot_sync(0xffffffffu, eq);
    const int g_rank = gt_before + __popc(bg & below);
    const int e_rank = eq_before + __popc(be & below);
    if (gt || (eq && e_rank < take_eq)) out[guard(g_rank + min(e_rank, take_eq), 1, K, status)] = t;
    gt_before += __popc(bg);
    eq_before += __popc(be);
  }
}

// ---------------------------------------------------------------------------
// The same selection spread over a cluster of kCluster CTAs per unit: CTA r
// pools and keeps keys [r S, (r + 1) S) in its shared memory; per radix round
// each CTA builds the histogram of its keys, and after a cluster barrier every
// CTA reads all the cluster's histograms through distributed shared memory and
// derives the same digit; the compaction offsets of a CTA are the counts of
// the lower-ranked CTAs. Same result as select_kernel, bit for bit.

constexpr int kCluster = 8;
constexpr int kCThreads = 512;
constexpr int kCWarps = kCThreads / 32;
constexpr int kCMaxKeys = 40 * 1024;  // keys per CTA held in shared memory

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Shared::cluster address of the same shared-memory word in CTA `rank`.
__device__ __forceinline__ uint32_t cluster_addr(const void *p, uint32_t rank) {
  uint32_t out;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(out) : "r"(smem_u32(p)), "r"(rank));
  return out;
}
__device__ __forceinline__ uint4 ld_cluster_v4(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared::cluster.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}
__device__ __forceinline__ uint2 ld_cluster_v2(uint32_t addr) {
  uint2 v;
  asm volatile("ld.shared::cluster.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(addr) : "memory");
  return v;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Exclusive prefix sum of one int per thread over kCThreads threads.
__device__ __forceinline__ int cta_exclusive_scan(int x, int *warp_tot, int *total) {
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
    const int t = lane < kCWarps ? warp_tot[lane] : 0;
    int ti = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, ti, o);
      if (lane >= o) ti += y;
    }
    if (lane < kCWarps) warp_tot[lane] = ti - t;
    if (lane == 31) warp_tot[32] = ti;
  }
  __syncthreads();
  const int res = warp_tot[wid] + incl - x;
  *total = warp_tot[32];
  __syncthreads();
  return res;
}

// Layers of one launch: units per layer, and per layer the kept count and the
// index output [upl][n_keep].
struct SelTable {
  int upl;
  int n_keep[kCompressMaxLayers];
  int32_t *idx[kCompressMaxLayers];
  int32_t *status;
  // select_unit_kernel with gather != 0 also copies each unit's kept rows
  int gather, row_bytes;
  const uint8_t *k[kCompressMaxLayers];
  const uint8_t *v[kCompressMaxLayers];
  uint8_t *k_out[kCompressMaxLayers];
  uint8_t *v_out[kCompressMaxLayers];
  int cap[kCompressMaxLayers];
};

__global__ void __cluster_dims__(kCluster, 1, 1) __launch_bounds__(kCThreads)
    select_cluster_kernel(LayerGeom g, const float *votes, const __grid_constant__ SelTable tab) {
  extern __shared__ uint32_t sm[];
  uint32_t *hist2 = sm;                            // [2][kBins], one per round parity
  int *warp_tot = (int *)(sm + 2 * kBins);         // [33]
  int *ctrl = warp_tot + 40;                       // [8]
  int *cnt = ctrl + 8;                             // [2]: this CTA's (> tau, == tau) counts
  int *wgt = cnt + 8, *weq = wgt + 32;             // [32] each
  uint32_t *keys = sm + 2 * kBins + kCtrlWords;    // [S]

  const uint32_t rank = cluster_rank();
  const int unit = blockIdx.x / kCluster;  // over all layers of the launch
  const int layer = unit / tab.upl;
  const int n_keep = tab.n_keep[layer];
  const int P = g.P, K = n_keep - g.W;
  const int S = ((P + kCluster - 1) / kCluster + 31) & ~31;
  const int k0 = min(P, (int)rank * S), k1 = min(P, k0 + S);
  const float *v = votes + (size_t)unit * P;
  int32_t *out = tab.idx[layer] + (size_t)(unit % tab.upl) * n_keep;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;

  if (rank == 0)
    for (int j = tid; j < g.W; j += kCThreads) out[K + j] = P + j;
  if (K <= 0) return;
  if (K >= P) {
    for (int t = k0 + tid; t < k1; t += kCThreads) out[t] = t;
    return;
  }

  // This CTA's votes and the pooling halo, staged in shared memory with all
  // loads in flight at once (one memory latency instead of one per step).
  const int half = g.pool_kernel / 2;
  const int lo = max(0, k0 - half), hi = min(P, k1 + half);
  float *vs = reinterpret_cast<float *>(keys + S);  // [S + 2 * half]
  {
    constexpr int kU = 8;
    for (int b0 = lo; b0 < hi; b0 += kU * kCThreads) {
      float x[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int j = b0 + u * kCThreads + tid;
        x[u] = j < hi ? __ldcg(v + j) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int j = b0 + u * kCThreads + tid;
        if (j < hi) vs[j - lo] = x[u];
      }
    }
  }
  __syncthreads();
  // Pooled keys of this CTA's range (the window reads across range edges).
  const int step = 32 - 2 * half;
  for (int seg = k0 + wid * step; seg < k1; seg += kCWarps * step) {
    const int src = seg - half + lane;
    const bool in = src >= 0 && src < P;
    const float x = in ? vs[src - lo] : 0.f;
    float r;
    if (g.pool_type == RIPPLE_POOL_MAX) {
      r = in ? x : -INFINITY;
      const float own = r;
      for (int d = 1; d <= half; ++d) {
        r = fmaxf(r, __shfl_up_sync(0xffffffffu, own, d));
        r = fmaxf(r, __shfl_down_sync(0xffffffffu, own, d));
      }
    } else if (g.pool_type == RIPPLE_POOL_AVG) {
      float s = 0.f;
      int c = 0;
      for (int d = -half; d <= half; ++d) {
        const float xv = d < 0 ? __shfl_up_sync(0xffffffffu, x, -d)
                               : __shfl_down_sync(0xffffffffu, x, d);
        const int pos = src + d;
        if (pos >= 0 && pos < P) {
          s = __fadd_rn(s, d == 0 ? x : xv);
          ++c;
        }
      }
      r = __fdiv_rn(s, (float)c);
    } else {
      r = x;
    }
    if (lane >= half && lane < 32 - half && src >= k0 && src < k1)
      keys[src - k0] = order_key(r);
  }
  __syncthreads();

  // Radix select of the K-th largest key over the whole unit.
  uint32_t prefix = 0, mask = 0;
  int remaining = K;
  const int shifts[3] = {21, 10, 0};
  const int widths[3] = {11, 11, 10};
  const int n_local = k1 - k0;
  for (int round = 0; round < 3; ++round) {
    const int shift = shifts[round];
    const uint32_t dmask = (1u << widths[round]) - 1u;
    uint32_t *hist = hist2 + (round & 1) * kBins;
    for (int i = tid; i < kBins; i += kCThreads) hist[i] = 0;
    __syncthreads();
    for (int base = 0; base < n_local; base += kCThreads) {
      const int t = base + tid;
      const uint32_t u = t < n_local ? keys[t] : 0u;
      if (t < n_local && (u & mask) == prefix) atomicAdd(&hist[(u >> shift) & dmask], 1u);
    }
    cluster_sync_all();  // every CTA's histogram of this round is complete
    // Thread j sums digits 2047-4j .. 2044-4j (descending) over the cluster:
    // one 16-byte load from every CTA's histogram, all in flight together.
    int c[4] = {0, 0, 0, 0};
    const int d0 = kBins - 1 - 4 * tid;
    {
      uint4 h[kCluster];
#pragma unroll
      for (uint32_t r = 0; r < kCluster; ++r) h[r] = ld_cluster_v4(cluster_addr(hist + d0 - 3, r));
#pragma unroll
      for (uint32_t r = 0; r < kCluster; ++r) {
        c[0] += (int)h[r].w;
        c[1] += (int)h[r].z;
        c[2] += (int)h[r].y;
        c[3] += (int)h[r].x;
      }
    }
    int total;
    int above = cta_exclusive_scan(c[0] + c[1] + c[2] + c[3], warp_tot, &total);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      if (above < remaining && remaining <= above + c[q]) {
        ctrl[0] = d0 - q;
        ctrl[1] = remaining - above;
      }
      above += c[q];
    }
    __syncthreads();
    prefix |= (uint32_t)ctrl[0] << shift;
    mask |= dmask << shift;
    remaining = ctrl[1];
    __syncthreads();
  }
  const uint32_t tau = prefix;
  const int take_eq = remaining;

  // Ordered compaction over the cluster: counts per warp range, per CTA,
  // then offsets from the lower-ranked CTAs.
  const int per = ((n_local + kCWarps - 1) / kCWarps + 31) & ~31;
  const int r0 = min(n_local, wid * per), r1 = min(n_local, r0 + per);
  int cgt = 0, ceq = 0;
  for (int b = r0; b < r1; b += 32) {
    const int t = b + lane;
    const uint32_t u = t < r1 ? keys[t] : 0u;
    cgt += __popc(__ballot_sync(0xffffffffu, t < r1 && u > tau));
    ceq += __popc(__ballot_sync(0xffffffffu, t < r1 && u == tau));
  }
  if (lane == 0) {
    wgt[wid] = cgt;
    weq[wid] = ceq;
  }
  __syncthreads();
  if (wid == 0) {
    const int a = lane < kCWarps ? wgt[lane] : 0, e = lane < kCWarps ? weq[lane] : 0;
    int ia = a, ie = e;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int ya = __shfl_up_sync(0xffffffffu, ia, o), ye = __shfl_up_sync(0xffffffffu, ie, o);
      if (lane >= o) {
        ia += ya;
        ie += ye;
      }
    }
    if (lane < kCWarps) {
      wgt[lane] = ia - a;
      weq[lane] = ie - e;
    }
    if (lane == 31) {
      cnt[0] = ia;
      cnt[1] = ie;
    }
  }
  cluster_sync_all();  // every CTA's counts are published
  int gt_cta = 0, eq_cta = 0;
  for (uint32_t r = 0; r < rank; ++r) {
    const uint2 c = ld_cluster_v2(cluster_addr(cnt, r));
    gt_cta += (int)c.x;
    eq_cta += (int)c.y;
  }
  int gt_before = gt_cta + wgt[wid], eq_before = eq_cta + weq[wid];
  const uint32_t below = (1u << lane) - 1u;
  for (int b = r0; b < r1; b += 32) {
    const int t = b + lane;
    const uint32_t u = t < r1 ? keys[t] : 0u;
    const bool gt = t < r1 && u > tau, eq = t < r1 && u == tau;
    const uint32_t bg = __ballot_sync(0xffffffffu, gt), be = __ballot_sync(0xffffffffu, eq);
    const int g_rank = gt_before + __popc(bg & below);
    const int e_rank = eq_before + __popc(be & below);
    if (gt || (eq && e_rank < take_eq))
      out[guard(g_rank + min(e_rank, take_eq), 1, K, tab.status)] = k0 + t;
    gt_before += __popc(bg);
    eq_before += __popc(be);
  }
  cluster_sync_all();  // no CTA leaves while others may still read its memory
}

// Prefixes up to kUMaxP tokens: one 1024-thread CTA per unit and no cluster
// (a launch covers every unit of every layer, so the GPU is filled by units).
// Thread t keeps the pooled keys of tokens 32t .. 32t + 31 in registers: the
// votes are staged in shared memory with a pad word after every 32 (coalesced
// stores, conflict-free reads of a thread's run), the 7-wide max pooling is
// three maxima per key over the run and its halo, four radix rounds of 8 bits
// count into per-warp histograms (no contention between warps), and the
// ordered compaction is one block scan over the threads' counts followed by
// each thread writing its kept tokens in order. Same result as select_kernel,
// bit for bit.
constexpr int kUThreads = 1024;
constexpr int kUWarps = kUThreads / 32;
constexpr int kUKeys = 32;                    // keys per thread
constexpr int kUMaxP = kUThreads * kUKeys;
constexpr int kUBins = 256;
constexpr int kUMinUnits = 256;               // units per launch for this kernel
constexpr int kUCand = 128;                   // bucket size that ends the radix rounds
// shared words before the staged votes: per-warp histograms, bin totals,
// scan scratch and control
constexpr int kUHead = kUWarps * kUBins + kUBins + 64;

// Shared-memory word of staged vote j: one pad word after every 32.
__device__ __forceinline__ int upad(int j) { return j + (j >> 5); }

// Pooling, radix select and ordered compaction of one unit's prefix tokens
// (0 < K < P): writes out[0 .. K).
__device__ __forceinline__ void select_unit_keys(const LayerGeom &g, const float *v, int32_t *out,
                                                 int K, uint32_t *sm, int32_t *status) {
  uint32_t *hist = sm;                                   // [kUWarps][kUBins]
  int *tot = (int *)(hist + kUWarps * kUBins);           // [kUBins]
  int *warp_tot = tot + kUBins;                          // [33]
  int *ctl = warp_tot + 40;                              // [6]
  float *vs = reinterpret_cast<float *>(sm + kUHead);    // [P + P / 32], padded
  const int P = g.P;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;

  // Votes into shared memory (coalesced, sixteen loads of a thread in flight),
  // with one pad word after every 32: thread t then reads its run of keys
  // 32t .. 32t + 31 (and the pooling halo) without bank conflicts.
#pragma unroll
  for (int i0 = 0; i0 < kUKeys; i0 += 16) {
    float x[16];
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      const int j = (i0 + u) * kUThreads + tid;
      x[u] = j < P ? __ldcg(v + j) : 0.f;
    }
#pragma unroll
    for (int u = 0; u < 16; ++u) {
      const int j = (i0 + u) * kUThreads + tid;
      if (j < P) vs[upad(j)] = x[u];
    }
  }
  __syncthreads();

  // Pooled keys of this thread's tokens j0 .. j0 + 31 (window clipped to the
  // prefix).
  const int half = g.pool_kernel / 2;
  const int j0 = tid * kUKeys;
  uint32_t key[kUKeys];
  if (g.pool_type == RIPPLE_POOL_MAX && half == 3) {
    // the 7-wide max from the votes w = v[j0 - 3 .. j0 + 34] (-inf outside
    // the prefix): b[i] = max(w[i .. i + 3]) and pooled(j0 + i) = max(b[i], b[i + 3])
    float w[kUKeys + 6];
#pragma unroll
    for (int i = 0; i < kUKeys + 6; ++i) {
      const int j = j0 - 3 + i;
      w[i] = j >= 0 && j < P ? vs[upad(j)] : -INFINITY;
    }
    float a[kUKeys + 5];
#pragma unroll
    for (int i = 0; i < kUKeys + 5; ++i) a[i] = fmaxf(w[i], w[i + 1]);
    float b[kUKeys + 3];
#pragma unroll
    for (int i = 0; i < kUKeys + 3; ++i) b[i] = fmaxf(a[i], a[i + 2]);
#pragma unroll
    for (int i = 0; i < kUKeys; ++i) key[i] = order_key(fmaxf(b[i], b[i + 3]));
  } else {
#pragma unroll
    for (int i = 0; i < kUKeys; ++i) {
      const int j = j0 + i;
      float r = 0.f;
      if (j < P) {
        if (g.pool_type == RIPPLE_POOL_MAX) {
          r = vs[upad(j)];
          for (int d = 1; d <= half; ++d) {
            if (j - d >= 0) r = fmaxf(r, vs[upad(j - d)]);
            if (j + d < P) r = fmaxf(r, vs[upad(j + d)]);
          }
        } else if (g.pool_type == RIPPLE_POOL_AVG) {
          float sum = 0.f;
          int c = 0;
          for (int d = -half; d <= half; ++d) {
            const int pos = j + d;
            if (pos >= 0 && pos < P) {
              sum = __fadd_rn(sum, vs[upad(pos)]);
              ++c;
            }
          }
          r = __fdiv_rn(sum, (float)c);
        } else {
          r = vs[upad(j)];
        }
      }
      key[i] = order_key(r);
    }
  }

  // Radix select of the K-th largest key: up to 4 rounds of 8 bits from the
  // top; once the bucket that holds it has at most kUCand keys, the rest is
  // found among that bucket's keys directly (tau is then the same key).
  uint32_t prefix = 0, mask = 0;
  int remaining = K;
  uint32_t tau = 0;
  int take_eq = -1;
  uint32_t *hw = hist + wid * kUBins;
  for (int round = 0; round < 4; ++round) {
    const int shift = 24 - 8 * round;
#pragma unroll
    for (int b = lane; b < kUBins; b += 32) hw[b] = 0;
    __syncwarp();
#pragma unroll
    for (int i = 0; i < kUKeys; ++i)
      if (j0 + i < P && (key[i] & mask) == prefix) atomicAdd(&hw[(key[i] >> shift) & 255u], 1u);
    __syncthreads();
    if (tid < kUBins) {
      int sum = 0;
#pragma unroll 8
      for (int w = 0; w < kUWarps; ++w) sum += (int)hist[w * kUBins + tid];
      tot[tid] = sum;
    }
    __syncthreads();
    if (wid == 0) {
      // lane l holds digits 255 - 8l down to 248 - 8l
      int c[8], sum = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        c[q] = tot[kUBins - 1 - 8 * lane - q];
        sum += c[q];
      }
      int incl = sum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      int above = incl - sum;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (above < remaining && remaining <= above + c[q]) {
          ctl[0] = kUBins - 1 - 8 * lane - q;
          ctl[1] = remaining - above;
          ctl[2] = c[q];
        }
        above += c[q];
      }
      if (lane == 0) ctl[3] = 0;
    }
    __syncthreads();
    prefix |= (uint32_t)ctl[0] << shift;
    mask |= 255u << shift;
    remaining = ctl[1];
    if (round < 3 && ctl[2] <= kUCand) {
      // the bucket's keys into a list (any order); each of them counts the
      // keys above and equal to it, and the one with remaining - 1 above
      // and at least remaining above or equal is tau
      uint32_t *cand = hist;  // the histograms are not needed any more
#pragma unroll
      for (int i = 0; i < kUKeys; ++i)
        if (j0 + i < P && (key[i] & mask) == prefix) cand[atomicAdd(&ctl[3], 1)] = key[i];
      __syncthreads();
      const int nc = ctl[2];
      if (tid < nc) {
        const uint32_t x = cand[tid];
        int above = 0, same = 0;
        for (int c = 0; c < nc; ++c) {
          const uint32_t y = cand[c];
          above += y > x;
          same += y == x;
        }
        if (above < remaining && remaining <= above + same) {
          ctl[4] = (int)x;
          ctl[5] = remaining - above;
        }
      }
      __syncthreads();
      tau = (uint32_t)ctl[4];
      take_eq = ctl[5];
      break;
    }
  }
  if (take_eq < 0) {
    tau = prefix;
    take_eq = remaining;
  }

  // Ordered compaction: this thread's counts of keys above and equal to tau,
  // one block scan over the threads (token order), then its kept tokens in
  // order: every key above tau and the first take_eq keys equal to it.
  int gt = 0, eq = 0;
#pragma unroll
  for (int i = 0; i < kUKeys; ++i) {
    gt += j0 + i < P && key[i] > tau;
    eq += j0 + i < P && key[i] == tau;
  }
  int total;
  const int off = block_exclusive_scan((gt << 16) | eq, warp_tot, &total);
  int g_rank = off >> 16, e_rank = off & 0xffff;
#pragma unroll
  for (int i = 0; i < kUKeys; ++i) {
    const bool is_gt = j0 + i < P && key[i] > tau, is_eq = j0 + i < P && key[i] == tau;
    if (is_gt || (is_eq && e_rank < take_eq))
      out[guard(g_rank + min(e_rank, take_eq), 1, K, status)] = j0 + i;
    g_rank += is_gt;
    e_rank += is_eq;
  }
}

__global__ void __launch_bounds__(kUThreads, 1)
    select_unit_kernel(LayerGeom g, const float *votes, const __grid_constant__ SelTable tab) {
  extern __shared__ uint32_t sm[];
  const int unit = blockIdx.x;  // over all layers of the launch
  const int layer = unit / tab.upl;
  const int n_keep = tab.n_keep[layer];
  const int P = g.P, K = n_keep - g.W;
  int32_t *out = tab.idx[layer] + (size_t)(unit % tab.upl) * n_keep;
  const int tid = threadIdx.x;

  for (int j = tid; j < g.W; j += kUThreads) out[K + j] = P + j;
  if (K >= P) {
    for (int t = tid; t < P; t += kUThreads) out[t] = t;
  } else if (K > 0) {
    select_unit_keys(g, votes + (size_t)unit * P, out, K, sm, tab.status);
  }
  if (tab.gather) {
    // the unit's kept K and V rows into its compact cache rows 0 .. n_keep - 1:
    // row_bytes / 16 consecutive threads copy one row 16 bytes each, four rows
    // a thread in flight
    __syncthreads();  // out[] of this CTA written
    const int rb = tab.row_bytes, lpr = rb >> 4, rpp = kUThreads / lpr;
    const int r_in = tid / lpr, c16 = (tid % lpr) * 16;
    const size_t local = (size_t)(unit % tab.upl);
    const uint8_t *kin = tab.k[layer] + local * g.T * rb;
    const uint8_t *vin = tab.v[layer] + local * g.T * rb;
    uint8_t *kout = tab.k_out[layer] + local * tab.cap[layer] * rb;
    uint8_t *vout = tab.v_out[layer] + local * tab.cap[layer] * rb;
    for (int r0 = 0; r0 < n_keep; r0 += 4 * rpp) {
      uint4 xk[4], xv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int r = r0 + u * rpp + r_in;
        if (r < n_keep) {
          const long long t = guard(__ldcg(&out[r]), 1, g.T, tab.status);
          xk[u] = __ldcs(reinterpret_cast<const uint4 *>(kin + t * rb + c16));
          xv[u] = __ldcs(reinterpret_cast<const uint4 *>(vin + t * rb + c16));
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int r = r0 + u * rpp + r_in;
        if (r < n_keep) {
          *reinterpret_cast<uint4 *>(kout + (size_t)r * rb + c16) = xk[u];
          *reinterpret_cast<uint4 *>(vout + (size_t)r * rb + c16) = xv[u];
        }
      }
    }
  }
}

}  // namespace

cudaError_t launch_select(const LayerGeom &g, int n_layers, const float *votes,
                          const CompressWs &ws, const int *n_keep, int32_t *const *idx,
                          int32_t *status, cudaStream_t st, const GatherArgs *gather,
                          bool *gathered) {
  if (n_layers < 1 || n_layers > kCompressMaxLayers) return cudaErrorInvalidValue;
  if (gathered != nullptr) *gathered = false;
  // One CTA per unit once the launch has enough units to fill the GPU;
  // fewer units (a single layer) are spread over 8-CTA clusters instead.
  if (g.P <= kUMaxP && (long long)g.units * n_layers >= kUMinUnits) {
    SelTable tab;
    tab.upl = g.units;
    tab.status = status;
    tab.gather = gather != nullptr && gathered != nullptr;
    tab.row_bytes = g.D * (g.dtype == RIPPLE_F32 ? 4 : 2);
    for (int l = 0; l < n_layers; ++l) {
      tab.n_keep[l] = n_keep[l];
      tab.idx[l] = idx[l];
      if (tab.gather) {
        tab.k[l] = (const uint8_t *)gather->k[l];
        tab.v[l] = (const uint8_t *)gather->v[l];
        tab.k_out[l] = (uint8_t *)gather->k_out[l];
        tab.v_out[l] = (uint8_t *)gather->v_out[l];
        tab.cap[l] = gather->cap[l];
      }
    }
    const size_t smem = sizeof(uint32_t) * ((size_t)kUHead + g.P + g.P / 32 + 1);
    cudaError_t e = cudaFuncSetAttribute(select_unit_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    select_unit_kernel<<<g.units * n_layers, kUThreads, smem, st>>>(g, votes, tab);
    count_launches(1);
    e = cudaGetLastError();
    if (e == cudaSuccess && gathered != nullptr) *gathered = tab.gather != 0;
    return e;
  }
  const int per_cta = ((g.P + kCluster - 1) / kCluster + 31) & ~31;
  if (per_cta <= kCMaxKeys && (long long)g.units * n_layers * kCluster <= 0x7fffffff) {
    SelTable tab;
    tab.upl = g.units;
    tab.status = status;
    tab.gather = 0;
    for (int l = 0; l < n_layers; ++l) {
      tab.n_keep[l] = n_keep[l];
      tab.idx[l] = idx[l];
    }
    // histograms, control words, keys, staged votes (with the pooling halo)
    const size_t smem = sizeof(uint32_t) * (2 * kBins + kCtrlWords + 2 * per_cta + 32);
    cudaError_t e = cudaFuncSetAttribute(select_cluster_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    select_cluster_kernel<<<g.units * n_layers * kCluster, kCThreads, smem, st>>>(g, votes, tab);
    count_launches(1);
    return cudaGetLastError();
  }
  // Very long prefixes: one CTA per unit, layer by layer.
  const int in_smem = g.P <= kSelectSmemKeys;
  const size_t smem = sizeof(uint32_t) * (kBins + kCtrlWords + (in_smem ? g.P : 0));
  cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  for (int l = 0; l < n_layers; ++l) {
    select_kernel<<<g.units, kThreads, smem, st>>>(g, votes + (size_t)l * g.units * g.P, ws.keys,
                                                   n_keep[l], in_smem, idx[l], status);
    count_launches(1);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
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
