// GQA decode attention over the ragged compressed caches (Sec. 4.1: each new
// query attends to the cached states), with the append of the new token.
//
// One persistent launch per step covers every layer; one CTA per SM with 8
// compute warps and one producer warp. Work item = up to p.item_rows cache rows
// of one (layer, batch row, KV head) group; items are fetched with an atomic
// counter (one ahead), layers with the longest caches first. The producer
// stages each item's G query rows and then its sub-chunks of K and V rows in
// shared memory with bulk-async copies (TMA engine) through a ring of stages;
// the new token's key and value rows are copied into the stage behind the
// cached rows, and appended to the cache from there.
//
// Lane layout (the same for Q.K and P.V): the rows of a warp step are split
// over R row groups of S lanes; each lane owns DL head dims (its 16-byte
// pieces of the row) of every query head of the group: it reads those dims of
// the scaled fp32 queries from shared memory (converted once per item, in the
// order the lanes read them) and keeps those dims of the output accumulator
// in registers. Per row:
//   scores   fp32x2 FMAs over the lane's dims, then a reduce-scatter over the
//            S lanes of the row group (warp shuffles) that leaves each lane
//            with the full dot product of one head;
//   softmax  each (row group, head) keeps its own running max and sum (online
//            softmax; scores are in log2 units and the max is moved, and the
//            state rescaled, only when a score exceeds it by more than 8, a
//            probability factor of 2^8, so rescaling is rare);
//            the probability is computed once per head and all-gathered over
//            the row group (warp shuffles);
//   output   fp32x2 FMAs of the probabilities with the lane's value dims.
// At an item's end the row groups of a warp are merged by a shuffle butterfly
// and the 8 warps through shared memory. An item covering its whole group
// writes the output; otherwise its unnormalised partial is stored and the
// group's last finishing item (atomic count) combines the partials in item
// order (deterministic).
//
// The step's counters live in the caller's workspace, whose contents are
// arbitrary: CTA 0 zeroes them at the start of every call and then raises an
// init flag tagged with the call's epoch; the other CTAs use no counter
// before they see it (their first item needs none). Each launch is a
// programmatic dependent of the previous one on the stream: its CTAs take
// SMs as the previous step's CTAs leave and wait (griddepcontrol.wait) until
// that step has completed.
// CTA b's first item is item b, so that before that wait it can already
// prefetch its first sub-chunks into L2.
// Every wait is bounded; on timeout the CTA raises RIPPLE_ETIMEOUT and all
// roles leave their loops together.
#include <math.h>

#include <atomic>
#include <chrono>
#include <mutex>

#include "common.cuh"
#include "decode.cuh"
#include "kernels.cuh"

namespace ripple {
namespace {

constexpr int kWarps = 8;                     // compute warps
constexpr int kThreads = (kWarps + 1) * 32;   // + one producer warp
constexpr int kMaxStageBytes = 32768;         // K (or V) bytes of one sub-chunk, at most
constexpr int kRowsPerGroup = 4;              // rows per row group and sub-chunk (warp steps)
constexpr int kItemSlots = 4;
constexpr int kMaxStages = 6;
// Lazy rescaling: a running max (log2 units) is only moved when a score
// exceeds it by more than kRescaleLog2, so probabilities relative to a stale
// max stay <= 2^kRescaleLog2.
constexpr float kRescaleLog2 = 8.f;
constexpr int kSmemBudget = 226 * 1024;
constexpr int kMiscBytes = 4096;              // barriers, work list, merge statistics
constexpr unsigned kFull = 0xffffffffu;

constexpr int cmax(int a, int b) { return a > b ? a : b; }
constexpr int cmin(int a, int b) { return a < b ? a : b; }

template <typename Tin, int D, int G>
struct DecCfg {
  static constexpr int ROW_BYTES = D * (int)sizeof(Tin);
  static constexpr int NPIECE = ROW_BYTES / 16;             // 16-byte pieces per row
  static constexpr int PE = 16 / (int)sizeof(Tin);          // elements per piece
  // lanes per row: the queries and accumulators of a lane stay at 64
  // registers each, at least one lane per head, and a warp step's rows fit a
  // sub-chunk
  static constexpr int S = cmax(cmax(G * D / 64, G), cmax(ROW_BYTES / 128, 1));
  static constexpr int R = 32 / S;                          // row groups (rows per warp step)
  static constexpr int NIT =                                // warp steps per sub-chunk
      cmax(1, cmin(kRowsPerGroup, kMaxStageBytes / (kWarps * R * ROW_BYTES)));
  static constexpr int RPW = R * NIT;                       // rows per warp per sub-chunk
  static constexpr int CR = RPW * kWarps;                   // rows per sub-chunk
  static constexpr int STAGE_BYTES = CR * ROW_BYTES;
  static constexpr int PPL = NPIECE / S;                    // pieces per lane
  static constexpr int DL = PPL * PE;                       // head dims per lane
  static constexpr int HL = S / G;                          // lanes per head after the reduce-scatter
  static constexpr int QBYTES = G * ROW_BYTES;              // one group's queries
  static constexpr int NH = PE / 4;                         // float4 per piece in fp32
  static constexpr int STAGES =
      cmin(kMaxStages, (kSmemBudget - kMiscBytes - kItemSlots * QBYTES - (kWarps + 2) * G * D * 4) /
                           (2 * STAGE_BYTES));
  static_assert(kMinItemRows % CR == 0, "items are whole sub-chunks");
  static_assert(S <= 32 && S <= NPIECE && NPIECE % S == 0, "lanes per row");
  static_assert(STAGE_BYTES <= kMaxStageBytes, "stage size");
  static_assert(DL % 2 == 0 && PE % 2 == 0, "fp32x2 pairs");
  static_assert(STAGES >= 2, "shared memory budget");
};

template <typename Tin, int D, int G>
struct DecSmem {
  using C = DecCfg<Tin, D, G>;
  alignas(128) uint8_t kv[C::STAGES][2][C::STAGE_BYTES];  // [stage][K, V]
  alignas(128) uint8_t qs[kItemSlots][C::QBYTES];      // each item's query rows
  alignas(16) float qf[2][G * D];                      // scaled fp32 queries, lane-piece order
  alignas(16) float red_o[kWarps][G * D];              // per-warp outputs at an item's end
  float red_m[kWarps][G], red_l[kWarps][G];
  uint64_t full[C::STAGES], empty[C::STAGES], item_full[kItemSlots], item_empty[kItemSlots];
  int item_id[kItemSlots];
  int len[RIPPLE_MAX_LAYERS];    // by work-order position; -1 = full layer
  int nch[RIPPLE_MAX_LAYERS];    // items per group, by work-order position
  int base[RIPPLE_MAX_LAYERS + 1];
  int abort_flag;
  int last;
  int init_seen;  // this CTA has seen the init flag (consumer thread 0's view)
};

struct ItemInfo {
  int pos, layer, group, b, h, chunk, nch, len, r0, rows, full;
};

template <typename S>
__device__ __forceinline__ ItemInfo item_info(const DecParams &p, const S &s, int it) {
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
  f.r0 = f.chunk * p.item_rows;
  // rows 0..len: the cached rows and the new token
  f.rows = f.full ? 0 : min(p.item_rows, f.len + 1 - f.r0);
  return f;
}

// Bounded wait on an mbarrier phase. Gives up when another role of the CTA
// has given up, or after p.wait_cycles (then raises the CTA's abort flag and
// reports RIPPLE_ETIMEOUT).
__device__ __forceinline__ bool wait_bar(uint64_t *bar, uint32_t parity, int *abort_flag,
                                         const DecParams &p) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*(volatile int *)abort_flag) return false;
    if (clock64() - t0 > p.wait_cycles) {
      *(volatile int *)abort_flag = 1;
      report(p.status, RIPPLE_ETIMEOUT);
      return false;
    }
  }
}

// Waits until CTA 0 has zeroed this call's counters (the init flag holds the
// call's epoch). Bounded like wait_bar.
__device__ __forceinline__ bool wait_init(const DecParams &p, int *abort_flag) {
  if (ld_acquire(&p.ctrl[kCtrlFlag]) == p.epoch) return true;
  const long long t0 = clock64();
  for (;;) {
    if (ld_acquire(&p.ctrl[kCtrlFlag]) == p.epoch) return true;
    if (*(volatile int *)abort_flag) return false;
    if (clock64() - t0 > p.wait_cycles) {
      *(volatile int *)abort_flag = 1;
      report(p.status, RIPPLE_ETIMEOUT);
      return false;
    }
    __nanosleep(32);
  }
}

// Named barrier over the compute warps that also ORs a predicate over them.
__device__ __forceinline__ bool compute_bar_or(bool pred) {
  __syncwarp();
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n"
      " setp.ne.u32 p, %1, 0;\n"
      " barrier.red.or.pred q, 1, %2, p;\n"
      " selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r)
      : "r"((uint32_t)pred), "n"(kWarps * 32)
      : "memory");
  return r != 0;
}

// 2*NP consecutive elements (one aligned load of 4 * NP bytes for bf16, or
// 8 * NP bytes for fp32) as fp32 pairs; bf16 widens by placing its 16 bits in
// the upper half of an fp32.
__device__ __forceinline__ float2 bf16x2_pair(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}
template <int NP>
__device__ __forceinline__ void load_pairs(const __nv_bfloat16 *p, float2 (&o)[NP]) {
  static_assert(NP == 4, "one 16-byte piece");
  const uint4 u = *reinterpret_cast<const uint4 *>(p);
  o[0] = bf16x2_pair(u.x); o[1] = bf16x2_pair(u.y);
  o[2] = bf16x2_pair(u.z); o[3] = bf16x2_pair(u.w);
}
template <int NP>
__device__ __forceinline__ void load_pairs(const float *p, float2 (&o)[NP]) {
  static_assert(NP == 2, "one 16-byte piece");
  const float4 u = *reinterpret_cast<const float4 *>(p);
  o[0] = make_float2(u.x, u.y);
  o[1] = make_float2(u.z, u.w);
}

// Per-head values of a lane are kept in an order permuted by the lane's own
// head hq = (lane % S) / (S / G): entry j holds head j ^ hq. Then every step
// of the reduce-scatter and of the all-gather over the S lanes of a row group
// is a plain shuffle (the partner's entry that this lane needs sits at a fixed
// index), with no per-lane selects.
//
// Reduce-scatter of G per-lane partial sums: afterwards v[0] of every lane is
// the full sum of its head hq. At the step over lane bit o the partner's head
// differs from this lane's in the head bit being split, which is bit
// log2(nv / 2) of the entry index.
template <int S, int G>
__device__ __forceinline__ void reduce_scatter(float (&v)[G]) {
#pragma unroll
  for (int o = S / 2, nv = G; o >= 1; o >>= 1) {
    if (nv > 1) {
#pragma unroll
      for (int i = 0; i < G / 2; ++i)
        if (i < nv / 2) v[i] += __shfl_xor_sync(kFull, v[i + nv / 2], o);
      nv /= 2;
    } else {
      v[0] += __shfl_xor_sync(kFull, v[0], o);
    }
  }
}

// Inverse of the head split of reduce_scatter: from x (the value of head hq)
// every lane of the row group receives o[j] = the value of head j ^ hq.
template <int S, int G>
__device__ __forceinline__ void all_gather(float x, float (&o)[G]) {
  o[0] = x;
#pragma unroll
  for (int lev = 0; (1 << lev) < G; ++lev)
#pragma unroll
    for (int i = 0; i < (1 << lev); ++i)
      o[(1 << lev) + i] = __shfl_xor_sync(kFull, o[i], (S / G) << lev);
}

// ------------------------------------------------------------ producer
// Holds the producer until the bulk copies it has issued have landed (the
// last phase armed on each stage and item slot), so that no copy writes into
// shared memory after the CTA has left even when the consumers gave up early;
// when they did not, these phases have long completed. Fixed bound,
// independent of the launch's wait limit.
template <typename Tin, int D, int G>
__device__ __forceinline__ void drain(DecSmem<Tin, D, G> &s, uint32_t j,
                                      const int (&last_use)[kItemSlots]) {
  using C = DecCfg<Tin, D, G>;
  for (uint32_t jj = j > (uint32_t)C::STAGES ? j - C::STAGES : 0; jj < j; ++jj)
    mbar_wait(&s.full[jj % C::STAGES], (jj / C::STAGES) & 1, nullptr);
  for (int slot = 0; slot < kItemSlots; ++slot)
    if (last_use[slot] >= 0)
      mbar_wait(&s.item_full[slot], (last_use[slot] / kItemSlots) & 1, nullptr);
}

template <typename Tin, int D, int G>
__device__ __forceinline__ void produce(const DecParams &p, DecSmem<Tin, D, G> &s, int total) {
  using C = DecCfg<Tin, D, G>;
  const int units = p.B * p.Hkv;
  uint32_t j = 0;                                // sub-chunk stages armed
  int last_use[kItemSlots] = {-1, -1, -1, -1};   // last item count that armed each slot
  static_assert(kItemSlots == 4, "last_use initialiser");
  // The item after `cur`, fetched from the counter once CTA 0 has zeroed it.
  auto next_of = [&](int cur) {
    if (cur >= total || !wait_init(p, &s.abort_flag)) return total;
    return atomicAdd(&p.ctrl[kCtrlItem], 1) + (int)gridDim.x;
  };
  // The first item of CTA b is item b; later ones come from the counter, one
  // item ahead (for the first item, once its first loads are issued).
  int it = min((int)blockIdx.x, total);
  for (int icount = 0;; ++icount) {
    const int slot = icount % kItemSlots;
    int nxt = icount > 0 ? next_of(it) : -1;
    if (!wait_bar(&s.item_empty[slot], ((icount / kItemSlots) & 1) ^ 1, &s.abort_flag, p)) {
      drain(s, j, last_use);
      return;
    }
    const int cur = min(it, total);
    s.item_id[slot] = cur;
    last_use[slot] = icount;
    if (cur >= total) {
      mbar_arrive(&s.item_full[slot]);
      drain(s, j, last_use);  // returns at once unless the consumers gave up
      return;
    }
    const ItemInfo f = item_info(p, s, cur);
    if (f.full) {
      mbar_arrive(&s.item_full[slot]);
    } else {
      const size_t qrow = ((size_t)f.layer * p.B + f.b) * p.Hq + (size_t)f.h * G;
      mbar_arrive_expect_tx(&s.item_full[slot], C::QBYTES);
      const long long qr = guard((long long)qrow, G, (long long)p.L * p.B * p.Hq, p.status);
      bulk_g2s(s.qs[slot], (const uint8_t *)p.q + qr * C::ROW_BYTES, C::QBYTES,
               &s.item_full[slot]);
      const int nsub = (f.rows + C::CR - 1) / C::CR;
      const size_t gbase = (size_t)(f.b * p.Hkv + f.h) * p.cap[f.layer];
      const size_t nb = guard((long long)f.layer * units + f.b * p.Hkv + f.h, 1,
                              (long long)p.L * units, p.status) *
                        C::ROW_BYTES;
      for (int sub = 0; sub < nsub; ++sub, ++j) {
        const int stage = j % C::STAGES;
        if (sub == 1 && nxt < 0) nxt = next_of(it);
        if (!wait_bar(&s.empty[stage], ((j / C::STAGES) & 1) ^ 1, &s.abort_flag, p)) {
          drain(s, j, last_use);
          return;
        }
        const int rs = f.r0 + sub * C::CR;
        const int re = min(rs + C::CR, f.len);  // rows >= len are not in the cache yet
        const int nk = re > rs ? re - rs : 0;
        const bool has_new = f.len >= rs && f.len < rs + C::CR;
        mbar_arrive_expect_tx(&s.full[stage], 2u * (nk + (has_new ? 1 : 0)) * C::ROW_BYTES);
        if (nk > 0) {
          const size_t off =
              guard((long long)(gbase + rs), nk, (long long)units * p.cap[f.layer], p.status) *
              C::ROW_BYTES;
          bulk_g2s(s.kv[stage][0], (const uint8_t *)p.kc[f.layer] + off, nk * C::ROW_BYTES,
                   &s.full[stage]);
          bulk_g2s(s.kv[stage][1], (const uint8_t *)p.vc[f.layer] + off, nk * C::ROW_BYTES,
                   &s.full[stage]);
        }
        if (has_new) {
          const int r = f.len - rs;
          bulk_g2s(s.kv[stage][0] + r * C::ROW_BYTES, (const uint8_t *)p.k_new + nb,
                   C::ROW_BYTES, &s.full[stage]);
          bulk_g2s(s.kv[stage][1] + r * C::ROW_BYTES, (const uint8_t *)p.v_new + nb,
                   C::ROW_BYTES, &s.full[stage]);
        }
      }
    }
    if (nxt < 0) nxt = next_of(it);
    it = nxt;
  }
}

// ------------------------------------------------------------ compute warps
template <typename Tin, int D, int G>
__device__ __forceinline__ void consume(const DecParams &p, DecSmem<Tin, D, G> &s, int total,
                                        int warp, int lane) {
  using C = DecCfg<Tin, D, G>;
  constexpr int S = C::S, R = C::R, NIT = C::NIT, PPL = C::PPL, PE = C::PE, DL = C::DL;
  const int tid = warp * 32 + lane;
  const int sl = lane % S;              // lane within its row group
  const int rg = lane / S;              // row group
  const int hq = sl / C::HL;            // head of this lane after the reduce-scatter;
                                        // per-head arrays hold head j ^ hq at entry j
  const int rw0 = warp * C::RPW;        // this warp's first row in a sub-chunk
  uint32_t j = 0;
  for (int icount = 0;; ++icount) {
    const int slot = icount % kItemSlots;
    bool ok = wait_bar(&s.item_full[slot], (icount / kItemSlots) & 1, &s.abort_flag, p);
    ok = __all_sync(kFull, ok);
    const int it = ok ? s.item_id[slot] : total;
    // Queries to fp32, scaled to log2 units, in the order the lanes read them:
    // [entry j][piece k][half h][lane sl][4], entry j of lane sl being head
    // j ^ hq(sl).
    float *qf = s.qf[icount & 1];
    if (it < total) {
      const Tin *qg = (const Tin *)s.qs[slot];
      for (int e = tid; e < G * D; e += kWarps * 32) {
        const int c = e % 4, l4 = (e / 4) % S, h = (e / (4 * S)) % C::NH;
        const int k = (e / (4 * S * C::NH)) % PPL, jj = e / (4 * S * C::NH * PPL);
        const int g = jj ^ (l4 / C::HL);
        qf[e] = to_f32(qg[g * D + (l4 + k * S) * PE + h * 4 + c]) * p.scale2;
      }
    }
    // All compute warps leave together (the item's merge has named barriers);
    // this barrier also frees the merge buffers of the previous item and
    // publishes the fp32 queries.
    if (compute_bar_or(it >= total || *(volatile int *)&s.abort_flag)) {
      if (lane == 0) mbar_arrive(&s.item_empty[slot]);
      break;
    }
    const ItemInfo f = item_info(p, s, it);
    const size_t qrow = ((size_t)f.layer * p.B + f.b) * p.Hq + (size_t)f.h * G;
    if (f.full) {
      if (lane == 0) mbar_arrive(&s.item_empty[slot]);
      for (int e = tid; e < G * D; e += kWarps * 32)
        p.out[guard(qrow * D + e, 1, (long long)p.L * p.B * p.Hq * D, p.status)] = 0.f;
      continue;
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&s.item_empty[slot]);

    float2 acc[G][DL / 2];  // entry j: head j ^ hq, the lane's dims
#pragma unroll
    for (int g = 0; g < G; ++g)
#pragma unroll
      for (int e = 0; e < DL / 2; ++e) acc[g][e] = make_float2(0.f, 0.f);
    float m_run = -INFINITY, l_run = 0.f;  // of head hq over this row group's rows

    // One sub-chunk of this warp's rows; kMask: some rows are past nrows
    // (their index is clamped to a valid row and their probability is 0).
    auto rows_step = [&](const Tin *ks, const Tin *vs, int nrows, auto mask_tag) {
      constexpr bool kMask = decltype(mask_tag)::value;
      float2 d2[NIT][G];
#pragma unroll
      for (int t = 0; t < NIT; ++t)
#pragma unroll
        for (int g = 0; g < G; ++g) d2[t][g] = make_float2(0.f, 0.f);
#pragma unroll
      for (int k = 0; k < PPL; ++k) {
        float2 kp[NIT][PE / 2];
#pragma unroll
        for (int t = 0; t < NIT; ++t) {
          const int row = rw0 + t * R + rg;
          const int rr = kMask ? min(row, nrows - 1) : row;
          load_pairs<PE / 2>(ks + (size_t)rr * D + (sl + k * S) * PE, kp[t]);
        }
#pragma unroll
        for (int g = 0; g < G; ++g) {
          float2 qp[PE / 2];
#pragma unroll
          for (int h = 0; h < C::NH; ++h) {
            const float4 x =
                *reinterpret_cast<const float4 *>(&qf[(((g * PPL + k) * C::NH + h) * S + sl) * 4]);
            qp[2 * h] = make_float2(x.x, x.y);
            qp[2 * h + 1] = make_float2(x.z, x.w);
          }
#pragma unroll
          for (int t = 0; t < NIT; ++t)
#pragma unroll
            for (int e = 0; e < PE / 2; ++e) d2[t][g] = __ffma2_rn(qp[e], kp[t][e], d2[t][g]);
        }
      }
      float sc[NIT];
#pragma unroll
      for (int t = 0; t < NIT; ++t) {
        const int row = rw0 + t * R + rg;
        float v[G];
#pragma unroll
        for (int g = 0; g < G; ++g) v[g] = d2[t][g].x + d2[t][g].y;
        reduce_scatter<S, G>(v);
        sc[t] = (!kMask || row < nrows) ? v[0] : -INFINITY;
      }
      float mb = sc[0];
#pragma unroll
      for (int t = 1; t < NIT; ++t) mb = fmaxf(mb, sc[t]);
      const bool grow = mb > m_run + kRescaleLog2;  // true for the first rows (m_run = -inf)
      if (__any_sync(kFull, grow)) {
        const float mn = grow ? mb : m_run;
        const float a = grow ? fast_exp2(m_run - mn) : 1.f;
        l_run *= a;
        float ag[G];
        all_gather<S, G>(a, ag);
#pragma unroll
        for (int g = 0; g < G; ++g)
#pragma unroll
          for (int e = 0; e < DL / 2; ++e) acc[g][e] = __fmul2_rn(acc[g][e], make_float2(ag[g], ag[g]));
        m_run = mn;
      }
#pragma unroll
      for (int t = 0; t < NIT; ++t) {
        const int row = rw0 + t * R + rg;
        const int rr = kMask ? min(row, nrows - 1) : row;
        const float pt =
            (!kMask || sc[t] > -INFINITY) ? fast_exp2(sc[t] - m_run) : 0.f;  // m_run is finite
        l_run += pt;
        float pg[G];
        all_gather<S, G>(pt, pg);
#pragma unroll
        for (int k = 0; k < PPL; ++k) {
          float2 vp[PE / 2];
          load_pairs<PE / 2>(vs + (size_t)rr * D + (sl + k * S) * PE, vp);
#pragma unroll
          for (int g = 0; g < G; ++g)
#pragma unroll
            for (int e = 0; e < PE / 2; ++e)
              acc[g][k * PE / 2 + e] =
                  __ffma2_rn(make_float2(pg[g], pg[g]), vp[e], acc[g][k * PE / 2 + e]);
        }
      }
    };

    const int nsub = (f.rows + C::CR - 1) / C::CR;
    for (int sub = 0; sub < nsub; ++sub, ++j) {
      const int stage = j % C::STAGES;
      wait_bar(&s.full[stage], (j / C::STAGES) & 1, &s.abort_flag, p);
      __syncwarp();
      const int nrows = min(C::CR, f.rows - sub * C::CR);
      const Tin *ks = (const Tin *)s.kv[stage][0];
      const Tin *vs = (const Tin *)s.kv[stage][1];
      if (rw0 + C::RPW <= nrows)
        rows_step(ks, vs, nrows, std::false_type{});
      else if (rw0 < nrows)
        rows_step(ks, vs, nrows, std::true_type{});
      // The new token's rows, staged behind the cached rows, go to the cache.
      const int rs = f.r0 + sub * C::CR;
      if (warp == 0 && f.len >= rs && f.len < rs + C::CR) {
        const size_t dst =
            guard((long long)(f.b * p.Hkv + f.h) * p.cap[f.layer] + f.len, 1,
                  (long long)p.B * p.Hkv * p.cap[f.layer], p.status) *
            C::ROW_BYTES;
        for (int e = lane; e < 2 * C::NPIECE; e += 32) {
          const int kvsel = e >= C::NPIECE, pc = e % C::NPIECE;
          const uint4 val = reinterpret_cast<const uint4 *>(
              s.kv[stage][kvsel] + (size_t)(f.len - rs) * C::ROW_BYTES)[pc];
          reinterpret_cast<uint4 *>((uint8_t *)(kvsel ? p.vc[f.layer] : p.kc[f.layer]) + dst)[pc] =
              val;
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.empty[stage]);
    }

    // Item end. (1) Merge the warp's row groups (butterfly over lanes with
    // the same position in their row group, hence the same head).
#pragma unroll
    for (int o = S; o < 32; o <<= 1) {
      const float mo = __shfl_xor_sync(kFull, m_run, o);
      const float lo = __shfl_xor_sync(kFull, l_run, o);
      const float M = fmaxf(m_run, mo);
      const float as = m_run == -INFINITY ? 0.f : fast_exp2(m_run - M);
      const float ao = mo == -INFINITY ? 0.f : fast_exp2(mo - M);
      l_run = l_run * as + lo * ao;
      m_run = M;
      float gs[G], go[G];
      all_gather<S, G>(as, gs);
      all_gather<S, G>(ao, go);
#pragma unroll
      for (int g = 0; g < G; ++g)
#pragma unroll
        for (int e = 0; e < DL / 2; ++e) {
          float2 other;
          other.x = __shfl_xor_sync(kFull, acc[g][e].x, o);
          other.y = __shfl_xor_sync(kFull, acc[g][e].y, o);
          acc[g][e] = __ffma2_rn(acc[g][e], make_float2(gs[g], gs[g]),
                                 __fmul2_rn(other, make_float2(go[g], go[g])));
        }
    }
    // (2) Merge the 8 warps through shared memory.
    if (rg == 0) {
#pragma unroll
      for (int g = 0; g < G; ++g)
#pragma unroll
        for (int k = 0; k < PPL; ++k)
#pragma unroll
          for (int e = 0; e < PE / 2; ++e)
            *reinterpret_cast<float2 *>(
                &s.red_o[warp][(g ^ hq) * D + (sl + k * S) * PE + 2 * e]) = acc[g][k * PE / 2 + e];
      if (sl % C::HL == 0) {
        s.red_m[warp][hq] = m_run;
        s.red_l[warp][hq] = l_run;
      }
    }
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
        const float wgt = fast_exp2(s.red_m[w][g] - M);  // M is finite: row 0 is in warp 0
        num += wgt * s.red_o[w][e];
        den += wgt * s.red_l[w][g];
      }
      if (single) {
        p.out[guard(qrow * D + e, 1, (long long)p.L * p.B * p.Hq * D, p.status)] = num / den;
      } else {
        const long long wi = guard(item, 1, p.ws_items, p.status);
        p.ws_o[wi * G * D + e] = num;
        if (e % D == 0) p.ws_ml[wi * G + g] = make_float2(M, den);
      }
    }
    if (!single) {
      __threadfence();
      named_bar_sync(1, kWarps * 32);
      if (tid == 0) {
        if (!s.init_seen) s.init_seen = wait_init(p, &s.abort_flag);
        // without the counters (a wait gave up) no item combines the group
        s.last = s.init_seen && atomicAdd(&p.ctrl[guard(kCtrlGroup + f.group, 1, p.n_ctrl,
                                                        p.status)],
                                          1) == f.nch - 1;
      }
      named_bar_sync(1, kWarps * 32);
      if (s.last) {
        __threadfence();
        const long long ib = guard(item_base, f.nch, p.ws_items, p.status);
        for (int e = tid; e < G * D; e += kWarps * 32) {
          const int g = e / D;
          float M = -INFINITY;
          for (int c = 0; c < f.nch; ++c)
            M = fmaxf(M, __ldcg(&p.ws_ml[(size_t)(ib + c) * G + g]).x);
          float num = 0.f, den = 0.f;
          for (int c = 0; c < f.nch; ++c) {
            const float2 ml = __ldcg(&p.ws_ml[(size_t)(ib + c) * G + g]);
            const float wgt = fast_exp2(ml.x - M);
            den += wgt * ml.y;
            num += wgt * __ldcg(&p.ws_o[(size_t)(ib + c) * G * D + e]);
          }
          p.out[guard(qrow * D + e, 1, (long long)p.L * p.B * p.Hq * D, p.status)] = num / den;
        }
      }
    }
  }
}

// Before the previous step has completed: the first sub-chunks of this CTA's
// first item (item blockIdx.x) into L2, from the lengths as they read now
// (one less than this step's if the previous step has not yet advanced
// them; a prefetch is only a hint), so that this step's first loads do not
// start from DRAM after the previous step's tail.
template <typename Tin, int D, int G>
__device__ __forceinline__ void prefetch_first_item(const DecParams &p) {
  using C = DecCfg<Tin, D, G>;
  const int units = p.B * p.Hkv;
  int rest = (int)blockIdx.x;
  for (int t = 0; t < p.L; ++t) {
    const int l = p.order[t];
    const int len = *(volatile const int32_t *)&p.lens[l];
    const bool full = len < 0 || len >= p.cap[l];
    const int nch = full ? 1 : (len + p.item_rows) / p.item_rows;
    if (rest >= units * nch) {
      rest -= units * nch;
      continue;
    }
    if (full) return;
    const int unit = rest / nch, chunk = rest % nch;
    const int r0 = chunk * p.item_rows, r1 = min(len, r0 + p.item_rows);
    const int rows = min(r1 - r0, C::STAGES * C::CR);
    if (rows <= 0) return;
    const size_t off = guard((long long)unit * p.cap[l] + r0, rows, (long long)units * p.cap[l],
                             p.status) *
                       C::ROW_BYTES;
    bulk_prefetch_l2((const uint8_t *)p.kc[l] + off, (uint32_t)rows * C::ROW_BYTES);
    bulk_prefetch_l2((const uint8_t *)p.vc[l] + off, (uint32_t)rows * C::ROW_BYTES);
    return;
  }
}

template <typename Tin, int D, int G>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(const __grid_constant__ DecParams p) {
  using C = DecCfg<Tin, D, G>;
  extern __shared__ __align__(128) uint8_t smem_raw[];
  DecSmem<Tin, D, G> &s = *reinterpret_cast<DecSmem<Tin, D, G> *>(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int units = p.B * p.Hkv;

  // Launched as a programmatic dependent of the previous step: let the next
  // step's CTAs take SMs as this grid's CTAs leave, and wait here until the
  // previous grid has completed and its writes (lengths, appended rows,
  // counters) are visible.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  if (tid == 0) prefetch_first_item<Tin, D, G>(p);
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // Work list of this step from the current lengths (read once, before any
  // CTA can advance them: that happens after every CTA has exited).
  if (tid < p.L) {
    const int l = p.order[tid];
    const int len = p.lens[l];
    const bool full = len < 0 || len >= p.cap[l];
    s.len[tid] = full ? -1 : len;
    s.nch[tid] = full ? 1 : (len + p.item_rows) / p.item_rows;
    if (full && blockIdx.x == 0) report(p.status, RIPPLE_EFULL);
  }
  if (tid == 0) {
    for (int i = 0; i < C::STAGES; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], kWarps);
    }
    for (int i = 0; i < kItemSlots; ++i) {
      mbar_init(&s.item_full[i], 1);
      mbar_init(&s.item_empty[i], kWarps);
    }
    s.abort_flag = 0;
    s.init_seen = 0;
    fence_mbar_init();
  }
  // CTA 0 zeroes this call's counters (the workspace may hold anything),
  // then raises the init flag; the other CTAs use no counter before they see
  // it (wait_init).
  const int n_ctrl = (kCtrlGroup - kCtrlItem) + p.L * units;
  if (blockIdx.x == 0)
    for (int i = tid; i < n_ctrl; i += kThreads) p.ctrl[kCtrlItem + i] = 0;
  __syncthreads();
  if (blockIdx.x == 0 && tid == 0) {
    __threadfence();
    st_release(&p.ctrl[kCtrlFlag], p.epoch);
  }
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
    if (lane == 0) produce<Tin, D, G>(p, s, total);
  } else {
    consume<Tin, D, G>(p, s, total, warp, lane);
  }

  // The last CTA to leave advances the lengths of the layers it appended to
  // and lowers the init flag (a replay of this launch starts from CTA 0's
  // zeroing again). A CTA that never saw the flag (its wait gave up) leaves
  // the counters alone; the call has then reported RIPPLE_ETIMEOUT.
  __syncwarp();
  __syncthreads();
  if (tid == 0) {
    if (!s.init_seen) s.init_seen = wait_init(p, &s.abort_flag);
    __threadfence();
    if (s.init_seen && atomicAdd(&p.ctrl[kCtrlExit], 1) == (int)gridDim.x - 1) {
      for (int t = 0; t < p.L; ++t)
        if (s.len[t] >= 0) p.lens[p.order[t]] = s.len[t] + 1;
      __threadfence();
      st_release(&p.ctrl[kCtrlFlag], 0);
    }
  }
}

// ------------------------------------------------------------ host side

constexpr int kMaxDevices = 64;

// Per-device caches of the SM count and of the kernels' shared-memory
// attribute; atomics, as several host threads may make their first calls at
// once (a repeated look-up or attribute set is harmless).
int sm_count(int dev) {
  static std::atomic<int> n[kMaxDevices];
  if (dev < 0 || dev >= kMaxDevices) return 1;
  int v = n[dev].load(std::memory_order_relaxed);
  if (v == 0) {
    cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
    v = v > 0 ? v : 1;
    n[dev].store(v, std::memory_order_relaxed);
  }
  return v;
}

template <typename Tin, int D, int G>
cudaError_t launch_g(const DecParams &p, int dev, cudaStream_t st) {
  static std::atomic<bool> attr_set[kMaxDevices];
  const int smem = (int)sizeof(DecSmem<Tin, D, G>);
  static_assert(sizeof(DecSmem<Tin, D, G>) <= 227 * 1024, "shared memory per CTA");
  if (!attr_set[dev].load(std::memory_order_acquire)) {
    const cudaError_t e = cudaFuncSetAttribute(decode_kernel<Tin, D, G>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr_set[dev].store(true, std::memory_order_release);
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(sm_count(dev));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, decode_kernel<Tin, D, G>, p);
  count_launches(1);
  return e;
}

template <typename Tin, int D>
cudaError_t launch_d(const DecParams &p, int dev, cudaStream_t st) {
  switch (p.G) {
    case 1: return launch_g<Tin, D, 1>(p, dev, st);
    case 2: return launch_g<Tin, D, 2>(p, dev, st);
    case 4: return launch_g<Tin, D, 4>(p, dev, st);
    case 8: return launch_g<Tin, D, 8>(p, dev, st);
    default: return cudaErrorInvalidValue;
  }
}

// Epoch of a call: a per-process sequence (never 0) that starts at a value
// taken from the clock, so that an init flag left in reused memory by an
// earlier call or process is unlikely to match.
int next_epoch() {
  static std::atomic<uint32_t> seq{(uint32_t)std::chrono::steady_clock::now()
                                       .time_since_epoch()
                                       .count() *
                                   2654435761u};
  uint32_t e;
  do {
    e = seq.fetch_add(1, std::memory_order_relaxed) + 1;
  } while (e == 0);
  return (int)e;
}

// Cache rows per work item (the workspace holds one partial per item).
// Cache rows per work item for these capacities: kMaxItemRows when that
// already gives at least one item per SM; otherwise (a single layer's step,
// short caches) the smallest power of two down to kMinItemRows whose items
// still fit in one wave of one CTA per SM, so that no CTA takes two items one
// after the other. A step's lengths are at most its capacities, so the plan's
// item count bounds the kernel's.
int item_rows(const ripple_decode_desc *d, const int32_t *caps) {
  int dev = 0;
  cudaGetDevice(&dev);
  const long long sms = sm_count(dev);
  auto items = [&](int rows) {
    long long n = 0;
    for (int l = 0; l < d->n_layers; ++l)
      n += (long long)d->batch * d->n_kv_heads * ((caps[l] + rows - 1) / rows);
    return n;
  };
  int rows = kMaxItemRows;
  if (items(rows) >= sms) return rows;
  while (rows > kMinItemRows && items(rows / 2) <= sms) rows /= 2;
  return rows;
}

static size_t round_up(size_t x) { return (x + 255) & ~(size_t)255; }

// Workspace layout for these capacities: control block, partial (max, sum),
// partial outputs. Returns the total bytes; fills p's pointers if given.
size_t plan(const ripple_decode_desc *d, const int32_t *caps, void *ws, DecParams *p) {
  const int G = d->n_q_heads / d->n_kv_heads;
  const int rows = item_rows(d, caps);
  size_t items = 0;
  for (int l = 0; l < d->n_layers; ++l)
    items += (size_t)d->batch * d->n_kv_heads * ((caps[l] + rows - 1) / rows);
  const size_t groups = (size_t)d->n_layers * d->batch * d->n_kv_heads;
  const size_t ctrl = round_up(sizeof(int) * (kCtrlGroup + groups));
  const size_t ml = round_up(sizeof(float2) * items * G);
  const size_t o = round_up(sizeof(float) * items * G * d->head_dim);
  if (p != nullptr) {
    uint8_t *base = (uint8_t *)ws;
    p->item_rows = rows;
    p->ws_items = (long long)items;
    p->n_ctrl = (int)(kCtrlGroup + groups);
    p->ctrl = (int *)base;
    p->ws_ml = (float2 *)(base + ctrl);
    p->ws_o = (float *)(base + ctrl + ml);
  }
  return ctrl + ml + o;
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

ripple_status run(const ripple_decode_desc *desc, DecParams &p, void *stream) {
  p.epoch = next_epoch();
  p.wait_cycles = wait_limit_cycles();
  cudaStream_t st = (cudaStream_t)stream;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return RIPPLE_ECUDA;
  cudaError_t e;
  if (desc->dtype == RIPPLE_F32)
    e = desc->head_dim == 64 ? launch_d<float, 64>(p, dev, st) : launch_d<float, 128>(p, dev, st);
  else
    e = desc->head_dim == 64 ? launch_d<__nv_bfloat16, 64>(p, dev, st)
                             : launch_d<__nv_bfloat16, 128>(p, dev, st);
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
// keeps it until the process exits; all calls on a device share it. Every
// call zeroes the counters it uses before using them, and every partial a call
// reads it has written itself, so no state carries over from the previous call
// (not even from one that ended with RIPPLE_ETIMEOUT). Calls that overlap on
// the GPU race on it.

static __device__ __align__(256) float
    g_decode_scratch[RIPPLE_DECODE_NOALLOC_SCRATCH_BYTES / sizeof(float)];

namespace {

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
