// Gather of the kept K/V rows into the compact per-layer cache (Eq. 4: the
// compressed cache holds exactly the (k, v) of the retained positions, which
// compression never alters).
//
// Staged through shared memory with the bulk-async (TMA) engine: each CTA
// takes a tile of up to kTileRows output rows of one unit; one lane per row
// issues a cp.async.bulk global->shared copy of that K row and V row, all
// completing on one mbarrier; one thread then writes the two contiguous
// output tiles back with cp.async.bulk shared->global.
#include "common.cuh"
#include "kernels.cuh"

namespace ripple {
namespace {

constexpr int kTileRows = 64;
constexpr int kThreads = 64;

// Layers of one launch: units per layer, and per layer the input caches
// [upl][T][d], the kept indices [upl][n_keep], the outputs [upl][cap][d].
struct GatherTable {
  int upl;
  const uint8_t *k[kCompressMaxLayers];
  const uint8_t *v[kCompressMaxLayers];
  const int32_t *idx[kCompressMaxLayers];
  uint8_t *k_out[kCompressMaxLayers];
  uint8_t *v_out[kCompressMaxLayers];
  int n_keep[kCompressMaxLayers];
  int cap[kCompressMaxLayers];
};

__global__ void __launch_bounds__(kThreads) gather_kernel(const __grid_constant__ GatherTable tab,
                                                          int T, int row_bytes,
                                                          int32_t *status,
                                                          long long wait_cycles) {
  extern __shared__ __align__(128) uint8_t tile[];
  __shared__ __align__(8) uint64_t bar;
  const int layer = blockIdx.y / tab.upl, unit = blockIdx.y % tab.upl;
  const int n_keep = tab.n_keep[layer], cap = tab.cap[layer];
  const uint8_t *k = tab.k[layer], *v = tab.v[layer];
  uint8_t *k_out = tab.k_out[layer], *v_out = tab.v_out[layer];
  const int32_t *idx = tab.idx[layer];
  const int j0 = blockIdx.x * kTileRows;
  if (j0 >= n_keep) return;  // this layer keeps fewer rows than the longest one
  const int rows = min(kTileRows, n_keep - j0);
  uint8_t *tk = tile;
  uint8_t *tv = tile + (size_t)kTileRows * row_bytes;
  const int32_t *uidx = idx + (size_t)unit * n_keep;
  __shared__ int bad;
  if (threadIdx.x == 0) {
    bad = 0;
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_arrive_expect_tx(&bar, (uint32_t)(2 * rows * row_bytes));
  __syncthreads();
  const size_t unit_in = (size_t)unit * T;
  for (int r = threadIdx.x; r < rows; r += kThreads) {
    int t = uidx[j0 + r];
    if (t < 0 || t >= T) {  // never produced by the selection; keeps the copy in bounds
      bad = 1;
      t = 0;
    }
    bulk_g2s(tk + (size_t)r * row_bytes, k + (unit_in + t) * row_bytes, row_bytes, &bar);
    bulk_g2s(tv + (size_t)r * row_bytes, v + (unit_in + t) * row_bytes, row_bytes, &bar);
  }
  const bool ok = mbar_wait(&bar, 0, status, wait_cycles);
  // After a wait that gave up, hold the block until its copies have landed
  // (fixed bound), so that none writes into shared memory after it has left.
  if (!ok) mbar_wait(&bar, 0, nullptr);
  __syncthreads();
  if (bad) report(status, RIPPLE_EBOUNDS);
  if (threadIdx.x == 0 && ok) {
    const size_t dst = ((size_t)unit * cap + j0) * row_bytes;
    bulk_s2g(k_out + dst, tk, (uint32_t)(rows * row_bytes));
    bulk_s2g(v_out + dst, tv, (uint32_t)(rows * row_bytes));
    bulk_commit();
    bulk_wait_all();
  }
}

}  // namespace

cudaError_t launch_gather(const LayerGeom &g, int n_layers, const void *const *k,
                          const void *const *v, const int32_t *const *idx, const int *n_keep,
                          void *const *k_out, void *const *v_out, const int *cap,
                          int32_t *status, cudaStream_t st) {
  if (n_layers < 1 || n_layers > kCompressMaxLayers ||
      (long long)g.units * n_layers > 65535)
    return cudaErrorInvalidValue;
  GatherTable tab;
  tab.upl = g.units;
  int max_keep = 0;
  for (int l = 0; l < n_layers; ++l) {
    tab.k[l] = (const uint8_t *)k[l];
    tab.v[l] = (const uint8_t *)v[l];
    tab.idx[l] = idx[l];
    tab.k_out[l] = (uint8_t *)k_out[l];
    tab.v_out[l] = (uint8_t *)v_out[l];
    tab.n_keep[l] = n_keep[l];
    tab.cap[l] = cap[l];
    max_keep = n_keep[l] > max_keep ? n_keep[l] : max_keep;
  }
  if (max_keep == 0) return cudaSuccess;
  const int row_bytes = g.D * (g.dtype == RIPPLE_F32 ? 4 : 2);
  const size_t smem = (size_t)2 * kTileRows * row_bytes;
  cudaError_t e = cudaFuncSetAttribute(gather_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  const dim3 grid((max_keep + kTileRows - 1) / kTileRows, g.units * n_layers);
  gather_kernel<<<grid, kThreads, smem, st>>>(tab, g.T, row_bytes, status, wait_limit_cycles());
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace ripple
