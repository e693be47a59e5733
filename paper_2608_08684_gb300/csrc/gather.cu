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

__global__ void __launch_bounds__(kThreads) gather_kernel(const uint8_t *k, const uint8_t *v,
                                                          const int32_t *idx, int T, int n_keep,
                                                          int row_bytes, uint8_t *k_out,
                                                          uint8_t *v_out, int cap,
                                                          int32_t *status) {
  extern __shared__ __align__(128) uint8_t tile[];
  __shared__ __align__(8) uint64_t bar;
  const int unit = blockIdx.y;
  const int j0 = blockIdx.x * kTileRows;
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
  const bool ok = mbar_wait(&bar, 0, status);
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

cudaError_t launch_gather(const LayerGeom &g, const void *k, const void *v, const int32_t *idx,
                          int n_keep, void *k_out, void *v_out, int cap, int32_t *status,
                          cudaStream_t st) {
  const int row_bytes = g.D * (g.dtype == RIPPLE_F32 ? 4 : 2);
  const size_t smem = (size_t)2 * kTileRows * row_bytes;
  cudaError_t e = cudaFuncSetAttribute(gather_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  const dim3 grid((n_keep + kTileRows - 1) / kTileRows, g.units);
  gather_kernel<<<grid, kThreads, smem, st>>>((const uint8_t *)k, (const uint8_t *)v, idx, g.T,
                                              n_keep, row_bytes, (uint8_t *)k_out,
                                              (uint8_t *)v_out, cap, status);
  count_launches(1);
  return cudaGetLastError();
}

}  // namespace ripple
