// Finishing kernel of the split-K FFN down GEMM.  Launches with few output tiles
// (a decode step: 64 tokens give the router contraction 2 tiles and the FFN down
// GEMM 16) split K so that every SM streams weights; the k_splits fp32 partial
// slices are added in a fixed order, so results do not depend on scheduling (the
// router kernel adds the router contraction's slices the same way as it reads them).
#include "hero_device.cuh"

namespace hero {
namespace {

// Block-closing epilogue over the summed partials: one warp per (row, partial-sum
// slot of kTcPartCols columns); lane owns 4 consecutive columns and the slot's
// sums are reduced over the warp in a fixed order.
__global__ void __launch_bounds__(256) k_splitk_close(const float* __restrict__ part, int splits,
                                                      long split_stride, int ld, const int* m_dev,
                                                      int m_max, const LayerOutArgs lo) {
  pdl_enter();
  static_assert(kTcPartCols == 128, "one warp covers one 128-column slot with float4 lanes");
  int M = *m_dev;
  if (M < 0 || M > m_max) M = 0;
  const int slots = lo.d / kTcPartCols;
  const long w = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (w >= (long)M * slots) return;
  const int m = (int)(w / slots);
  const int slot = (int)(w - (long)m * slots);
  const int n = slot * kTcPartCols + 4 * lane;
  const size_t off = (size_t)m * ld + n;
  float4 y = *reinterpret_cast<const float4*>(part + off);
  for (int s = 1; s < splits; ++s) {
    const float4 v = *reinterpret_cast<const float4*>(part + (size_t)s * split_stride + off);
    y.x += v.x; y.y += v.y; y.z += v.z; y.w += v.w;
  }
  const int t = lo.idx[m];
  const float sc = lo.scale[m];
  const LayerOutIn in = layer_out_load(lo, t, n);
  float ss = 0.f, dd = 0.f, dp = 0.f;
  layer_out_store(lo, t, n, in, y, sc, ss, dd, dp);
  if (!lo.last) {
    ss = warp_sum(ss);
    dd = warp_sum(dd);
    dp = warp_sum(dp);
    if (lane == 0)
      *reinterpret_cast<float4*>(lo.part + ((size_t)t * lo.np + slot) * 4) =
          make_float4(ss, dd, dp, 0.f);
  }
}

}  // namespace

cudaError_t launch_splitk_close(const float* part, int splits, long split_stride, int ld,
                                const int* m_dev, int m_max, const LayerOutArgs& lo,
                                cudaStream_t st) {
  if (m_max <= 0) return cudaSuccess;
  if (lo.d % kTcPartCols) return cudaErrorInvalidValue;
  const long warps = (long)m_max * (lo.d / kTcPartCols);
  return launch_pdl(k_splitk_close, dim3((unsigned)((warps + 7) / 8)), dim3(256), 0, st, part, splits,
                    split_stride, ld, m_dev, m_max, lo);
}

}  // namespace hero
