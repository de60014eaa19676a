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
                                                      int m_max, const LayerOutArgs lo,
                                                      const SplitkAdapter ad) {
  pdl_enter();
  static_assert(kTcPartCols == 128, "one warp covers one 128-column slot with float4 lanes");
  int M = *m_dev;
  if (M < 0 || M > m_max) M = 0;
  const int slots = lo.d / kTcPartCols;
  const long w = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  const long rows = ad.ah ? m_max : M;
  if (w >= rows * slots) return;
  const int m = (int)(w / slots);
  const int slot = (int)(w - (long)m * slots);
  const int n = slot * kTcPartCols + 4 * lane;
  const bool ffn = m < M;
  const LayerOutArgs& p = ffn ? lo : ad.lo;
  const int row = ffn ? m : m - M;
  const int t = p.idx[row];
  const float sc = p.scale[row];
  const LayerOutIn in = layer_out_load(p, t, n);   // in flight with the loads below
  float4 y;
  if (ffn) {
    const size_t off = (size_t)(ad.by_token ? t : m) * ld + n;
    y = *reinterpret_cast<const float4*>(part + off);
    // up to 8 slices' loads in flight, added in slice order
    for (int s0 = 1; s0 < splits; s0 += 8) {
      float4 v[8];
#pragma unroll
      for (int i = 0; i < 8; ++i)
        v[i] = s0 + i < splits
                   ? *reinterpret_cast<const float4*>(part + (size_t)(s0 + i) * split_stride + off)
                   : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int i = 0; i < 8; ++i)
        if (s0 + i < splits) {
          y.x += v[i].x; y.y += v[i].y; y.z += v[i].z; y.w += v[i].w;
        }
    }
  } else {   // adapter row: y = W_2 ah[row] over the lane's 4 columns
    const uint16_t* ar = static_cast<const uint16_t*>(ad.ah) + (size_t)(ad.by_token ? t : row) * ad.d_r;
    const uint16_t* wr = static_cast<const uint16_t*>(ad.w2) + (size_t)n * ad.d_r;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
    for (int k = 0; k < ad.d_r; k += 8) {
      const uint4 xa = __ldg(reinterpret_cast<const uint4*>(ar + k));
      const uint32_t xs[4] = {xa.x, xa.y, xa.z, xa.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint4 wv = __ldg(reinterpret_cast<const uint4*>(wr + (size_t)i * ad.d_r + k));
        const uint32_t ws[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          acc[i] = fmaf(__uint_as_float(xs[e] << 16), __uint_as_float(ws[e] << 16), acc[i]);
          acc[i] = fmaf(__uint_as_float(xs[e] & 0xffff0000u), __uint_as_float(ws[e] & 0xffff0000u),
                        acc[i]);
        }
      }
    }
    y = make_float4(acc[0], acc[1], acc[2], acc[3]);
  }
  float ss = 0.f, dd = 0.f, dp = 0.f;
  layer_out_store(p, t, n, in, y, sc, ss, dd, dp);
  if (!p.last) {
    ss = warp_sum(ss);
    dd = warp_sum(dd);
    dp = warp_sum(dp);
    if (lane == 0)
      *reinterpret_cast<float4*>(p.part + ((size_t)t * p.np + slot) * 4) =
          make_float4(ss, dd, dp, 0.f);
  }
}

// Decoding step, split-K q/k/v projection: one warp per (token, head); lane owns
// columns lane + 32 k (k = 0..3), i.e. RoPE pairs (lane, lane + 64) and
// (lane + 32, lane + 96).  The slices are added in order, q and k heads rotated at
// the token's position, and bf16 values stored as the fused epilogue stores them.
__global__ void __launch_bounds__(256) k_qkv_close(const float* __restrict__ part, int splits,
                                                   long split_stride, int B, const RopeArgs r,
                                                   uint32_t* err) {
  pdl_enter();
  const int heads = r.H + 2 * r.Hkv, N = heads * 128;
  const long w = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (w >= (long)B * heads) return;
  const int m = (int)(w / heads), head = (int)(w - (long)m * heads);
  const int s = r.pos[m];
  if (s < 0 || s >= r.S_kv) {
    if (head == 0 && lane == 0) atomicOr(err, ERR_BAD_INDEX);
    return;
  }
  float x[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const size_t off = (size_t)m * N + head * 128 + lane + 32 * k;
    float a = part[off];
    for (int sp = 1; sp < splits; ++sp) a += part[(size_t)sp * split_stride + off];
    x[k] = a;
  }
  uint16_t* dst;
  if (head < r.H)
    dst = static_cast<uint16_t*>(r.q) + ((size_t)m * r.H + head) * r.S_q * 128;
  else if (head < r.H + r.Hkv)
    dst = static_cast<uint16_t*>(r.k) + (((size_t)m * r.Hkv + head - r.H) * r.S_kv + s) * 128;
  else
    dst = static_cast<uint16_t*>(r.v) + (((size_t)m * r.Hkv + head - r.H - r.Hkv) * r.S_kv + s) * 128;
  if (head < r.H + r.Hkv) {
#pragma unroll
    for (int k = 0; k < 2; ++k) {   // pair (i, i + 64), i = lane + 32 k
      const int i = lane + 32 * k;
      const float cs = r.cs[((size_t)s * 64 + i) * 2], sn = r.cs[((size_t)s * 64 + i) * 2 + 1];
      const float a = x[k], b = x[k + 2];
      x[k] = a * cs - b * sn;
      x[k + 2] = b * cs + a * sn;
    }
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) dst[lane + 32 * k] = (uint16_t)(pack_bf16x2(x[k], 0.f) & 0xffffu);
}

// Split-K output projection closing into the block entry (the EPI_ATTN_ENTRY
// arithmetic): one warp per (token, 128-column slot), lane owns 4 columns.
__global__ void __launch_bounds__(256) k_entry_close(const float* __restrict__ part, int splits,
                                                     long split_stride, int B,
                                                     const float* __restrict__ resid,
                                                     const LayerOutArgs p) {
  pdl_enter();
  const int slots = p.d / kTcPartCols;
  const long w = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (w >= (long)B * slots) return;
  const int t = (int)(w / slots), slot = (int)(w - (long)t * slots);
  const int n = slot * kTcPartCols + 4 * lane;
  const size_t off = (size_t)t * p.d + n;
  float4 y = *reinterpret_cast<const float4*>(part + off);
  for (int sp = 1; sp < splits; ++sp) {
    const float4 v = *reinterpret_cast<const float4*>(part + (size_t)sp * split_stride + off);
    y.x += v.x; y.y += v.y; y.z += v.z; y.w += v.w;
  }
  const float4 hr = *reinterpret_cast<const float4*>(resid + off);
  const float4 hn = make_float4(hr.x + y.x, hr.y + y.y, hr.z + y.z, hr.w + y.w);
  float ss = hn.x * hn.x + hn.y * hn.y + hn.z * hn.z + hn.w * hn.w, dd = 0.f, dp = 0.f;
  if (p.router) {
    float4 dl = make_float4(0.f, 0.f, 0.f, 0.f);
    if (!p.first) {
      const float4 hp = *reinterpret_cast<const float4*>(p.hbar + off);
      const float4 dv = *reinterpret_cast<const float4*>(p.delta + off);
      dl = make_float4(hn.x - hp.x, hn.y - hp.y, hn.z - hp.z, hn.w - hp.w);
      dp = dl.x * dv.x + dl.y * dv.y + dl.z * dv.z + dl.w * dv.w;
    }
    dd = dl.x * dl.x + dl.y * dl.y + dl.z * dl.z + dl.w * dl.w;
    *reinterpret_cast<float4*>(p.delta + off) = dl;
    store_xl4(p.xl, p.xl_bf16, p.d, t, n, hn);
  }
  *reinterpret_cast<float4*>(p.hbar + off) = hn;
  ss = warp_sum(ss);
  dd = warp_sum(dd);
  dp = warp_sum(dp);
  if (lane == 0)
    *reinterpret_cast<float4*>(p.part + ((size_t)t * p.np + slot) * 4) = make_float4(ss, dd, dp, 0.f);
}

}  // namespace

cudaError_t launch_qkv_close(const float* part, int splits, long split_stride, int B,
                             const RopeArgs& r, uint32_t* err, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  if (!r.pos) return cudaErrorInvalidValue;   // decoding steps only
  const long warps = (long)B * (r.H + 2 * r.Hkv);
  return launch_pdl(k_qkv_close, dim3((unsigned)((warps + 7) / 8)), dim3(256), 0, st, part, splits,
                    split_stride, B, r, err);
}

cudaError_t launch_entry_close(const float* part, int splits, long split_stride, int B,
                               const float* resid, const LayerOutArgs& lo, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  if (lo.d % kTcPartCols) return cudaErrorInvalidValue;
  const long warps = (long)B * (lo.d / kTcPartCols);
  return launch_pdl(k_entry_close, dim3((unsigned)((warps + 7) / 8)), dim3(256), 0, st, part, splits,
                    split_stride, B, resid, lo);
}

cudaError_t launch_splitk_close(const float* part, int splits, long split_stride, int ld,
                                const int* m_dev, int m_max, const LayerOutArgs& lo,
                                const SplitkAdapter& ad, cudaStream_t st) {
  if (m_max <= 0) return cudaSuccess;
  if (lo.d % kTcPartCols) return cudaErrorInvalidValue;
  if (ad.ah && (ad.d_r <= 0 || ad.d_r % 8 || !ad.w2 || ad.lo.d != lo.d)) return cudaErrorInvalidValue;
  if (ad.by_token && !ad.ah) return cudaErrorInvalidValue;
  const long warps = (long)m_max * (lo.d / kTcPartCols);
  return launch_pdl(k_splitk_close, dim3((unsigned)((warps + 7) / 8)), dim3(256), 0, st, part, splits,
                    split_stride, ld, m_dev, m_max, lo, ad);
}

}  // namespace hero
