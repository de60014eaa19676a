// Adapter up-projection fused with the block-closing epilogue (Eqs. 2-3 for the
// tokens routed to the adapter):
//   y = W_2 SiLU(W_1 u)   (the SiLU(W_1 u) rows come from the adapter-down GEMM)
//   h = h_bar + (1 - g) y, then the next block's h_bar, delta and partial sums.
// Used by f32 models, and by bf16 models when the token count is small (decode),
// where the tensor-core launch's fixed latency dominates; large bf16 batches run
// the up projection as a tensor-core GEMM.  The contraction has depth d_r (<= 64),
// i.e. 2 d_r FLOP per output element against 22 bytes of epilogue traffic, so it
// runs on the FMA pipes with row-contiguous global access.
//
// CTA: 8 RPW adapter rows x 256 output columns, 256 threads.  Warp w owns rows
// RPW w .. RPW w + RPW - 1; lane x owns columns x + 32 j (j < 8), so every warp
// instruction of the epilogue touches 128 contiguous bytes of one row.  RPW = 4 for
// large batches; 1 when the row count is small (decode), so the few rows spread over
// four times the CTAs.  The rows the epilogue
// will update are bulk-prefetched into L2 at kernel start.
#include "hero_device.cuh"

namespace hero {
namespace {

constexpr int AU_COLS = 256;
constexpr int AU_DR = 64;          // largest supported rank
constexpr int AU_WLD = AU_DR + 2;  // row stride of the staged W_2 slice (conflict-free reads)

template <int RPW, typename WT>
constexpr size_t au_smem() {
  return sizeof(float) * 8 * RPW * AU_DR + sizeof(WT) * AU_COLS * AU_WLD;
}

__device__ __forceinline__ float to_f32(uint16_t b) { return __uint_as_float((uint32_t)b << 16); }
__device__ __forceinline__ float to_f32(float v) { return v; }

// WT: operand element type, uint16_t (bf16 bits) or float.  SLOT: columns per
// partial-sum slot of the model (64 or 256).
template <int SLOT, int RPW, typename WT>
__global__ void __launch_bounds__(256) k_adapter_up(const AdapterUpArgs a) {
  constexpr int AU_ROWS = 8 * RPW;
  pdl_enter();
  extern __shared__ __align__(16) float smem_au[];
  float* ahs = smem_au;                                         // [AU_ROWS][AU_DR] fp32
  WT* w2s = reinterpret_cast<WT*>(smem_au + AU_ROWS * AU_DR);   // [AU_COLS][AU_WLD]
  int M = *a.m_dev;
  if (M < 0 || M > a.m_max) M = 0;
  const int m0 = blockIdx.y * AU_ROWS;
  if (m0 >= M) return;
  const int n0 = blockIdx.x * AU_COLS;
  const int dr = a.d_r;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const LayerOutArgs& p = a.lo;
  const WT* ah = static_cast<const WT*>(a.ah);
  const WT* w2 = static_cast<const WT*>(a.w2);

  // Start pulling the epilogue's rows (h_bar, delta, P_{j+1} over this CTA's
  // columns) into L2 while the contraction runs.
  if (tid < AU_ROWS && m0 + tid < M) {
    const int t = p.idx[m0 + tid];
    const int cols = min(AU_COLS, a.d - n0);
    const size_t off = (size_t)t * p.d + n0;
    prefetch_l2(p.hbar + off, cols * 4);
    if (!p.last) {
      if (p.router && !p.first) prefetch_l2(p.delta + off, cols * 4);
      const int pes = p.p_bf16 ? 2 : 4;
      if (p.p_next) prefetch_l2(static_cast<const char*>(p.p_next) + off * pes, cols * pes);
    }
  }

  constexpr int V = 16 / (int)sizeof(WT);   // elements per 16-byte vector
  if (dr % V == 0) {   // 16-byte loads, several per thread in flight
    const int vr = dr / V;
#pragma unroll 4
    for (int e = tid; e < AU_ROWS * vr; e += 256) {
      const int r = e / vr, kv = (e - r * vr) * V;
      const int m = m0 + r;
      uint4 u = make_uint4(0u, 0u, 0u, 0u);
      if (m < M) u = __ldg(reinterpret_cast<const uint4*>(ah + (size_t)m * dr + kv));
      const WT* x = reinterpret_cast<const WT*>(&u);
#pragma unroll
      for (int i = 0; i < V; ++i) ahs[r * AU_DR + kv + i] = to_f32(x[i]);
    }
#pragma unroll 4
    for (int e = tid; e < AU_COLS * vr; e += 256) {
      const int c = e / vr, kv = (e - c * vr) * V;
      const int n = n0 + c;
      uint4 u = make_uint4(0u, 0u, 0u, 0u);
      if (n < a.d) u = __ldg(reinterpret_cast<const uint4*>(w2 + (size_t)n * dr + kv));
      const WT* x = reinterpret_cast<const WT*>(&u);
#pragma unroll
      for (int i = 0; i < V; ++i) w2s[c * AU_WLD + kv + i] = x[i];
    }
  } else {
    for (int e = tid; e < AU_ROWS * dr; e += 256) {
      const int r = e / dr, k = e % dr;
      const int m = m0 + r;
      ahs[r * AU_DR + k] = m < M ? to_f32(ah[(size_t)m * dr + k]) : 0.f;
    }
    for (int e = tid; e < AU_COLS * dr; e += 256) {
      const int c = e / dr, k = e % dr;
      const int n = n0 + c;
      w2s[c * AU_WLD + k] = n < a.d ? w2[(size_t)n * dr + k] : WT(0);
    }
  }
  __syncthreads();

  float acc[RPW][8];
#pragma unroll
  for (int i = 0; i < RPW; ++i)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[i][j] = 0.f;
  const float* arow = ahs + (warp * RPW) * AU_DR;
  for (int k = 0; k < dr; ++k) {
    float x[RPW], w[8];
#pragma unroll
    for (int i = 0; i < RPW; ++i) x[i] = arow[i * AU_DR + k];
#pragma unroll
    for (int j = 0; j < 8; ++j) w[j] = to_f32(w2s[(lane + 32 * j) * AU_WLD + k]);
#pragma unroll
    for (int i = 0; i < RPW; ++i)
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[i][j] = fmaf(x[i], w[j], acc[i][j]);
  }

  constexpr int spt = AU_COLS / SLOT;   // partial slots per tile
#pragma unroll 1
  for (int i = 0; i < RPW; ++i) {
    const int m = m0 + warp * RPW + i;
    if (m >= M) break;                     // warp-uniform
    const int t = p.idx[m];
    const float s = p.scale[m];
    LayerOutIn1 in[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int n = n0 + lane + 32 * j;
      if (n < a.d) in[j] = layer_out_load1(p, t, n);
    }
    float ss[4] = {0.f, 0.f, 0.f, 0.f}, dd[4] = {0.f, 0.f, 0.f, 0.f}, dp[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int n = n0 + lane + 32 * j;
      const int sl = (32 * j) / SLOT;
      if (n < a.d) layer_out_store1(p, t, n, in[j], acc[i][j], s, ss[sl], dd[sl], dp[sl]);
    }
    if (!p.last) {
#pragma unroll
      for (int sl = 0; sl < spt; ++sl) {
        const float v0 = warp_sum(ss[sl]), v1 = warp_sum(dd[sl]), v2 = warp_sum(dp[sl]);
        const int slot = n0 / SLOT + sl;
        if (lane == 0 && slot * SLOT < a.d)
          *reinterpret_cast<float4*>(p.part + ((size_t)t * p.np + slot) * 4) =
              make_float4(v0, v1, v2, 0.f);
      }
    }
  }
}

template <int SLOT, int RPW, typename WT>
cudaError_t launch_au(const AdapterUpArgs& a, cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_adapter_up<SLOT, RPW, WT>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)au_smem<RPW, WT>());
    if (e != cudaSuccess) return e;
    attr = true;
  }
  dim3 grid((a.d + AU_COLS - 1) / AU_COLS, (a.m_max + 8 * RPW - 1) / (8 * RPW));
  return launch_pdl(k_adapter_up<SLOT, RPW, WT>, grid, dim3(256), au_smem<RPW, WT>(), st, a);
}

}  // namespace

cudaError_t launch_adapter_up(const AdapterUpArgs& a, cudaStream_t st) {
  if (a.m_max <= 0) return cudaSuccess;
  if (a.d_r > AU_DR) return cudaErrorInvalidValue;
  const bool few = a.m_max <= 256;
  if (a.bf16 && a.slot_cols == 128)
    return few ? launch_au<128, 1, uint16_t>(a, st) : launch_au<128, 4, uint16_t>(a, st);
  if (!a.bf16 && a.slot_cols == 64)
    return few ? launch_au<64, 1, float>(a, st) : launch_au<64, 4, float>(a, st);
  return cudaErrorInvalidValue;
}

}  // namespace hero
