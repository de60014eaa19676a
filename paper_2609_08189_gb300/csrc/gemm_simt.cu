// fp32 SIMT GEMM with the routed stack's epilogues, for f32 models (whose parity
// bound rules out reduced-precision tensor-core operands).
//
//   C[M, N] = A[M, K] * B[N, K]^T   (A, B row-major fp32; M may be device-resident)
//
// 64 x 64 output tile per 256-thread block, 4 x 4 outputs per thread, K in steps
// of 16 staged through shared memory.  EPI_SWIGLU computes the gate (B) and up (B2)
// products of the same tile at once.
#include "hero_device.cuh"

namespace hero {
namespace {

constexpr int TM = 64, TN = kSimtTileN, TK = 16;

template <int EPI>
__global__ void __launch_bounds__(256) k_gemm_simt(const GemmArgs a) {
  pdl_enter();
  constexpr bool DUAL = EPI == EPI_SWIGLU;
  __shared__ float As[TK][TM + 4];
  __shared__ float Bs[TK][TN + 4];
  __shared__ float B2s[DUAL ? TK : 1][TN + 4];
  __shared__ float red[TM][16][3];

  int M = a.m_dev ? *a.m_dev : a.m_static;
  if (M < 0 || M > a.m_max) M = 0;
  const int m0 = blockIdx.y * TM;
  const int n0 = blockIdx.x * TN;
  if (m0 >= M) return;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const float* A = static_cast<const float*>(a.A);
  const float* B = static_cast<const float*>(a.B);
  const float* B2 = static_cast<const float*>(a.B2);

  float acc[4][4] = {};
  float acc2[DUAL ? 4 : 1][4] = {};
  for (int k0 = 0; k0 < a.K; k0 += TK) {
    for (int i = threadIdx.x; i < TM * TK; i += 256) {
      const int r = i / TK, k = i % TK;
      const int gm = m0 + r, gk = k0 + k;
      As[k][r] = (gm < M && gk < a.K) ? A[(size_t)gm * a.lda + gk] : 0.f;
      const int gn = n0 + r;
      Bs[k][r] = (gn < a.N && gk < a.K) ? B[(size_t)gn * a.ldb + gk] : 0.f;
      if constexpr (DUAL) B2s[k][r] = (gn < a.N && gk < a.K) ? B2[(size_t)gn * a.ldb + gk] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < TK; ++k) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) av[i] = As[k][ty * 4 + i];
#pragma unroll
      for (int i = 0; i < 4; ++i) bv[i] = Bs[k][tx * 4 + i];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) acc[i][jj] = fmaf(av[i], bv[jj], acc[i][jj]);
      if constexpr (DUAL) {
#pragma unroll
        for (int i = 0; i < 4; ++i) bv[i] = B2s[k][tx * 4 + i];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int jj = 0; jj < 4; ++jj) acc2[i][jj] = fmaf(av[i], bv[jj], acc2[i][jj]);
      }
    }
    __syncthreads();
  }

  const int nc = n0 + tx * 4;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int rl = ty * 4 + i;
    const int m = m0 + rl;
    const bool valid = m < M;
    if constexpr (EPI == EPI_STORE_F32) {
      if (valid)
        for (int jj = 0; jj < 4; ++jj)
          if (nc + jj < a.N) a.out_f32[(size_t)m * a.ldo + nc + jj] = acc[i][jj];
    } else if constexpr (EPI == EPI_SWIGLU) {
      if (valid)
        for (int jj = 0; jj < 4; ++jj)
          if (nc + jj < a.N)
            static_cast<float*>(a.out)[(size_t)m * a.ldo + nc + jj] =
                siluf_(acc[i][jj]) * acc2[i][jj];
    } else if constexpr (EPI == EPI_SILU) {
      if (valid)
        for (int jj = 0; jj < 4; ++jj)
          if (nc + jj < a.N) static_cast<float*>(a.out)[(size_t)m * a.ldo + nc + jj] = siluf_(acc[i][jj]);
    } else {
      float ss = 0.f, dd = 0.f, dp = 0.f;
      if (valid && nc < a.N) {
        const int t = a.lo.idx[m];
        const float s = a.lo.scale[m];
        layer_out4(a.lo, t, nc, make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]), s, ss,
                   dd, dp);
      }
      red[rl][tx][0] = ss;
      red[rl][tx][1] = dd;
      red[rl][tx][2] = dp;
    }
  }
  if constexpr (EPI == EPI_LAYER_OUT) {
    __syncthreads();
    if (threadIdx.x < TM && !a.lo.last) {
      const int m = m0 + threadIdx.x;
      if (m < M) {
        float s0 = 0.f, s1 = 0.f, s2 = 0.f;
        for (int x = 0; x < 16; ++x) {
          s0 += red[threadIdx.x][x][0];
          s1 += red[threadIdx.x][x][1];
          s2 += red[threadIdx.x][x][2];
        }
        const int t = a.lo.idx[m];
        *reinterpret_cast<float4*>(a.lo.part + ((size_t)t * a.lo.np + blockIdx.x) * 4) =
            make_float4(s0, s1, s2, 0.f);
      }
    }
  }
}

}  // namespace

cudaError_t launch_gemm_simt(EpiKind epi, const GemmArgs& a, cudaStream_t st) {
  if (a.m_max <= 0) return cudaSuccess;
  dim3 grid((a.N + TN - 1) / TN, (a.m_max + TM - 1) / TM);
  cudaError_t e = cudaErrorInvalidValue;
  switch (epi) {
    case EPI_STORE_F32: e = launch_pdl(k_gemm_simt<EPI_STORE_F32>, grid, dim3(256), 0, st, a); break;
    case EPI_SWIGLU: e = launch_pdl(k_gemm_simt<EPI_SWIGLU>, grid, dim3(256), 0, st, a); break;
    case EPI_SILU: e = launch_pdl(k_gemm_simt<EPI_SILU>, grid, dim3(256), 0, st, a); break;
    case EPI_LAYER_OUT: e = launch_pdl(k_gemm_simt<EPI_LAYER_OUT>, grid, dim3(256), 0, st, a); break;
    default: break;
  }
  return e;
}

}  // namespace hero
