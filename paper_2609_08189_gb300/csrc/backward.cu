// Training path of a routed block (Sec. 3.1, Sec. 3.3): the backward of its branch
// part with the decisions fixed, and the gradient of the skip penalty L_skip.
//
// A routed block computes h = h_bar + s Branch(u), u = LN_ffn(h_bar), with s = g and
// Branch = the frozen SwiGLU FFN for the tokens with g >= tau, s = 1 - g and Branch =
// the adapter W_2 SiLU(W_1 u) for the rest (Eqs. 2-3).  The threshold is not
// differentiated; the scale carries the gradient to the router.  Given G = dL/dh:
//   FFN rows      e = G W_down, dL/dg = <e, act>, dact = g e,
//                 dgate = dact up SiLU'(gate), dup = dact SiLU(gate),
//                 du = dgate W_gate + dup W_up
//   adapter rows  ga = G W_2, hid = SiLU(a), a = W_1 u, dL/dg = -<ga, hid>,
//                 da = (1 - g) ga SiLU'(a), du = da W_1,
//                 dL/dW_2 += (1 - g) G hid^T, dL/dW_1 += da u^T
//   every row     dL/dh_bar = G + RMSNorm backward of du (the residual plus the branch)
// The GEMMs run on the tensor-core kernel (gemm_tc.cu) against transposed copies of
// the frozen weights; the kernels here do the row-wise and reduction steps.
#include "hero_device.cuh"

namespace hero {
namespace {

constexpr int kRowWarps = 8;   // rows (one warp each) per 256-thread CTA

// Compacted row m of the block -> (token, branch): FFN rows are 0 .. n_f - 1, then the
// adapter rows; false past the last adapter row.
__device__ __forceinline__ bool row_of(int m, const int* counts, const int* idx_f,
                                       const int* idx_a, int& t, bool& ffn, int& mr) {
  const int nf = counts[0], na = counts[1];
  if (m < nf) {
    t = idx_f[m];
    ffn = true;
    mr = m;
    return true;
  }
  mr = m - nf;
  if (mr >= na) return false;
  t = idx_a[mr];
  ffn = false;
  return true;
}

// u = bf16(LN_ffn(h_bar)) and bf16(G) into the branch's compacted rows; 1/rms per token.
__global__ void __launch_bounds__(256) k_bw_prep(const BwPrepArgs a) {
  pdl_enter();
  const int m = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (m >= a.T) return;
  int t, mr;
  bool ffn;
  if (!row_of(m, a.counts, a.idx_f, a.idx_a, t, ffn, mr)) return;
  const float* h = a.hbar + (size_t)t * a.d;
  const float* G = a.G + (size_t)t * a.d;
  float ss = 0.f;
  for (int c = 4 * lane; c < a.d; c += 128) {
    const float4 v = *reinterpret_cast<const float4*>(h + c);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = warp_sum(ss);
  const float rinv = 1.0f / sqrtf(ss / (float)a.d + a.rms_eps);
  if (lane == 0) a.rinv[t] = rinv;
  uint16_t* u = (ffn ? a.u_f : a.u_a) + (size_t)mr * a.d;
  uint16_t* g = (ffn ? a.g_f : a.g_a) + (size_t)mr * a.d;
  for (int c = 4 * lane; c < a.d; c += 128) {
    const float4 v = *reinterpret_cast<const float4*>(h + c);
    const float4 w = *reinterpret_cast<const float4*>(a.gain + c);
    const float4 q = *reinterpret_cast<const float4*>(G + c);
    *reinterpret_cast<uint2*>(u + c) =
        make_uint2(pack_bf16x2(v.x * rinv * w.x, v.y * rinv * w.y),
                   pack_bf16x2(v.z * rinv * w.z, v.w * rinv * w.w));
    *reinterpret_cast<uint2*>(g + c) = make_uint2(pack_bf16x2(q.x, q.y), pack_bf16x2(q.z, q.w));
  }
}

// Per compacted row: dL/dg of FFN rows (the per-tile sums of the SwiGLU-backward
// epilogue added in tile order) and the adapter rows' hidden-layer backward.
__global__ void __launch_bounds__(256) k_bw_rows(const BwRowsArgs a) {
  pdl_enter();
  const int m = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (m >= a.T) return;
  int t, mr;
  bool ffn;
  if (!row_of(m, a.counts, a.idx_f, a.idx_a, t, ffn, mr)) return;
  if (ffn) {
    if (!a.grad_gate) return;
    const float* p = a.dgpart + (size_t)mr * a.part_ld;
    float s = 0.f;
    for (int i = lane; i < a.n_parts; i += 32) s += p[i];
    s = warp_sum(s);
    if (lane == 0) a.grad_gate[t] = s;
    return;
  }
  const float sc = a.scale_a[mr];   // 1 - g
  const float* ar = a.pre + (size_t)mr * a.d_r;
  const float* gr = a.ga + (size_t)mr * a.d_r;
  float dgs = 0.f;
  for (int r = lane; r < a.d_r; r += 32) {
    const float x = ar[r], e = gr[r];
    const float sg = sigmoidf_(x);
    const float hid = __bfloat162float(__float2bfloat16_rn(x * sg));   // what W_2 read
    dgs = fmaf(e, hid, dgs);
    const float da = sc * e * sg * (1.f + x * (1.f - sg));
    a.da_f32[(size_t)mr * a.d_r + r] = da;
    a.da_bf16[(size_t)mr * a.d_r + r] = __float2bfloat16_rn(da);
    a.y2[(size_t)mr * a.d_r + r] = sc * hid;
  }
  dgs = warp_sum(dgs);
  if (lane == 0 && a.grad_gate) a.grad_gate[t] = -dgs;
}

// Partial weight gradients over chunks of kChunk compacted adapter rows:
//   part[c, n, r] = sum_{m in chunk c, m < rows} X(m, n) Y[m, r]
// X(m, n) = Xf[idx[m], n] (fp32, gathered) or Xb[m, n] (bf16, compacted).  64 x 64
// outputs per 256-thread CTA, 4 x 4 per thread, rows staged 16 at a time.
template <bool XBF16>
__global__ void __launch_bounds__(256) k_bw_wgrad(const BwWgradArgs a) {
  pdl_enter();
  __shared__ float Xs[16][64 + 4];
  __shared__ float Ys[16][64 + 4];
  const int rows = *a.rows;
  const int c = blockIdx.z;
  const int m0 = c * kBwChunk;
  if (m0 >= rows) return;
  const int m1 = min(rows, m0 + kBwChunk);
  const int n0 = blockIdx.x * 64, r0 = blockIdx.y * 64;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int mb = m0; mb < m1; mb += 16) {
    for (int i = threadIdx.x; i < 16 * 64; i += 256) {
      const int k = i >> 6, col = i & 63;
      const int m = mb + k;
      float xv = 0.f, yv = 0.f;
      if (m < m1) {
        const int n = n0 + col, r = r0 + col;
        if (n < a.N) {
          if constexpr (XBF16)
            xv = __bfloat162float(static_cast<const __nv_bfloat16*>(a.X)[(size_t)m * a.N + n]);
          else
            xv = static_cast<const float*>(a.X)[(size_t)a.idx[m] * a.N + n];
        }
        if (r < a.R) yv = a.Y[(size_t)m * a.R + r];
      }
      Xs[k][col] = xv;
      Ys[k][col] = yv;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      float xv[4], yv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) xv[i] = Xs[k][ty * 4 + i];
#pragma unroll
      for (int i = 0; i < 4; ++i) yv[i] = Ys[k][tx * 4 + i];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int jj = 0; jj < 4; ++jj) acc[i][jj] = fmaf(xv[i], yv[jj], acc[i][jj]);
    }
    __syncthreads();
  }
  float* out = a.part + (size_t)c * a.N * a.R;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int n = n0 + ty * 4 + i;
    if (n >= a.N) continue;
#pragma unroll
    for (int jj = 0; jj < 4; ++jj) {
      const int r = r0 + tx * 4 + jj;
      if (r < a.R) out[(size_t)n * a.R + r] = acc[i][jj];
    }
  }
}

// out = sum over the used chunks (in chunk order) of part[c, n, r]; out[n, r], or
// out[r, n] when transposed.  Zero when there are no rows.
__global__ void __launch_bounds__(256) k_bw_wreduce(const float* __restrict__ part,
                                                    const int* __restrict__ rows, int max_ch, int N,
                                                    int R, int transposed, float* __restrict__ out) {
  pdl_enter();
  const int nch = min(max_ch, (max(*rows, 0) + kBwChunk - 1) / kBwChunk);
  const size_t total = (size_t)N * R;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    // transposed: i indexes out[r, n] (n fastest) so the writes are coalesced
    const size_t n = transposed ? i % N : i / R;
    const size_t r = transposed ? i / N : i % R;
    float s = 0.f;
    for (int c = 0; c < nch; ++c) s += part[(size_t)c * total + n * R + r];
    out[i] = s;
  }
}

// dL/dh_bar = G + r (du gain) - h_bar r^3 mean(h_bar du gain), r = 1/rms(h_bar).
__global__ void __launch_bounds__(256) k_bw_out(const BwOutArgs a) {
  pdl_enter();
  const int m = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (m >= a.T) return;
  int t, mr;
  bool ffn;
  if (!row_of(m, a.counts, a.idx_f, a.idx_a, t, ffn, mr)) return;
  const float* h = a.hbar + (size_t)t * a.d;
  const float* du = (ffn ? a.du_f : a.du_a) + (size_t)mr * a.d;
  float dot = 0.f;
  for (int c = 4 * lane; c < a.d; c += 128) {
    const float4 x = *reinterpret_cast<const float4*>(h + c);
    const float4 v = *reinterpret_cast<const float4*>(du + c);
    const float4 w = *reinterpret_cast<const float4*>(a.gain + c);
    dot += x.x * v.x * w.x + x.y * v.y * w.y + x.z * v.z * w.z + x.w * v.w * w.w;
  }
  dot = warp_sum(dot);
  const float r = a.rinv[t];
  const float k = r * r * r * dot / (float)a.d;
  const float* G = a.G + (size_t)t * a.d;
  float* o = a.grad_hbar + (size_t)t * a.d;
  for (int c = 4 * lane; c < a.d; c += 128) {
    const float4 x = *reinterpret_cast<const float4*>(h + c);
    const float4 v = *reinterpret_cast<const float4*>(du + c);
    const float4 w = *reinterpret_cast<const float4*>(a.gain + c);
    const float4 g = *reinterpret_cast<const float4*>(G + c);
    *reinterpret_cast<float4*>(o + c) =
        make_float4(g.x + r * v.x * w.x - x.x * k, g.y + r * v.y * w.y - x.y * k,
                    g.z + r * v.z * w.z - x.z * k, g.w + r * v.w * w.w - x.w * k);
  }
}

// dL_skip/dg (Sec. 3.3), scaled by alpha: 2 alpha / (B (S - 1)) times the token's summed
// routed gates at its S - 1 next-token positions, 0 at a sequence's last position and
// in the rows of the dense prefix.
__global__ void __launch_bounds__(256) k_skip_grad(const float* __restrict__ gates, int L, int n_dense,
                                                   int n_seqs, int seq_len, float alpha,
                                                   float* __restrict__ out) {
  pdl_enter();
  const int T = n_seqs * seq_len;
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  float tot = 0.f;
  for (int l = n_dense; l < L; ++l) tot += gates[(size_t)l * T + t];
  const bool next = t % seq_len < seq_len - 1;
  const float v = next ? 2.f * alpha / ((float)n_seqs * (float)(seq_len - 1)) * tot : 0.f;
  for (int l = 0; l < L; ++l) out[(size_t)l * T + t] = l < n_dense ? 0.f : v;
}

// out[z][c][r] = in[z][r][c] for bf16 matrices [R][C], 32 x 32 tiles through shared memory.
__global__ void __launch_bounds__(256) k_transpose_bf16(const uint16_t* __restrict__ in,
                                                        uint16_t* __restrict__ out, int R, int C) {
  __shared__ uint16_t tile[32][33];
  const size_t zoff = (size_t)blockIdx.z * R * C;
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  for (int k = ty; k < 32; k += 8) {
    const int r = r0 + k, c = c0 + tx;
    if (r < R && c < C) tile[k][tx] = in[zoff + (size_t)r * C + c];
  }
  __syncthreads();
  for (int k = ty; k < 32; k += 8) {
    const int c = c0 + k, r = r0 + tx;
    if (r < R && c < C) out[zoff + (size_t)c * R + r] = tile[tx][k];
  }
}

unsigned row_blocks(int T) { return (unsigned)((T + kRowWarps - 1) / kRowWarps); }

}  // namespace

cudaError_t launch_bw_prep(const BwPrepArgs& a, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  if (a.d % 4) return cudaErrorInvalidValue;
  return launch_pdl(k_bw_prep, dim3(row_blocks(a.T)), dim3(256), 0, st, a);
}

cudaError_t launch_bw_rows(const BwRowsArgs& a, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  return launch_pdl(k_bw_rows, dim3(row_blocks(a.T)), dim3(256), 0, st, a);
}

cudaError_t launch_bw_wgrad(const BwWgradArgs& a, bool x_bf16, int max_rows, cudaStream_t st) {
  const int chunks = (max_rows + kBwChunk - 1) / kBwChunk;
  if (chunks <= 0) return cudaSuccess;
  const dim3 grid((a.N + 63) / 64, (a.R + 63) / 64, chunks);
  return x_bf16 ? launch_pdl(k_bw_wgrad<true>, grid, dim3(256), 0, st, a)
                : launch_pdl(k_bw_wgrad<false>, grid, dim3(256), 0, st, a);
}

cudaError_t launch_bw_wreduce(const float* part, const int* rows, int max_rows, int N, int R,
                              int transposed, float* out, int num_sms, cudaStream_t st) {
  const long total = (long)N * R;
  long blocks = (total + 255) / 256;
  if (blocks > 8L * num_sms) blocks = 8L * num_sms;
  if (blocks <= 0) return cudaSuccess;
  const int max_ch = (max_rows + kBwChunk - 1) / kBwChunk;
  return launch_pdl(k_bw_wreduce, dim3((unsigned)blocks), dim3(256), 0, st, part, rows, max_ch, N,
                    R, transposed, out);
}

cudaError_t launch_bw_out(const BwOutArgs& a, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  if (a.d % 4) return cudaErrorInvalidValue;
  return launch_pdl(k_bw_out, dim3(row_blocks(a.T)), dim3(256), 0, st, a);
}

cudaError_t launch_skip_grad(const float* gates, int L, int n_dense, int n_seqs, int seq_len,
                             float alpha, float* out, cudaStream_t st) {
  const int T = n_seqs * seq_len;
  if (T <= 0) return cudaSuccess;
  return launch_pdl(k_skip_grad, dim3((T + 255) / 256), dim3(256), 0, st, gates, L, n_dense,
                    n_seqs, seq_len, alpha, out);
}

cudaError_t launch_transpose_bf16(const void* in, void* out, int R, int C, int batch,
                                  cudaStream_t st) {
  if (R <= 0 || C <= 0 || batch <= 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((C + 31) / 32, (R + 31) / 32, batch);
  cfg.blockDim = dim3(256);
  cfg.stream = st;
  return cudaLaunchKernelEx(&cfg, k_transpose_bf16, static_cast<const uint16_t*>(in),
                            static_cast<uint16_t*>(out), R, C);
}

}  // namespace hero
