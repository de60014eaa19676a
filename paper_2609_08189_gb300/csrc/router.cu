// Router, memory and bookkeeping kernels of the routed FFN stack.
//
//   k_init      h_bar_1 = h_0 + P_1, its operand copy and sum of squares; reset of
//               the per-token memory (S = 0, zeta = 0) and path state (p = m = 1).
//   k_router    steps 1, 2 and 6 of a routed block for TB tokens per CTA:
//               transition features (Eqs. 7-8), path vector (Eqs. 4, 6), hidden and
//               path encoders (Eqs. 5, 9), q/k/v (Eq. 10), memory read (Eq. 11)
//               fused with the memory write (Eq. 12; S read once, written once),
//               nu (Eq. 13), f_theta / p_hist / m_hist (Eqs. 14-15), f_psi and the
//               gate (Eq. 16), and the decision g >= tau_exec (Eq. 3).
//   k_compact   stable scan of the decisions into FFN / adapter index lists.
//   k_norm      u = LN_ffn(h_bar) (Eq. 1) of each token into its branch's rows.
//   k_convert   weight conversion / repacking at load time.
#include "hero_device.cuh"

namespace hero {
namespace {

// ------------------------------------------------------------------------------
// k_init: one warp per token.
// ------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_init(const InitArgs a) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= a.T) return;
  const int t = warp;
  const size_t row = (size_t)t * a.d;
  float ss = 0.f;
  for (int n = lane * 4; n < a.d; n += 128) {
    float4 h = *reinterpret_cast<const float4*>(a.h_in + row + n);
    if (a.p0) {
      const float4 p = load4(a.p0, row + n, a.p_bf16);
      h.x += p.x; h.y += p.y; h.z += p.z; h.w += p.w;
    }
    *reinterpret_cast<float4*>(a.hbar + row + n) = h;
    store4(a.xl, row + n, h, a.xl_bf16);
    ss += h.x * h.x + h.y * h.y + h.z * h.z + h.w * h.w;
  }
  ss = warp_sum(ss);
  for (int s = lane; s < a.np; s += 32)
    *reinterpret_cast<float4*>(a.part + ((size_t)t * a.np + s) * 4) =
        make_float4(s == 0 ? ss : 0.f, 0.f, 0.f, 0.f);
  if (a.reset_router) {
    const int dm2 = a.d_m * a.d_m;
    float* S = a.S + (size_t)t * dm2;
    for (int i = lane * 4; i < dm2; i += 128)
      *reinterpret_cast<float4*>(S + i) = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int i = lane; i < a.d_m; i += 32) a.zeta[(size_t)t * a.d_m + i] = 0.f;
    if (lane == 0) {
      a.pst[t] = 1.f;   // p_hist_{l_0} = 1
      a.mst[t] = 1.f;   // m_hist_{l_0} = 1
      a.dprev[t] = 0.f;
    }
  }
}

// ------------------------------------------------------------------------------
// Block-level small matmul: out[t][o] = act(sum_i in[t][i] * Wt[i][o] + bias[o])
// for t < TB tokens held in shared memory.  Each work item owns one output column
// for a group of TPG tokens so every weight is loaded once per group.
// ------------------------------------------------------------------------------
constexpr int TB = 16;        // tokens per CTA
constexpr int NTHR = 256;

template <int TPG>
__device__ __forceinline__ void bmm_tpg(const float* in, int in_ld, int NI,
                                        const float* __restrict__ Wt, int NO,
                                        const float* __restrict__ bias, float* out, int out_ld,
                                        bool silu_act) {
  constexpr int G = TB / TPG;
  for (int w = threadIdx.x; w < NO * G; w += NTHR) {
    const int o = w % NO;
    const int g = w / NO;
    float acc[TPG];
    const float b = bias ? __ldg(bias + o) : 0.f;
#pragma unroll
    for (int t = 0; t < TPG; ++t) acc[t] = b;
    const float* inb = in + g * TPG * in_ld;
    for (int i = 0; i < NI; ++i) {
      const float wv = __ldg(Wt + (size_t)i * NO + o);
#pragma unroll
      for (int t = 0; t < TPG; ++t) acc[t] = fmaf(inb[t * in_ld + i], wv, acc[t]);
    }
#pragma unroll
    for (int t = 0; t < TPG; ++t) out[(g * TPG + t) * out_ld + o] = silu_act ? siluf_(acc[t]) : acc[t];
  }
}

__device__ __forceinline__ void bmm(const float* in, int in_ld, int NI, const float* Wt, int NO,
                                    const float* bias, float* out, int out_ld, bool silu_act) {
  if (NO >= 128)
    bmm_tpg<16>(in, in_ld, NI, Wt, NO, bias, out, out_ld, silu_act);
  else if (NO >= 32)
    bmm_tpg<4>(in, in_ld, NI, Wt, NO, bias, out, out_ld, silu_act);
  else
    bmm_tpg<1>(in, in_ld, NI, Wt, NO, bias, out, out_ld, silu_act);
}

// Shared-memory layout of k_router (floats).
constexpr int LD_ENC = 256 + 1;   // encoder / psi hidden rows (<= 256 wide)
constexpr int LD_S = 128 + 128 + 2;  // [s ; c ; nu] rows (d_s <= 128, d_m <= 128)
constexpr int LD_QKV = 3 * 128 + 1;
constexpr int LD_HID = 256 + 1;

template <int DM>
__global__ void __launch_bounds__(NTHR) k_router(const RouterArgs a) {
  extern __shared__ float sm[];
  float* enc = sm;                          // [TB][LD_ENC]  SiLU(W_hd RMSNorm(h_bar))
  float* psi = enc + TB * LD_ENC;           // [TB][LD_ENC]  SiLU(f_psi first layer)
  float* scn = psi + TB * LD_ENC;           // [TB][LD_S]    s | c | nu
  float* qkv = scn + TB * LD_S;             // [TB][LD_QKV]  q | k | v
  float* hid = qkv + TB * LD_QKV;           // [TB][LD_HID]  f_theta hidden / scratch
  float* sc = hid + TB * LD_HID;            // [TB][16] per-token scalars
  // sc: 0 rinv, 1 d_j, 2 gamma_j, 3 p_prev, 4 m_prev, 5 a, 6 b, 8.. path x (6)

  const int ds = a.d_h + a.d_a;
  const int t0 = blockIdx.x * TB;
  const int nY = a.d_enc + a.d_head;
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;

  // 1. per-token scalars from the partial sums of the previous block's epilogue
  if (tid < TB) {
    const int t = t0 + tid;
    float ss = 0.f, dd = 0.f, dp = 0.f, dprev = 0.f, pp = 1.f, mp = 1.f;
    if (t < a.T) {
      for (int s = 0; s < a.np; ++s) {
        const float4 v = *reinterpret_cast<const float4*>(a.part + ((size_t)t * a.np + s) * 4);
        ss += v.x;
        dd += v.y;
        dp += v.z;
      }
      dprev = a.dprev[t];
      pp = a.pst[t];
      mp = a.mst[t];
    }
    const float rinv = rsqrtf(ss / (float)a.d + a.rms_eps);
    const float dj = a.j == 1 ? 0.f : sqrtf(dd);                       // Eq. 7
    const float gam = a.j > 2 ? dp / (dj * dprev + a.eps) : 0.f;       // Eq. 8
    float* s_ = sc + tid * 16;
    s_[0] = rinv;
    s_[1] = dj;
    s_[2] = gam;
    s_[3] = pp;
    s_[4] = mp;
    // path vector, Eq. 4 with Eq. 6
    s_[8] = (float)a.j / (float)a.L;
    s_[9] = (float)(a.L - a.j) / (float)a.L;
    s_[10] = dj;
    s_[11] = gam;
    s_[12] = pp;
    s_[13] = mp;
  }
  __syncthreads();

  // 2. encoder hidden SiLU(rinv * (W_hd diag(g_r)) h_bar) and f_psi hidden
  for (int i = tid; i < TB * nY; i += NTHR) {
    const int tl = i / nY, c = i % nY;
    const int t = t0 + tl;
    const float y = t < a.T ? a.Y[(size_t)t * nY + c] : 0.f;
    if (c < a.d_enc)
      enc[tl * LD_ENC + c] = siluf_(y * sc[tl * 16]);
    else
      psi[tl * LD_ENC + (c - a.d_enc)] = siluf_(y + a.w.ps_b1[c - a.d_enc]);
  }
  __syncthreads();

  // 3. z_h = W_hu enc (Eq. 5) -> s[0, d_h);  path encoder hidden -> hid
  bmm(enc, LD_ENC, a.d_enc, a.w.w_hu_t, a.d_h, nullptr, scn, LD_S, false);
  bmm(sc + 8, 16, 6, a.w.path_w1_t, a.d_path, a.w.path_b1, hid, LD_HID, true);
  __syncthreads();
  // z_a = W_a2 hid + b_a2 (Eq. 9) -> s[d_h, d_s)
  bmm(hid, LD_HID, a.d_path, a.w.path_w2_t, a.d_a, a.w.path_b2, scn + a.d_h, LD_S, false);
  __syncthreads();

  // 4. q | k | v = W_{q,k,v} s (Eq. 10)
  bmm(scn, LD_S, ds, a.w.w_qkv_t, 3 * DM, nullptr, qkv, LD_QKV, false);
  __syncthreads();

  // 5. memory read (Eq. 11) fused with the write (Eq. 12), one warp per token.
  //    Lane owns a 4-column group and every (32/LPR)-th row of S.
  {
    constexpr int LPR = DM / 4;          // lanes per S row
    constexpr int RPI = 32 / LPR;        // rows per iteration
    const int cq = lane % LPR;
    const int r0 = lane / LPR;
    for (int tl = warp; tl < TB; tl += NTHR / 32) {
      const int t = t0 + tl;
      if (t >= a.T) continue;
      const float* q = qkv + tl * LD_QKV;
      const float* k = q + DM;
      const float* v = q + 2 * DM;
      float* S = a.S + (size_t)t * DM * DM;
      float* z = a.zeta + (size_t)t * DM;
      float den = 0.f;
      for (int m = lane; m < DM; m += 32) {
        const float zo = z[m];
        den += phif_(q[m]) * zo;
        z[m] = a.rho * zo + phif_(k[m]);
      }
      den = warp_sum(den);
      float4 c = make_float4(0.f, 0.f, 0.f, 0.f);
      const float4 vv = make_float4(v[4 * cq], v[4 * cq + 1], v[4 * cq + 2], v[4 * cq + 3]);
#pragma unroll 4
      for (int r = r0; r < DM; r += RPI) {
        float4* p = reinterpret_cast<float4*>(S + r * DM + 4 * cq);
        const float4 so = *p;
        const float fq = phif_(q[r]);
        const float fk = phif_(k[r]);
        c.x += fq * so.x; c.y += fq * so.y; c.z += fq * so.z; c.w += fq * so.w;
        *p = make_float4(a.rho * so.x + fk * vv.x, a.rho * so.y + fk * vv.y,
                         a.rho * so.z + fk * vv.z, a.rho * so.w + fk * vv.w);
      }
#pragma unroll
      for (int o = LPR; o < 32; o <<= 1) {
        c.x += __shfl_xor_sync(0xffffffffu, c.x, o);
        c.y += __shfl_xor_sync(0xffffffffu, c.y, o);
        c.z += __shfl_xor_sync(0xffffffffu, c.z, o);
        c.w += __shfl_xor_sync(0xffffffffu, c.w, o);
      }
      if (r0 == 0) {
        const float inv = 1.0f / (den + a.eps);
        float* cdst = scn + tl * LD_S + ds + 4 * cq;
        cdst[0] = c.x * inv;
        cdst[1] = c.y * inv;
        cdst[2] = c.z * inv;
        cdst[3] = c.w * inv;
      }
    }
  }
  __syncthreads();

  // 6. nu = 1 - cos(W_n s, W_c c) for j > 1 (Eq. 13); nu_1 = 0
  if (a.j > 1) {
    float* nv = hid;                 // [TB][LD_HID]: cols [0, DM) W_n s, [128, 128+DM) W_c c
    bmm(scn, LD_S, ds, a.w.w_n_t, DM, nullptr, nv, LD_HID, false);
    bmm(scn + ds, LD_S, DM, a.w.w_c_t, DM, nullptr, nv + 128, LD_HID, false);
    __syncthreads();
    for (int tl = warp; tl < TB; tl += NTHR / 32) {
      const float* x = nv + tl * LD_HID;
      float xy = 0.f, xx = 0.f, yy = 0.f;
      for (int i = lane; i < DM; i += 32) {
        const float u = x[i], w = x[128 + i];
        xy += u * w;
        xx += u * u;
        yy += w * w;
      }
      xy = warp_sum(xy);
      xx = warp_sum(xx);
      yy = warp_sum(yy);
      if (lane == 0) scn[tl * LD_S + ds + DM] = 1.f - xy / (sqrtf(xx) * sqrtf(yy) + a.eps);
    }
  } else {
    if (tid < TB) scn[tid * LD_S + ds + DM] = 0.f;
  }
  __syncthreads();

  // 7. f_theta hidden = SiLU(W_th1 [s; c; nu] + b)
  bmm(scn, LD_S, ds + DM + 1, a.w.th_w1_t, a.d_head, a.w.th_b1, hid, LD_HID, true);
  __syncthreads();

  // 8. a = w_th2 . hidden + b (Eq. 14), b = w_ps2 . psi + b (Eq. 16); gate and decision
  for (int tl = warp; tl < TB; tl += NTHR / 32) {
    float sa = 0.f, sb = 0.f;
    for (int i = lane; i < a.d_head; i += 32) {
      sa += a.w.th_w2[i] * hid[tl * LD_HID + i];
      sb += a.w.ps_w2[i] * psi[tl * LD_ENC + i];
    }
    sa = warp_sum(sa);
    sb = warp_sum(sb);
    const int t = t0 + tl;
    if (lane == 0 && t < a.T) {
      const float av = sa + a.w.th_b2[0];
      const float bv = sb + a.w.ps_b2[0];
      const float p = sigmoidf_(av / a.t_hist);      // Eq. 14
      const float m = sc[tl * 16 + 4] * p;          // Eq. 15
      const float g = sigmoidf_(av + bv);            // Eq. 16
      uint8_t dec;
      if (a.mask_in)
        dec = a.mask_in[t] ? 1 : 0;
      else
        dec = g >= a.tau ? 1 : 0;                    // Eq. 3 (ties run the FFN)
      a.pst[t] = p;
      a.mst[t] = m;
      a.dprev[t] = sc[tl * 16 + 1];
      a.gate[t] = g;
      a.mask[t] = dec;
      if (a.gate_out) a.gate_out[t] = g;
      if (a.mask_out) a.mask_out[t] = dec;
    }
  }
}

constexpr size_t kRouterSmem =
    sizeof(float) * (size_t)TB * (2 * LD_ENC + LD_S + LD_QKV + LD_HID + 16);

// ------------------------------------------------------------------------------
// k_compact: one CTA; stable exclusive scan of the decisions, chunks of 8192.
// ------------------------------------------------------------------------------
constexpr int CT = 1024, CPT = 8;

__global__ void __launch_bounds__(CT) k_compact(const CompactArgs a) {
  __shared__ int wsum[CT / 32];
  __shared__ int carry_s;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) carry_s = 0;
  __syncthreads();
  for (int base = 0; base < a.T; base += CT * CPT) {
    uint8_t f[CPT];
    int cnt = 0;
#pragma unroll
    for (int i = 0; i < CPT; ++i) {
      const int t = base + tid * CPT + i;
      f[i] = (t < a.T) ? (a.dense ? 1 : (a.mask[t] ? 1 : 0)) : 2;
      cnt += f[i] == 1;
    }
    // inclusive warp scan of the per-thread counts
    int x = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) wsum[warp] = x;
    __syncthreads();
    if (warp == 0) {
      int w = wsum[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      wsum[lane] = w;  // inclusive over warps
    }
    __syncthreads();
    const int carry = carry_s;
    int pos_f = carry + (warp ? wsum[warp - 1] : 0) + x - cnt;  // exclusive
    int t = base + tid * CPT;
    int pos_a = t - pos_f;  // tokens before t that went to the adapter
#pragma unroll
    for (int i = 0; i < CPT; ++i, ++t) {
      if (f[i] == 2) break;
      if (f[i]) {
        a.idx_f[pos_f] = t;
        a.scale_f[pos_f] = a.dense ? 1.f : a.gate[t];
        ++pos_f;
      } else {
        a.idx_a[pos_a] = t;
        a.scale_a[pos_a] = 1.f - a.gate[t];
        ++pos_a;
      }
      if (a.dense) {
        if (a.gate_out) a.gate_out[t] = 1.f;
        if (a.mask_out) a.mask_out[t] = 1;
      }
    }
    __syncthreads();
    if (tid == 0) carry_s = carry + wsum[CT / 32 - 1];
    __syncthreads();
  }
  if (tid == 0) {
    const int nf = carry_s;
    a.counts[0] = nf;
    a.counts[1] = a.T - nf;
    if (a.count_out) *a.count_out = nf;
  }
}

// ------------------------------------------------------------------------------
// k_norm: 8 consecutive elements per thread; slot s < n_f is FFN row s (token
// idx_f[s]), slot s >= n_f is adapter row s - n_f.
// ------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_norm(const NormArgs a) {
  const int per_row = a.d / 8;
  const long gid = (long)blockIdx.x * blockDim.x + threadIdx.x;
  const long slot = gid / per_row;
  if (slot >= a.T) return;
  const int c = (int)(gid % per_row) * 8;
  const int nf = a.counts[0];
  int t;
  void* dst;
  long r;
  if (slot < nf) {
    t = a.idx_f[slot];
    dst = a.u_f;
    r = slot;
  } else {
    t = a.idx_a[slot - nf];
    dst = a.u_a;
    r = slot - nf;
  }
  float ss = 0.f;
  for (int s = 0; s < a.np; ++s) ss += a.part[((size_t)t * a.np + s) * 4];
  const float rinv = rsqrtf(ss / (float)a.d + a.rms_eps);
  const float* h = a.hbar + (size_t)t * a.d + c;
  const float4 h0 = *reinterpret_cast<const float4*>(h);
  const float4 h1 = *reinterpret_cast<const float4*>(h + 4);
  const float4 g0 = *reinterpret_cast<const float4*>(a.gain + c);
  const float4 g1 = *reinterpret_cast<const float4*>(a.gain + c + 4);
  const float4 u0 = make_float4(h0.x * rinv * g0.x, h0.y * rinv * g0.y, h0.z * rinv * g0.z,
                                h0.w * rinv * g0.w);
  const float4 u1 = make_float4(h1.x * rinv * g1.x, h1.y * rinv * g1.y, h1.z * rinv * g1.z,
                                h1.w * rinv * g1.w);
  const size_t off = (size_t)r * a.d + c;
  store4(dst, off, u0, a.out_bf16);
  store4(dst, off + 4, u1, a.out_bf16);
}

// ------------------------------------------------------------------------------
// k_convert: weight conversion / repacking (load time only).
// ------------------------------------------------------------------------------
__global__ void k_convert(const void* src, int src_bf16, void* dst, int dst_bf16, long rows,
                          long cols, long grp, long grp_stride, long offset,
                          const float* col_scale) {
  const long n = rows * cols;
  for (long i = (long)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (long)gridDim.x * blockDim.x) {
    const long r = i / cols, c = i % cols;
    float v = src_bf16 ? __uint_as_float((uint32_t)static_cast<const uint16_t*>(src)[i] << 16)
                       : static_cast<const float*>(src)[i];
    if (col_scale) v *= col_scale[c];
    const long dr = (r / grp) * grp_stride + (r % grp) + offset;
    const long di = dr * cols + c;
    if (dst_bf16)
      static_cast<__nv_bfloat16*>(dst)[di] = __float2bfloat16_rn(v);
    else
      static_cast<float*>(dst)[di] = v;
  }
}

}  // namespace

cudaError_t launch_init(const InitArgs& a, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  const int warps_per_block = 8;
  k_init<<<(a.T + warps_per_block - 1) / warps_per_block, 256, 0, st>>>(a);
  return cudaGetLastError();
}

template <int DM>
static cudaError_t launch_router_dm(const RouterArgs& a, cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_router<DM>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kRouterSmem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  k_router<DM><<<(a.T + TB - 1) / TB, NTHR, kRouterSmem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_router(int d_m, const RouterArgs& a, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  switch (d_m) {
    case 16: return launch_router_dm<16>(a, st);
    case 32: return launch_router_dm<32>(a, st);
    case 64: return launch_router_dm<64>(a, st);
    case 128: return launch_router_dm<128>(a, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_compact(const CompactArgs& a, cudaStream_t st) {
  k_compact<<<1, CT, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_norm(const NormArgs& a, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  const long threads = (long)a.T * (a.d / 8);
  k_norm<<<(unsigned)((threads + 255) / 256), 256, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_convert_rows(const void* src, int src_bf16, void* dst, int dst_bf16, long rows,
                                long cols, long grp, long grp_stride, long offset,
                                const float* col_scale, cudaStream_t st) {
  const long n = rows * cols;
  if (n <= 0) return cudaSuccess;
  long blocks = (n + 255) / 256;
  if (blocks > 65536) blocks = 65536;
  k_convert<<<(unsigned)blocks, 256, 0, st>>>(src, src_bf16, dst, dst_bf16, rows, cols, grp,
                                              grp_stride, offset, col_scale);
  return cudaGetLastError();
}

}  // namespace hero
