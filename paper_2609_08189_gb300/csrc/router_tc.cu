// Step 4 of the router on the tensor cores (RouterTcArgs): the per-token part between the
// q/k/v product and f_theta's first layer, one warp per token.
//   c = phi(q)^T S / (phi(q)^T zeta + eps)                Eq. 11 (before the write)
//   S = rho S + phi(k) v^T, zeta = rho zeta + phi(k)      Eq. 12
//   nu = 1 - cos(W_n s, W_c c) for j > 1, else 0          Eq. 13
//   f_theta's input [s; c; nu] as three bf16 terms per value (zero padded to kf columns)
// S is read once and written once; its lanes and the order in which c's partial sums are
// added follow the fused router's memory step.  k_rt_hist is the same step in its history
// form (see there), for a forward pass over all routed blocks.
#include "hero_device.cuh"

namespace hero {
namespace {

constexpr int kRtMaxF = 64 + 128 + 1;   // [s; c; nu] for d_s = 64, d_m <= 128

__device__ __forceinline__ uint16_t bf16_term(float x, int term) {
  __nv_bfloat16 h = __float2bfloat16_rn(x);
  for (int p = 0; p < term; ++p) {
    x -= __bfloat162float(h);
    h = __float2bfloat16_rn(x);
  }
  return *reinterpret_cast<const uint16_t*>(&h);
}

// W_c c and nu = 1 - cos(W_n s, W_c c) (Eq. 13), then f_theta's input [s; c; nu] as three
// bf16 terms (term p of element e at column p F + e, zero padded to kf): the part of the
// memory step after c, shared by the two memory kernels.  xin is this warp's [s; c; nu]
// (s and c stored, nu stored here), wc W_c ([in][out], read through L1), wnr
// the lane's elements lane + 32 u of W_n s.  The sums run in the order of the plain loops.
template <int DM>
__device__ __forceinline__ void rt_tail(const RouterTcArgs& a, int t, int lane, float* xin,
                                        const float* wc, const float (&wnr)[(DM + 31) / 32]) {
  constexpr int NO = (DM + 31) / 32;
  const int ds = a.d_h + a.d_a, F = ds + DM + 1;
  const float* c = xin + ds;
  __syncwarp();
  float cv[NO];
#pragma unroll
  for (int u = 0; u < NO; ++u) cv[u] = 0.f;
#pragma unroll 8
  for (int i = 0; i < DM; ++i) {
    const float ci = c[i];
#pragma unroll
    for (int u = 0; u < NO; ++u)
      if (lane + 32 * u < DM) cv[u] = fmaf(wc[i * DM + lane + 32 * u], ci, cv[u]);
  }
  float nu = 0.f;
  if (a.j > 1) {
    float xy = 0.f, xx = 0.f, yy = 0.f;
#pragma unroll
    for (int u = 0; u < NO; ++u)
      if (lane + 32 * u < DM) {
        const float x = wnr[u], y = cv[u];
        xy += x * y;
        xx += x * x;
        yy += y * y;
      }
    xy = warp_sum(xy);
    xx = warp_sum(xx);
    yy = warp_sum(yy);
    nu = 1.f - xy / (sqrtf(xx) * sqrtf(yy) + a.eps);
  }
  if (lane == 0) xin[ds + DM] = nu;
  __syncwarp();
  // two columns per 32-bit store
  uint32_t* fin = reinterpret_cast<uint32_t*>(a.fin3 + (size_t)t * a.kf);
  for (int cp = lane; cp < a.kf / 2; cp += 32) {
    uint32_t pk = 0;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int col = 2 * cp + h, p = col / F, e = col - p * F;
      if (p < 3) pk |= (uint32_t)bf16_term(xin[e], p) << (16 * h);
    }
    fin[cp] = pk;
  }
}

// The warp's start: s into its [s; c; nu] row, W_n s into registers.
template <int DM>
__device__ __forceinline__ void rt_tail_load(const RouterTcArgs& a, int t, int lane, float* xin,
                                             const float* wn, float (&wnr)[(DM + 31) / 32]) {
  const int ds = a.d_h + a.d_a;
  const float* sr = a.s + (size_t)t * ds;
  for (int e = lane; e < ds; e += 32) xin[e] = sr[e];
#pragma unroll
  for (int u = 0; u < (DM + 31) / 32; ++u) wnr[u] = lane + 32 * u < DM ? wn[lane + 32 * u] : 0.f;
}

template <int DM>
__global__ void __launch_bounds__(256) k_rt_mem(const RouterTcArgs a) {
  static_assert(DM <= 128, "DM / 4 lanes per S row");
  __shared__ float xin_s[8][kRtMaxF];
  pdl_enter();
  const float* wc = a.w.w_c_t;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * 8 + w;
  if (t >= a.T) return;   // whole warps only; nothing below synchronises the CTA
  float* xin = xin_s[w];
  const float* q = a.qkvn + (size_t)t * 4 * DM;
  const float* k = q + DM;
  const float* v = q + 2 * DM;
  const float* wn = q + 3 * DM;   // W_n s
  float wnr[(DM + 31) / 32];
  rt_tail_load<DM>(a, t, lane, xin, wn, wnr);
  const int ds = a.d_h + a.d_a;
  float* S = a.S + (size_t)t * DM * DM;
  float* z = a.zeta + (size_t)t * DM;
  float den = 0.f;
  for (int m = lane; m < DM; m += 32) {
    const float zo = z[m];
    den += phif_(q[m]) * zo;
    z[m] = a.rho * zo + phif_(k[m]);
  }
  den = warp_sum(den);
  const float inv = 1.0f / (den + a.eps);
  constexpr int LPR = DM / 4;          // lanes per S row
  constexpr int RPI = 32 / LPR;        // rows per iteration
  constexpr int NIT = DM / RPI;        // S rows handled by this lane
  constexpr int BATCH = NIT < 8 ? NIT : 8;
  const int cq = lane % LPR;
  const int r0 = lane / LPR;
  float4 c = make_float4(0.f, 0.f, 0.f, 0.f);
  const float4 vv = *reinterpret_cast<const float4*>(v + 4 * cq);
#pragma unroll 1
  for (int i0 = 0; i0 < NIT; i0 += BATCH) {
    float4 so[BATCH];
#pragma unroll
    for (int i = 0; i < BATCH; ++i)
      so[i] = *reinterpret_cast<const float4*>(S + (r0 + (i0 + i) * RPI) * DM + 4 * cq);
#pragma unroll
    for (int i = 0; i < BATCH; ++i) {
      const int r = r0 + (i0 + i) * RPI;
      const float fq = phif_(q[r]);
      const float fk = phif_(k[r]);
      c.x += fq * so[i].x; c.y += fq * so[i].y; c.z += fq * so[i].z; c.w += fq * so[i].w;
      *reinterpret_cast<float4*>(S + r * DM + 4 * cq) =
          make_float4(a.rho * so[i].x + fk * vv.x, a.rho * so[i].y + fk * vv.y,
                      a.rho * so[i].z + fk * vv.z, a.rho * so[i].w + fk * vv.w);
    }
  }
#pragma unroll
  for (int o = LPR; o < 32; o <<= 1) {
    c.x += __shfl_xor_sync(0xffffffffu, c.x, o);
    c.y += __shfl_xor_sync(0xffffffffu, c.y, o);
    c.z += __shfl_xor_sync(0xffffffffu, c.z, o);
    c.w += __shfl_xor_sync(0xffffffffu, c.w, o);
  }
  if (r0 == 0) {
    xin[ds + 4 * cq] = c.x * inv;
    xin[ds + 4 * cq + 1] = c.y * inv;
    xin[ds + 4 * cq + 2] = c.z * inv;
    xin[ds + 4 * cq + 3] = c.w * inv;
  }
  rt_tail<DM>(a, t, lane, xin, wc, wnr);
}

// The memory step in its history form, for a forward pass that runs every routed block in
// order from S_0 = 0, zeta_0 = 0 (the fused stack and the decoder forward).  Unrolling Eq. 12,
//   S_{j-1} = sum_{i<j} w_ji phi(k_i) v_i^T,  zeta_{j-1} = sum_{i<j} w_ji phi(k_i),
//   w_ji = rho_{i+1} ... rho_{j-1}  (1 for i = j - 1),
// so Eq. 11's read is c = sum_i w_ji s_i v_i / (sum_i w_ji s_i + eps) with s_i = phi(q).phi(k_i):
// the same quantity in exact arithmetic, computed from the token's earlier (phi(k_i), v_i)
// (2 d_m floats per routed block) instead of its d_m x d_m state.  Block j appends its own
// pair.  One warp per token; lane owns elements EL lane .. EL lane + EL - 1 of each vector;
// history entries are taken in order (bitwise reproducible).
template <int DM>
__global__ void __launch_bounds__(256) k_rt_hist(const RouterTcArgs a) {
  static_assert(DM % 64 == 0 && DM <= 128, "two or four elements per lane");
  constexpr int EL = DM / 32;
  __shared__ float xin_s[8][kRtMaxF];
  pdl_enter();
  const float* wc = a.w.w_c_t;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t = blockIdx.x * 8 + w;
  if (t >= a.T) return;   // whole warps only; nothing below synchronises the CTA
  float* xin = xin_s[w];
  const float* q = a.qkvn + (size_t)t * 4 * DM;
  const float* k = q + DM;
  const float* v = q + 2 * DM;
  const float* wn = q + 3 * DM;   // W_n s
  float wnr[(DM + 31) / 32];
  rt_tail_load<DM>(a, t, lane, xin, wn, wnr);
  const int ds = a.d_h + a.d_a;
  float fq[EL], fk[EL], vv[EL];
#pragma unroll
  for (int e = 0; e < EL; ++e) {
    const int m = lane * EL + e;
    fq[e] = phif_(q[m]);
    fk[e] = phif_(k[m]);
    vv[e] = v[m];
  }
  float* H = a.hist + (size_t)t * a.hist_ld;   // entry i: phi(k_i) [DM] | v_i [DM]
  const float* wj = a.hw + (size_t)(a.j - 1) * a.L;
  const int nh = a.j - 1;
  float c[EL], den = 0.f;
#pragma unroll
  for (int e = 0; e < EL; ++e) c[e] = 0.f;
  constexpr int HB = 8;   // entries per batch of loads
#pragma unroll 1
  for (int i0 = 0; i0 < nh; i0 += HB) {
    float hk[HB][EL], hv[HB][EL];
#pragma unroll
    for (int u = 0; u < HB; ++u)
#pragma unroll
      for (int e = 0; e < EL; ++e) {
        const bool in = i0 + u < nh;
        hk[u][e] = in ? H[(size_t)(i0 + u) * 2 * DM + lane * EL + e] : 0.f;
        hv[u][e] = in ? H[(size_t)(i0 + u) * 2 * DM + DM + lane * EL + e] : 0.f;
      }
#pragma unroll
    for (int u = 0; u < HB; ++u) {
      if (i0 + u >= nh) break;   // warp-uniform
      float sp = 0.f;
#pragma unroll
      for (int e = 0; e < EL; ++e) sp = fmaf(fq[e], hk[u][e], sp);
      const float ws = __ldg(wj + i0 + u) * warp_sum(sp);
      den += ws;
#pragma unroll
      for (int e = 0; e < EL; ++e) c[e] = fmaf(ws, hv[u][e], c[e]);
    }
  }
  const float inv = 1.0f / (den + a.eps);
  float* Hj = H + (size_t)nh * 2 * DM;   // this block's entry
#pragma unroll
  for (int e = 0; e < EL; ++e) {
    xin[ds + lane * EL + e] = c[e] * inv;
    Hj[lane * EL + e] = fk[e];
    Hj[DM + lane * EL + e] = vv[e];
  }
  rt_tail<DM>(a, t, lane, xin, wc, wnr);
}

}  // namespace

cudaError_t launch_rt_mem(const RouterTcArgs& a, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  const dim3 grid((a.T + 7) / 8);
  switch (a.dm) {
    case 16: return launch_pdl(k_rt_mem<16>, grid, dim3(256), 0, st, a);
    case 32: return launch_pdl(k_rt_mem<32>, grid, dim3(256), 0, st, a);
    case 64: return launch_pdl(k_rt_mem<64>, grid, dim3(256), 0, st, a);
    case 128: return launch_pdl(k_rt_mem<128>, grid, dim3(256), 0, st, a);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_rt_hist(const RouterTcArgs& a, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  if (!a.hist || !a.hw || a.j < 1 || a.j > a.L || a.hist_ld < (long)a.L * 2 * a.dm)
    return cudaErrorInvalidValue;
  const dim3 grid((a.T + 7) / 8);
  switch (a.dm) {
    case 64: return launch_pdl(k_rt_hist<64>, grid, dim3(256), 0, st, a);
    case 128: return launch_pdl(k_rt_hist<128>, grid, dim3(256), 0, st, a);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace hero
