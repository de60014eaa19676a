// The router of one routed block (Sec. 3.2: Eqs. 4-16, the encoders, the memory read and
// write, the heads, the gate and the decision) at small and medium token counts, one launch
// per block.  The router's parameters (about 134 KB of bf16 matrices for d_m = 64: W_hu,
// [W_q; W_k; W_v; W_n], W_c, W_th1, plus the fp32 vectors) are staged in shared memory by
// four bulk copies per CTA, issued before the kernel waits on its predecessor; each CTA then
// runs TB tokens (1 to 16: as many CTAs as the token count allows, up to one per SM) through
// phases that read only shared memory, separated by CTA barriers:
//   1 per-token scalars from the previous block's partial sums (rinv, d_j, gamma; Eqs. 7-8)
//   2 the router contraction's output: encoder input SiLU(rinv y) and f_psi's logit b
//   3 z_h = W_hu enc (Eq. 5) beside the path encoder (Eqs. 4, 6, 9): s = [z_h; z_a]
//   4 q | k | v | W_n s (Eqs. 10, 13)
//   5 memory read (Eq. 11) fused with the write (Eq. 12), S read and written once
//   6 nu = 1 - cos(W_n s, W_c c) (Eq. 13)
//   7 f_theta's hidden layer SiLU(W_th1 [s; c; nu] + b)
//   8-9 a (Eq. 14), p_hist, m_hist (Eq. 15), g (Eq. 16), the decision (Eq. 3)
// Each matrix-vector phase gives a thread two adjacent outputs (one 32-bit load of a bf16
// pair per input) over a fixed slice of the inputs for all TB tokens; the slices' partial
// sums are added in slice order, so results are bitwise reproducible.
#include "hero_device.cuh"

namespace hero {
namespace {

constexpr int kThr = 256;   // threads per CTA

template <int DM, int TB>
struct RsmAct {   // fp32 activations after the blob, offsets in floats; rows are [..][TB]
  static constexpr int F = RsmBlob<DM>::F;
  static constexpr int enc = 0;                          // [256] encoder input, then f_theta hidden
  static constexpr int sv = enc + kRsmEnc * TB;          // [F] s | c | nu
  static constexpr int x = sv + (F * TB + 3) / 4 * 4;    // [8] path features (6 used)
  static constexpr int ph = x + 8 * TB;                  // [16] path hidden
  static constexpr int q4 = ph + kRsmPath * TB;          // [4 DM] q | k | v | W_n s
  static constexpr int cv = q4 + 4 * DM * TB;            // [DM] W_c c
  static constexpr int scr = cv + DM * TB;               // [512] partial sums of a phase
  static constexpr int red = scr + 512 * TB;             // [8 warps] per-warp sums
  static constexpr int sc = red + 8 * TB;                // [TB][4] rinv, d_j, m_prev, den
  static constexpr int ab = sc + 4 * TB;                 // [2] a | b
  static constexpr int floats = ab + 2 * TB;
};

constexpr int kBlobAt = 128;   // mbarriers and the abort flag below, the blob from here

template <int DM, int TB>
constexpr size_t rsm_smem_bytes() {
  return kBlobAt + RsmBlob<DM>::bytes + sizeof(float) * RsmAct<DM, TB>::floats;
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                         uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(dst), "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// Partial products of one phase: thread (op, ks), op < NO / 2, ks < KS, sums inputs
// [ks kc, (ks + 1) kc) of outputs 2 op and 2 op + 1 for the TB tokens into
// P[(ks NO + o) TB + t].  W is [NI][NO] bf16 (pairs of outputs as one 32-bit word), X is
// [NI][TB] fp32.
template <int TB, int NO, int KS>
__device__ __forceinline__ void mv_part(const uint32_t* __restrict__ W, int NI,
                                        const float* __restrict__ X, float* __restrict__ P,
                                        int tid) {
  constexpr int NP = NO / 2;
  static_assert(NP * KS <= kThr, "one work item per thread");
  if (tid >= NP * KS) return;
  const int op = tid % NP, ks = tid / NP;
  const int kc = (NI + KS - 1) / KS;
  const int k0 = ks * kc, k1 = min(NI, k0 + kc);
  float a0[TB], a1[TB];
#pragma unroll
  for (int t = 0; t < TB; ++t) a0[t] = a1[t] = 0.f;
#pragma unroll 2
  for (int k = k0; k < k1; ++k) {
    const uint32_t w = W[k * NP + op];
    const float w0 = __uint_as_float(w << 16), w1 = __uint_as_float(w & 0xffff0000u);
    float xv[TB];
    if constexpr (TB % 4 == 0) {
#pragma unroll
      for (int q = 0; q < TB / 4; ++q) {
        const float4 v = *reinterpret_cast<const float4*>(X + k * TB + 4 * q);
        xv[4 * q] = v.x;
        xv[4 * q + 1] = v.y;
        xv[4 * q + 2] = v.z;
        xv[4 * q + 3] = v.w;
      }
    } else {
#pragma unroll
      for (int t = 0; t < TB; ++t) xv[t] = X[k * TB + t];
    }
#pragma unroll
    for (int t = 0; t < TB; ++t) {
      a0[t] = fmaf(w0, xv[t], a0[t]);
      a1[t] = fmaf(w1, xv[t], a1[t]);
    }
  }
#pragma unroll
  for (int t = 0; t < TB; ++t) {
    P[(ks * NO + 2 * op) * TB + t] = a0[t];
    P[(ks * NO + 2 * op + 1) * TB + t] = a1[t];
  }
}

// out[o][t] = act(sum over ks of P, in ks order, + bias[o]) for the phase's NO x TB outputs.
template <int TB, int NO, int KS, bool SILU>
__device__ __forceinline__ void mv_finish(const float* __restrict__ P, const float* bias,
                                          float* __restrict__ out, int tid) {
  for (int e = tid; e < NO * TB; e += kThr) {
    float v = 0.f;
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) v += P[ks * NO * TB + e];
    if (bias) v += bias[e / TB];
    out[e] = SILU ? siluf_(v) : v;
  }
}

template <int DM, int TB>
__global__ void __launch_bounds__(kThr, 1) k_router_sm(const RouterArgs a) {
  using B = RsmBlob<DM>;
  using A = RsmAct<DM, TB>;
  constexpr int F = B::F;
  extern __shared__ __align__(128) unsigned char smraw[];
  uint64_t* bars = reinterpret_cast<uint64_t*>(smraw);   // 4 mbarriers, one per blob part
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smraw + 64);
  unsigned char* blob = smraw + kBlobAt;
  float* act = reinterpret_cast<float*>(smraw + kBlobAt + B::bytes);
  const uint32_t* w_hu = reinterpret_cast<const uint32_t*>(blob + B::hu);
  const uint32_t* w_q4 = reinterpret_cast<const uint32_t*>(blob + B::q4);
  const uint32_t* w_c = reinterpret_cast<const uint32_t*>(blob + B::wc);
  const uint32_t* w_t1 = reinterpret_cast<const uint32_t*>(blob + B::t1);
  const float* vf = reinterpret_cast<const float*>(blob + B::f32);
  float* enc = act + A::enc;
  float* sv = act + A::sv;
  float* xf = act + A::x;
  float* ph = act + A::ph;
  float* q4 = act + A::q4;
  float* cv = act + A::cv;
  float* scr = act + A::scr;
  float* red = act + A::red;
  float* sc = act + A::sc;
  float* ab = act + A::ab;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t0 = blockIdx.x * TB;
  const int nvalid = min(TB, a.T - t0);

  // 0. the blob (model parameters, written before any launch) in four parts, each on its
  //    own mbarrier, and this CTA's memory rows into L2, all before the wait on the
  //    previous launch
  if (tid == 0) {
    for (int i = 0; i < 4; ++i) mbar_init(smem_u32(&bars[i]), 1);
    fence_mbar_init();
    *abort_flag = 0;
    const char* g = static_cast<const char*>(a.wsm);
    const uint32_t s0 = smem_u32(blob);
    mbar_arrive_expect_tx(smem_u32(&bars[0]), B::q4 + (B::bytes - B::f32));
    bulk_g2s(s0 + B::hu, g + B::hu, B::q4 - B::hu, smem_u32(&bars[0]));
    bulk_g2s(s0 + B::f32, g + B::f32, B::bytes - B::f32, smem_u32(&bars[0]));
    mbar_arrive_expect_tx(smem_u32(&bars[1]), B::wc - B::q4);
    bulk_g2s(s0 + B::q4, g + B::q4, B::wc - B::q4, smem_u32(&bars[1]));
    mbar_arrive_expect_tx(smem_u32(&bars[2]), B::t1 - B::wc);
    bulk_g2s(s0 + B::wc, g + B::wc, B::t1 - B::wc, smem_u32(&bars[2]));
    mbar_arrive_expect_tx(smem_u32(&bars[3]), B::f32 - B::t1);
    bulk_g2s(s0 + B::t1, g + B::t1, B::f32 - B::t1, smem_u32(&bars[3]));
    const char* Sb = reinterpret_cast<const char*>(a.S + (size_t)t0 * DM * DM);
    for (int i = 0; i < nvalid; ++i) prefetch_l2(Sb + (size_t)i * DM * DM * 4, DM * DM * 4);
  }
  // Blob part i present: every thread waits on its mbarrier (bounded); on expiry the CTA
  // records the error, drains the copies in flight and returns (a uniform decision, taken
  // after the barrier that follows).
  auto wait_part = [&](int i) {
    if (!mbar_wait(smem_u32(&bars[i]), 0, a.wait_ns)) *abort_flag = 1;
  };
  auto aborted = [&]() -> bool {
    if (!*abort_flag) return false;
    if (tid == 0) {
      atomicOr(a.err, ERR_WAIT_PRODUCER);
      for (int i = 0; i < 4; ++i)
        if (!mbar_wait(smem_u32(&bars[i]), 0, kDrainLimitNs)) atomicOr(a.err, ERR_WAIT_DRAIN);
    }
    return true;
  };
  __syncthreads();   // barrier initialisation visible to every waiting thread
  pdl_enter();

  // 1. per-token scalars from the partial sums of the previous block's epilogue
  for (int tl = warp; tl < TB; tl += kThr / 32) {
    const int t = t0 + tl;
    float ss = 0.f, dd = 0.f, dp = 0.f;
    if (t < a.T)
      for (int s = lane; s < a.np; s += 32) {
        const float4 v = *reinterpret_cast<const float4*>(a.part + ((size_t)t * a.np + s) * 4);
        ss += v.x;
        dd += v.y;
        dp += v.z;
      }
    ss = warp_sum(ss);
    dd = warp_sum(dd);
    dp = warp_sum(dp);
    if (lane == 0) {
      float dprev = 0.f, pp = 1.f, mp = 1.f;
      if (t < a.T) {
        dprev = a.dprev[t];
        pp = a.pst[t];
        mp = a.mst[t];
      }
      const float rinv = rsqrtf(ss / (float)a.d + a.rms_eps);
      const float dj = a.j == 1 ? 0.f : sqrtf(dd);                    // Eq. 7
      const float gam = a.j > 2 ? dp / (dj * dprev + a.eps) : 0.f;    // Eq. 8
      sc[tl * 4 + 0] = rinv;
      sc[tl * 4 + 1] = dj;
      sc[tl * 4 + 2] = mp;
      xf[0 * TB + tl] = (float)a.j / (float)a.L;
      xf[1 * TB + tl] = (float)(a.L - a.j) / (float)a.L;
      xf[2 * TB + tl] = dj;
      xf[3 * TB + tl] = gam;
      xf[4 * TB + tl] = pp;
      xf[5 * TB + tl] = mp;
    }
  }
  __syncthreads();

  // 2. thread tid takes columns 2 tid, 2 tid + 1 of the contraction's 512 (split-K slices
  //    added in slice order): encoder input SiLU(rinv y) below 256, f_psi's hidden
  //    SiLU(y + b_1) dotted with w_2 above (Eq. 16).  The loads are issued before the wait
  //    on the blob's first part (f_psi's vectors).
  {
    const int c0 = 2 * tid;
    float2 y[TB];
#pragma unroll
    for (int tl = 0; tl < TB; ++tl) y[tl] = make_float2(0.f, 0.f);
    const long sstride = a.y_split_stride / 2;
    const int yr = a.y_rows > 1 ? 2 : 1;   // rows per token (the stacked operand pair)
    const int parts = a.y_splits * yr;     // part p: slice p / yr, row p % yr of the token
    // SB parts x TB tokens of loads in flight before they are added (in part order)
    constexpr int SB = TB >= 8 ? 1 : 16 / TB;
    for (int p0 = 0; p0 < parts; p0 += SB) {
      float2 v[SB][TB];
#pragma unroll
      for (int i = 0; i < SB; ++i)
#pragma unroll
        for (int tl = 0; tl < TB; ++tl) {
          const int p = p0 + i;
          v[i][tl] = p < parts && tl < nvalid
                         ? __ldg(reinterpret_cast<const float2*>(
                                     a.Y + ((size_t)(t0 + tl) * yr + p % yr) * 512) +
                                 (p / yr) * sstride + tid)
                         : make_float2(0.f, 0.f);
        }
#pragma unroll
      for (int i = 0; i < SB; ++i)
#pragma unroll
        for (int tl = 0; tl < TB; ++tl) {
          y[tl].x += v[i][tl].x;
          y[tl].y += v[i][tl].y;
        }
    }
    wait_part(0);
    __syncthreads();
    if (aborted()) return;
    if (c0 < kRsmEnc) {
#pragma unroll
      for (int tl = 0; tl < TB; ++tl) {
        const float r = sc[tl * 4];
        enc[c0 * TB + tl] = siluf_(y[tl].x * r);
        enc[(c0 + 1) * TB + tl] = siluf_(y[tl].y * r);
      }
    } else {
      const int e = c0 - kRsmEnc;
      const float w0 = vf[B::psw2 + e], w1 = vf[B::psw2 + e + 1];
      const float b0 = vf[B::psb1 + e], b1 = vf[B::psb1 + e + 1];
#pragma unroll
      for (int tl = 0; tl < TB; ++tl) {
        float v = w0 * siluf_(y[tl].x + b0);
        v = fmaf(w1, siluf_(y[tl].y + b1), v);
        v = warp_sum(v);
        if (lane == 0) red[(warp - 4) * TB + tl] = v;
      }
    }
  }
  __syncthreads();
  if (tid < TB) ab[TB + tid] = ((red[tid] + red[TB + tid]) + red[2 * TB + tid]) + red[3 * TB + tid];

  // 3. z_h = W_hu enc -> s[0, 48) on warps 0-5; the path encoder on warps 6-7:
  //    SiLU(W_1 x + b_1), then z_a = W_2 (.) + b_2 -> s[48, 64)
  if (tid < 192) {
    mv_part<TB, kRsmDh, 8>(w_hu, kRsmEnc, enc, scr, tid);
  } else {
    const int g = tid - 192;
    for (int e = g; e < kRsmPath * TB; e += 64) {
      const int o = e / TB, tl = e - o * TB;
      float v = 0.f;
#pragma unroll
      for (int i = 0; i < 6; ++i) v = fmaf(vf[B::p1 + i * kRsmPath + o], xf[i * TB + tl], v);
      ph[e] = siluf_(v + vf[B::pb1 + o]);
    }
    asm volatile("bar.sync 1, 64;" ::: "memory");
    for (int e = g; e < kRsmDa * TB; e += 64) {
      const int o = e / TB, tl = e - o * TB;
      float v = 0.f;
#pragma unroll
      for (int i = 0; i < kRsmPath; ++i) v = fmaf(vf[B::p2 + i * kRsmDa + o], ph[i * TB + tl], v);
      sv[(kRsmDh + o) * TB + tl] = v + vf[B::pb2 + o];
    }
  }
  __syncthreads();
  mv_finish<TB, kRsmDh, 8, false>(scr, nullptr, sv, tid);
  wait_part(1);
  __syncthreads();
  if (aborted()) return;

  // 4. q | k | v | W_n s
  constexpr int KS4 = kThr / (2 * DM) < 8 ? kThr / (2 * DM) : 8;
  mv_part<TB, 4 * DM, KS4>(w_q4, kRsmDs, sv, scr, tid);
  __syncthreads();
  mv_finish<TB, 4 * DM, KS4, false>(scr, nullptr, q4, tid);
  __syncthreads();

  // 5. memory read fused with the write.  Unit (token, sub) of a warp covers RW rows of the
  //    token's S: a lane owns a float4 column group of every RPI-th row; its partial c goes
  //    to scr [TB][WPT][DM] and sub 0 also takes den = phi(q) . zeta and the zeta update.
  {
    constexpr int LPR = DM / 4, RPI = 32 / LPR;
    constexpr int WA = 8 / TB > 0 ? 8 / TB : 1;
    constexpr int WB = DM * DM / 128 > 0 ? DM * DM / 128 : 1;
    constexpr int WPT = WA < WB ? WA : WB;   // warps per token
    constexpr int RW = DM / WPT;             // rows per unit
    constexpr int NI = RW / RPI;             // rows per lane
    constexpr int BATCH = NI < 16 ? NI : 16;
    static_assert(RW % RPI == 0 && NI % BATCH == 0, "whole row iterations per unit");
    for (int u = warp; u < TB * WPT; u += kThr / 32) {
      const int tl = u / WPT, sub = u - tl * WPT;
      const int t = t0 + tl;
      if (t >= a.T) continue;
      const float* qc = q4 + tl;                // q[r] = qc[r TB]
      const float* kc = q4 + DM * TB + tl;
      const float* vc = q4 + 2 * DM * TB + tl;
      if (sub == 0) {
        float* z = a.zeta + (size_t)t * DM;
        float den = 0.f;
        for (int m = lane; m < DM; m += 32) {
          const float zo = z[m];
          den += phif_(qc[m * TB]) * zo;
          z[m] = a.rho * zo + phif_(kc[m * TB]);
        }
        den = warp_sum(den);
        if (lane == 0) sc[tl * 4 + 3] = den;
      }
      float* S = a.S + (size_t)t * DM * DM;
      const int cq = lane % LPR, r0 = lane / LPR;
      const float4 vv = make_float4(vc[(4 * cq) * TB], vc[(4 * cq + 1) * TB], vc[(4 * cq + 2) * TB],
                                    vc[(4 * cq + 3) * TB]);
      float4 c = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 1
      for (int i0 = 0; i0 < NI; i0 += BATCH) {
        float4 so[BATCH];
#pragma unroll
        for (int i = 0; i < BATCH; ++i)
          so[i] = *reinterpret_cast<const float4*>(S + (sub * RW + r0 + (i0 + i) * RPI) * DM + 4 * cq);
#pragma unroll
        for (int i = 0; i < BATCH; ++i) {
          const int r = sub * RW + r0 + (i0 + i) * RPI;
          const float fq = phif_(qc[r * TB]), fk = phif_(kc[r * TB]);
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
      if (r0 == 0) *reinterpret_cast<float4*>(scr + (tl * WPT + sub) * DM + 4 * cq) = c;
    }
    __syncthreads();
    for (int e = tid; e < TB * DM; e += kThr) {
      const int tl = e / DM, col = e - tl * DM;
      float v = 0.f;
      if (tl < nvalid) {
#pragma unroll
        for (int sub = 0; sub < WPT; ++sub) v += scr[(tl * WPT + sub) * DM + col];
        v /= sc[tl * 4 + 3] + a.eps;
      }
      sv[(kRsmDs + col) * TB + tl] = v;
    }
  }
  wait_part(2);
  __syncthreads();
  if (aborted()) return;

  // 6. nu = 1 - cos(W_n s, W_c c) for j > 1; nu_1 = 0
  float* nuv = sv + (kRsmDs + DM) * TB;
  if (a.j > 1) {
    constexpr int KSC = kThr / (DM / 2) < 8 ? kThr / (DM / 2) : 8;
    mv_part<TB, DM, KSC>(w_c, DM, sv + kRsmDs * TB, scr, tid);
    __syncthreads();
    mv_finish<TB, DM, KSC, false>(scr, nullptr, cv, tid);
    __syncthreads();
    for (int tl = warp; tl < TB; tl += kThr / 32) {
      float xy = 0.f, xx = 0.f, yy = 0.f;
      for (int i = lane; i < DM; i += 32) {
        const float u = q4[(3 * DM + i) * TB + tl], w = cv[i * TB + tl];
        xy += u * w;
        xx += u * u;
        yy += w * w;
      }
      xy = warp_sum(xy);
      xx = warp_sum(xx);
      yy = warp_sum(yy);
      if (lane == 0) nuv[tl] = 1.f - xy / (sqrtf(xx) * sqrtf(yy) + a.eps);
    }
  } else if (tid < TB) {
    nuv[tid] = 0.f;
  }
  wait_part(3);
  __syncthreads();
  if (aborted()) return;

  // 7. f_theta hidden = SiLU(W_th1 [s; c; nu] + b_1) -> the encoder input's rows
  mv_part<TB, kRsmHead, 2>(w_t1, F, sv, scr, tid);
  __syncthreads();
  mv_finish<TB, kRsmHead, 2, true>(scr, vf + B::tb1, enc, tid);
  __syncthreads();

  // 8. a = w_2 . hidden (Eq. 14): thread tid holds hidden unit tid of every token
  {
    const float w2 = vf[B::tw2 + tid];
#pragma unroll
    for (int tl = 0; tl < TB; ++tl) {
      const float v = warp_sum(w2 * enc[tid * TB + tl]);
      if (lane == 0) red[warp * TB + tl] = v;
    }
  }
  __syncthreads();

  // 9. history score, cumulative score, gate and decision
  if (tid < nvalid) {
    const int t = t0 + tid;
    float sa = 0.f;
#pragma unroll
    for (int w = 0; w < kThr / 32; ++w) sa += red[w * TB + tid];
    const float av = sa + vf[B::tb2];
    const float bv = ab[TB + tid] + vf[B::psb2];
    const float p = sigmoidf_(av / a.t_hist);     // Eq. 14
    const float m = sc[tid * 4 + 2] * p;          // Eq. 15
    const float g = sigmoidf_(av + bv);           // Eq. 16
    uint8_t dec;
    if (a.mask_in)
      dec = a.mask_in[t] ? 1 : 0;
    else
      dec = g >= a.tau ? 1 : 0;                   // Eq. 3 (ties run the FFN)
    a.pst[t] = p;
    a.mst[t] = m;
    a.dprev[t] = sc[tid * 4 + 1];
    a.gate[t] = g;
    a.mask[t] = dec;
    if (a.gate_out) a.gate_out[t] = g;
    if (a.mask_out) a.mask_out[t] = dec;
  }
}

template <int DM, int TB>
cudaError_t launch_tb(const RouterArgs& a, cudaStream_t st) {
  constexpr size_t smem = rsm_smem_bytes<DM, TB>();
  static_assert(smem <= 232448, "shared memory per CTA");
  static bool attr = false;
  if (!attr) {
    const cudaError_t e =
        cudaFuncSetAttribute(k_router_sm<DM, TB>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  return launch_pdl(k_router_sm<DM, TB>, dim3((a.T + TB - 1) / TB), dim3(kThr), smem, st, a);
}

template <int DM>
cudaError_t launch_dm(const RouterArgs& a, int num_sms, cudaStream_t st) {
  auto ctas = [&](int tb) { return (a.T + tb - 1) / tb; };
  if (ctas(1) <= num_sms) return launch_tb<DM, 1>(a, st);
  if (ctas(2) <= num_sms) return launch_tb<DM, 2>(a, st);
  if (ctas(4) <= num_sms) return launch_tb<DM, 4>(a, st);
  if (ctas(8) <= num_sms) return launch_tb<DM, 8>(a, st);
  return launch_tb<DM, 16>(a, st);
}

}  // namespace

bool router_sm_supported(int d_enc, int d_head, int d_h, int d_a, int d_path, int d_m) {
  return d_enc == kRsmEnc && d_head == kRsmHead && d_h == kRsmDh && d_a == kRsmDa &&
         d_path == kRsmPath && (d_m == 16 || d_m == 32 || d_m == 64);
}

size_t router_sm_blob_bytes(int d_m) {
  switch (d_m) {
    case 16: return RsmBlob<16>::bytes;
    case 32: return RsmBlob<32>::bytes;
    case 64: return RsmBlob<64>::bytes;
    default: return 0;
  }
}

cudaError_t launch_router_sm(int d_m, const RouterArgs& a, int num_sms, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  if (!a.wsm || a.variant != 0 || a.d_enc + a.d_head != 512) return cudaErrorInvalidValue;
  switch (d_m) {
    case 16: return launch_dm<16>(a, num_sms, st);
    case 32: return launch_dm<32>(a, num_sms, st);
    case 64: return launch_dm<64>(a, num_sms, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace hero
