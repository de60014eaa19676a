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
  pdl_enter();
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
    store_xl4(a.xl, a.xl_bf16, a.d, t, n, h);
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
// k_block_entry: one warp per token, for one routed block run on its own.
// delta_j = h_bar_j - h_bar_{j-1} (Eq. 7, zero for j = 1); partial sums
// (sum h_bar^2, sum delta^2, sum delta . delta_{j-1}) into slot 0; the router's
// operand copy of h_bar; then the carried h_bar_prev / delta_prev become this
// block's (each element is read before it is overwritten by the same lane).
// ------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_block_entry(const BlockEntryArgs a) {
  pdl_enter();
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= a.T) return;
  const int t = warp;
  const size_t row = (size_t)t * a.d;
  float ss = 0.f, dd = 0.f, dp = 0.f;
  for (int n = lane * 4; n < a.d; n += 128) {
    const float4 h = *reinterpret_cast<const float4*>(a.h_bar + row + n);
    float4 dl = make_float4(0.f, 0.f, 0.f, 0.f);
    if (a.router) {
      if (a.j > 1) {
        const float4 hp = *reinterpret_cast<const float4*>(a.h_bar_prev + row + n);
        dl = make_float4(h.x - hp.x, h.y - hp.y, h.z - hp.z, h.w - hp.w);
      }
      if (a.j > 2) {
        const float4 dv = *reinterpret_cast<const float4*>(a.delta_prev + row + n);
        dp += dl.x * dv.x + dl.y * dv.y + dl.z * dv.z + dl.w * dv.w;
      }
      dd += dl.x * dl.x + dl.y * dl.y + dl.z * dl.z + dl.w * dl.w;
      *reinterpret_cast<float4*>(a.h_bar_prev + row + n) = h;
      *reinterpret_cast<float4*>(a.delta_prev + row + n) = dl;
      store_xl4(a.xl, a.xl_bf16, a.d, t, n, h);
    }
    ss += h.x * h.x + h.y * h.y + h.z * h.z + h.w * h.w;
  }
  ss = warp_sum(ss);
  dd = warp_sum(dd);
  dp = warp_sum(dp);
  for (int s = lane; s < a.np; s += 32)
    *reinterpret_cast<float4*>(a.part + ((size_t)t * a.np + s) * 4) =
        s == 0 ? make_float4(ss, dd, dp, 0.f) : make_float4(0.f, 0.f, 0.f, 0.f);
}

// Router state reset for a new forward pass (S = 0, zeta = 0, p = m = 1, d_prev = 0).
__global__ void __launch_bounds__(256) k_state_reset(float* S, float* zeta, float* pst, float* mst,
                                                     float* dprev, int T, int dm) {
  pdl_enter();
  const long n_s = (long)T * dm * dm;
  for (long i = (long)blockIdx.x * blockDim.x + threadIdx.x; i < n_s; i += (long)gridDim.x * blockDim.x) {
    S[i] = 0.f;
    if (i < (long)T * dm) zeta[i] = 0.f;
    if (i < T) {
      pst[i] = 1.f;
      mst[i] = 1.f;
      dprev[i] = 0.f;
    }
  }
}

// ------------------------------------------------------------------------------
// k_router: TB tokens per CTA.  Activations live in shared memory transposed,
// [feature][TB], so a block matmul loads one float4 of weights (four outputs) and
// one float4 of activations (four tokens) per 16 FMAs.
// ------------------------------------------------------------------------------
// Tokens per CTA: 16 for large token counts, 4 when T/16 CTAs would not fill the
// GPU twice over (decode and short prefill), where the per-CTA chain of dependent
// phases is the critical path and the head matmuls split K more widely.
constexpr int TB_LARGE = 16, TB_SMALL = 4;
// Threads per CTA: 256 with 16 tokens; 1024 with 4 tokens, where each phase's split-K
// and per-token reductions spread over four times the threads to shorten the chain.
template <int TB>
constexpr int nthr() { return TB < 16 ? 1024 : 256; }

// Shared-memory layout (floats), computed from the model's widths on host and
// device alike.  Regions are reused once their contents are dead:
//   big   [max(d_enc, d_head)][TB]: encoder input (steps 2-3), split-K scratch of
//         W_n / W_c (step 6), f_theta hidden (steps 7-8)
//   s     [d_s + d_m + 1][TB]: s | c | nu
//   qkv   [TB][3 d_m] token-major
//   aux   [max(3072, 2 d_m TB)]: split-K scratch of W_hu (step 3), W_n s | W_c c (step 6)
template <int TB>
struct RouterLayout {
  int big, s, qkv, aux, x, ph, red, sc, ab, sk, floats;
  // sk: split-K scratch of q/k/v and f_theta (small TB only; with TB = 16 those
  // products have enough output tiles to occupy every thread without a split)
  static constexpr int kSplitScratch = TB < 16 ? 16384 : 0;
  __host__ __device__ RouterLayout(int d_enc, int d_head, int ds, int dm, int d_path) {
    const int nbig = (d_enc > d_head ? d_enc : d_head) * TB;
    const int ns = ((ds + dm + 1 + 3) & ~3) * TB;
    const int naux = (3072 > 2 * dm * TB ? 3072 : 2 * dm * TB);
    big = 0;
    s = big + nbig;
    qkv = s + ns;
    aux = qkv + TB * 3 * dm;
    x = aux + naux;
    ph = x + 8 * TB;
    red = ph + d_path * TB;
    sc = red + 3 * nthr<TB>();
    ab = sc + TB * 16;
    sk = ab + 2 * TB;
    floats = sk + kSplitScratch;
  }
};

// out[o][t] = sum_i Wt[i][o] in[i][t]  (+ bias[o], then optional SiLU), o < NO,
// t < TB; `in` is [NI][TB]; `out` is [NO][TB] or, if out_tok_ld > 0, token-major
// [TB][out_tok_ld].  Narrow outputs split K across threads; the partial sums go to
// `scratch` ([ks][NO][TB], at most scratch_cap floats) and are added in a fixed
// order, so results are bitwise reproducible.  NO must be a multiple of 4.  Run by the
// gn threads from g0 (default: the whole CTA), which it synchronises: __syncthreads for
// the whole CTA, else the named barrier `bar` (two groups may run concurrently).
__device__ __forceinline__ void group_sync(int bar, int gn) {
  if (bar == 0)
    __syncthreads();
  else
    asm volatile("bar.sync %0, %1;" ::"r"(bar), "r"(gn) : "memory");
}

template <int TB>
__device__ void bmm4(const float* in, int NI, const float* __restrict__ Wt, int NO,
                     const float* __restrict__ bias, float* out, int out_tok_ld, bool silu_act,
                     float* scratch = nullptr, int scratch_cap = 0, int g0 = 0,
                     int gn = nthr<TB>(), int bar = 0) {
  const int no4 = NO >> 2;
  const int base = no4 * (TB / 4);
  const int gt = threadIdx.x - g0;   // index in the group
  int ks = 1;
  if (scratch)
    while (base * ks * 2 <= gn && NI / (ks * 2) >= (TB < 16 ? 8 : 16) &&
           (ks * 2) * NO * TB <= scratch_cap)
      ks <<= 1;
  const int kchunk = (NI + ks - 1) / ks;
  auto oidx = [&](int o, int t) { return out_tok_ld > 0 ? t * out_tok_ld + o : o * TB + t; };
  for (int w = gt; w < base * ks; w += gn) {
    const int o4 = (w % no4) * 4;
    const int rest = w / no4;
    const int t4 = (rest % (TB / 4)) * 4;
    const int kk = rest / (TB / 4);
    const int i0 = kk * kchunk;
    const int i1 = min(NI, i0 + kchunk);
    float acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;
#pragma unroll 4
    for (int i = i0; i < i1; ++i) {
      const float4 wv = __ldg(reinterpret_cast<const float4*>(Wt + (size_t)i * NO + o4));
      const float4 xv = *reinterpret_cast<const float4*>(in + i * TB + t4);
      const float wa[4] = {wv.x, wv.y, wv.z, wv.w};
      const float xb[4] = {xv.x, xv.y, xv.z, xv.w};
#pragma unroll
      for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(wa[a], xb[b], acc[a][b]);
    }
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        if (ks > 1) {
          scratch[(kk * NO + o4 + a) * TB + t4 + b] = acc[a][b];
        } else {
          float v = acc[a][b] + (bias ? __ldg(bias + o4 + a) : 0.f);
          out[oidx(o4 + a, t4 + b)] = silu_act ? siluf_(v) : v;
        }
      }
  }
  group_sync(bar, gn);
  if (ks > 1) {
    for (int e = gt; e < NO * TB; e += gn) {
      const int o = e / TB, t = e % TB;
      float v = 0.f;
      for (int kk = 0; kk < ks; ++kk) v += scratch[(kk * NO + o) * TB + t];
      v += bias ? __ldg(bias + o) : 0.f;
      out[oidx(o, t)] = silu_act ? siluf_(v) : v;
    }
    group_sync(bar, gn);
  }
}

// Within a warp, add the partials of the lanes that serve the same token (lane %
// TB) with a fixed shuffle tree; lanes < TB then hold the warp's sum per token.
template <int TB>
__device__ __forceinline__ float warp_part_sum(float v) {
#pragma unroll
  for (int o = TB; o < 32; o <<= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Sum the nthr<TB>() / TB per-thread partials of each token (thread tid holds a partial of
// token tid % TB): a shuffle tree inside each warp, then the warps' sums in warp
// order (fixed, so bitwise reproducible); contains __syncthreads.
template <int TB>
__device__ __forceinline__ void reduce16(float* red, float v, float* out) {
  v = warp_part_sum<TB>(v);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane < TB) red[warp * TB + lane] = v;
  __syncthreads();
  if (threadIdx.x < TB) {
    float s = 0.f;
    for (int w = 0; w < nthr<TB>() / 32; ++w) s += red[w * TB + threadIdx.x];
    out[threadIdx.x] = s;
  }
  __syncthreads();
}

// Memory read (Eq. 11) fused with the write (Eq. 12) for the CTA's TB tokens, one
// warp per token: c[n] = sum_m phi(q)_m S[m][n] / (phi(q) . zeta + eps), then
// S = rho S + phi(k) v^T and zeta = rho zeta + phi(k); S is read once and written
// once.  c goes to cT ([DM][TB], transposed).  DM <= 128: lane owns a 4-column
// group and every (32 / (DM/4))-th row, partial c summed over the lanes of a
// column group; DM = 256: lane owns column groups lane and lane + 32 over all
// rows (a warp instruction covers 512 contiguous bytes of one row).
template <int DM, int TB>
__device__ __forceinline__ void memory_read_write(const RouterArgs& a, const float* qkv, float* cT,
                                                  int t0, int warp, int lane) {
  for (int tl = warp; tl < TB; tl += nthr<TB>() / 32) {
    const int t = t0 + tl;
    if (t >= a.T) continue;
    const float* q = qkv + tl * 3 * DM;
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
    const float inv = 1.0f / (den + a.eps);
    if constexpr (DM <= 128) {
      constexpr int LPR = DM / 4;          // lanes per S row
      constexpr int RPI = 32 / LPR;        // rows per iteration
      constexpr int NIT = DM / RPI;        // S rows handled by this lane
      constexpr int BATCH = NIT < 8 ? NIT : 8;  // loads kept in flight
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
        float* cdst = cT + (4 * cq) * TB + tl;
        cdst[0 * TB] = c.x * inv;
        cdst[1 * TB] = c.y * inv;
        cdst[2 * TB] = c.z * inv;
        cdst[3 * TB] = c.w * inv;
      }
    } else {
      constexpr int NCG = DM / 128;        // column groups per lane
      constexpr int RB = 8;                // rows per batch: 64 KB of S in flight per CTA
      float4 c[NCG], vv[NCG];
#pragma unroll
      for (int i = 0; i < NCG; ++i) {
        c[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        vv[i] = *reinterpret_cast<const float4*>(v + 4 * (lane + 32 * i));
      }
#pragma unroll 1
      for (int r0 = 0; r0 < DM; r0 += RB) {
        float4 so[RB][NCG];
#pragma unroll
        for (int rr = 0; rr < RB; ++rr)
#pragma unroll
          for (int i = 0; i < NCG; ++i)
            so[rr][i] = *reinterpret_cast<const float4*>(S + (r0 + rr) * DM + 4 * (lane + 32 * i));
#pragma unroll
        for (int rr = 0; rr < RB; ++rr) {
          const float fq = phif_(q[r0 + rr]);
          const float fk = phif_(k[r0 + rr]);
#pragma unroll
          for (int i = 0; i < NCG; ++i) {
            const float4 x = so[rr][i];
            c[i].x += fq * x.x; c[i].y += fq * x.y; c[i].z += fq * x.z; c[i].w += fq * x.w;
            *reinterpret_cast<float4*>(S + (r0 + rr) * DM + 4 * (lane + 32 * i)) =
                make_float4(a.rho * x.x + fk * vv[i].x, a.rho * x.y + fk * vv[i].y,
                            a.rho * x.z + fk * vv[i].z, a.rho * x.w + fk * vv[i].w);
          }
        }
      }
#pragma unroll
      for (int i = 0; i < NCG; ++i) {
        float* cdst = cT + (4 * (lane + 32 * i)) * TB + tl;
        cdst[0 * TB] = c[i].x * inv;
        cdst[1 * TB] = c[i].y * inv;
        cdst[2 * TB] = c[i].z * inv;
        cdst[3 * TB] = c[i].w * inv;
      }
    }
  }
}

// Memory step at small token counts (every warp of the CTA busy): the nthr / 32 / TB
// warps of a token each take DM / WPT rows of its S, write them back updated and leave
// their partial read of c in scratch ([TB][WPT][DM]); warp 0 of a token also reads
// den = phi(q) . zeta and updates zeta, its den in scratch[TB WPT DM + token].
// memory_split_finish adds the partials in warp order once the CTA has synchronised.
template <int DM, int TB>
constexpr int mem_wpt() { return nthr<TB>() / 32 / TB; }

// The split memory step applies when every warp of a token gets whole row iterations.
template <int DM, int TB>
constexpr bool mem_split() {
  if (TB >= 16 || DM > 128) return false;
  constexpr int wpt = mem_wpt<DM, TB>() > 0 ? mem_wpt<DM, TB>() : 1;
  return mem_wpt<DM, TB>() > 0 && DM / wpt >= 32 / (DM / 4);
}

template <int DM, int TB>
__device__ __forceinline__ void memory_split(const RouterArgs& a, const float* qkv, float* scratch,
                                             int t0, int warp, int lane) {
  constexpr int WPT = mem_wpt<DM, TB>();
  constexpr int RW = DM / WPT;            // rows of S per warp
  constexpr int LPR = DM / 4;             // lanes per S row (float4 columns)
  constexpr int RPI = 32 / LPR;           // rows per iteration
  static_assert(RW % RPI == 0, "whole iterations per warp");
  const int tl = warp / WPT, sub = warp - tl * WPT;
  const int t = t0 + tl;
  if (tl >= TB || t >= a.T) return;
  const float* q = qkv + tl * 3 * DM;
  const float* k = q + DM;
  const float* v = q + 2 * DM;
  if (sub == 0) {
    float* z = a.zeta + (size_t)t * DM;
    float den = 0.f;
    for (int m = lane; m < DM; m += 32) {
      const float zo = z[m];
      den += phif_(q[m]) * zo;
      z[m] = a.rho * zo + phif_(k[m]);
    }
    den = warp_sum(den);
    if (lane == 0) scratch[TB * WPT * DM + tl] = den;
  }
  float* S = a.S + (size_t)t * DM * DM;
  const int cq = lane % LPR, r0 = lane / LPR;
  const float4 vv = *reinterpret_cast<const float4*>(v + 4 * cq);
  float4 so[RW / RPI];
#pragma unroll
  for (int i = 0; i < RW / RPI; ++i)
    so[i] = *reinterpret_cast<const float4*>(S + (sub * RW + r0 + i * RPI) * DM + 4 * cq);
  float4 c = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int i = 0; i < RW / RPI; ++i) {
    const int r = sub * RW + r0 + i * RPI;
    const float fq = phif_(q[r]), fk = phif_(k[r]);
    c.x += fq * so[i].x; c.y += fq * so[i].y; c.z += fq * so[i].z; c.w += fq * so[i].w;
    *reinterpret_cast<float4*>(S + r * DM + 4 * cq) =
        make_float4(a.rho * so[i].x + fk * vv.x, a.rho * so[i].y + fk * vv.y,
                    a.rho * so[i].z + fk * vv.z, a.rho * so[i].w + fk * vv.w);
  }
#pragma unroll
  for (int o = LPR; o < 32; o <<= 1) {
    c.x += __shfl_xor_sync(0xffffffffu, c.x, o);
    c.y += __shfl_xor_sync(0xffffffffu, c.y, o);
    c.z += __shfl_xor_sync(0xffffffffu, c.z, o);
    c.w += __shfl_xor_sync(0xffffffffu, c.w, o);
  }
  if (r0 == 0)
    *reinterpret_cast<float4*>(scratch + (tl * WPT + sub) * DM + 4 * cq) = c;
}

template <int DM, int TB>
__device__ __forceinline__ void memory_split_finish(const RouterArgs& a, const float* scratch,
                                                    float* cT, int t0) {
  constexpr int WPT = mem_wpt<DM, TB>();
  for (int e = threadIdx.x; e < TB * DM; e += nthr<TB>()) {
    const int tl = e / DM, col = e - tl * DM;
    if (t0 + tl >= a.T) continue;
    float c = 0.f;
#pragma unroll
    for (int sub = 0; sub < WPT; ++sub) c += scratch[(tl * WPT + sub) * DM + col];
    cT[col * TB + tl] = c / (scratch[TB * WPT * DM + tl] + a.eps);
  }
}

template <int DM, int TB>
__global__ void __launch_bounds__(nthr<TB>(), (DM >= 256 || TB < 16) ? 1 : 4) k_router(const RouterArgs a) {
  pdl_enter();
  extern __shared__ __align__(16) float sm[];
  const int ds = a.d_h + a.d_a;
  const RouterLayout<TB> lay(a.d_enc, a.d_head, ds, DM, a.d_path);
  float* skT = RouterLayout<TB>::kSplitScratch ? sm + lay.sk : nullptr;
  float* bigT = sm + lay.big;
  float* sT = sm + lay.s;      // rows [0, d_s) s, [d_s, d_s + DM) c, d_s + DM nu
  float* qkv = sm + lay.qkv;   // [TB][3 DM]
  float* aux = sm + lay.aux;
  float* xT = sm + lay.x;
  float* phT = sm + lay.ph;
  float* red = sm + lay.red;
  float* sc = sm + lay.sc;     // per token: 0 rinv, 1 d_j, 4 m_prev
  float* ab = sm + lay.ab;     // a[TB] | b[TB]
  const int t0 = blockIdx.x * TB;
  const int nY = a.d_enc + a.d_head;
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int nvalid = min(TB, a.T - t0);

  const bool no_history = a.variant & RV_NO_HISTORY;
  const bool no_memread = a.variant & RV_NO_MEMREAD;

  // 0. pull this CTA's memory block into L2 while the heads run (read in step 5)
  if (tid == 0 && !no_history && !no_memread) {
    const char* Sb = reinterpret_cast<const char*>(a.S + (size_t)t0 * DM * DM);
    const uint32_t bytes = (uint32_t)(DM * DM * sizeof(float));
    for (int i = 0; i < nvalid; ++i)
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(Sb + (size_t)i * bytes),
                   "r"(bytes)
                   : "memory");
  }

  // Thread tid serves token tl = tid % TB as part pt = tid / TB of nthr / TB in the
  // two input phases; the parts of a token are added in a fixed order.
  const int tl0 = tid % TB, pt0 = tid / TB;
  const int tok0 = t0 + tl0;

  // 1. per-token scalars from the partial sums of the previous block's epilogue;
  //    transition features (Eqs. 7-8) and the path vector (Eqs. 4, 6)
  {
    float ss = 0.f, dd = 0.f, dp = 0.f;
    if (tok0 < a.T)
      for (int s = pt0; s < a.np; s += nthr<TB>() / TB) {
        const float4 v = *reinterpret_cast<const float4*>(a.part + ((size_t)tok0 * a.np + s) * 4);
        ss += v.x;
        dd += v.y;
        dp += v.z;
      }
    ss = warp_part_sum<TB>(ss);
    dd = warp_part_sum<TB>(dd);
    dp = warp_part_sum<TB>(dp);
    if (lane < TB) {
      red[warp * TB + lane] = ss;
      red[nthr<TB>() + warp * TB + lane] = dd;
      red[2 * nthr<TB>() + warp * TB + lane] = dp;
    }
  }
  __syncthreads();
  if (tid < TB) {
    const int t = t0 + tid;
    float ss = 0.f, dd = 0.f, dp = 0.f, dprev = 0.f, pp = 1.f, mp = 1.f;
    for (int w = 0; w < nthr<TB>() / 32; ++w) {
      ss += red[w * TB + tid];
      dd += red[nthr<TB>() + w * TB + tid];
      dp += red[2 * nthr<TB>() + w * TB + tid];
    }
    if (t < a.T) {
      dprev = a.dprev[t];
      pp = a.pst[t];
      mp = a.mst[t];
    }
    const float rinv = rsqrtf(ss / (float)a.d + a.rms_eps);
    const float dj = a.j == 1 ? 0.f : sqrtf(dd);                       // Eq. 7
    const float gam = a.j > 2 ? dp / (dj * dprev + a.eps) : 0.f;       // Eq. 8
    sc[tid * 16 + 0] = rinv;
    sc[tid * 16 + 1] = dj;
    sc[tid * 16 + 4] = mp;
    const bool pos = !(a.variant & RV_NO_POS);   // ablation: no progress / transition
    xT[0 * TB + tid] = pos ? (float)a.j / (float)a.L : 0.f;
    xT[1 * TB + tid] = pos ? (float)(a.L - a.j) / (float)a.L : 0.f;
    xT[2 * TB + tid] = pos ? dj : 0.f;
    xT[3 * TB + tid] = pos ? gam : 0.f;
    xT[4 * TB + tid] = pp;
    xT[5 * TB + tid] = mp;
  }
  __syncthreads();

  // 2. encoder hidden SiLU(rinv (W_hd diag(g_r)) h_bar), transposed; f_psi's
  //    second layer reduced on the fly (b = w_ps2 . SiLU(W_ps1 h_bar + b_ps1), Eq. 16).
  //    Part pt reads float4 column groups pt, pt + 16, ... of its token's Y row; a
  //    warp instruction covers 16 rows x 32 contiguous bytes, and up to eight
  //    loads per thread are in flight.  d_enc is a multiple of 4, so no group
  //    straddles the encoder / f_psi boundary.
  {
    constexpr int YB = 8;
    float bpart = 0.f;
    const int ng = nY >> 2;
    const float rinv = sc[tl0 * 16];
    const float4* yrow = reinterpret_cast<const float4*>(a.Y + (size_t)tok0 * nY);
    for (int g0 = pt0; g0 < ng; g0 += YB * (nthr<TB>() / TB)) {
      float4 yv[YB];
#pragma unroll
      for (int k = 0; k < YB; ++k) {
        const int g = g0 + k * (nthr<TB>() / TB);
        yv[k] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (tok0 < a.T && g < ng) {
          yv[k] = __ldg(yrow + g);
          for (int sp = 1; sp < a.y_splits; ++sp) {   // split-K slices, in slice order
            const float4 v = __ldg(yrow + (size_t)sp * (a.y_split_stride / 4) + g);
            yv[k].x += v.x; yv[k].y += v.y; yv[k].z += v.z; yv[k].w += v.w;
          }
        }
      }
#pragma unroll
      for (int k = 0; k < YB; ++k) {
        const int g = g0 + k * (nthr<TB>() / TB);
        if (g >= ng) break;
        const int c = 4 * g;
        const float y4[4] = {yv[k].x, yv[k].y, yv[k].z, yv[k].w};
        if (c < a.d_enc) {
#pragma unroll
          for (int i = 0; i < 4; ++i) bigT[(c + i) * TB + tl0] = siluf_(y4[i] * rinv);
        } else {
          const int e = c - a.d_enc;
#pragma unroll
          for (int i = 0; i < 4; ++i)
            bpart = fmaf(__ldg(a.w.ps_w2 + e + i), siluf_(y4[i] + __ldg(a.w.ps_b1 + e + i)), bpart);
        }
      }
    }
    reduce16<TB>(red, bpart, ab + TB);   // also orders step 2's writes before step 3
  }

  if (no_history) {   // ablation: g = sigma(b), the local logit alone; state untouched
    if (tid < TB) {
      const int t = t0 + tid;
      if (t < a.T) {
        const float g = sigmoidf_(ab[TB + tid] + __ldg(a.w.ps_b2));
        const uint8_t dec = a.mask_in ? (a.mask_in[t] ? 1 : 0) : (g >= a.tau ? 1 : 0);
        a.gate[t] = g;
        a.mask[t] = dec;
        if (a.gate_out) a.gate_out[t] = g;
        if (a.mask_out) a.mask_out[t] = dec;
      }
    }
    return;
  }

  // 3. z_h = W_hu enc (Eq. 5) -> s[0, d_h); FFN_path hidden; z_a (Eq. 9) -> s[d_h, d_s).
  //    Small token counts: the two are independent and run on the two halves of the CTA.
  if (TB < 16 && !(a.variant & RV_NO_AUX)) {
    constexpr int half = nthr<TB>() / 2;
    if (tid < half) {
      bmm4<TB>(bigT, a.d_enc, a.w.w_hu_t, a.d_h, nullptr, sT, 0, false, aux, 3072, 0, half, 1);
    } else {
      bmm4<TB>(xT, 6, a.w.path_w1_t, a.d_path, a.w.path_b1, phT, 0, true, nullptr, 0, half, half, 2);
      bmm4<TB>(phT, a.d_path, a.w.path_w2_t, a.d_a, a.w.path_b2, sT + a.d_h * TB, 0, false,
               nullptr, 0, half, half, 2);
    }
    __syncthreads();
  } else {
    bmm4<TB>(bigT, a.d_enc, a.w.w_hu_t, a.d_h, nullptr, sT, 0, false, aux, 3072);
    if (a.variant & RV_NO_AUX) {   // ablation: no auxiliary path encoder, z_a = 0
      for (int e = tid; e < a.d_a * TB; e += nthr<TB>()) sT[a.d_h * TB + e] = 0.f;
      __syncthreads();
    } else {
      bmm4<TB>(xT, 6, a.w.path_w1_t, a.d_path, a.w.path_b1, phT, 0, true);
      bmm4<TB>(phT, a.d_path, a.w.path_w2_t, a.d_a, a.w.path_b2, sT + a.d_h * TB, 0, false);
    }
  }

  // 4. q | k | v = W_{q,k,v} s (Eq. 10), token-major for the memory step.  Small token
  //    counts: W_n s of step 6 (it needs s only) runs beside it on the other half.
  const bool need_nu = a.j > 1 && !no_memread;
  const bool nu_early = TB < 16 && need_nu;
  const int cap_big = (a.d_enc > a.d_head ? a.d_enc : a.d_head) * TB;
  if (nu_early) {
    constexpr int half = nthr<TB>() / 2;
    if (tid < half)
      bmm4<TB>(sT, ds, a.w.w_qkv_t, 3 * DM, nullptr, qkv, 3 * DM, false, skT,
               RouterLayout<TB>::kSplitScratch, 0, half, 1);
    else   // W_n s -> aux [DM][TB] (aux and the big region are free after step 3)
      bmm4<TB>(sT, ds, a.w.w_n_t, DM, nullptr, aux, 0, false, bigT, cap_big, half, half, 2);
    __syncthreads();
  } else {
    bmm4<TB>(sT, ds, a.w.w_qkv_t, 3 * DM, nullptr, qkv, 3 * DM, false, skT,
             RouterLayout<TB>::kSplitScratch);
  }

  // 5. memory read (Eq. 11) fused with the write (Eq. 12), one warp per token.
  if (no_memread) {   // ablation: c = 0; the memory is neither read nor written
    for (int e = tid; e < DM * TB; e += nthr<TB>()) sT[ds * TB + e] = 0.f;
  } else if constexpr (mem_split<DM, TB>()) {
    memory_split<DM, TB>(a, qkv, skT, t0, warp, lane);   // skT is free between steps 4 and 7
    __syncthreads();
    memory_split_finish<DM, TB>(a, skT, sT + ds * TB, t0);
  } else {
    memory_read_write<DM, TB>(a, qkv, sT + ds * TB, t0, warp, lane);
  }
  __syncthreads();

  // 6. nu = 1 - cos(W_n s, W_c c) for j > 1 (Eq. 13); nu_1 = 0
  float* nuT = sT + (ds + DM) * TB;
  if (need_nu) {   // the ablation without memory access sees nu = 0
    float* nv = aux;               // [DM][TB]
    float* cv = aux + DM * TB;     // [DM][TB]
    if (!nu_early) bmm4<TB>(sT, ds, a.w.w_n_t, DM, nullptr, nv, 0, false, bigT, cap_big);
    bmm4<TB>(sT + ds * TB, DM, a.w.w_c_t, DM, nullptr, cv, 0, false, bigT, cap_big);
    // thread (part, t) sums DM/16 products; fixed-order reduction per token
    const int tl = tid % TB, part = tid / TB;
    float xy = 0.f, xx = 0.f, yy = 0.f;
    for (int i = part; i < DM; i += nthr<TB>() / TB) {
      const float u = nv[i * TB + tl], w = cv[i * TB + tl];
      xy += u * w;
      xx += u * u;
      yy += w * w;
    }
    xy = warp_part_sum<TB>(xy);    // the three sums reduced in one pass
    xx = warp_part_sum<TB>(xx);
    yy = warp_part_sum<TB>(yy);
    if (lane < TB) {
      red[warp * TB + lane] = xy;
      red[nthr<TB>() + warp * TB + lane] = xx;
      red[2 * nthr<TB>() + warp * TB + lane] = yy;
    }
    __syncthreads();
    if (tid < TB) {
      float sxy = 0.f, sxx = 0.f, syy = 0.f;
      for (int w = 0; w < nthr<TB>() / 32; ++w) {
        sxy += red[w * TB + tid];
        sxx += red[nthr<TB>() + w * TB + tid];
        syy += red[2 * nthr<TB>() + w * TB + tid];
      }
      nuT[tid] = 1.f - sxy / (sqrtf(sxx) * sqrtf(syy) + a.eps);
    }
  } else {
    if (tid < TB) nuT[tid] = 0.f;
  }
  __syncthreads();

  // 7. f_theta hidden = SiLU(W_th1 [s; c; nu] + b) -> big region
  bmm4<TB>(sT, ds + DM + 1, a.w.th_w1_t, a.d_head, a.w.th_b1, bigT, 0, true, skT,
           RouterLayout<TB>::kSplitScratch);

  // 8. a = w_th2 . hidden + b (Eq. 14)
  {
    const int tl = tid % TB, part = tid / TB;
    float sa = 0.f;
    for (int i = part; i < a.d_head; i += nthr<TB>() / TB) sa = fmaf(__ldg(a.w.th_w2 + i), bigT[i * TB + tl], sa);
    reduce16<TB>(red, sa, ab);
  }

  // 9. history score, cumulative score, gate and decision
  if (tid < TB) {
    const int t = t0 + tid;
    if (t < a.T) {
      const float av = ab[tid] + __ldg(a.w.th_b2);
      const float bv = ab[TB + tid] + __ldg(a.w.ps_b2);
      const float p = sigmoidf_(av / a.t_hist);     // Eq. 14
      const float m = sc[tid * 16 + 4] * p;         // Eq. 15
      const float g = sigmoidf_(av + bv);           // Eq. 16
      uint8_t dec;
      if (a.mask_in)
        dec = a.mask_in[t] ? 1 : 0;
      else
        dec = g >= a.tau ? 1 : 0;                   // Eq. 3 (ties run the FFN)
      a.pst[t] = p;
      a.mst[t] = m;
      a.dprev[t] = sc[tid * 16 + 1];
      a.gate[t] = g;
      a.mask[t] = dec;
      if (a.gate_out) a.gate_out[t] = g;
      if (a.mask_out) a.mask_out[t] = dec;
    }
  }
}

// ------------------------------------------------------------------------------
// k_compact: one CTA; stable exclusive scan of the decisions in chunks of
// CT * SEGS tokens.  A warp owns SEGS consecutive 32-token segments: one ballot
// per segment gives its FFN count (pass 1, then a block scan of the warp totals)
// and each lane's rank inside the segment (pass 2), so every load and every
// index write of a segment is one coalesced warp access.
// ------------------------------------------------------------------------------
constexpr int CT = 1024, SEGS = 16;

__global__ void __launch_bounds__(CT) k_compact(const CompactArgs a) {
  pdl_enter();
  __shared__ int wsum[CT / 32];
  __shared__ int carry_s;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t lt_mask = (1u << lane) - 1u;
  if (tid == 0) carry_s = 0;
  __syncthreads();
  for (int base = 0; base < a.T; base += CT * SEGS) {
    const int wbase = base + warp * 32 * SEGS;
    uint32_t bal[SEGS];
    int wtot = 0;
#pragma unroll
    for (int sg = 0; sg < SEGS; ++sg) {
      const int t = wbase + sg * 32 + lane;
      const bool f = t < a.T && (a.dense || a.mask[t] != 0);
      bal[sg] = __ballot_sync(0xffffffffu, f);
      wtot += __popc(bal[sg]);
    }
    if (lane == 0) wsum[warp] = wtot;
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
    int pos0 = carry + (warp ? wsum[warp - 1] : 0);   // FFN tokens before this warp's tokens
#pragma unroll
    for (int sg = 0; sg < SEGS; ++sg) {
      const int t = wbase + sg * 32 + lane;
      if (t < a.T) {
        const bool f = (bal[sg] >> lane) & 1u;
        const int pf = pos0 + __popc(bal[sg] & lt_mask);
        if (f) {
          a.idx_f[pf] = t;
          a.scale_f[pf] = a.dense ? 1.f : a.gate[t];
        } else {
          const int pa = t - pf;   // tokens before t that went to the adapter
          a.idx_a[pa] = t;
          a.scale_a[pa] = 1.f - a.gate[t];
        }
        if (a.dense) {
          if (a.gate_out) a.gate_out[t] = 1.f;
          if (a.mask_out) a.mask_out[t] = 1;
        }
      }
      pos0 += __popc(bal[sg]);
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
// k_norm: wpr warps per branch row (1 for large T; more when few rows would leave
// the GPU idle), each over a contiguous column range; slot s < n_f is FFN row s
// (token idx_f[s]), slot s >= n_f is adapter row s - n_f.  The row's 1/rms comes
// from the epilogue's partial sums (lane-parallel loads, fixed-order warp
// reduction); the columns are streamed with up to eight float4 loads per lane in
// flight.
// ------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_norm(const NormArgs a, int wpr) {
  pdl_enter();
  const long gw = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const long slot = gw / wpr;
  const int part = (int)(gw - slot * wpr);
  const int lane = threadIdx.x & 31;
  if (slot >= a.T) return;
  const int nf = a.counts ? a.counts[0] : a.T;   // no counts: every token, in token order
  int t;
  void* dst;
  long r;
  if (!a.counts) {
    t = (int)slot;
    dst = a.u_f;
    r = slot;
  } else if (slot < nf) {
    t = a.idx_f[slot];
    dst = a.u_f;
    r = slot;
  } else {
    t = a.idx_a[slot - nf];
    dst = a.u_a;
    r = slot - nf;
  }
  float ss = 0.f;
  for (int s = lane; s < a.np; s += 32) ss += a.part[((size_t)t * a.np + s) * 4];
  ss = warp_sum(ss);
  const float rinv = rsqrtf(ss / (float)a.d + a.rms_eps);
  const int cols = a.d / wpr;
  const int c_lo = part * cols, c_hi = c_lo + cols;
  const float* h = a.hbar + (size_t)t * a.d;
  const size_t ro = (size_t)r * a.d;
  constexpr int NB = 8;
  for (int c0 = c_lo + lane * 4; c0 < c_hi; c0 += 128 * NB) {
    float4 hv[NB];
#pragma unroll
    for (int k = 0; k < NB; ++k) {
      const int c = c0 + 128 * k;
      if (c < c_hi) hv[k] = *reinterpret_cast<const float4*>(h + c);
    }
#pragma unroll
    for (int k = 0; k < NB; ++k) {
      const int c = c0 + 128 * k;
      if (c < c_hi) {
        const float4 g = __ldg(reinterpret_cast<const float4*>(a.gain + c));
        store4(dst, ro + c,
               make_float4(hv[k].x * rinv * g.x, hv[k].y * rinv * g.y, hv[k].z * rinv * g.z,
                           hv[k].w * rinv * g.w),
               a.out_bf16);
      }
    }
  }
}

// ------------------------------------------------------------------------------
// k_route_norm: k_compact and k_norm in one launch for token counts up to
// kRouteNormMaxT, or any count when the router left per-32-token FFN counts (chunk_cnt).
// Warp gw serves token t = gw / wpr (column range gw % wpr); it counts the FFN decisions
// of the tokens before t (the chunks' counts, then one ballot per 32 tokens; without
// counts every warp repeats the ballot scan, which at those token counts costs less than a
// launch), so that
// token t's branch row is its rank among the tokens of its branch, as in k_compact.
// The column-range-0 warp of a token writes the token's index and scale entries; the
// warp of the last token writes the counts.  Outputs equal those of the two kernels.
// ------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_route_norm(const CompactArgs c, const NormArgs a, int wpr) {
  pdl_enter();
  const long gw = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int t = (int)(gw / wpr);
  const int part = (int)(gw - (long)t * wpr);
  const int lane = threadIdx.x & 31;
  if (t >= a.T) return;
  int pf = t;   // FFN tokens before t
  bool f = true;
  if (!c.dense) {
    pf = 0;
    int b0 = 0;
    if (c.chunk_cnt) {   // whole 32-token chunks before t's from their counts
      const int nc = t >> 5;
      int sum = 0;
#pragma unroll 4
      for (int i = lane; i < nc; i += 32) sum += c.chunk_cnt[i];
      pf = __reduce_add_sync(0xffffffffu, sum);
      b0 = nc << 5;
    }
    for (int b = b0; b < t; b += 128) {
      int n = 0;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int u = b + 32 * q + lane;
        n += __popc(__ballot_sync(0xffffffffu, u < t && c.mask[u] != 0));
      }
      pf += n;
    }
    f = c.mask[t] != 0;
  }
  if (part == 0 && lane == 0) {
    if (f) {
      c.idx_f[pf] = t;
      c.scale_f[pf] = c.dense ? 1.f : c.gate[t];
    } else {
      c.idx_a[t - pf] = t;
      c.scale_a[t - pf] = 1.f - c.gate[t];
    }
    if (c.dense) {
      if (c.gate_out) c.gate_out[t] = 1.f;
      if (c.mask_out) c.mask_out[t] = 1;
    }
    if (t == a.T - 1) {
      const int nf = pf + (f ? 1 : 0);
      c.counts[0] = nf;
      c.counts[1] = a.T - nf;
      if (c.count_out) *c.count_out = nf;
    }
  }
  void* dst = f ? a.u_f : a.u_a;
  const long r = f ? pf : t - pf;
  float ss = 0.f;
  for (int s = lane; s < a.np; s += 32) ss += a.part[((size_t)t * a.np + s) * 4];
  ss = warp_sum(ss);
  const float rinv = rsqrtf(ss / (float)a.d + a.rms_eps);
  const int cols = a.d / wpr;
  const int c_lo = part * cols, c_hi = c_lo + cols;
  const float* h = a.hbar + (size_t)t * a.d;
  const size_t ro = (size_t)r * a.d;
  constexpr int NB = 8;
  for (int c0 = c_lo + lane * 4; c0 < c_hi; c0 += 128 * NB) {
    float4 hv[NB];
#pragma unroll
    for (int k = 0; k < NB; ++k) {
      const int cc = c0 + 128 * k;
      if (cc < c_hi) hv[k] = *reinterpret_cast<const float4*>(h + cc);
    }
#pragma unroll
    for (int k = 0; k < NB; ++k) {
      const int cc = c0 + 128 * k;
      if (cc < c_hi) {
        const float4 g = __ldg(reinterpret_cast<const float4*>(a.gain + cc));
        store4(dst, ro + cc,
               make_float4(hv[k].x * rinv * g.x, hv[k].y * rinv * g.y, hv[k].z * rinv * g.z,
                           hv[k].w * rinv * g.w),
               a.out_bf16);
      }
    }
  }
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
  return launch_pdl(k_init, dim3((a.T + warps_per_block - 1) / warps_per_block), dim3(256), 0, st, a);
}

cudaError_t launch_block_entry(const BlockEntryArgs& a, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  return launch_pdl(k_block_entry, dim3((a.T + 7) / 8), dim3(256), 0, st, a);
}

cudaError_t launch_state_reset(float* S, float* zeta, float* pst, float* mst, float* dprev, int T,
                               int dm, cudaStream_t st) {
  if (T <= 0) return cudaSuccess;
  long n = (long)T * dm * dm;
  long blocks = (n + 255) / 256;
  if (blocks > 8192) blocks = 8192;
  return launch_pdl(k_state_reset, dim3((unsigned)blocks), dim3(256), 0, st, S, zeta, pst, mst, dprev,
                    T, dm);
}

template <int DM, int TB>
static cudaError_t launch_router_tb(const RouterArgs& a, cudaStream_t st) {
  const RouterLayout<TB> lay(a.d_enc, a.d_head, a.d_h + a.d_a, DM, a.d_path);
  const size_t smem = sizeof(float) * (size_t)lay.floats;
  static size_t attr = 0;
  if (smem > attr) {
    cudaError_t e = cudaFuncSetAttribute(k_router<DM, TB>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr = smem;
  }
  return launch_pdl(k_router<DM, TB>, dim3((a.T + TB - 1) / TB), dim3(nthr<TB>()), smem, st, a);
}

template <int DM>
static cudaError_t launch_router_dm(const RouterArgs& a, int num_sms, cudaStream_t st) {
  if ((a.T + TB_LARGE - 1) / TB_LARGE < 2 * num_sms) return launch_router_tb<DM, TB_SMALL>(a, st);
  return launch_router_tb<DM, TB_LARGE>(a, st);
}

cudaError_t launch_router(int d_m, const RouterArgs& a, int num_sms, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  switch (d_m) {
    case 16: return launch_router_dm<16>(a, num_sms, st);
    case 32: return launch_router_dm<32>(a, num_sms, st);
    case 64: return launch_router_dm<64>(a, num_sms, st);
    case 128: return launch_router_dm<128>(a, num_sms, st);
    case 256: return launch_router_dm<256>(a, num_sms, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_compact(const CompactArgs& a, cudaStream_t st) {
  return launch_pdl(k_compact, dim3(1), dim3(CT), 0, st, a);
}

// Warps per row of the norm: split rows across warps until there are ~16 warps per SM
// (column ranges stay whole multiples of 4 elements).
static int norm_wpr(const NormArgs& a, int num_sms) {
  int wpr = 1;
  while ((long)a.T * wpr * 2 <= 16L * num_sms && (a.d / (wpr * 2)) % 4 == 0 && a.d / (wpr * 2) >= 128)
    wpr *= 2;
  return wpr;
}

cudaError_t launch_norm(const NormArgs& a, int num_sms, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  const int wpr = norm_wpr(a, num_sms);
  const long warps = (long)a.T * wpr;
  return launch_pdl(k_norm, dim3((unsigned)((warps + 7) / 8)), dim3(256), 0, st, a, wpr);
}

cudaError_t launch_route_norm(const CompactArgs& c, const NormArgs& a, int num_sms, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  if ((a.T > kRouteNormMaxT && !c.chunk_cnt) || c.T != a.T) return cudaErrorInvalidValue;
  const int wpr = norm_wpr(a, num_sms);
  const long warps = (long)a.T * wpr;
  return launch_pdl(k_route_norm, dim3((unsigned)((warps + 7) / 8)), dim3(256), 0, st, c, a, wpr);
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
