// Persistent tensor-core GEMM for sm_103a: TMA-fed shared-memory ring, tcgen05.mma
// with the accumulator in TMEM (double buffered), and fused epilogues.
//
//   C[M, N] = A[M, K] * B[N, K]^T        (bf16 operands, fp32 accumulation)
//
// A launch may carry a second, independent problem (grouped launch): the FFN and
// the adapter branch of a routed block touch disjoint token rows, so the adapter's
// GEMM tiles are spread evenly among the FFN's tiles of the same launch and their
// epilogues overlap the FFN's tensor-core work.
//
// One CTA per SM, 6 warps:
//   warp 0      TMA producer (one elected lane) - A and B tiles into a STAGES-deep ring
//   warp 1      TMEM allocator and MMA issuer (one elected lane)
//   warps 2..5  epilogue: each owns the 32 TMEM lanes (= tile rows) of its quadrant
// Tiles are 128 x BN with K-blocks of 64 bf16 (one 128-byte swizzle row).  The row
// count M may live in device memory (the compacted token count of a routed block),
// so no host synchronisation is needed between routing and the GEMMs; tiles past M
// do no work.  Every mbarrier wait is bounded (%globaltimer) and reports through
// the error word instead of hanging.
#include "hero_device.cuh"

namespace hero {
namespace {

constexpr int BM = 128;
constexpr int BK = 64;
// raster: kGroupM M-tiles share each wave of N-tiles (L2 reuse); CTA-pair tiles are twice
// as tall, so the pair kernel groups half as many (the same rows per group)
constexpr int kGroupM = 16;

constexpr int EPI_NONE = -1;   // no second problem

// CG = 1: one CTA computes a 128 x BN tile.  CG = 2: a CTA pair (thread-block cluster
// of 2) computes a 256 x BN tile with the 2-SM MMA: each CTA holds 128 rows of A, BN / 2
// rows of B and 128 rows of the accumulator, so per FLOP each SM stages a third less
// operand data through its shared memory.
// INB = 1 (the wide block-closing epilogue of the adapter's rank-d_r up projection, one
// K-block per tile): a single ring stage, and per epilogue warp a 12 KB buffer that the
// epilogue's row inputs (h_bar, delta, P) are copied into with cp.async.
template <int BN, int EPIW, int CG = 1, int INB = 0>
struct TcCfg {
  static constexpr int B_ROWS = BN / CG;   // rows of B staged by this CTA
  static constexpr int STAGES = INB ? 1 : (CG == 2 ? 6 : (BN == 256 ? 4 : 6));
  static constexpr uint32_t A_BYTES = BM * BK * 2;
  static constexpr uint32_t B_BYTES = B_ROWS * BK * 2;
  static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr uint32_t TMEM_COLS = 2 * BN < 32 ? 32 : 2 * BN;
  // instruction descriptor, kind::f16: D fp32 (bit 4), A bf16 (bits 7-9 = 1),
  // B bf16 (bits 10-12 = 1), both K-major, N >> 3 at bit 17, M >> 4 at bit 24
  // (M = 256 for the pair).
  static constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) |
                                    ((uint32_t)(BN >> 3) << 17) | ((uint32_t)((BM * CG) >> 4) << 24);
  // EPIW epilogue warps: one (4 warps) or two (8 warps, each taking half of the
  // tile's columns) per TMEM lane quadrant.
  static constexpr int EPI_WARPS = EPIW;
  static constexpr int THREADS = 64 + 32 * EPI_WARPS;
  // ring | barriers (256 B) | per-epilogue-warp staging tiles (32 x 32 fp32 each)
  static constexpr uint32_t EPI_STAGE_OFF = STAGES * STAGE_BYTES + 256;
  static constexpr uint32_t IN_OFF = EPI_STAGE_OFF + EPI_WARPS * 32 * 32 * 4;
  static constexpr uint32_t IN_BYTES = INB ? 3 * 8 * 32 * 16 : 0;   // per epilogue warp
  static constexpr size_t SMEM = (size_t)IN_OFF + EPI_WARPS * IN_BYTES + 1024;
  static_assert(SMEM <= 232448, "shared memory per CTA");
};

// The wide block-closing epilogue loads its row inputs with cp.async (epi_layer_out_async);
// -DHERO_WIDE_INBUF=0 keeps the register-held loads of epi_layer_out.
#ifndef HERO_WIDE_INBUF
#define HERO_WIDE_INBUF 1
#endif
template <int EPI>
constexpr int epi_inbuf() { return EPI == EPI_LAYER_OUT_WIDE && HERO_WIDE_INBUF ? 1 : 0; }

template <int EPI>
constexpr int epi_warps() {
  return EPI == EPI_LAYER_OUT_WIDE || EPI == EPI_ATTN_ENTRY || EPI == EPI_RT_HEAD ? 8 : 4;
}

__device__ __forceinline__ void tile_coords(int tile, int m_tiles, int n_tiles, int& mb, int& nb,
                                            int group_m) {
  const int group = group_m * n_tiles;
  const int g = tile / group;
  const int first_m = g * group_m;
  const int gm = min(group_m, m_tiles - first_m);
  const int local = tile - g * group;
  mb = first_m + local % gm;
  nb = local / gm;
}

// ---- epilogues: one thread = one tile row; TMEM read in 32 or 16 column chunks ----

// Stage one warp's 32 rows x 32 fp32 columns through shared memory so that the
// global accesses that follow are row-contiguous: lane l then owns float4 slot
// (l & 7) of rows (l >> 3) + 4k, k = 0..7 (128 contiguous bytes per row per
// instruction).  Float4 slots are XOR-swizzled by row to avoid bank conflicts.
__device__ __forceinline__ void stage_rows(float4* st, const uint32_t (&r)[32], int lane) {
#pragma unroll
  for (int c4 = 0; c4 < 8; ++c4)
    st[lane * 8 + (c4 ^ (lane & 7))] =
        make_float4(__uint_as_float(r[4 * c4]), __uint_as_float(r[4 * c4 + 1]),
                    __uint_as_float(r[4 * c4 + 2]), __uint_as_float(r[4 * c4 + 3]));
}

__device__ __forceinline__ float4 staged(const float4* st, int row, int slot) {
  return st[row * 8 + (slot ^ (row & 7))];
}

template <int BN, bool RESID = false>
__device__ __forceinline__ void epi_store_f32(const GemmArgs& a, uint32_t tbase, int row0, int M,
                                              int nb, int split, float4* st) {
  float* out = a.out_f32 + (size_t)split * a.split_stride;
  const int lane = threadIdx.x & 31;
  const int sub = lane >> 3, slot = lane & 7;
#pragma unroll 1
  for (int c0 = 0; c0 < BN; c0 += 32) {
    uint32_t r[32];
    tmem_ld32(tbase + c0, r);
    stage_rows(st, r, lane);
    __syncwarp();
    const int n = nb * BN + c0 + 4 * slot;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int rr = sub + 4 * k;
      const int m = row0 + rr;
      if (m < M && n < a.N) {
        float4 v = staged(st, rr, slot);
        if constexpr (RESID) {
          const float4 r = *reinterpret_cast<const float4*>(a.resid + (size_t)m * a.ldo + n);
          v.x += r.x; v.y += r.y; v.z += r.z; v.w += r.w;
        }
        *reinterpret_cast<float4*>(out + (size_t)m * a.ldo + n) = v;
      }
    }
    __syncwarp();
  }
}

// Gate/up columns are interleaved per 256-wide tile: [0,128) gate, [128,256) up of
// the same 128 intermediate features; output act[m, nb*128 + c].
__device__ __forceinline__ void epi_swiglu(const GemmArgs& a, uint32_t tbase, int m, bool valid,
                                           int nb) {
#pragma unroll 1
  for (int c0 = 0; c0 < 128; c0 += 16) {
    uint32_t g[16], u[16];
    tmem_ld16(tbase + c0, g);
    tmem_ld16(tbase + 128 + c0, u);
    if (valid) {
      uint32_t pk[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float g0 = __uint_as_float(g[2 * i]), g1 = __uint_as_float(g[2 * i + 1]);
        const float u0 = __uint_as_float(u[2 * i]), u1 = __uint_as_float(u[2 * i + 1]);
        pk[i] = pack_bf16x2(siluf_(g0) * u0, siluf_(g1) * u1);
      }
      uint4* dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(a.out) + (size_t)m * a.ldo +
                                            nb * 128 + c0);
      dst[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
      dst[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
    }
  }
}

// Columns past N (a multiple of 32) are not written: the adapter's rank can be
// narrower than the tile.
template <int BN>
__device__ __forceinline__ void epi_silu(const GemmArgs& a, uint32_t tbase, int m, bool valid,
                                         int nb) {
  const int ncols = min(BN, a.N - nb * BN);
#pragma unroll 1
  for (int c0 = 0; c0 < ncols; c0 += 32) {
    uint32_t r[32];
    tmem_ld32(tbase + c0, r);
    if (valid) {
      uint32_t pk[16];
#pragma unroll
      for (int i = 0; i < 16; ++i)
        pk[i] = pack_bf16x2(siluf_(__uint_as_float(r[2 * i])), siluf_(__uint_as_float(r[2 * i + 1])));
      uint4* dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(a.out) + (size_t)m * a.ldo +
                                            nb * BN + c0);
#pragma unroll
      for (int i = 0; i < 4; ++i) dst[i] = make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
    }
  }
}

// Plain bf16 store of the accumulator (columns past N, a multiple of 32, skipped).
template <int BN>
__device__ __forceinline__ void epi_store_bf16(const GemmArgs& a, uint32_t tbase, int m, bool valid,
                                               int nb) {
  const int ncols = min(BN, a.N - nb * BN);
#pragma unroll 1
  for (int c0 = 0; c0 < ncols; c0 += 32) {
    uint32_t r[32];
    tmem_ld32(tbase + c0, r);
    if (valid) {
      uint32_t pk[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) pk[i] = pack_bf16x2(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1]));
      uint4* dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(a.out) + (size_t)m * a.ldo +
                                            nb * BN + c0);
#pragma unroll
      for (int i = 0; i < 4; ++i) dst[i] = make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
    }
  }
}

// Backward of act = SiLU(gate) up (training path, decisions fixed).  The accumulator
// holds e = dL/dy W_down for features f = nb BN + c of compacted FFN row m, where
// dL/dy = G (the upstream gradient; the branch scale g is applied here):
//   dact = g e,  dgate = dact up SiLU'(gate),  dup = dact SiLU(gate),
//   dL/dg contribution: sum_f e_f act_f with act = bf16(SiLU(gate) up), the value the
//   forward fed to W_down.
// gate and up (bf16 pre-activations) sit in the interleaved gate/up layout (per 128
// features: 128 gate columns, then 128 up columns) of row m of a.out and are replaced
// there by dgate and dup (bf16): the A operand of the input-gradient GEMM.
template <int BN>
__device__ __forceinline__ void epi_bw_swiglu(const GemmArgs& a, uint32_t tbase, int m, bool valid,
                                              int nb) {
  const int ncols = min(BN, a.N - nb * BN);
  uint16_t* row = static_cast<uint16_t*>(a.out) + (size_t)m * a.ldo;
  const float s = valid ? a.row_scale[m] : 0.f;
  float dgs = 0.f;
#pragma unroll 1
  for (int c0 = 0; c0 < ncols; c0 += 32) {
    uint32_t r[32];
    tmem_ld32(tbase + c0, r);
    if (valid) {
      const int f = nb * BN + c0;   // 32 features inside one 128-feature group
      uint4* gp = reinterpret_cast<uint4*>(row + (f >> 7) * 256 + (f & 127));
      uint4* upp = reinterpret_cast<uint4*>(row + (f >> 7) * 256 + 128 + (f & 127));
      uint4 gr[4], ur[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        gr[i] = gp[i];
        ur[i] = upp[i];
      }
      const uint32_t* gw = reinterpret_cast<const uint32_t*>(gr);
      const uint32_t* uw = reinterpret_cast<const uint32_t*>(ur);
      uint32_t dgw[16], duw[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        float g0, g1, u0, u1;
        unpack_bf16x2(gw[i], g0, g1);
        unpack_bf16x2(uw[i], u0, u1);
        const float e0 = __uint_as_float(r[2 * i]), e1 = __uint_as_float(r[2 * i + 1]);
        const float s0 = sigmoidf_(g0), s1 = sigmoidf_(g1);
        const float sl0 = g0 * s0, sl1 = g1 * s1;
        const float a0 = __bfloat162float(__float2bfloat16_rn(sl0 * u0));
        const float a1 = __bfloat162float(__float2bfloat16_rn(sl1 * u1));
        dgs = fmaf(e0, a0, dgs);
        dgs = fmaf(e1, a1, dgs);
        const float d0 = s * e0, d1 = s * e1;
        dgw[i] = pack_bf16x2(d0 * u0 * s0 * (1.f + g0 * (1.f - s0)),
                             d1 * u1 * s1 * (1.f + g1 * (1.f - s1)));
        duw[i] = pack_bf16x2(d0 * sl0, d1 * sl1);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        gp[i] = make_uint4(dgw[4 * i], dgw[4 * i + 1], dgw[4 * i + 2], dgw[4 * i + 3]);
        upp[i] = make_uint4(duw[4 * i], duw[4 * i + 1], duw[4 * i + 2], duw[4 * i + 3]);
      }
    }
  }
  if (valid) a.row_part[(size_t)m * a.part_ld + nb] = dgs;
}

// ---- the router on the tensor cores (RouterTcArgs) ----
// x = t0 + t1 + t2 exactly, each a bf16 number (8 significant bits per term; the
// remainders x - t0 and x - t0 - t1 are exact in fp32).
__device__ __forceinline__ void split3(float x, uint16_t (&t)[3]) {
  const __nv_bfloat16 h0 = __float2bfloat16_rn(x);
  const float r0 = x - __bfloat162float(h0);
  const __nv_bfloat16 h1 = __float2bfloat16_rn(r0);
  const float r1 = r0 - __bfloat162float(h1);
  const __nv_bfloat16 h2 = __float2bfloat16_rn(r1);
  t[0] = *reinterpret_cast<const uint16_t*>(&h0);
  t[1] = *reinterpret_cast<const uint16_t*>(&h1);
  t[2] = *reinterpret_cast<const uint16_t*>(&h2);
}

// Store 32 fp32 values of row `row` (bf16 terms at columns col, col + stride, col + 2 stride).
__device__ __forceinline__ void store_split32(uint16_t* row, int col, int stride, const float (&x)[32]) {
  uint32_t w[3][16];
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    uint16_t a[3], b[3];
    split3(x[2 * i], a);
    split3(x[2 * i + 1], b);
#pragma unroll
    for (int p = 0; p < 3; ++p) w[p][i] = (uint32_t)a[p] | ((uint32_t)b[p] << 16);
  }
#pragma unroll
  for (int p = 0; p < 3; ++p) {
    uint4* dst = reinterpret_cast<uint4*>(row + col + p * stride);
#pragma unroll
    for (int q = 0; q < 4; ++q) dst[q] = make_uint4(w[p][4 * q], w[p][4 * q + 1], w[p][4 * q + 2], w[p][4 * q + 3]);
  }
}

// Step 1 (the router contraction, Eq. 5 and f_psi's first layer, Eq. 16): column tile 0
// holds (W_hd diag(g_r)) h_bar, tile 1 W_psi1 h_bar.  Tile 0: 1/rms, d_j and gamma
// (Eqs. 7-8) from the partial sums, and the encoder hidden SiLU(acc / rms) as three bf16
// terms; tile 1: f_psi's second layer without its bias.  One thread = one token row.
template <int BN>
__device__ __forceinline__ void epi_rt_enc(const GemmArgs& a, uint32_t tbase, int m, bool valid, int nb) {
  static_assert(BN == 256, "one tile per half of the contraction");
  const RouterTcArgs& r = a.rt;
  if (nb == 0) {
    float rinv = 0.f;
    if (valid) {
      float ss = 0.f, dd = 0.f, dp = 0.f;
      const float4* pp = reinterpret_cast<const float4*>(r.part + (size_t)m * r.np * 4);
      for (int s = 0; s < r.np; ++s) {
        const float4 v = pp[s];
        ss += v.x;
        dd += v.y;
        dp += v.z;
      }
      rinv = rsqrtf(ss / (float)r.d + r.rms_eps);
      const float dj = r.j == 1 ? 0.f : sqrtf(dd);                       // Eq. 7
      const float gam = r.j > 2 ? dp / (dj * r.dprev[m] + r.eps) : 0.f;   // Eq. 8
      r.scal[(size_t)m * 4 + 0] = dj;
      r.scal[(size_t)m * 4 + 1] = gam;
    }
    uint16_t* row = r.enc3 + (size_t)m * 768;
#pragma unroll 1
    for (int c0 = 0; c0 < 256; c0 += 32) {
      uint32_t v[32];
      tmem_ld32(tbase + c0, v);
      if (valid) {
        float x[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) x[i] = siluf_(__uint_as_float(v[i]) * rinv);
        store_split32(row, c0, 256, x);
      }
    }
  } else {
    float bsum = 0.f;
#pragma unroll 1
    for (int c0 = 0; c0 < 256; c0 += 32) {
      uint32_t v[32];
      tmem_ld32(tbase + c0, v);
      if (valid) {
#pragma unroll
        for (int i = 0; i < 32; ++i)
          bsum = fmaf(__ldg(r.w.ps_w2 + c0 + i), siluf_(__uint_as_float(v[i]) + __ldg(r.w.ps_b1 + c0 + i)), bsum);
      }
    }
    if (valid) r.scal[(size_t)m * 4 + 2] = bsum;
  }
}

// Step 2: acc = z_h = W_hu enc (Eq. 5); the path vector (Eqs. 4, 6) and its encoder z_a
// (Eq. 9); s = [z_h; z_a] in fp32 and as three bf16 terms.
template <int BN>
__device__ __forceinline__ void epi_rt_s(const GemmArgs& a, uint32_t tbase, int m, bool valid) {
  const RouterTcArgs& r = a.rt;
  constexpr int DH = 48, DA = 16, DP = 16;   // d_h, d_a, d_path of this form (checked on host)
  float s[DH + DA];
#pragma unroll
  for (int c0 = 0; c0 < DH; c0 += 16) {
    uint32_t v[16];
    tmem_ld16(tbase + c0, v);
#pragma unroll
    for (int i = 0; i < 16; ++i) s[c0 + i] = __uint_as_float(v[i]);
  }
  if (!valid) return;
  const float* sc = r.scal + (size_t)m * 4;
  const float x[6] = {(float)r.j / (float)r.L, (float)(r.L - r.j) / (float)r.L, sc[0], sc[1],
                      r.pst[m], r.mst[m]};
  float hid[DP];
#pragma unroll
  for (int o = 0; o < DP; ++o) {
    float acc = __ldg(r.w.path_b1 + o);
#pragma unroll
    for (int i = 0; i < 6; ++i) acc = fmaf(__ldg(r.w.path_w1_t + i * DP + o), x[i], acc);
    hid[o] = siluf_(acc);
  }
#pragma unroll
  for (int o = 0; o < DA; ++o) {
    float acc = __ldg(r.w.path_b2 + o);
#pragma unroll
    for (int i = 0; i < DP; ++i) acc = fmaf(__ldg(r.w.path_w2_t + i * DA + o), hid[i], acc);
    s[DH + o] = acc;
  }
  float4* so = reinterpret_cast<float4*>(r.s + (size_t)m * (DH + DA));
#pragma unroll
  for (int i = 0; i < (DH + DA) / 4; ++i) so[i] = make_float4(s[4 * i], s[4 * i + 1], s[4 * i + 2], s[4 * i + 3]);
  uint16_t* row = r.s3 + (size_t)m * 3 * (DH + DA);
  float x32[32];
#pragma unroll
  for (int h = 0; h < (DH + DA) / 32; ++h) {
#pragma unroll
    for (int i = 0; i < 32; ++i) x32[i] = s[32 * h + i];
    store_split32(row, 32 * h, DH + DA, x32);
  }
}

// Step 5: acc = W_th1 [s; c; nu] (Eq. 14); a = w_th2 . SiLU(acc + b_th1) + b_th2,
// p_hist = sigma(a / T_hist), m_hist *= p_hist (Eq. 15), g = sigma(a + b) (Eq. 16) and the
// decision g >= tau (Eq. 3; ties run the FFN) or the caller's.
template <int BN>
__device__ __forceinline__ void epi_rt_head(const GemmArgs& a, uint32_t tbase, int m, bool valid,
                                            int ew, float4* stg, uint32_t* qcnt, int parity) {
  static_assert(BN == 256, "f_theta's hidden width is one tile");
  const RouterTcArgs& r = a.rt;
  // two epilogue warps per TMEM lane quadrant (8 warps): warp ew takes hidden units
  // [128 (ew >> 2), + 128) of its 32 rows
  const int lane = threadIdx.x & 31;
  const int c_lo = (ew >> 2) * 128;
  float asum = 0.f;
#pragma unroll 1
  for (int c0 = c_lo; c0 < c_lo + 128; c0 += 32) {
    uint32_t v[32];
    tmem_ld32(tbase + c0, v);
    if (valid) {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        asum = fmaf(__ldg(r.w.th_w2 + c0 + i), siluf_(__uint_as_float(v[i]) + __ldg(r.w.th_b1 + c0 + i)), asum);
    }
  }
  // The two halves of a row meet in the warps' staging areas, in a slot per tile parity, and
  // are counted on a counter per tile parity: a warp is at most one tile ahead of its
  // partner (it cannot reuse an accumulator before the partner released it), so a slot and
  // a counter only ever see the two arrivals of one tile at a time.  A counter grows by 2 per
  // use; the warp that finds it odd arrives second, adds the halves (lower half first) and
  // finishes the row.  No barrier between the warps.
  float* mine = reinterpret_cast<float*>(stg) + parity * 32;
  mine[lane] = asum;
  __syncwarp();
  __threadfence_block();
  uint32_t old = 0;
  if (lane == 0) old = atomicAdd(qcnt + parity, 1u);
  old = __shfl_sync(0xffffffffu, old, 0);
  if ((old & 1u) == 0) return;   // first of the two
  __threadfence_block();
  const float4* st0 = ew < 4 ? stg : stg - 4 * 256;   // the lower half's warp
  const float* lo = reinterpret_cast<const float*>(st0) + parity * 32;
  const float* hi = reinterpret_cast<const float*>(st0 + 4 * 256) + parity * 32;
  asum = lo[lane] + hi[lane];
  float p = 0.f, mm = 0.f, g = 0.f;
  const float* sc = r.scal + (size_t)m * 4;
  uint8_t dec = 0;
  if (valid) {
    const float av = asum + __ldg(r.w.th_b2);
    const float bv = sc[2] + __ldg(r.w.ps_b2);
    p = sigmoidf_(av / r.t_hist);
    mm = r.mst[m] * p;
    g = sigmoidf_(av + bv);
    dec = r.mask_in ? (r.mask_in[m] ? 1 : 0) : (g >= r.tau ? 1 : 0);
  }
  // the warp's 32 consecutive rows: their FFN count for the compaction
  const uint32_t bal = __ballot_sync(0xffffffffu, dec != 0);
  if (r.chunk_cnt && lane == 0 && m - lane < r.T) r.chunk_cnt[(m - lane) >> 5] = __popc(bal);
  if (!valid) return;
  r.pst[m] = p;
  r.mst[m] = mm;
  r.dprev[m] = sc[0];
  r.gate[m] = g;
  r.mask[m] = dec;
  if (r.gate_out) r.gate_out[m] = g;
  if (r.mask_out) r.mask_out[m] = dec;
}

// Fused q/k/v projection epilogue: one thread = one token row; the two halves of a
// head (columns i and i + 64) are read from TMEM together, q and k heads are
// rotated (RoPE, fp32), and each head's 128 values are stored as bf16 into its
// [sequence][head][position][128] array (64 contiguous bytes per store group).
template <int BN>
__device__ __forceinline__ void epi_qkv_rope(const GemmArgs& a, uint32_t tbase, int m, bool valid,
                                             int nb) {
  static_assert(BN % 128 == 0, "whole heads per tile");
  const RopeArgs& r = a.rope;
  const int heads = r.H + 2 * r.Hkv;
  int bq = 0, s = 0, sq = 0;
  if (valid) {
    if (r.pos) {   // decoding step: row = sequence, its position from memory
      bq = m;
      s = r.pos[m];
      if (s < 0 || s >= r.S_kv) {   // outside the cache: report, store nothing
        if (nb == 0) atomicOr(a.err, ERR_BAD_INDEX);
        valid = false;
      }
    } else {
      bq = m / r.S;
      s = m - bq * r.S;
      sq = s;
    }
  }
#pragma unroll 1
  for (int hb = 0; hb < BN; hb += 128) {
    const int head = (nb * BN + hb) >> 7;
    if (head >= heads) break;                      // uniform over the warp
#pragma unroll 1
    for (int c0 = 0; c0 < 64; c0 += 32) {
      uint32_t x1[32], x2[32];
      tmem_ld32(tbase + hb + c0, x1);
      tmem_ld32(tbase + hb + c0 + 64, x2);
      if (!valid) continue;
      uint16_t* dst;
      const bool rot = head < r.H + r.Hkv;
      if (!rot && r.vt) {   // v transposed: element e of this token at [e][s]
        uint16_t* vt = static_cast<uint16_t*>(r.vt) +
                       ((size_t)bq * r.Hkv + head - r.H - r.Hkv) * 128 * (size_t)r.S_pad + s;
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          vt[(size_t)(c0 + e) * r.S_pad] =
              (uint16_t)(pack_bf16x2(__uint_as_float(x1[e]), 0.f) & 0xffffu);
          vt[(size_t)(c0 + 64 + e) * r.S_pad] =
              (uint16_t)(pack_bf16x2(__uint_as_float(x2[e]), 0.f) & 0xffffu);
        }
      }
      if (!rot && !r.v) continue;
      if (head < r.H)
        dst = static_cast<uint16_t*>(r.q) + (((size_t)bq * r.H + head) * r.S_q + sq) * 128;
      else if (rot)
        dst = static_cast<uint16_t*>(r.k) + (((size_t)bq * r.Hkv + head - r.H) * r.S_kv + s) * 128;
      else
        dst = static_cast<uint16_t*>(r.v) +
              (((size_t)bq * r.Hkv + head - r.H - r.Hkv) * r.S_kv + s) * 128;
      uint32_t p1[16], p2[16];
      const float4* cs = reinterpret_cast<const float4*>(r.cs + ((size_t)s * 64 + c0) * 2);
#pragma unroll
      for (int e = 0; e < 32; e += 2) {
        float a0 = __uint_as_float(x1[e]), a1 = __uint_as_float(x1[e + 1]);
        float b0 = __uint_as_float(x2[e]), b1 = __uint_as_float(x2[e + 1]);
        if (rot) {
          const float4 t = __ldg(cs + (e >> 1));   // (cos, sin) of pairs e and e + 1
          const float y0 = a0 * t.x - b0 * t.y, z0 = b0 * t.x + a0 * t.y;
          const float y1 = a1 * t.z - b1 * t.w, z1 = b1 * t.z + a1 * t.w;
          a0 = y0; b0 = z0; a1 = y1; b1 = z1;
        }
        p1[e >> 1] = pack_bf16x2(a0, a1);
        p2[e >> 1] = pack_bf16x2(b0, b1);
      }
      uint4* d1 = reinterpret_cast<uint4*>(dst + c0);
      uint4* d2 = reinterpret_cast<uint4*>(dst + c0 + 64);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        d1[i] = make_uint4(p1[4 * i], p1[4 * i + 1], p1[4 * i + 2], p1[4 * i + 3]);
        d2[i] = make_uint4(p2[4 * i], p2[4 * i + 1], p2[4 * i + 2], p2[4 * i + 3]);
      }
    }
  }
}

// Block-closing epilogue over columns [c_begin, c_begin + NCOLS) of the tile,
// row-contiguous through the staging tile.  Each lane keeps the partial sums of
// its 8 rows; every kTcPartCols columns they are reduced over the 8 lanes that
// share a row and stored as one partial-sum slot.
template <int BN, int NCOLS>
__device__ __forceinline__ void flush_partials(const LayerOutArgs& p, const int (&tok)[8],
                                               float (&ss)[8], float (&dd)[8], float (&dp)[8],
                                               int slot_lane, int pslot) {
#pragma unroll
  for (int k = 0; k < 8; ++k) {
#pragma unroll
    for (int o = 1; o < 8; o <<= 1) {
      ss[k] += __shfl_xor_sync(0xffffffffu, ss[k], o);
      dd[k] += __shfl_xor_sync(0xffffffffu, dd[k], o);
      dp[k] += __shfl_xor_sync(0xffffffffu, dp[k], o);
    }
    if (slot_lane == 0 && tok[k] >= 0)
      *reinterpret_cast<float4*>(p.part + ((size_t)tok[k] * p.np + pslot) * 4) =
          make_float4(ss[k], dd[k], dp[k], 0.f);
    ss[k] = dd[k] = dp[k] = 0.f;
  }
}

template <int BN, int NCOLS>
__device__ __forceinline__ void epi_layer_out(const GemmArgs& a, uint32_t tbase, int row0, int M,
                                              int nb, int c_begin, float4* st) {
  static_assert(NCOLS % kTcPartCols == 0, "whole partial-sum slots per warp");
  const int lane = threadIdx.x & 31;
  const int sub = lane >> 3, slot = lane & 7;
  const LayerOutArgs& p = a.lo;
  int tok[8];
  float scl[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int m = row0 + sub + 4 * k;
    tok[k] = m < M ? p.idx[m] : -1;
    scl[k] = m < M ? p.scale[m] : 0.f;
  }
  float ss[8], dd[8], dp[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) ss[k] = dd[k] = dp[k] = 0.f;
#pragma unroll 1
  for (int c0 = c_begin; c0 < c_begin + NCOLS; c0 += 32) {
    uint32_t r[32];
    tmem_ld32(tbase + c0, r);
    stage_rows(st, r, lane);
    __syncwarp();
    const int n = nb * BN + c0 + 4 * slot;
    // two groups of 4 rows: issue every load of a group before any store
#pragma unroll
    for (int k0 = 0; k0 < 8; k0 += 4) {
      LayerOutIn in[4];
#pragma unroll
      for (int k = 0; k < 4; ++k)
        if (tok[k0 + k] >= 0) in[k] = layer_out_load(p, tok[k0 + k], n);
#pragma unroll
      for (int k = 0; k < 4; ++k)
        if (tok[k0 + k] >= 0)
          layer_out_store(p, tok[k0 + k], n, in[k], staged(st, sub + 4 * (k0 + k), slot),
                          scl[k0 + k], ss[k0 + k], dd[k0 + k], dp[k0 + k]);
    }
    __syncwarp();
    if (!p.last && (c0 + 32) % kTcPartCols == 0)
      flush_partials<BN, NCOLS>(p, tok, ss, dd, dp, slot, (nb * BN + c0 + 32) / kTcPartCols - 1);
  }
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async8(uint32_t dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(dst), "l"(src) : "memory");
}

// The block-closing epilogue with its row inputs copied into shared memory (inb: this
// warp's [3][8][32] 16-byte slots: h_bar, delta, P_{j+1} of the lane's 4 columns of its 8
// rows) by cp.async, issued for a whole 32-column chunk before the accumulator is read from
// TMEM, so that a chunk's loads are in flight together without holding registers.  The
// arithmetic and its order are epi_layer_out's.
template <int BN, int NCOLS>
__device__ __forceinline__ void epi_layer_out_async(const GemmArgs& a, uint32_t tbase, int row0,
                                                    int M, int nb, int c_begin, float4* st,
                                                    float4* inb) {
  static_assert(NCOLS % kTcPartCols == 0, "whole partial-sum slots per warp");
  const int lane = threadIdx.x & 31;
  const int sub = lane >> 3, slot = lane & 7;
  const LayerOutArgs& p = a.lo;
  const bool need_pn = !p.last && p.p_next;
  const bool need_dv = !p.last && p.router && !p.first;
  int tok[8];
  float scl[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int m = row0 + sub + 4 * k;
    tok[k] = m < M ? p.idx[m] : -1;
    scl[k] = m < M ? p.scale[m] : 0.f;
  }
  float ss[8], dd[8], dp[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) ss[k] = dd[k] = dp[k] = 0.f;
  const uint32_t ib = smem_u32(inb);
  auto slot_addr = [&](int arr, int k) { return ib + (uint32_t)(((arr * 8 + k) * 32 + lane) * 16); };
#pragma unroll 1
  for (int c0 = c_begin; c0 < c_begin + NCOLS; c0 += 32) {
    const int n = nb * BN + c0 + 4 * slot;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if (tok[k] < 0) continue;
      const size_t off = (size_t)tok[k] * p.d + n;
      cp_async16(slot_addr(0, k), p.hbar + off);
      if (need_dv) cp_async16(slot_addr(1, k), p.delta + off);
      if (need_pn) {
        if (p.p_bf16)
          cp_async8(slot_addr(2, k), static_cast<const uint16_t*>(p.p_next) + off);
        else
          cp_async16(slot_addr(2, k), static_cast<const float*>(p.p_next) + off);
      }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    uint32_t r[32];
    tmem_ld32(tbase + c0, r);
    stage_rows(st, r, lane);
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncwarp();
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      if (tok[k] < 0) continue;
      LayerOutIn in;
      in.hb = inb[(0 * 8 + k) * 32 + lane];
      in.dprev = need_dv ? inb[(1 * 8 + k) * 32 + lane] : make_float4(0.f, 0.f, 0.f, 0.f);
      in.pn = make_float4(0.f, 0.f, 0.f, 0.f);
      if (need_pn) {
        if (p.p_bf16) {
          const uint2 u = *reinterpret_cast<const uint2*>(&inb[(2 * 8 + k) * 32 + lane]);
          in.pn = make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u),
                              __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
        } else {
          in.pn = inb[(2 * 8 + k) * 32 + lane];
        }
      }
      layer_out_store(p, tok[k], n, in, staged(st, sub + 4 * k, slot), scl[k], ss[k], dd[k], dp[k]);
    }
    __syncwarp();
    if (!p.last && (c0 + 32) % kTcPartCols == 0)
      flush_partials<BN, NCOLS>(p, tok, ss, dd, dp, slot, (nb * BN + c0 + 32) / kTcPartCols - 1);
  }
}

// Attention output projection closing into the block entry (Eq. 7): per element
// h_bar_j = h_{j-1} + acc, delta_j = h_bar_j - h_bar_{j-1} (zero in the first routed
// block); h_bar_j and delta_j overwrite the carried h_bar_{j-1} and delta_{j-1}
// after the same thread has read them; partial sums of h_bar_j^2, delta_j^2 and
// delta_j . delta_{j-1} per 128-column slot.  Rows are tokens.
template <int BN, int NCOLS>
__device__ __forceinline__ void epi_attn_entry(const GemmArgs& a, uint32_t tbase, int row0, int M,
                                               int nb, int c_begin, float4* st) {
  static_assert(NCOLS % kTcPartCols == 0, "whole partial-sum slots per warp");
  const int lane = threadIdx.x & 31;
  const int sub = lane >> 3, slot = lane & 7;
  const LayerOutArgs& p = a.lo;
  const bool rt = p.router, carry = p.router && !p.first;
  int tok[8];
  float ss[8], dd[8], dp[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const int m = row0 + sub + 4 * k;
    tok[k] = m < M ? m : -1;
    ss[k] = dd[k] = dp[k] = 0.f;
  }
#pragma unroll 1
  for (int c0 = c_begin; c0 < c_begin + NCOLS; c0 += 32) {
    uint32_t r[32];
    tmem_ld32(tbase + c0, r);
    stage_rows(st, r, lane);
    __syncwarp();
    const int n = nb * BN + c0 + 4 * slot;
#pragma unroll
    for (int k0 = 0; k0 < 8; k0 += 4) {
      float4 hr[4], hp[4], dv[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int t = tok[k0 + k];
        if (t < 0) continue;
        const size_t off = (size_t)t * p.d + n;
        hr[k] = *reinterpret_cast<const float4*>(a.resid + off);
        if (carry) {
          hp[k] = *reinterpret_cast<const float4*>(p.hbar + off);
          dv[k] = *reinterpret_cast<const float4*>(p.delta + off);
        }
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int t = tok[k0 + k];
        if (t < 0) continue;
        const size_t off = (size_t)t * p.d + n;
        const float4 y = staged(st, sub + 4 * (k0 + k), slot);
        const float4 hn = make_float4(hr[k].x + y.x, hr[k].y + y.y, hr[k].z + y.z, hr[k].w + y.w);
        *reinterpret_cast<float4*>(p.hbar + off) = hn;
        ss[k0 + k] += hn.x * hn.x + hn.y * hn.y + hn.z * hn.z + hn.w * hn.w;
        if (rt) {
          float4 dl = make_float4(0.f, 0.f, 0.f, 0.f);
          if (carry) {
            dl = make_float4(hn.x - hp[k].x, hn.y - hp[k].y, hn.z - hp[k].z, hn.w - hp[k].w);
            dp[k0 + k] += dl.x * dv[k].x + dl.y * dv[k].y + dl.z * dv[k].z + dl.w * dv[k].w;
          }
          dd[k0 + k] += dl.x * dl.x + dl.y * dl.y + dl.z * dl.z + dl.w * dl.w;
          *reinterpret_cast<float4*>(p.delta + off) = dl;
          store_xl4(p.xl, p.xl_bf16, p.d, t, n, hn);
        }
      }
    }
    __syncwarp();
    if ((c0 + 32) % kTcPartCols == 0)
      flush_partials<BN, NCOLS>(p, tok, ss, dd, dp, slot, (nb * BN + c0 + 32) / kTcPartCols - 1);
  }
}

// Sizes of one problem of a launch (the row count may be device-resident).  With
// split-K the tile index runs over splits x M-tiles x N-tiles and split s covers
// K-blocks [s * kpb, min((s + 1) * kpb, kblocks)).
struct ProbSize {
  int M, m_tiles, n_tiles, kblocks, tiles, kpb;
};

// Tile `local` of a problem -> coordinates and K-block range.
template <int CG = 1>
__device__ __forceinline__ void tile_work(const ProbSize& p, int local, int& mb, int& nb, int& s,
                                          int& kb0, int& kb1);

template <int BN, int CG = 1>
__device__ __forceinline__ ProbSize prob_size(const GemmArgs& a) {
  ProbSize p;
  int M = a.m_dev ? *a.m_dev : a.m_static;
  if (M < 0 || M > a.m_max) {
    if (threadIdx.x == 0) atomicOr(a.err, ERR_BAD_INDEX);
    M = 0;
  }
  p.M = M;
  p.m_tiles = (M + BM * CG - 1) / (BM * CG);   // M-tiles of the CTA or the CTA pair
  p.n_tiles = (a.N + BN - 1) / BN;
  p.kblocks = (a.K + BK - 1) / BK;
  const int splits = a.k_splits > 1 ? a.k_splits : 1;
  p.kpb = (p.kblocks + splits - 1) / splits;
  p.tiles = p.m_tiles * p.n_tiles * splits;
  return p;
}

template <int CG>
__device__ __forceinline__ void tile_work(const ProbSize& p, int local, int& mb, int& nb, int& s,
                                          int& kb0, int& kb1) {
  const int per_split = p.m_tiles * p.n_tiles;
  s = local / per_split;
  tile_coords(local - s * per_split, p.m_tiles, p.n_tiles, mb, nb, kGroupM / CG);
  kb0 = s * p.kpb;
  kb1 = min(p.kblocks, kb0 + p.kpb);
}

// Tile g of a grouped launch -> (problem, tile within it): the second problem's
// t1 tiles are spread evenly among all `total` tiles (Bresenham), so every
// persistent CTA gets its share of both.
__device__ __forceinline__ int split_tile(int g, int t1, int total, int& local) {
  if (t1 == 0) {
    local = g;
    return 0;
  }
  const int before = (int)(((long long)g * t1) / total);
  const int upto = (int)(((long long)(g + 1) * t1) / total);
  if (upto > before) {
    local = before;
    return 1;
  }
  local = g - before;
  return 0;
}

// Epilogue warp ew serves TMEM lane quadrant q = ew % 4; with 8 epilogue warps the
// second warp of a quadrant takes the upper half of the columns.
template <int BN, int EPI, int CG>
__device__ __forceinline__ void run_epilogue(const GemmArgs& a, uint32_t tbase, int q, int ew,
                                             int lane, int mb, int nb, int M, int split,
                                             float4* stg, int rank, uint32_t* qcnt = nullptr,
                                             int parity = 0, float4* inb = nullptr) {
  const int row0 = (mb * CG + rank) * BM + q * 32;
  if constexpr (EPI == EPI_STORE_F32) {
    epi_store_f32<BN>(a, tbase, row0, M, nb, split, stg);
  } else if constexpr (EPI == EPI_RESIDUAL) {
    epi_store_f32<BN, true>(a, tbase, row0, M, nb, split, stg);
  } else if constexpr (EPI == EPI_ATTN_ENTRY) {
    epi_attn_entry<BN, BN / 2>(a, tbase, row0, M, nb, (ew >> 2) * (BN / 2), stg);
  } else if constexpr (EPI == EPI_QKV_ROPE) {
    epi_qkv_rope<BN>(a, tbase, row0 + lane, row0 + lane < M, nb);
  } else if constexpr (EPI == EPI_SWIGLU) {
    epi_swiglu(a, tbase, row0 + lane, row0 + lane < M, nb);
  } else if constexpr (EPI == EPI_SILU) {
    epi_silu<BN>(a, tbase, row0 + lane, row0 + lane < M, nb);
  } else if constexpr (EPI == EPI_STORE_BF16) {
    epi_store_bf16<BN>(a, tbase, row0 + lane, row0 + lane < M, nb);
  } else if constexpr (EPI == EPI_BW_SWIGLU) {
    epi_bw_swiglu<BN>(a, tbase, row0 + lane, row0 + lane < M, nb);
  } else if constexpr (EPI == EPI_RT_ENC) {
    epi_rt_enc<BN>(a, tbase, row0 + lane, row0 + lane < M, nb);
  } else if constexpr (EPI == EPI_RT_S) {
    epi_rt_s<BN>(a, tbase, row0 + lane, row0 + lane < M);
  } else if constexpr (EPI == EPI_RT_HEAD) {
    epi_rt_head<BN>(a, tbase, row0 + lane, row0 + lane < M, ew, stg, qcnt + 2 * q, parity);
  } else if constexpr (EPI == EPI_LAYER_OUT) {
    epi_layer_out<BN, BN>(a, tbase, row0, M, nb, 0, stg);
  } else if constexpr (EPI == EPI_LAYER_OUT_WIDE && HERO_WIDE_INBUF) {
    epi_layer_out_async<BN, BN / 2>(a, tbase, row0, M, nb, (ew >> 2) * (BN / 2), stg, inb);
  } else {
    epi_layer_out<BN, BN / 2>(a, tbase, row0, M, nb, (ew >> 2) * (BN / 2), stg);
  }
}

template <int BN, int EPI0, int EPI1, int CG>
__global__ void __launch_bounds__(TcCfg<BN, epi_warps<EPI0>(), CG, epi_inbuf<EPI0>()>::THREADS, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmB0,
              const __grid_constant__ CUtensorMap tmA1, const __grid_constant__ CUtensorMap tmB1,
              const GemmArgs a0, const GemmArgs a1) {
  if (a0.pdl_mode != 2) pdl_enter();
  using C = TcCfg<BN, epi_warps<EPI0>(), CG, epi_inbuf<EPI0>()>;
  constexpr bool kGrouped = EPI1 != EPI_NONE;
  constexpr bool kPair = CG == 2;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::STAGES * C::STAGE_BYTES);
  // bars: full[STAGES], empty[STAGES], tfull[2], tempty[2], drain
  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (C::STAGES + s); };
  auto tfull_bar = [&](int a) { return bar0 + 8u * (2 * C::STAGES + a); };
  auto tempty_bar = [&](int a) { return bar0 + 8u * (2 * C::STAGES + 2 + a); };
  const uint32_t drain_bar = bar0 + 8u * (2 * C::STAGES + 4);
  volatile uint32_t* misc = reinterpret_cast<volatile uint32_t*>(bars + 2 * C::STAGES + 5);
  const uint32_t smem_base = smem_u32(smem);
  auto sA = [&](int s) { return smem_base + s * C::STAGE_BYTES; };
  auto sB = [&](int s) { return smem_base + s * C::STAGE_BYTES + C::A_BYTES; };
  uint32_t* err = a0.err;
  const uint64_t wait_ns = a0.wait_ns;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // A CTA pair works on one tile: the even CTA (rank 0) issues the MMAs, waits for both
  // CTAs' operand copies on its full barriers and for both CTAs' epilogues on its
  // accumulator-empty barriers; its commits arrive on the barriers of both CTAs.
  const int rank = kPair ? (int)cluster_ctarank() : 0;
  const bool issuer = rank == 0;
  const int unit = blockIdx.x / CG, n_units = gridDim.x / CG;
  // barrier addresses of the pair's even CTA (its own for rank 0)
  const uint32_t bar0_lead = kPair ? mapa_shared(bar0, 0) : bar0;

  const ProbSize P0 = prob_size<BN, CG>(a0);
  ProbSize P1{0, 0, 0, 0, 0};
  if constexpr (kGrouped) P1 = prob_size<BN, CG>(a1);
  const int total = P0.tiles + P1.tiles;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull_bar(a), 1);
      mbar_init(tempty_bar(a), C::EPI_WARPS * CG);
    }
    mbar_init(drain_bar, 1);
    misc[1] = 0;  // abort flag
    for (int i = 4; i < 12; ++i) misc[i] = 0;   // EPI_RT_HEAD: counters per quadrant and parity
    fence_mbar_init();
  }
  // both CTAs' barriers are initialised before either signals the other's (and before
  // the allocation below, so that no CTA waits on its partner while holding TMEM)
  if constexpr (kPair) cluster_sync();
  if (warp == 1) {
    if constexpr (kPair) {   // one warp of each CTA of the pair, collectively
      tmem_alloc_pair(smem_u32(const_cast<uint32_t*>(misc)), C::TMEM_COLS);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(smem_u32(const_cast<uint32_t*>(misc)), C::TMEM_COLS);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = misc[0];

  if (warp == 0) {
    // ------------------------------ TMA producer ------------------------------
    if (lane == 0 && total > 0) {
      tma_prefetch_desc(&tmA0);
      tma_prefetch_desc(&tmB0);
      if constexpr (kGrouped) {
        tma_prefetch_desc(&tmA1);
        tma_prefetch_desc(&tmB1);
      }
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0, last_par = 0;  // per-stage bit masks for the drain
      bool ok = true;
      for (int g = unit; g < total && ok; g += n_units) {
        int local;
        const int pr = split_tile(g, P1.tiles, total, local);
        int mb, nb, sp, kb0, kb1;
        tile_work<CG>(pr ? P1 : P0, local, mb, nb, sp, kb0, kb1);
        const CUtensorMap* tA = pr ? &tmA1 : &tmA0;
        const CUtensorMap* tB = pr ? &tmB1 : &tmB0;
        if (a0.pdl_mode == 1 && g + n_units >= total)   // this CTA's last tile
          asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
        const int ya = (mb * CG + rank) * BM, yb = nb * BN + rank * C::B_ROWS;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(empty_bar(stage), phase ^ 1u, wait_ns) || misc[1]) {
            ok = false;
            break;
          }
          if constexpr (kPair) {
            // both CTAs' copies complete on the even CTA's full barrier, which expects
            // the bytes of the pair
            const uint32_t fb = bar0_lead + 8u * stage;
            if (issuer) mbar_arrive_expect_tx(full_bar(stage), CG * C::STAGE_BYTES);
            tma_load_2d_pair(sA(stage), tA, kb * BK, ya, fb);
            tma_load_2d_pair(sB(stage), tB, kb * BK, yb, fb);
          } else {
            mbar_arrive_expect_tx(full_bar(stage), C::STAGE_BYTES);
            tma_load_2d(sA(stage), tA, kb * BK, ya, full_bar(stage));
            tma_load_2d(sB(stage), tB, kb * BK, yb, full_bar(stage));
          }
          issued |= 1u << stage;
          last_par = (last_par & ~(1u << stage)) | (phase << stage);
          if (++stage == C::STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        misc[1] = 1;
        atomicOr(err, ERR_WAIT_PRODUCER);
      }
      if (issuer) {
        // Let every copy issued into the stages land before the CTA can exit, also when
        // the loop ended normally: if another role gave up early, stages it never
        // consumed may still be in flight.  (Normally they have landed already.)
        for (int s = 0; s < C::STAGES; ++s)
          if ((issued & (1u << s)) && !mbar_wait(full_bar(s), (last_par >> s) & 1u, kDrainLimitNs))
            atomicOr(err, ERR_WAIT_DRAIN);
      } else if (!ok) {
        // the odd CTA's copies complete on the even CTA's barriers, which it cannot
        // wait on: after an abort, give copies in flight a fixed grace period
        const uint64_t t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < 2000000ull) {
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------ MMA issuer ------------------------------
    if (lane == 0 && total > 0 && issuer) {
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int g = unit; g < total && ok; g += n_units) {
        int local;
        const int pr = split_tile(g, P1.tiles, total, local);
        int mb, nb, sp, kb0, kb1;
        tile_work<CG>(pr ? P1 : P0, local, mb, nb, sp, kb0, kb1);
        if (!mbar_wait(tempty_bar(acc), acc_phase ^ 1u, wait_ns) || misc[1]) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(full_bar(stage), phase, wait_ns) || misc[1]) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t adesc = sw128_desc(sA(stage));
          const uint64_t bdesc = sw128_desc(sB(stage));
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            // +32 bytes per K step of 16 bf16 inside the 128-byte swizzle row
            if constexpr (kPair)
              umma_bf16_pair(d_tmem, adesc + 2u * k, bdesc + 2u * k, C::IDESC, (kb != kb0) || k != 0);
            else
              umma_bf16(d_tmem, adesc + 2u * k, bdesc + 2u * k, C::IDESC, (kb != kb0) || k != 0);
          }
          if constexpr (kPair)
            umma_commit_pair(empty_bar(stage));   // frees the stage in both CTAs
          else
            umma_commit(empty_bar(stage));
          if (++stage == C::STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        if constexpr (kPair)
          umma_commit_pair(tfull_bar(acc));
        else
          umma_commit(tfull_bar(acc));
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
      if (!ok) {
        misc[1] = 1;
        atomicOr(err, ERR_WAIT_MMA);
      }
      // Every MMA this thread issued completes before TMEM is freed, also when the
      // loop ended normally but an epilogue warp gave up on a tile still in flight.
      if constexpr (kPair)
        umma_commit_pair(drain_bar);   // arrives in both CTAs once every MMA has finished
      else
        umma_commit(drain_bar);
      if (!mbar_wait(drain_bar, 0, kDrainLimitNs)) atomicOr(err, ERR_WAIT_DRAIN);
    }
  } else {
    // ------------------------------ epilogue ------------------------------
    const int q = warp & 3;  // TMEM lane quadrant this warp may access
    const int ew = warp - 2;  // epilogue warp index
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int g = unit; g < total; g += n_units) {
      int local;
      const int pr = split_tile(g, P1.tiles, total, local);
      int mb, nb, sp, kb0, kb1;
      tile_work<CG>(pr ? P1 : P0, local, mb, nb, sp, kb0, kb1);
      bool ok = mbar_wait(tfull_bar(acc), acc_phase, wait_ns);
      ok = __all_sync(0xffffffffu, ok) && !misc[1];
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) {
        if (lane == 0) {
          misc[1] = 1;
          atomicOr(err, ERR_WAIT_EPILOGUE);
        }
        break;
      }
      tc_fence_after();
      const uint32_t tbase = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
      float4* stg = reinterpret_cast<float4*>(smem + C::EPI_STAGE_OFF) + ew * (32 * 8);
      if constexpr (kGrouped) {
        if (pr)
          run_epilogue<BN, EPI1, CG>(a1, tbase, q, ew, lane, mb, nb, P1.M, sp, stg, rank);
        else
          run_epilogue<BN, EPI0, CG>(a0, tbase, q, ew, lane, mb, nb, P0.M, sp, stg, rank);
      } else {
        run_epilogue<BN, EPI0, CG>(a0, tbase, q, ew, lane, mb, nb, P0.M, sp, stg, rank,
                                   const_cast<uint32_t*>(misc) + 4, acc,
                                   reinterpret_cast<float4*>(smem + C::IN_OFF + ew * C::IN_BYTES));
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if constexpr (kPair)
          mbar_arrive_cluster(bar0_lead + 8u * (2 * C::STAGES + 2 + acc));
        else
          mbar_arrive(tempty_bar(acc));
      }
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    if constexpr (kPair) {
      // the odd CTA's accumulator is written by the even CTA's MMAs: wait for their
      // completion (the even CTA's drain commit) before freeing TMEM
      if (!issuer && total > 0) {
        bool w = true;
        if (lane == 0) w = mbar_wait(drain_bar, 0, kDrainLimitNs);
        if (!__shfl_sync(0xffffffffu, w ? 1 : 0, 0) && lane == 0) atomicOr(err, ERR_WAIT_DRAIN);
      }
      tc_fence_after();
      tmem_dealloc_pair(tmem_base, C::TMEM_COLS);
    } else {
      tc_fence_after();
      tmem_dealloc(tmem_base, C::TMEM_COLS);
    }
  }
  if constexpr (kPair) cluster_sync();   // neither CTA exits while the other may signal it
  if (a0.pdl_mode == 2) pdl_enter();   // complete only after the previous kernel
}

template <int BN, int EPI0, int EPI1, int CG = 1>
cudaError_t launch_tc(const CUtensorMap& tmA0, const CUtensorMap& tmB0, const GemmArgs& a0,
                      const CUtensorMap& tmA1, const CUtensorMap& tmB1, const GemmArgs& a1,
                      int num_sms, cudaStream_t st) {
  using C = TcCfg<BN, epi_warps<EPI0>(), CG, epi_inbuf<EPI0>()>;
  auto kernel = k_gemm_tc<BN, EPI0, EPI1, CG>;
  static bool attr_set = false;  // per process; the attribute is per function
  static int pair_slots = 0;     // CG = 2: CTA pairs resident at once
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
    if (e != cudaSuccess) return e;
    if (CG == 2) {
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = CG;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = 1;
      cudaLaunchConfig_t q = {};
      q.gridDim = dim3(CG * (num_sms / CG));
      q.blockDim = dim3(C::THREADS);
      q.dynamicSmemBytes = C::SMEM;
      q.attrs = at;
      q.numAttrs = 1;
      e = cudaOccupancyMaxActiveClusters(&pair_slots, kernel, &q);
      if (e != cudaSuccess) return e;
      if (pair_slots < 1) return cudaErrorInvalidConfiguration;
    }
    attr_set = true;
  }
  if (a0.k_splits > 1 && (EPI0 != EPI_STORE_F32 || CG != 1)) return cudaErrorInvalidValue;
  const long kb0 = (a0.K + BK - 1) / BK;
  if (a0.k_splits > 1 && (a0.k_splits > kb0 || (long)(a0.k_splits - 1) *
                                                 ((kb0 + a0.k_splits - 1) / a0.k_splits) >= kb0))
    return cudaErrorInvalidValue;   // every split must own at least one K-block
  const long tile_rows = (long)BM * CG;
  long max_tiles = (long)((a0.m_max + tile_rows - 1) / tile_rows) * ((a0.N + BN - 1) / BN) *
                   (a0.k_splits > 1 ? a0.k_splits : 1);
  if (EPI1 != EPI_NONE)
    max_tiles += (long)((a1.m_max + tile_rows - 1) / tile_rows) * ((a1.N + BN - 1) / BN);
  if (max_tiles <= 0) return cudaSuccess;
  const long slots = CG == 2 ? (long)pair_slots : (long)num_sms;
  const int units = (int)(max_tiles < slots ? max_tiles : slots);
  GemmArgs b0 = a0;
  b0.wait_ns = wait_limit_ns();
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = CG;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(units * CG);
  cfg.blockDim = dim3(C::THREADS);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = CG == 2 ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kernel, tmA0, tmB0, tmA1, tmB1, b0, a1);
}

bool qkv_args_ok(const GemmArgs& a) {
  return a.N == (a.rope.H + 2 * a.rope.Hkv) * 128 && a.rope.S > 0 && a.rope.S_q > 0 &&
         a.rope.S_kv > 0 && (a.rope.pos || a.rope.S_kv >= a.rope.S);
}

bool bw_swiglu_args_ok(const GemmArgs& a) {
  return a.N % 32 == 0 && a.ldo >= 2 * a.N && a.row_scale && a.row_part &&
         a.part_ld >= (a.N + 255) / 256;
}

}  // namespace

cudaError_t launch_gemm_tc(int bn, EpiKind epi, const CUtensorMap& tmA, const CUtensorMap& tmB,
                           const GemmArgs& args, int num_sms, cudaStream_t st) {
  if (bn != 256) return cudaErrorInvalidValue;
  const GemmArgs none{};
  switch (epi) {
    case EPI_STORE_F32:
      return launch_tc<256, EPI_STORE_F32, EPI_NONE>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_SWIGLU:
      return launch_tc<256, EPI_SWIGLU, EPI_NONE>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_LAYER_OUT:
      return launch_tc<256, EPI_LAYER_OUT, EPI_NONE>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_LAYER_OUT_WIDE:
      return launch_tc<256, EPI_LAYER_OUT_WIDE, EPI_NONE>(tmA, tmB, args, tmA, tmB, none, num_sms,
                                                          st);
    case EPI_RESIDUAL:
      return launch_tc<256, EPI_RESIDUAL, EPI_NONE>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_QKV_ROPE:
      if (!qkv_args_ok(args)) return cudaErrorInvalidValue;
      return launch_tc<256, EPI_QKV_ROPE, EPI_NONE>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_ATTN_ENTRY:
      if (args.lo.d != args.N || args.ldo != args.N) return cudaErrorInvalidValue;
      return launch_tc<256, EPI_ATTN_ENTRY, EPI_NONE>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_STORE_BF16:
      if (args.N % 32 != 0) return cudaErrorInvalidValue;
      return launch_tc<256, EPI_STORE_BF16, EPI_NONE>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_BW_SWIGLU:
      if (!bw_swiglu_args_ok(args)) return cudaErrorInvalidValue;
      return launch_tc<256, EPI_BW_SWIGLU, EPI_NONE>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    default:
      return cudaErrorInvalidValue;
  }
}

cudaError_t launch_gemm_tc2(EpiKind epi, const CUtensorMap& tmA, const CUtensorMap& tmB,
                            const GemmArgs& args, int num_sms, cudaStream_t st) {
  const GemmArgs none{};
  switch (epi) {
    case EPI_STORE_F32:
      return launch_tc<256, EPI_STORE_F32, EPI_NONE, 2>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_SWIGLU:
      return launch_tc<256, EPI_SWIGLU, EPI_NONE, 2>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_LAYER_OUT:
      return launch_tc<256, EPI_LAYER_OUT, EPI_NONE, 2>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_RESIDUAL:
      return launch_tc<256, EPI_RESIDUAL, EPI_NONE, 2>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_QKV_ROPE:
      if (!qkv_args_ok(args)) return cudaErrorInvalidValue;
      return launch_tc<256, EPI_QKV_ROPE, EPI_NONE, 2>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_ATTN_ENTRY:
      if (args.lo.d != args.N || args.ldo != args.N) return cudaErrorInvalidValue;
      return launch_tc<256, EPI_ATTN_ENTRY, EPI_NONE, 2>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_STORE_BF16:
      if (args.N % 32 != 0) return cudaErrorInvalidValue;
      return launch_tc<256, EPI_STORE_BF16, EPI_NONE, 2>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_BW_SWIGLU:
      if (!bw_swiglu_args_ok(args)) return cudaErrorInvalidValue;
      return launch_tc<256, EPI_BW_SWIGLU, EPI_NONE, 2>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_RT_ENC:
      if (args.N != 512) return cudaErrorInvalidValue;
      return launch_tc<256, EPI_RT_ENC, EPI_NONE, 2>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_RT_S:
      if (args.N != 48 || args.rt.d_h != 48 || args.rt.d_a != 16 || args.rt.d_path != 16)
        return cudaErrorInvalidValue;
      return launch_tc<256, EPI_RT_S, EPI_NONE, 2>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    case EPI_RT_HEAD:
      if (args.N != 256) return cudaErrorInvalidValue;
      return launch_tc<256, EPI_RT_HEAD, EPI_NONE, 2>(tmA, tmB, args, tmA, tmB, none, num_sms, st);
    default:
      return cudaErrorInvalidValue;
  }
}

cudaError_t launch_gemm_tc2_pair(EpiKind epi0, const CUtensorMap& tmA0, const CUtensorMap& tmB0,
                                 const GemmArgs& a0, EpiKind epi1, const CUtensorMap& tmA1,
                                 const CUtensorMap& tmB1, const GemmArgs& a1, int num_sms,
                                 cudaStream_t st) {
  if (epi0 == EPI_SWIGLU && epi1 == EPI_SILU)
    return launch_tc<256, EPI_SWIGLU, EPI_SILU, 2>(tmA0, tmB0, a0, tmA1, tmB1, a1, num_sms, st);
  return cudaErrorInvalidValue;
}

cudaError_t launch_gemm_tc_pair(EpiKind epi0, const CUtensorMap& tmA0, const CUtensorMap& tmB0,
                                const GemmArgs& a0, EpiKind epi1, const CUtensorMap& tmA1,
                                const CUtensorMap& tmB1, const GemmArgs& a1, int num_sms,
                                cudaStream_t st) {
  if (epi0 == EPI_SWIGLU && epi1 == EPI_SILU)
    return launch_tc<256, EPI_SWIGLU, EPI_SILU>(tmA0, tmB0, a0, tmA1, tmB1, a1, num_sms, st);
  return cudaErrorInvalidValue;
}

}  // namespace hero
