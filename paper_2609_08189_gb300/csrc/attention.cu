// The attention sublayer of Eq. 1 (the full decoder forward), bf16 models:
//   x = LN_attn(h)                      k_attn_norm (bf16 rows, the projection operand)
//   q, k, v = x [W_q; W_k; W_v]^T,      tensor-core GEMM (gemm_tc.cu) whose epilogue
//   q, k <- RoPE(q), RoPE(k)            rotates and stores bf16 [sequence][head][position][128]
//                                       (and v transposed for k_flash_tc)
//   o = softmax(q k^T / sqrt(hd)) v     causal, grouped-query heads: k_flash_tc (tcgen05,
//                                       S >= 128), k_flash_attn (mma.sync, shorter), or one
//                                       query per sequence over the KV cache: k_attn_decode
//                                       + k_attn_combine
//   h_bar = h + o W_o^T                 tensor-core GEMM with the residual epilogue, which
//                                       in the decoder also closes into the block entry
#include "hero_device.cuh"

namespace hero {
namespace {

constexpr int HD = 128;       // head dimension
constexpr int FA_BM = 64;     // query rows per CTA (16 per warp)
constexpr int FA_BN = 64;     // keys per tile
constexpr int FA_THREADS = 128;

// ---------------------------------------------------------------------------------
// x = bf16(h * rsqrt(mean(h^2) + eps) * g), one warp per row.
// ---------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_attn_norm(const float* __restrict__ h,
                                                   const float* __restrict__ g, int T, int d,
                                                   float eps, uint16_t* __restrict__ x) {
  pdl_enter();
  const long row = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (row >= T) return;
  const float* hr = h + (size_t)row * d;
  float ss = 0.f;
  for (int c = lane * 4; c < d; c += 128) {
    const float4 v = *reinterpret_cast<const float4*>(hr + c);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = warp_sum(ss);
  const float rinv = rsqrtf(ss / (float)d + eps);
  for (int c = lane * 4; c < d; c += 128) {
    const float4 v = *reinterpret_cast<const float4*>(hr + c);
    const float4 gv = __ldg(reinterpret_cast<const float4*>(g + c));
    store4(x, (size_t)row * d + c,
           make_float4(v.x * rinv * gv.x, v.y * rinv * gv.y, v.z * rinv * gv.z, v.w * rinv * gv.w),
           1);
  }
}

// The same with one CTA of 8 warps per row (few rows: decoding steps), each warp
// 1/8 of the row held in registers; the 8 partial sums of squares are added in warp
// order.  d must be a multiple of 1024.
__global__ void __launch_bounds__(256) k_attn_norm_row(const float* __restrict__ h,
                                                       const float* __restrict__ g, int d,
                                                       float eps, uint16_t* __restrict__ x) {
  pdl_enter();
  __shared__ float part[8];
  const size_t row = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int seg = d / 8, c0 = warp * seg;
  const float* hr = h + row * d;
  constexpr int MAXV = 4;   // float4 per lane for d <= 4096
  float4 v[MAXV];
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < MAXV; ++i) {
    const int c = c0 + (i * 32 + lane) * 4;
    v[i] = (i * 128 < seg) ? *reinterpret_cast<const float4*>(hr + c) : make_float4(0.f, 0.f, 0.f, 0.f);
    ss += v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
  }
  for (int c = c0 + (MAXV * 32 + lane) * 4; c < c0 + seg; c += 128) {   // d > 4096
    const float4 w = *reinterpret_cast<const float4*>(hr + c);
    ss += w.x * w.x + w.y * w.y + w.z * w.z + w.w * w.w;
  }
  ss = warp_sum(ss);
  if (lane == 0) part[warp] = ss;
  __syncthreads();
  float tot = 0.f;
#pragma unroll
  for (int w = 0; w < 8; ++w) tot += part[w];
  const float rinv = rsqrtf(tot / (float)d + eps);
#pragma unroll
  for (int i = 0; i < MAXV; ++i) {
    const int c = c0 + (i * 32 + lane) * 4;
    if (i * 128 >= seg) break;
    const float4 gv = __ldg(reinterpret_cast<const float4*>(g + c));
    store4(x, row * d + c,
           make_float4(v[i].x * rinv * gv.x, v[i].y * rinv * gv.y, v[i].z * rinv * gv.z,
                       v[i].w * rinv * gv.w), 1);
  }
  for (int c = c0 + (MAXV * 32 + lane) * 4; c < c0 + seg; c += 128) {
    const float4 w = *reinterpret_cast<const float4*>(hr + c);
    const float4 gv = __ldg(reinterpret_cast<const float4*>(g + c));
    store4(x, row * d + c,
           make_float4(w.x * rinv * gv.x, w.y * rinv * gv.y, w.z * rinv * gv.z, w.w * rinv * gv.w), 1);
  }
}

// ---------------------------------------------------------------------------------
// Causal attention, FlashAttention-2 schedule on the mma.sync bf16 tensor path:
// CTA = 64 query rows of one (sequence, head), 4 warps of 16 rows; key/value tiles
// of 64 rows double-buffered in shared memory (cp.async); S = Q K^T and O += P V
// with m16n8k16 MMAs, fp32 accumulators in registers; online softmax in fp32 with
// exp2; P is rounded to bf16 as the A operand of P V (the FlashAttention rounding
// of exp(s - running max)); O / l is rounded to bf16 on store.
// Shared tiles are [row][128] bf16 with 16-byte chunks XOR-swizzled by row % 8.
// ---------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t swz(int r, int c) {   // element offset (c multiple of 8)
  return (uint32_t)(r * HD + (((c >> 3) ^ (r & 7)) << 3));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
  const int n = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Load rows [row0, row0 + 64) of a [S][128] bf16 matrix into a swizzled tile;
// rows at or past S are zero-filled (their source address is clamped to row 0).
__device__ __forceinline__ void load_tile(uint32_t tile, const uint16_t* src, int row0, int S,
                                          int tid) {
#pragma unroll
  for (int i = 0; i < (FA_BM * HD / 8) / FA_THREADS; ++i) {
    const int chunk = tid + i * FA_THREADS;
    const int r = chunk >> 4, c = (chunk & 15) << 3;
    const bool valid = row0 + r < S;
    const uint16_t* g = src + (size_t)(valid ? row0 + r : 0) * HD + c;
    cp_async16(tile + 2u * swz(r, c), g, valid);
  }
}

__global__ void __launch_bounds__(FA_THREADS) k_flash_attn(const uint16_t* __restrict__ Q,
                                                           const uint16_t* __restrict__ K,
                                                           const uint16_t* __restrict__ V, int H,
                                                           int Hkv, int S, int kv_stride,
                                                           float scale_log2,
                                                           uint16_t* __restrict__ O) {
  pdl_enter();
  extern __shared__ __align__(128) uint16_t fa_smem[];
  const uint32_t sQ = smem_u32(fa_smem);
  const uint32_t sK = sQ + 2u * FA_BM * HD;            // 2 buffers
  const uint32_t sV = sK + 2u * 2 * FA_BN * HD;        // 2 buffers
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int qt = gridDim.x - 1 - blockIdx.x;           // long rows first
  const int hh = blockIdx.y, b = blockIdx.z;
  const int kvh = hh / (H / Hkv);
  const int q0 = qt * FA_BM;
  const uint16_t* Qg = Q + ((size_t)b * H + hh) * S * HD;
  const uint16_t* Kg = K + ((size_t)b * Hkv + kvh) * kv_stride * HD;
  const uint16_t* Vg = V + ((size_t)b * Hkv + kvh) * kv_stride * HD;
  const int n_tiles = qt + 1;                          // causal: key tiles 0..qt

  load_tile(sQ, Qg, q0, S, tid);
  load_tile(sK, Kg, 0, S, tid);
  load_tile(sV, Vg, 0, S, tid);
  cp_async_commit();

  uint32_t qa[HD / 16][4];
  float o[HD / 8][4];
#pragma unroll
  for (int j = 0; j < HD / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;   // rows lane/4 and lane/4 + 8
  const int qrow0 = q0 + warp * 16 + (lane >> 2);

  for (int it = 0; it < n_tiles; ++it) {
    const int buf = it & 1;
    if (it + 1 < n_tiles) {   // prefetch the next key/value tile
      load_tile(sK + 2u * (buf ^ 1) * FA_BN * HD, Kg, (it + 1) * FA_BN, S, tid);
      load_tile(sV + 2u * (buf ^ 1) * FA_BN * HD, Vg, (it + 1) * FA_BN, S, tid);
      cp_async_commit();
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    if (it == 0) {   // the warp's 16 query rows as A fragments, once
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk) {
        const int r = warp * 16 + (lane & 15), c = kk * 16 + ((lane >> 4) << 3);
        ldsm_x4(sQ + 2u * swz(r, c), qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3]);
      }
    }
    const uint32_t kt = sK + 2u * buf * FA_BN * HD;
    const uint32_t vt = sV + 2u * buf * FA_BN * HD;

    // S = Q K^T for 16 rows x 64 keys
    float sc[FA_BN / 8][4];
#pragma unroll
    for (int j = 0; j < FA_BN / 8; ++j) sc[j][0] = sc[j][1] = sc[j][2] = sc[j][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int j = 0; j < FA_BN / 8; j += 2) {
        const int r = j * 8 + (lane & 7) + ((lane >> 4) << 3);
        const int c = kk * 16 + (((lane >> 3) & 1) << 3);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(kt + 2u * swz(r, c), b0, b1, b2, b3);
        mma_bf16(sc[j], qa[kk], b0, b1);
        mma_bf16(sc[j + 1], qa[kk], b2, b3);
      }
    }
    // causal / length mask, then the online softmax (scores in log2 units)
    const int k0 = it * FA_BN;
    float tmax0 = -INFINITY, tmax1 = -INFINITY;
#pragma unroll
    for (int j = 0; j < FA_BN / 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int kpos = k0 + j * 8 + ((lane & 3) << 1) + (e & 1);
        const int qpos = qrow0 + ((e >> 1) << 3);
        float v = sc[j][e] * scale_log2;
        if (kpos > qpos || kpos >= S) v = -INFINITY;
        sc[j][e] = v;
      }
      tmax0 = fmaxf(tmax0, fmaxf(sc[j][0], sc[j][1]));
      tmax1 = fmaxf(tmax1, fmaxf(sc[j][2], sc[j][3]));
    }
#pragma unroll
    for (int off = 1; off < 4; off <<= 1) {
      tmax0 = fmaxf(tmax0, __shfl_xor_sync(0xffffffffu, tmax0, off));
      tmax1 = fmaxf(tmax1, __shfl_xor_sync(0xffffffffu, tmax1, off));
    }
    const float mn0 = fmaxf(m0, tmax0), mn1 = fmaxf(m1, tmax1);   // finite: key 0 is in tile 0
    const float al0 = exp2f(m0 - mn0), al1 = exp2f(m1 - mn1);
    m0 = mn0;
    m1 = mn1;
    float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
    for (int j = 0; j < FA_BN / 8; ++j) {
      sc[j][0] = exp2f(sc[j][0] - mn0);
      sc[j][1] = exp2f(sc[j][1] - mn0);
      sc[j][2] = exp2f(sc[j][2] - mn1);
      sc[j][3] = exp2f(sc[j][3] - mn1);
      ps0 += sc[j][0] + sc[j][1];
      ps1 += sc[j][2] + sc[j][3];
    }
    l0 = l0 * al0 + ps0;
    l1 = l1 * al1 + ps1;
#pragma unroll
    for (int j = 0; j < HD / 8; ++j) {
      o[j][0] *= al0;
      o[j][1] *= al0;
      o[j][2] *= al1;
      o[j][3] *= al1;
    }
    // O += P V: P (bf16) as A fragments straight from the score accumulators
#pragma unroll
    for (int kk = 0; kk < FA_BN / 16; ++kk) {
      uint32_t pa[4];
      pa[0] = pack_bf16x2(sc[2 * kk][0], sc[2 * kk][1]);
      pa[1] = pack_bf16x2(sc[2 * kk][2], sc[2 * kk][3]);
      pa[2] = pack_bf16x2(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
      pa[3] = pack_bf16x2(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
      for (int j = 0; j < HD / 8; j += 2) {
        const int r = kk * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int c = j * 8 + ((lane >> 4) << 3);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(vt + 2u * swz(r, c), b0, b1, b2, b3);
        mma_bf16(o[j], pa, b0, b1);
        mma_bf16(o[j + 1], pa, b2, b3);
      }
    }
    __syncthreads();   // this buffer is refilled by the next iteration's prefetch
  }
  // rows' sums over the four lanes of a row, then O / l in bf16
#pragma unroll
  for (int off = 1; off < 4; off <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, off);
    l1 += __shfl_xor_sync(0xffffffffu, l1, off);
  }
  const float inv0 = 1.f / l0, inv1 = 1.f / l1;
  const int dcol = hh * HD + ((lane & 3) << 1);
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const int qpos = qrow0 + half * 8;
    if (qpos >= S) continue;
    uint32_t* orow = reinterpret_cast<uint32_t*>(O + ((size_t)b * S + qpos) * H * HD + dcol);
    const float inv = half ? inv1 : inv0;
#pragma unroll
    for (int j = 0; j < HD / 8; ++j)
      orow[j * 4] = pack_bf16x2(o[j][2 * half] * inv, o[j][2 * half + 1] * inv);
  }
}

// ---------------------------------------------------------------------------------
// Causal attention on the tcgen05 tensor cores (sequences of 128 tokens or more).
// CTA = two query tiles of 128 rows (A = 2p, B = 2p + 1) of one (sequence, head),
// sharing every K and V^T tile; 10 warps:
//   warp 0     TMA producer: Q_A, Q_B once, K tiles of 128 keys through a 2-stage ring,
//              V^T tiles through one stage
//   warp 1     TMEM allocator and MMA issuer, ping-pong between the tiles:
//              S_A(0) S_B(0) | PV_A(0) S_A(1) | PV_B(0) S_B(1) | PV_A(1) S_A(2) | ...
//              so the tensor pipe works on one tile while the other's softmax runs
//   warps 2-5  softmax of tile A, warps 6-9 of tile B: one thread per query row (its TMEM
//              lane) reads the row of S from TMEM, runs the online softmax in log2 units
//              (exp2 of one FMA; the running max is raised only when the row max grows
//              by more than 8, then that row's O and l are rescaled, otherwise the stale
//              max keeps every p <= 2^8), writes P as the bf16 A operand of P V (128-byte
//              swizzle) and finally O / l in bf16.
// TMEM: S_A | O_A | S_B | O_B, 128 columns each.  A tile's S(i + 1) is issued after its
// P V(i), and tcgen05.commit signals only when every earlier MMA of the issuing thread has
// completed, so once S(i + 1) is visible P V(i) has finished: the softmax may then
// overwrite P and rescale O without another barrier.  All operands are K-major (V^T from
// the q/k/v epilogue) in 128 x 64 bf16 panels.  Every mbarrier wait is bounded; on expiry
// the CTA drains its copies and MMAs, reports through err and frees its TMEM.
// ---------------------------------------------------------------------------------
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

namespace fa {
constexpr int BM = 128, BN = 128, THREADS = 320;
constexpr uint32_t PANEL = 128 * 128;   // [128 rows][64 bf16] = 16 KB
constexpr uint32_t TILE = 2 * PANEL;    // [128 rows][128 bf16]
constexpr uint32_t OFF_Q = 0, OFF_K = 2 * TILE, OFF_V = 4 * TILE, OFF_P = 5 * TILE,
                   OFF_BAR = 7 * TILE;  // Q_A Q_B | K0 K1 | V | P_A P_B
enum { Q_FULL = 0, K_FULL = 1, K_EMPTY = 3, V_FULL = 5, V_EMPTY = 6, S_FULL = 7, P_FULL = 9,
       FINAL = 11, DRAIN = 12, NBAR = 13 };
constexpr size_t SMEM = OFF_BAR + NBAR * 8 + 16 + 1024;
constexpr uint32_t TMEM_COLS = 512;
// kind::f16 instruction descriptor: fp32 D, bf16 A and B, K-major, N = 128, M = 128
constexpr uint32_t IDESC = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
                           ((uint32_t)(BM >> 4) << 24);
constexpr float RESCALE = 8.f;          // log2 units
static_assert(SMEM <= 232448, "shared memory per CTA");
}  // namespace fa

__global__ void __launch_bounds__(fa::THREADS, 1)
    k_flash_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
               const __grid_constant__ CUtensorMap tmV, int H, int Hkv, int S, int n_qt,
               float scale_log2, uint16_t* __restrict__ O, uint32_t* err, uint64_t wait_ns) {
  using namespace fa;
  pdl_enter();
  extern __shared__ uint8_t fa_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(fa_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sb = smem_u32(smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  const uint32_t bar0 = smem_u32(bars);
  auto bar = [&](int i) { return bar0 + 8u * i; };
  volatile uint32_t* misc = reinterpret_cast<volatile uint32_t*>(bars + NBAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int pr = gridDim.x - 1 - blockIdx.x;   // long rows first
  const int hh = blockIdx.y, b = blockIdx.z;
  const int kvh = hh / (H / Hkv);
  const int qtA = 2 * pr;
  const bool hasB = qtA + 1 < n_qt;
  const int nA = qtA + 1, nB = hasB ? qtA + 2 : 0;   // causal: key tiles 0 .. qt
  const int n = hasB ? nB : nA;
  if (threadIdx.x == 0) {
    mbar_init(bar(Q_FULL), 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(bar(K_FULL + s), 1);
      mbar_init(bar(K_EMPTY + s), 1);
      mbar_init(bar(S_FULL + s), 1);
      mbar_init(bar(P_FULL + s), 4);
    }
    mbar_init(bar(V_FULL), 1);
    mbar_init(bar(V_EMPTY), 1);
    mbar_init(bar(FINAL), 1);
    mbar_init(bar(DRAIN), 1);
    misc[1] = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(const_cast<uint32_t*>(misc)), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = misc[0];
  auto tS = [&](int x) { return tbase + 256u * x; };
  auto tO = [&](int x) { return tbase + 256u * x + 128u; };

  if (warp == 0) {
    // ------------------------------ TMA producer ------------------------------
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      const int zq = b * H + hh, zk = b * Hkv + kvh;
      mbar_arrive_expect_tx(bar(Q_FULL), hasB ? 2 * TILE : TILE);
      tma_load_3d(sb + OFF_Q, &tmQ, 0, qtA * BM, zq, bar(Q_FULL));
      tma_load_3d(sb + OFF_Q + PANEL, &tmQ, 64, qtA * BM, zq, bar(Q_FULL));
      if (hasB) {
        tma_load_3d(sb + OFF_Q + TILE, &tmQ, 0, (qtA + 1) * BM, zq, bar(Q_FULL));
        tma_load_3d(sb + OFF_Q + TILE + PANEL, &tmQ, 64, (qtA + 1) * BM, zq, bar(Q_FULL));
      }
      bool ok = true, kiss[2] = {false, false}, viss = false;
      uint32_t kpar[2] = {0, 0}, vpar = 0;
      for (int i = 0; i < n && ok; ++i) {
        const int st = i & 1;
        const uint32_t ph = (i >> 1) & 1;
        if (!mbar_wait(bar(K_EMPTY + st), ph ^ 1u, wait_ns) || misc[1]) {
          ok = false;
          break;
        }
        const uint32_t sk = sb + OFF_K + st * TILE;
        mbar_arrive_expect_tx(bar(K_FULL + st), TILE);
        tma_load_3d(sk, &tmK, 0, i * BN, zk, bar(K_FULL + st));
        tma_load_3d(sk + PANEL, &tmK, 64, i * BN, zk, bar(K_FULL + st));
        kiss[st] = true;
        kpar[st] = ph;
        if (!mbar_wait(bar(V_EMPTY), (i & 1) ^ 1u, wait_ns) || misc[1]) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(bar(V_FULL), TILE);
        tma_load_3d(sb + OFF_V, &tmV, i * BN, 0, zk, bar(V_FULL));
        tma_load_3d(sb + OFF_V + PANEL, &tmV, i * BN + 64, 0, zk, bar(V_FULL));
        viss = true;
        vpar = i & 1;
      }
      if (!ok) {
        misc[1] = 1;
        atomicOr(err, ERR_WAIT_PRODUCER);
      }
      // let every copy still in flight land before the CTA can exit, also after a
      // normal end (another role may have given up before consuming them)
      bool drained = mbar_wait(bar(Q_FULL), 0, kDrainLimitNs);
      for (int s = 0; s < 2; ++s)
        if (kiss[s]) drained = mbar_wait(bar(K_FULL + s), kpar[s], kDrainLimitNs) && drained;
      if (viss) drained = mbar_wait(bar(V_FULL), vpar, kDrainLimitNs) && drained;
      if (!drained) atomicOr(err, ERR_WAIT_DRAIN);
    }
  } else if (warp == 1) {
    // ------------------------------ MMA issuer ------------------------------
    if (lane == 0) {
      bool ok = mbar_wait(bar(Q_FULL), 0, wait_ns) && !misc[1];
      auto wait = [&](int id, uint32_t par) {
        ok = ok && mbar_wait(bar(id), par, wait_ns) && !misc[1];
        return ok;
      };
      auto issue_s = [&](int x, int i) {   // S_x(i) = Q_x K_i^T over the head dimension
        tc_fence_after();
        const uint32_t qx = sb + OFF_Q + x * TILE, kx = sb + OFF_K + (i & 1) * TILE;
#pragma unroll
        for (int kk = 0; kk < 128 / 16; ++kk)
          umma_bf16(tS(x), sw128_desc(qx + (kk >> 2) * PANEL) + 2u * (kk & 3),
                    sw128_desc(kx + (kk >> 2) * PANEL) + 2u * (kk & 3), IDESC, kk > 0 ? 1u : 0u);
        umma_commit(bar(S_FULL + x));
      };
      auto issue_pv = [&](int x, int i) {   // O_x += P_x(i) V_i
        tc_fence_after();
        const uint32_t px = sb + OFF_P + x * TILE;
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk)
          umma_bf16(tO(x), sw128_desc(px + (kk >> 2) * PANEL) + 2u * (kk & 3),
                    sw128_desc(sb + OFF_V + (kk >> 2) * PANEL) + 2u * (kk & 3), IDESC,
                    (i > 0 || kk > 0) ? 1u : 0u);
      };
      if (wait(K_FULL, 0)) {
        issue_s(0, 0);
        if (hasB) issue_s(1, 0);
        umma_commit(bar(K_EMPTY));
      }
      for (int i = 0; i < n && ok; ++i) {
        const int nst = (i + 1) & 1;
        const uint32_t nph = ((i + 1) >> 1) & 1;
        bool k_next = false;
        if (!wait(V_FULL, i & 1)) break;
        if (i < nA) {
          if (!wait(P_FULL + 0, i & 1)) break;
          issue_pv(0, i);
          if (i + 1 < nA) {
            if (!wait(K_FULL + nst, nph)) break;
            k_next = true;
            issue_s(0, i + 1);
          }
        }
        if (i < nB) {
          if (!wait(P_FULL + 1, i & 1)) break;
          issue_pv(1, i);
        }
        umma_commit(bar(V_EMPTY));   // V_i read by both tiles' P V
        if (i + 1 < n) {
          if (!k_next && !wait(K_FULL + nst, nph)) break;
          if (i + 1 < nB) issue_s(1, i + 1);
          umma_commit(bar(K_EMPTY + nst));
        }
      }
      if (ok) umma_commit(bar(FINAL));   // every MMA of the CTA has completed
      if (!ok) {
        misc[1] = 1;
        atomicOr(err, ERR_WAIT_MMA);
      }
      // every issued MMA completes before TMEM is freed, also after a normal end
      // (a softmax warp may have given up while MMAs were in flight)
      umma_commit(bar(DRAIN));
      if (!mbar_wait(bar(DRAIN), 0, kDrainLimitNs)) atomicOr(err, ERR_WAIT_DRAIN);
    }
  } else {
    // ------------------------------ softmax ------------------------------
    const int x = (warp - 2) >> 2;              // 0: tile A, 1: tile B
    const int quad = warp & 3;                  // TMEM lane quadrant of this warp
    const int r = quad * 32 + lane;             // query row in the tile
    const int nx = x ? nB : nA;
    const int qpos = (qtA + x) * BM + r;
    const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
    float m_used = -INFINITY, l = 0.f;          // m_used in raw score units
    bool ok = true;
    for (int i = 0; i < nx; ++i) {
      bool w = mbar_wait(bar(S_FULL + x), i & 1, wait_ns);
      w = __all_sync(0xffffffffu, w) && !misc[1];
      if (!__all_sync(0xffffffffu, w)) {
        ok = false;
        break;
      }
      tc_fence_after();
      // the row of S in one TMEM load; p = 2^(s scale - m) streamed into the P tile
      const bool diag = i == nx - 1;   // the diagonal tile: causal mask and the sequence end
      const int kvalid = min(qpos + 1, S) - i * BN;   // keys c < kvalid are visible
      uint32_t rr[BN];
      tmem_ld128(tS(x) + lane_off, rr);
      if (diag) {
#pragma unroll
        for (int c = 0; c < BN; ++c)
          if (c >= kvalid) rr[c] = 0xff800000u;   // -inf
      }
      float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
      for (int c = 0; c < BN; c += 8)   // three-input max: two new values per instruction
#pragma unroll
        for (int k = 0; k < 4; ++k)
          m4[k] = fmax3(m4[k], __uint_as_float(rr[c + 2 * k]), __uint_as_float(rr[c + 2 * k + 1]));
      const float mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
      float alpha = 1.f;
      if ((mx - m_used) * scale_log2 > RESCALE) {   // raise the running max (first tile: always)
        alpha = exp2f((m_used - mx) * scale_log2);
        m_used = mx;
        l *= alpha;
      }
      const float mb = -m_used * scale_log2;
      float ps[4] = {0.f, 0.f, 0.f, 0.f};
      // S(i) completing implies P V(i - 1) has: P and O are free
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) {
        uint32_t pk[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const float p0 = exp2f(fmaf(__uint_as_float(rr[32 * c + 2 * e]), scale_log2, mb));
          const float p1 = exp2f(fmaf(__uint_as_float(rr[32 * c + 2 * e + 1]), scale_log2, mb));
          ps[e & 3] += p0 + p1;
          pk[e] = pack_bf16x2(p0, p1);
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {   // 16-byte chunk ch = 4 c + q of the row, 128-byte swizzle
          const int ch = 4 * c + q;
          const uint32_t off = OFF_P + x * TILE + (ch >> 3) * PANEL + r * 128 + (((ch & 7) ^ (r & 7)) << 4);
          *reinterpret_cast<uint4*>(smem + off) = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
        }
      }
      l += (ps[0] + ps[1]) + (ps[2] + ps[3]);
      if (i >= 1 && __any_sync(0xffffffffu, alpha != 1.f)) {   // rescale this warp's rows of O
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t rr[32];
          tmem_ld32(tO(x) + lane_off + c * 32, rr);
#pragma unroll
          for (int e = 0; e < 32; ++e) rr[e] = __float_as_uint(__uint_as_float(rr[e]) * alpha);
          tmem_st32(tO(x) + lane_off + c * 32, rr);
        }
      }
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(P_FULL + x));
    }
    if (ok && nx > 0) {
      const bool w = mbar_wait(bar(FINAL), 0, wait_ns);
      ok = __all_sync(0xffffffffu, w);
      if (ok) {
        tc_fence_after();
        const float inv = 1.f / l;
        uint16_t* orow = O + ((size_t)b * S + qpos) * H * 128 + hh * 128;
        uint32_t rr[128];
        tmem_ld128(tO(x) + lane_off, rr);
        if (qpos < S) {
          uint4* dst = reinterpret_cast<uint4*>(orow);
#pragma unroll
          for (int q = 0; q < 16; ++q)
            dst[q] = make_uint4(pack_bf16x2(__uint_as_float(rr[8 * q]) * inv, __uint_as_float(rr[8 * q + 1]) * inv),
                                pack_bf16x2(__uint_as_float(rr[8 * q + 2]) * inv, __uint_as_float(rr[8 * q + 3]) * inv),
                                pack_bf16x2(__uint_as_float(rr[8 * q + 4]) * inv, __uint_as_float(rr[8 * q + 5]) * inv),
                                pack_bf16x2(__uint_as_float(rr[8 * q + 6]) * inv, __uint_as_float(rr[8 * q + 7]) * inv));
        }
      }
    }
    if (!ok && lane == 0) {
      misc[1] = 1;
      atomicOr(err, ERR_WAIT_EPILOGUE);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tbase, fa::TMEM_COLS);
  }
}

// ---------------------------------------------------------------------------------
// Decoding step attention (flash-decoding): one query per sequence, the G = H / H_kv
// query heads of a key/value head together, keys split into chunks of DC positions
// so that every SM streams the cache.  CTA = (chunk, kv head, sequence), 128 threads:
//   1. scores: warp w takes keys 64 w .. 64 w + 63; eight lanes share a 256-byte key
//      row (lane: row 4 i + lane / 8, 16-byte chunks lane % 8 and lane % 8 + 8; 16 loads
//      in flight), multiply by the G queries' matching 16 elements (held in registers)
//      and add up over the eight lanes by shuffles;
//   2. per query head (one warp each): chunk max m, p = 2^(s - m), l = sum p;
//   3. P V: thread t owns value columns 8 (t % 16) .. +7 of keys t / 16 + 8 i
//      (16-byte loads, 16 in flight), the 8 key groups added in shared memory.
// Partial (m, l, o[128]) per (sequence, head, chunk) are merged by k_attn_combine.
// ---------------------------------------------------------------------------------
constexpr int DC = 256;          // keys per chunk
constexpr int DEC_THREADS = 128;
constexpr int DEC_KPW = DC / (DEC_THREADS / 32);   // keys per warp in the score phase
constexpr int DEC_KG = 8;                          // key groups in the P V phase

template <int G>
__global__ void __launch_bounds__(DEC_THREADS) k_attn_decode(const uint16_t* __restrict__ Q,
                                                             const uint16_t* __restrict__ K,
                                                             const uint16_t* __restrict__ V,
                                                             const int* __restrict__ pos, int H,
                                                             int Hkv, int kv_stride, int max_pos,
                                                             float scale_log2, float* __restrict__ pm,
                                                             float* __restrict__ pl,
                                                             float* __restrict__ po, int n_chunks,
                                                             uint32_t* err) {
  pdl_enter();
  __shared__ float sc[G][DC];
  __shared__ __align__(16) float ored[DEC_KG][G][HD];
  const int c = blockIdx.x, kvh = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int len = pos[b] + 1;
  if (len < 1 || len > kv_stride || len > max_pos + 1) {   // bad position: no keys, reported
    if (c == 0 && kvh == 0 && threadIdx.x == 0) atomicOr(err, ERR_BAD_INDEX);
    len = 0;
  }
  const int j0 = c * DC, j1 = min(j0 + DC, len);
  const size_t part = ((size_t)b * H + (size_t)kvh * G) * n_chunks + c;   // + g * n_chunks
  if (j0 >= j1) {   // chunk past the sequence (or a bad position): an empty partial
    if (tid < G) {
      pm[part + (size_t)tid * n_chunks] = -INFINITY;
      pl[part + (size_t)tid * n_chunks] = 0.f;
    }
    return;
  }
  const uint16_t* Kg = K + ((size_t)b * Hkv + kvh) * kv_stride * HD;
  const uint16_t* Vg = V + ((size_t)b * Hkv + kvh) * kv_stride * HD;
  const int ch = lane & 7;   // this lane's 16-byte chunks ch and ch + 8 (elements 8 ch.., 64 + 8 ch..)
  float qr[G][16];
#pragma unroll
  for (int g = 0; g < G; ++g)
#pragma unroll
    for (int hlf = 0; hlf < 2; ++hlf) {
      const uint4 u = *reinterpret_cast<const uint4*>(Q + ((size_t)b * H + kvh * G + g) * HD +
                                                      (ch + 8 * hlf) * 8);
      const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
      for (int h2 = 0; h2 < 4; ++h2) {
        unpack_bf16x2(w[h2], qr[g][8 * hlf + 2 * h2], qr[g][8 * hlf + 2 * h2 + 1]);
        qr[g][8 * hlf + 2 * h2] *= scale_log2;
        qr[g][8 * hlf + 2 * h2 + 1] *= scale_log2;
      }
    }
  const int kw0 = warp * DEC_KPW;   // the warp's first key (offset in the chunk)
#pragma unroll 1
  for (int blk = 0; blk < DEC_KPW / 32; ++blk) {
    // 8 lanes per key row, 4 rows per instruction pair; 16 loads of 16 bytes in flight
    uint4 kr[8][2];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int j = j0 + kw0 + blk * 32 + 4 * i + (lane >> 3);
#pragma unroll
      for (int hlf = 0; hlf < 2; ++hlf)
        kr[i][hlf] = j < j1 ? __ldg(reinterpret_cast<const uint4*>(Kg + (size_t)j * HD + (ch + 8 * hlf) * 8))
                            : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float k16[16];
#pragma unroll
      for (int hlf = 0; hlf < 2; ++hlf) {
        const uint32_t w[4] = {kr[i][hlf].x, kr[i][hlf].y, kr[i][hlf].z, kr[i][hlf].w};
#pragma unroll
        for (int h2 = 0; h2 < 4; ++h2)
          unpack_bf16x2(w[h2], k16[8 * hlf + 2 * h2], k16[8 * hlf + 2 * h2 + 1]);
      }
      float acc[G];
#pragma unroll
      for (int g = 0; g < G; ++g) {
        float a0 = 0.f, a1 = 0.f;
#pragma unroll
        for (int e = 0; e < 16; e += 2) {
          a0 = fmaf(qr[g][e], k16[e], a0);
          a1 = fmaf(qr[g][e + 1], k16[e + 1], a1);
        }
        float a = a0 + a1;
#pragma unroll
        for (int o = 4; o > 0; o >>= 1) a += __shfl_xor_sync(0xffffffffu, a, o);
        acc[g] = a;
      }
      if (ch == 0) {
        const int r = kw0 + blk * 32 + 4 * i + (lane >> 3);
#pragma unroll
        for (int g = 0; g < G; ++g) sc[g][r] = j0 + r < j1 ? acc[g] : -INFINITY;
      }
    }
  }
  __syncthreads();
  for (int g = warp; g < G; g += DEC_THREADS / 32) {
    float mx = -INFINITY;
    for (int i = lane; i < DC; i += 32) mx = fmaxf(mx, sc[g][i]);
    mx = warp_max(mx);
    float l = 0.f;
    for (int i = lane; i < DC; i += 32) {
      const float p = exp2f(sc[g][i] - mx);   // 0 past the sequence
      sc[g][i] = p;
      l += p;
    }
    l = warp_sum(l);
    if (lane == 0) {
      pm[part + (size_t)g * n_chunks] = mx;
      pl[part + (size_t)g * n_chunks] = l;
    }
  }
  __syncthreads();
  const int cg = tid & 15, kg = tid >> 4;
  float o[G][8];
#pragma unroll
  for (int g = 0; g < G; ++g)
#pragma unroll
    for (int e = 0; e < 8; ++e) o[g][e] = 0.f;
#pragma unroll
  for (int h16 = 0; h16 < DC / DEC_KG; h16 += 16) {
    uint4 vr[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int j = j0 + kg + DEC_KG * (h16 + i);
      vr[i] = j < j1 ? __ldg(reinterpret_cast<const uint4*>(Vg + (size_t)j * HD + cg * 8))
                     : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int jj = kg + DEC_KG * (h16 + i);   // p is 0 past the sequence
      const uint32_t w[4] = {vr[i].x, vr[i].y, vr[i].z, vr[i].w};
#pragma unroll
      for (int h2 = 0; h2 < 4; ++h2) {
        float v0, v1;
        unpack_bf16x2(w[h2], v0, v1);
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const float p = sc[g][jj];
          o[g][2 * h2] += p * v0;
          o[g][2 * h2 + 1] += p * v1;
        }
      }
    }
  }
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float4* dst = reinterpret_cast<float4*>(&ored[kg][g][cg * 8]);
    dst[0] = make_float4(o[g][0], o[g][1], o[g][2], o[g][3]);
    dst[1] = make_float4(o[g][4], o[g][5], o[g][6], o[g][7]);
  }
  __syncthreads();
#pragma unroll
  for (int g = 0; g < G; ++g) {
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < DEC_KG; ++k) acc += ored[k][g][tid];
    po[(part + (size_t)g * n_chunks) * HD + tid] = acc;
  }
}

// Merge of the chunk partials: one warp per (sequence, head), lane owns 4 columns;
// o = sum_c 2^(m_c - M) o_c / sum_c 2^(m_c - M) l_c, stored bf16 into O [B][H 128].
__global__ void __launch_bounds__(256) k_attn_combine(const float* __restrict__ pm,
                                                      const float* __restrict__ pl,
                                                      const float* __restrict__ po, int BH,
                                                      int n_chunks, uint16_t* __restrict__ O) {
  pdl_enter();
  const int w = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (w >= BH) return;
  const size_t base = (size_t)w * n_chunks;
  float M = -INFINITY;
  for (int c = 0; c < n_chunks; ++c) M = fmaxf(M, pm[base + c]);
  float L = 0.f;
  float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
  if (M > -INFINITY) {
    for (int c = 0; c < n_chunks; ++c) {
      const float mc = pm[base + c];
      if (mc == -INFINITY) continue;
      const float f = exp2f(mc - M);
      L += f * pl[base + c];
      const float4 v = *reinterpret_cast<const float4*>(po + (base + c) * HD + 4 * lane);
      o.x += f * v.x; o.y += f * v.y; o.z += f * v.z; o.w += f * v.w;
    }
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  store4(O, (size_t)w * HD + 4 * lane, make_float4(o.x * inv, o.y * inv, o.z * inv, o.w * inv), 1);
}

}  // namespace

cudaError_t launch_attn_norm(const float* h, const float* g, int T, int d, float eps, void* x,
                             cudaStream_t st) {
  if (T <= 0) return cudaSuccess;
  if (d % 128) return cudaErrorInvalidValue;
  if (T <= 512 && d % 1024 == 0)   // few rows: a CTA per row
    return launch_pdl(k_attn_norm_row, dim3((unsigned)T), dim3(256), 0, st, h, g, d, eps,
                      static_cast<uint16_t*>(x));
  return launch_pdl(k_attn_norm, dim3((unsigned)((T + 7) / 8)), dim3(256), 0, st, h, g, T, d, eps,
                    static_cast<uint16_t*>(x));
}

cudaError_t launch_flash_attn(const void* Q, const void* K, const void* V, int B, int S, int H,
                              int Hkv, int kv_stride, void* O, cudaStream_t st) {
  if (B <= 0 || S <= 0) return cudaSuccess;
  if (H % Hkv || H > 65535 || B > 65535 || kv_stride < S) return cudaErrorInvalidValue;
  constexpr size_t smem = 2u * (FA_BM * HD + 2 * 2 * FA_BN * HD);   // 80 KB
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_flash_attn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)HD);
  dim3 grid((unsigned)((S + FA_BM - 1) / FA_BM), (unsigned)H, (unsigned)B);
  return launch_pdl(k_flash_attn, grid, dim3(FA_THREADS), smem, st,
                    static_cast<const uint16_t*>(Q), static_cast<const uint16_t*>(K),
                    static_cast<const uint16_t*>(V), H, Hkv, S, kv_stride, scale_log2,
                    static_cast<uint16_t*>(O));
}

}  // namespace hero

namespace hero {

int attn_decode_chunks(int max_pos) { return (max_pos + 1 + DC - 1) / DC; }

cudaError_t launch_attn_decode(const void* Q, const void* K, const void* V, const int* pos, int B,
                               int H, int Hkv, int kv_stride, int max_pos, float* pm, float* pl,
                               float* po, void* O, uint32_t* err, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  if (H % Hkv || Hkv > 65535 || B > 65535 || max_pos < 0 || max_pos >= kv_stride)
    return cudaErrorInvalidValue;
  const int G = H / Hkv, nc = attn_decode_chunks(max_pos);
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)HD);
  const dim3 grid((unsigned)nc, (unsigned)Hkv, (unsigned)B);
  cudaError_t e;
  const uint16_t *q = static_cast<const uint16_t*>(Q), *k = static_cast<const uint16_t*>(K),
                 *v = static_cast<const uint16_t*>(V);
  switch (G) {
    case 1: e = launch_pdl(k_attn_decode<1>, grid, dim3(DEC_THREADS), 0, st, q, k, v, pos, H, Hkv, kv_stride, max_pos, scale_log2, pm, pl, po, nc, err); break;
    case 2: e = launch_pdl(k_attn_decode<2>, grid, dim3(DEC_THREADS), 0, st, q, k, v, pos, H, Hkv, kv_stride, max_pos, scale_log2, pm, pl, po, nc, err); break;
    case 4: e = launch_pdl(k_attn_decode<4>, grid, dim3(DEC_THREADS), 0, st, q, k, v, pos, H, Hkv, kv_stride, max_pos, scale_log2, pm, pl, po, nc, err); break;
    case 8: e = launch_pdl(k_attn_decode<8>, grid, dim3(DEC_THREADS), 0, st, q, k, v, pos, H, Hkv, kv_stride, max_pos, scale_log2, pm, pl, po, nc, err); break;
    default: return cudaErrorInvalidValue;
  }
  if (e != cudaSuccess) return e;
  const int BH = B * H;
  return launch_pdl(k_attn_combine, dim3((unsigned)((BH + 7) / 8)), dim3(256), 0, st,
                    static_cast<const float*>(pm), static_cast<const float*>(pl),
                    static_cast<const float*>(po), BH, nc, static_cast<uint16_t*>(O));
}

}  // namespace hero

namespace hero {

cudaError_t launch_flash_tc(const CUtensorMap& tmQ, const CUtensorMap& tmK, const CUtensorMap& tmV,
                            int B, int S, int H, int Hkv, void* O, uint32_t* err, cudaStream_t st) {
  if (B <= 0 || S <= 0) return cudaSuccess;
  if (H % Hkv || H > 65535 || B > 65535) return cudaErrorInvalidValue;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_flash_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)fa::SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const float scale_log2 = 1.4426950408889634f / sqrtf((float)HD);
  const int n_qt = (S + fa::BM - 1) / fa::BM;
  const dim3 grid((unsigned)((n_qt + 1) / 2), (unsigned)H, (unsigned)B);   // query tile pairs
  return launch_pdl(k_flash_tc, grid, dim3(fa::THREADS), fa::SMEM, st, tmQ, tmK, tmV, H, Hkv, S,
                    n_qt, scale_log2, static_cast<uint16_t*>(O), err, wait_limit_ns());
}

}  // namespace hero
