// Device-side helpers: math, bf16 packing, PTX wrappers for mbarrier / TMA /
// tcgen05, and the shared block-closing epilogue.
#pragma once

#include "hero_internal.cuh"

namespace hero {

__device__ __forceinline__ float sigmoidf_(float x) { return 1.0f / (1.0f + expf(-x)); }
__device__ __forceinline__ float siluf_(float x) { return x / (1.0f + expf(-x)); }
// phi(x) = ELU(x) + 1, alpha = 1 (Sec. 3.2)
__device__ __forceinline__ float phif_(float x) { return x > 0.0f ? x + 1.0f : expf(x); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&b);
}

__device__ __forceinline__ void unpack_bf16x2(uint32_t u, float& lo, float& hi) {
  lo = __uint_as_float(u << 16);
  hi = __uint_as_float(u & 0xffff0000u);
}

// Load 4 consecutive elements (16-byte aligned fp32, 8-byte aligned bf16) as fp32.
__device__ __forceinline__ float4 load4(const void* base, size_t idx, int is_bf16) {
  if (is_bf16) {
    uint2 u = *reinterpret_cast<const uint2*>(static_cast<const uint16_t*>(base) + idx);
    float4 r;
    unpack_bf16x2(u.x, r.x, r.y);
    unpack_bf16x2(u.y, r.z, r.w);
    return r;
  }
  return *reinterpret_cast<const float4*>(static_cast<const float*>(base) + idx);
}

__device__ __forceinline__ void store4(void* base, size_t idx, float4 v, int is_bf16) {
  if (is_bf16) {
    uint2 u;
    u.x = pack_bf16x2(v.x, v.y);
    u.y = pack_bf16x2(v.z, v.w);
    *reinterpret_cast<uint2*>(static_cast<uint16_t*>(base) + idx) = u;
  } else {
    *reinterpret_cast<float4*>(static_cast<float*>(base) + idx) = v;
  }
}

// Operand copy of h_bar for the router contraction.  bf16 models keep it as a
// pair per element, hi = bf16(x) and lo = bf16(x - hi) (16 significant bits), in
// a [T, 2d] row: hi in columns [0, d), lo in [d, 2d).  f32 models: [T, d] fp32.
__device__ __forceinline__ void store_xl4(void* xl, int xl_bf16, int d, int t, int n, float4 v) {
  if (xl_bf16) {
    const __nv_bfloat162 h01 = __floats2bfloat162_rn(v.x, v.y);
    const __nv_bfloat162 h23 = __floats2bfloat162_rn(v.z, v.w);
    const float2 f01 = __bfloat1622float2(h01), f23 = __bfloat1622float2(h23);
    const __nv_bfloat162 l01 = __floats2bfloat162_rn(v.x - f01.x, v.y - f01.y);
    const __nv_bfloat162 l23 = __floats2bfloat162_rn(v.z - f23.x, v.w - f23.y);
    uint16_t* row = static_cast<uint16_t*>(xl) + (size_t)t * 2 * d;
    *reinterpret_cast<uint2*>(row + n) = make_uint2(*reinterpret_cast<const uint32_t*>(&h01),
                                                    *reinterpret_cast<const uint32_t*>(&h23));
    *reinterpret_cast<uint2*>(row + d + n) = make_uint2(*reinterpret_cast<const uint32_t*>(&l01),
                                                        *reinterpret_cast<const uint32_t*>(&l23));
  } else {
    *reinterpret_cast<float4*>(static_cast<float*>(xl) + (size_t)t * d + n) = v;
  }
}

__device__ __forceinline__ void store_xl1(void* xl, int xl_bf16, int d, int t, int n, float v) {
  if (xl_bf16) {
    const __nv_bfloat16 h = __float2bfloat16_rn(v);
    const __nv_bfloat16 l = __float2bfloat16_rn(v - __bfloat162float(h));
    __nv_bfloat16* row = static_cast<__nv_bfloat16*>(xl) + (size_t)t * 2 * d;
    row[n] = h;
    row[d + n] = l;
  } else {
    static_cast<float*>(xl)[(size_t)t * d + n] = v;
  }
}

// ---------------------------------------------------------------------------
// Block-closing epilogue on 4 consecutive columns n..n+3 of token t.
// y: GEMM outputs, s: branch scale.  Accumulates the partial sums.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void layer_out4(const LayerOutArgs& p, int t, int n, float4 y, float s,
                                           float& ss, float& dd, float& dp) {
  const size_t off = (size_t)t * p.d + n;
  float4 hb = *reinterpret_cast<const float4*>(p.hbar + off);
  float4 h;
  h.x = hb.x + s * y.x;
  h.y = hb.y + s * y.y;
  h.z = hb.z + s * y.z;
  h.w = hb.w + s * y.w;
  if (p.last) {
    *reinterpret_cast<float4*>(p.h_out + off) = h;
    return;
  }
  float4 pn = make_float4(0.f, 0.f, 0.f, 0.f);
  if (p.p_next) pn = load4(p.p_next, off, p.p_bf16);
  float4 hn;
  hn.x = h.x + pn.x; hn.y = h.y + pn.y; hn.z = h.z + pn.z; hn.w = h.w + pn.w;
  *reinterpret_cast<float4*>(p.hbar + off) = hn;
  ss += hn.x * hn.x + hn.y * hn.y + hn.z * hn.z + hn.w * hn.w;
  if (p.router) {  // the router of the next block needs delta and the operand copy
    float4 dprev = make_float4(0.f, 0.f, 0.f, 0.f);
    if (!p.first) dprev = *reinterpret_cast<const float4*>(p.delta + off);
    float4 dn;
    dn.x = s * y.x + pn.x; dn.y = s * y.y + pn.y; dn.z = s * y.z + pn.z; dn.w = s * y.w + pn.w;
    *reinterpret_cast<float4*>(p.delta + off) = dn;
    store_xl4(p.xl, p.xl_bf16, p.d, t, n, hn);
    dd += dn.x * dn.x + dn.y * dn.y + dn.z * dn.z + dn.w * dn.w;
    dp += dn.x * dprev.x + dn.y * dprev.y + dn.z * dprev.z + dn.w * dprev.w;
  }
}

// The same epilogue split into a load phase and a compute/store phase so that a
// caller can keep several rows' loads in flight.  (Streaming cache hints on these
// accesses measured 7% slower for the FFN down GEMM, so none are used.)
struct LayerOutIn {
  float4 hb, pn, dprev;
};

__device__ __forceinline__ LayerOutIn layer_out_load(const LayerOutArgs& p, int t, int n) {
  const size_t off = (size_t)t * p.d + n;
  LayerOutIn in;
  in.hb = *reinterpret_cast<const float4*>(p.hbar + off);
  in.pn = make_float4(0.f, 0.f, 0.f, 0.f);
  in.dprev = make_float4(0.f, 0.f, 0.f, 0.f);
  if (!p.last) {
    if (p.p_next) in.pn = load4(p.p_next, off, p.p_bf16);
    if (p.router && !p.first) in.dprev = *reinterpret_cast<const float4*>(p.delta + off);
  }
  return in;
}

__device__ __forceinline__ void layer_out_store(const LayerOutArgs& p, int t, int n,
                                                const LayerOutIn& in, float4 y, float s,
                                                float& ss, float& dd, float& dp) {
  const size_t off = (size_t)t * p.d + n;
  float4 h;
  h.x = in.hb.x + s * y.x;
  h.y = in.hb.y + s * y.y;
  h.z = in.hb.z + s * y.z;
  h.w = in.hb.w + s * y.w;
  if (p.last) {
    *reinterpret_cast<float4*>(p.h_out + off) = h;
    return;
  }
  const float4 pn = in.pn;
  float4 hn;
  hn.x = h.x + pn.x; hn.y = h.y + pn.y; hn.z = h.z + pn.z; hn.w = h.w + pn.w;
  *reinterpret_cast<float4*>(p.hbar + off) = hn;
  ss += hn.x * hn.x + hn.y * hn.y + hn.z * hn.z + hn.w * hn.w;
  if (p.router) {
    float4 dn;
    dn.x = s * y.x + pn.x; dn.y = s * y.y + pn.y; dn.z = s * y.z + pn.z; dn.w = s * y.w + pn.w;
    *reinterpret_cast<float4*>(p.delta + off) = dn;
    store_xl4(p.xl, p.xl_bf16, p.d, t, n, hn);
    const float4 dv = in.dprev;
    dd += dn.x * dn.x + dn.y * dn.y + dn.z * dn.z + dn.w * dn.w;
    dp += dn.x * dv.x + dn.y * dv.y + dn.z * dv.z + dn.w * dv.w;
  }
}

// Scalar form (one column n of token t).
struct LayerOutIn1 {
  float hb, pn, dprev;
};

__device__ __forceinline__ LayerOutIn1 layer_out_load1(const LayerOutArgs& p, int t, int n) {
  const size_t off = (size_t)t * p.d + n;
  LayerOutIn1 in;
  in.hb = p.hbar[off];
  in.pn = 0.f;
  in.dprev = 0.f;
  if (!p.last) {
    if (p.p_next)
      in.pn = p.p_bf16 ? __uint_as_float((uint32_t)static_cast<const uint16_t*>(p.p_next)[off] << 16)
                       : static_cast<const float*>(p.p_next)[off];
    if (p.router && !p.first) in.dprev = p.delta[off];
  }
  return in;
}

__device__ __forceinline__ void layer_out_store1(const LayerOutArgs& p, int t, int n,
                                                 const LayerOutIn1& in, float y, float s,
                                                 float& ss, float& dd, float& dp) {
  const size_t off = (size_t)t * p.d + n;
  const float h = in.hb + s * y;
  if (p.last) {
    p.h_out[off] = h;
    return;
  }
  const float hn = h + in.pn;
  p.hbar[off] = hn;
  ss += hn * hn;
  if (p.router) {
    const float dn = s * y + in.pn;
    p.delta[off] = dn;
    store_xl1(p.xl, p.xl_bf16, p.d, t, n, hn);
    dd += dn * dn;
    dp += dn * in.dprev;
  }
}

// Programmatic dependent launch: wait until the previous kernel of the stream has
// completed and its writes are visible.  Every hot-path kernel calls this first,
// before any global access, so the stream order of memory effects is unchanged
// while the kernel's launch overlaps its predecessor's tail; without the launch
// attribute it is a no-op.  (No early launch_dependents trigger: it let chains of
// waiting CTAs occupy SMs that the persistent GEMMs need, +7% per decode step.)
__device__ __forceinline__ void pdl_enter() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

// ---------------------------------------------------------------------------
// PTX wrappers (sm_100 family: mbarrier, TMA, tcgen05)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: true when the phase with the given parity completed, false after
// limit_ns of %globaltimer.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (globaltimer_ns() - t0 > limit_ns) return false;
  }
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* tm, int x, int y,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* tm, int x, int y, int z,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(z), "r"(bar)
      : "memory");
}

// ---- CTA pairs (thread-block clusters of 2) for the 2-SM tensor-core MMA ----
__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_id_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_count_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}
// Shared::cluster address of the same shared-memory offset in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
// Arrive on an mbarrier that may live in another CTA of the cluster.
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr)
               : "memory");
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                   : "memory");
}
// TMA tile load into this CTA's shared memory whose completion (complete_tx) is signalled
// on an mbarrier of either CTA of the pair (bar: shared::cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* tm, int x, int y,
                                                 uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
// D[tmem] (+)= A B^T over the CTA pair: M = 256 (128 rows of A and of D in each CTA), B
// split along N between the two CTAs' shared memory at the same offsets.  Issued by one
// thread of the even CTA.
__device__ __forceinline__ void umma_bf16_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                               uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on the mbarrier at this offset in both CTAs of the pair once every tcgen05
// operation issued so far by this thread has completed.
__device__ __forceinline__ void umma_commit_pair(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(bar),
      "h"((uint16_t)3)
      : "memory");
}

// Make this thread's generic-proxy shared-memory writes visible to the async proxy
// (a tcgen05.mma that reads them as an operand).
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Bulk prefetch of [p, p + bytes) into L2 (p 16-byte aligned, bytes a multiple of 16).
__device__ __forceinline__ void prefetch_l2(const void* p, int bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

__device__ __forceinline__ void tma_prefetch_desc(const CUtensorMap* tm) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tm)) : "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, bf16 x bf16 -> fp32, M = 128, one CTA.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                          uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on an mbarrier once every tcgen05 operation issued so far by this thread
// has completed.
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}

// Shared-memory matrix descriptor of a K-major tile stored with the 128-byte
// swizzle (rows of 128 bytes, 8-row groups 1024 bytes apart).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);  // start address
  d |= (uint64_t)1 << 16;                    // leading byte offset (unused with swizzle)
  d |= (uint64_t)(1024 >> 4) << 32;          // stride byte offset: 8 rows x 128 B
  d |= (uint64_t)1 << 46;                    // descriptor version
  d |= (uint64_t)2 << 61;                    // 128-byte swizzle
  return d;
}

#define HERO_R8(i) "=r"(r[i]), "=r"(r[i + 1]), "=r"(r[i + 2]), "=r"(r[i + 3]), \
                   "=r"(r[i + 4]), "=r"(r[i + 5]), "=r"(r[i + 6]), "=r"(r[i + 7])

// 32 lanes x 32 consecutive fp32 columns from TMEM (lane quadrant of this warp),
// waiting for the load inside the same asm statement.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : HERO_R8(0), HERO_R8(8), HERO_R8(16), HERO_R8(24)
      : "r"(taddr)
      : "memory");
}

// 128 consecutive fp32 columns in one load, waited for in the same asm statement.
__device__ __forceinline__ void tmem_ld128(uint32_t taddr, uint32_t (&r)[128]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x128.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63, %64, %65, %66, %67, %68, %69, %70, %71, %72, %73, %74, %75, %76, %77, %78, %79, %80, %81, %82, %83, %84, %85, %86, %87, %88, %89, %90, %91, %92, %93, %94, %95, %96, %97, %98, %99, %100, %101, %102, %103, %104, %105, %106, %107, %108, %109, %110, %111, %112, %113, %114, %115, %116, %117, %118, %119, %120, %121, %122, %123, %124, %125, %126, %127}, [%128];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63]), "=r"(r[64]), "=r"(r[65]), "=r"(r[66]), "=r"(r[67]), "=r"(r[68]), "=r"(r[69]), "=r"(r[70]), "=r"(r[71]), "=r"(r[72]), "=r"(r[73]), "=r"(r[74]), "=r"(r[75]), "=r"(r[76]), "=r"(r[77]), "=r"(r[78]), "=r"(r[79]), "=r"(r[80]), "=r"(r[81]), "=r"(r[82]), "=r"(r[83]), "=r"(r[84]), "=r"(r[85]), "=r"(r[86]), "=r"(r[87]), "=r"(r[88]), "=r"(r[89]), "=r"(r[90]), "=r"(r[91]), "=r"(r[92]), "=r"(r[93]), "=r"(r[94]), "=r"(r[95]), "=r"(r[96]), "=r"(r[97]), "=r"(r[98]), "=r"(r[99]), "=r"(r[100]), "=r"(r[101]), "=r"(r[102]), "=r"(r[103]), "=r"(r[104]), "=r"(r[105]), "=r"(r[106]), "=r"(r[107]), "=r"(r[108]), "=r"(r[109]), "=r"(r[110]), "=r"(r[111]), "=r"(r[112]), "=r"(r[113]), "=r"(r[114]), "=r"(r[115]), "=r"(r[116]), "=r"(r[117]), "=r"(r[118]), "=r"(r[119]), "=r"(r[120]), "=r"(r[121]), "=r"(r[122]), "=r"(r[123]), "=r"(r[124]), "=r"(r[125]), "=r"(r[126]), "=r"(r[127])
      : "r"(taddr)
      : "memory");
}

// Store 32 consecutive fp32 columns of this warp's lane quadrant, and wait for it.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};\n\t"
      "tcgen05.wait::st.sync.aligned;" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]),
      "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]),
      "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

// 16 consecutive fp32 columns.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : HERO_R8(0), HERO_R8(8)
      : "r"(taddr)
      : "memory");
}

}  // namespace hero
