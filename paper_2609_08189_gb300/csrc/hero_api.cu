// Host runtime of libhero: parameter loading and repacking, workspace, the
// per-block launch sequence of the routed FFN stack, profiling and the C ABI.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <atomic>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/hero.h"
#include "hero_internal.cuh"

using namespace hero;

namespace {

thread_local std::string g_last_error;

hero_status fail(hero_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

#define CUDA_TRY(expr)                                                                    \
  do {                                                                                    \
    cudaError_t e_ = (expr);                                                              \
    if (e_ != cudaSuccess)                                                                \
      return fail(e_ == cudaErrorMemoryAllocation ? HERO_ERR_NOMEM : HERO_ERR_CUDA,        \
                  "%s failed: %s (%s:%d)", #expr, cudaGetErrorString(e_), __FILE__, __LINE__); \
  } while (0)

// ---- cuTensorMapEncodeTiled through the runtime's driver entry point -----------
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool get_encoder() {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return g_encode != nullptr;
}

// 2-D bf16 tensor [outer, inner] (inner contiguous), box [box_outer, 64] with the
// 128-byte swizzle expected by the tcgen05 shared-memory descriptors.
bool encode_bf16_2d(CUtensorMap* tm, const void* ptr, uint64_t inner, uint64_t outer,
                    uint32_t box_outer) {
  if (!get_encoder()) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {64, box_outer};
  cuuint32_t es[2] = {1, 1};
  CUresult r = g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// The same with rows ld elements apart (ld >= inner): a view of the first `inner` columns.
bool encode_bf16_2d_ld(CUtensorMap* tm, const void* ptr, uint64_t inner, uint64_t outer, uint64_t ld,
                       uint32_t box_outer) {
  if (!get_encoder()) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {64, box_outer};
  cuuint32_t es[2] = {1, 1};
  CUresult r = g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 3-D bf16 map with 64 x 128 x 1 boxes (128-byte swizzle; out-of-range elements read 0):
// dims d0 (contiguous) x d1 x d2, byte strides s1 (between d1 rows) and s2.
bool encode_bf16_3d(CUtensorMap* tm, const void* ptr, uint64_t d0, uint64_t d1, uint64_t d2,
                    uint64_t s1, uint64_t s2) {
  if (!get_encoder()) return false;
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {s1, s2};
  cuuint32_t box[3] = {64, 128, 1};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Nearest bf16 (ties to even) of an fp32 value, as its 16-bit pattern.
uint16_t bf16_bits(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  if ((u & 0x7fffffffu) > 0x7f800000u) return (uint16_t)((u >> 16) | 0x40u);   // NaN stays NaN
  return (uint16_t)((u + 0x7fffu + ((u >> 16) & 1u)) >> 16);
}

float bf16_value(float f) {
  const uint32_t u = (uint32_t)bf16_bits(f) << 16;
  float r;
  memcpy(&r, &u, 4);
  return r;
}

// The router's parameters laid out as RsmBlob<DM> from the packed fp32 copy (already
// rounded to bf16 values on bf16 models, so the bf16 matrices are exact).
struct RouterPackAt {
  size_t hu, p1, pb1, p2, pb2, qkv, n, c, t1, tb1, t2, tb2, psb1, psw2, psb2;
};

template <int DM>
std::vector<uint8_t> router_sm_blob(const std::vector<float>& pk, const RouterPackAt& o) {
  using B = RsmBlob<DM>;
  std::vector<uint8_t> b(B::bytes, 0);
  auto put16 = [&](int region, size_t i, float v) {
    const uint16_t h = bf16_bits(v);
    std::memcpy(&b[region + 2 * i], &h, 2);
  };
  auto put32 = [&](int at, size_t src, int n) {
    std::memcpy(&b[B::f32 + 4 * (size_t)at], &pk[src], 4 * (size_t)n);
  };
  for (size_t i = 0; i < (size_t)kRsmEnc * kRsmDh; ++i) put16(B::hu, i, pk[o.hu + i]);
  for (int k = 0; k < kRsmDs; ++k) {
    for (int q = 0; q < 3 * DM; ++q) put16(B::q4, (size_t)k * 4 * DM + q, pk[o.qkv + (size_t)k * 3 * DM + q]);
    for (int q = 0; q < DM; ++q) put16(B::q4, (size_t)k * 4 * DM + 3 * DM + q, pk[o.n + (size_t)k * DM + q]);
  }
  for (size_t i = 0; i < (size_t)DM * DM; ++i) put16(B::wc, i, pk[o.c + i]);
  for (size_t i = 0; i < (size_t)B::F * kRsmHead; ++i) put16(B::t1, i, pk[o.t1 + i]);
  put32(B::p1, o.p1, 6 * kRsmPath);
  put32(B::pb1, o.pb1, kRsmPath);
  put32(B::p2, o.p2, kRsmPath * kRsmDa);
  put32(B::pb2, o.pb2, kRsmDa);
  put32(B::tb1, o.tb1, kRsmHead);
  put32(B::tw2, o.t2, kRsmHead);
  put32(B::psb1, o.psb1, kRsmHead);
  put32(B::psw2, o.psw2, kRsmHead);
  put32(B::tb2, o.tb2, 1);
  put32(B::psb2, o.psb2, 1);
  return b;
}

std::vector<float> host_f32(const void* p, size_t n, hero_dtype dt) {
  std::vector<float> v(n);
  if (dt == HERO_BF16) {
    const uint16_t* s = static_cast<const uint16_t*>(p);
    for (size_t i = 0; i < n; ++i) {
      uint32_t u = (uint32_t)s[i] << 16;
      memcpy(&v[i], &u, 4);
    }
  } else {
    memcpy(v.data(), p, n * sizeof(float));
  }
  return v;
}

struct ProfEvent {
  int cls;
  cudaEvent_t e0, e1;
};

}  // namespace

struct hero_model {
  hero_config cfg{};
  int device = 0;
  int num_sms = 0;
  bool bf16 = false;
  size_t esz = 4;  // operand element size
  int np = 1;      // partial-sum slots per token

  // parameters
  void* wgu = nullptr;     // bf16: [L][2I][d] gate/up interleaved per 128 rows; f32: gate
  void* wup = nullptr;     // f32 only: [L][I][d]
  void* wdown = nullptr;   // [L][d][I]
  void* w1 = nullptr;      // [L][d_r][d]
  void* w2 = nullptr;      // [L][d][d_r]
  void* wr = nullptr;      // [d_enc + d_head][d]: W_hd diag(g_r) ; f_psi first layer
  float* ffn_gain = nullptr;  // [L][d]
  float* router_small = nullptr;
  RouterWeights rw{};
  std::vector<float> rho;  // [L]

  // workspace
  void* ws = nullptr;
  size_t ws_bytes = 0;
  float *hbar, *delta, *part, *Y, *S, *zeta, *pst, *mst, *dprev, *gate, *scale_f, *scale_a;
  float* splitk_ws = nullptr;   // bf16: partial slices of split-K GEMMs (few-tile launches)
  // the router on the tensor cores (RouterTcArgs): weights, maps and per-token buffers
  // the router at small and medium token counts (launch_router_sm): its parameters as one
  // RsmBlob, or nullptr where that kernel does not serve the model
  void* rsm_w = nullptr;
  bool rtc = false;
  int rt_kf = 0;
  void* rt_w = nullptr;
  CUtensorMap tm_whu3, tm_wq3, tm_th3, tm_enc3, tm_s3, tm_fin3;
  uint16_t *rt_enc3 = nullptr, *rt_s3 = nullptr, *rt_fin3 = nullptr;
  float *rt_scal = nullptr, *rt_s = nullptr, *rt_qkvn = nullptr;
  int* chunk_cnt = nullptr;   // [ceil(T / 32)] FFN decisions per 32 tokens (RouterTcArgs)
  // the history form of the memory (d_m = 64 or 128 on the tensor-core router): per token
  // [L_R][2 d_m] entries phi(k_i) | v_i, and the decay weights [L_R][L_R] (RouterTcArgs)
  float *hist = nullptr, *hw = nullptr;
  void *xl, *u_f, *u_a, *act, *ah;
  uint8_t* mask;
  int *idx_f, *idx_a, *counts;
  uint32_t* err;

  // host-IO staging (lazily grown) and the attention stand-in's upload pipeline
  void* io = nullptr;
  size_t io_bytes = 0;
  cudaStream_t copy_stream = nullptr;
  std::vector<cudaEvent_t> ev_ready, ev_consumed;  // per routed block
  // recorded on the compute stream after the last kernel of every call: the next
  // host-IO call's uploads into the workspace wait for it, not for the previous
  // call's result downloads, so both directions overlap
  cudaEvent_t ev_kernels_done = nullptr;
  // batches of one 128-row tile (bf16, shared-memory router): the router's launches run on
  // side_stream, forked after the block entry (ev_fork) and joined before the block-closing
  // launch (ev_join); rws holds their split-K router contraction slices
  cudaStream_t side_stream = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  float* rws = nullptr;

  // tensor maps (bf16 only)
  CUtensorMap tm_xl, tm_uf, tm_ua, tm_act, tm_ah, tm_wr;
  // the router operand pair stacked along M: xl viewed as [2T][d] (rows 2t = hi, 2t + 1 = lo
  // of token t) against the first copy of the router weight, wr viewed as [nY][d]
  CUtensorMap tm_xl2, tm_wr1;
  std::vector<CUtensorMap> tm_wgu, tm_wd, tm_w1, tm_w2;
  // the same weights with 128-row boxes: the B operands of the CTA-pair GEMM
  CUtensorMap tm_wr_p;
  std::vector<CUtensorMap> tm_wgu_p, tm_wd_p, tm_w1_p;

  // attention sublayer of the full decoder forward (hero_attn_init; bf16 models)
  bool attn = false;
  int n_heads = 0, n_kv_heads = 0;
  float rope_theta = 0.f;
  void* wqkv = nullptr;        // [L][(H + 2 H_kv) 128][d]: W_q | W_k | W_v rows
  void* wo = nullptr;          // [L][d][H 128]
  float* attn_gain = nullptr;  // [L][d]
  void* aws = nullptr;         // attention workspace
  void *ax = nullptr, *aq = nullptr, *ak = nullptr, *av = nullptr, *ao = nullptr;
  void* avt = nullptr;         // v transposed for the tensor-core attention (S >= 128)
  size_t avt_elems = 0;
  float *hcur = nullptr, *dlprev = nullptr;
  float* rope_cs = nullptr;    // [rope_rows][64][2] RoPE cos, sin (own allocation)
  long rope_rows = 0;
  // KV cache (hero_kv_cache_init): per layer [max_seqs][H_kv][max_len][128] bf16, K then V
  void* kv = nullptr;
  int kv_seqs = 0, kv_len = 0;
  float *dec_pm = nullptr, *dec_pl = nullptr, *dec_po = nullptr;   // decode attention partials
  int* dec_pos = nullptr;      // positions staged for HERO_FLAG_HOST_IO
  float* dec_ws = nullptr;     // split-K slices of the decoding step's projections
  size_t dec_ws_floats = 0;
  size_t kv_layer_elems() const { return (size_t)kv_seqs * n_kv_heads * kv_len * 128; }
  uint16_t* kv_k(int jj) { return static_cast<uint16_t*>(kv) + (size_t)jj * 2 * kv_layer_elems(); }
  uint16_t* kv_v(int jj) { return kv_k(jj) + kv_layer_elems(); }
  CUtensorMap tm_ax, tm_ao;
  std::vector<CUtensorMap> tm_wqkv, tm_wo, tm_wqkv_p, tm_wo_p;   // _p: 128-row boxes (pair GEMM)

  // training path (hero_backward_init; bf16 models): transposed copies of the frozen
  // weights, whose rows are the K-major operands of the input-gradient GEMMs, and the
  // backward workspace
  bool bw = false;
  void *wdT = nullptr, *wguT = nullptr, *w1T = nullptr, *w2T = nullptr;
  void* bws = nullptr;
  uint16_t *bw_gu = nullptr, *bw_gf = nullptr, *bw_ga = nullptr;
  __nv_bfloat16* bw_da = nullptr;
  float *bw_rinv = nullptr, *bw_dgpart = nullptr, *bw_a = nullptr, *bw_gaf = nullptr,
        *bw_daf = nullptr, *bw_y2 = nullptr, *bw_duf = nullptr, *bw_dua = nullptr,
        *bw_wpart = nullptr;
  int bw_part_ld = 0;
  CUtensorMap tm_bwgf, tm_bwga, tm_bwgu, tm_bwda;
  std::vector<CUtensorMap> tm_wdT, tm_wguT, tm_w1T, tm_w2T, tm_wdT_p, tm_wguT_p;

  // measurement
  bool profiling = false;
  std::vector<ProfEvent> pending;
  std::vector<cudaEvent_t> event_pool;
  double prof_ms[HERO_K_COUNT] = {};
  int64_t launches[HERO_K_COUNT] = {};
};

namespace {

cudaEvent_t take_event(hero_model* m) {
  if (!m->event_pool.empty()) {
    cudaEvent_t e = m->event_pool.back();
    m->event_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Run one launch of kernel class `cls`, bracketed by events when profiling.
template <class F>
cudaError_t timed(hero_model* m, int cls, cudaStream_t st, F&& launch) {
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  if (m->profiling) {
    e0 = take_event(m);
    cudaEventRecord(e0, st);
  }
  cudaError_t e = launch();
  m->launches[cls]++;
  if (m->profiling) {
    e1 = take_event(m);
    cudaEventRecord(e1, st);
    m->pending.push_back({cls, e0, e1});
  }
  return e;
}

hero_status validate_config(const hero_config* c) {
  if (!c) return fail(HERO_ERR_ARG, "config is NULL");
  if (c->n_layers < 1 || c->d_model < 8 || c->d_ff < 1 || c->d_r < 1 || c->d_m < 1 || c->d_h < 1 ||
      c->d_a < 1 || c->d_enc < 1 || c->d_head < 1 || c->d_path < 1 || c->max_tokens < 1)
    return fail(HERO_ERR_ARG, "config has a non-positive dimension");
  if (c->dtype != HERO_F32 && c->dtype != HERO_BF16) return fail(HERO_ERR_ARG, "unknown dtype");
  if (c->n_dense < 0 || c->n_dense >= c->n_layers)
    return fail(HERO_ERR_ARG, "need 0 <= n_dense < n_layers (got %d)", c->n_dense);
  if (!(c->rms_eps >= 0.f) || !(c->eps >= 0.f) || !(c->t_hist > 0.f))
    return fail(HERO_ERR_ARG, "eps must be >= 0 and t_hist > 0");
  if (c->d_m != 16 && c->d_m != 32 && c->d_m != 64 && c->d_m != 128 && c->d_m != 256)
    return fail(HERO_ERR_UNSUPPORTED, "d_m must be 16, 32, 64, 128 or 256 (got %d)", c->d_m);
  if (c->router_variant & ~(uint32_t)(HERO_ROUTER_NO_HISTORY | HERO_ROUTER_NO_MEMREAD |
                                      HERO_ROUTER_NO_AUX | HERO_ROUTER_NO_POS))
    return fail(HERO_ERR_ARG, "unknown router_variant bits 0x%x", c->router_variant);
  if (c->d_h + c->d_a > 128 || c->d_enc > 256 || c->d_head > 256 || c->d_path > 64)
    return fail(HERO_ERR_UNSUPPORTED, "router widths exceed d_s<=128, d_enc,d_head<=256, d_path<=64");
  if (c->d_h % 4 || c->d_a % 4 || c->d_enc % 4 || c->d_head % 4 || c->d_path % 4)
    return fail(HERO_ERR_UNSUPPORTED, "router widths d_h, d_a, d_enc, d_head, d_path must be multiples of 4");
  if (c->d_model % 8 != 0) return fail(HERO_ERR_UNSUPPORTED, "d_model must be a multiple of 8");
  if (c->dtype == HERO_F32 && c->d_r > 64)
    return fail(HERO_ERR_UNSUPPORTED, "f32 models need d_r <= 64");
  if (c->dtype == HERO_BF16) {
    if (c->d_model % 256 != 0 || c->d_ff % 128 != 0 || c->d_r % 32 != 0 || c->d_r > 4096)
      return fail(HERO_ERR_UNSUPPORTED,
                  "bf16 needs d_model %% 256 == 0, d_ff %% 128 == 0 and d_r %% 32 == 0 (<= 4096)");
    if ((c->d_enc + c->d_head) % 8 != 0)
      return fail(HERO_ERR_UNSUPPORTED, "bf16 needs d_enc + d_head to be a multiple of 8");
  }
  return HERO_OK;
}

// K splits for a tensor-core launch of `tiles` 128x256 output tiles over `kblocks`
// 64-wide K-blocks (`rows` x `n` outputs), from a wave-quantisation cost model: the
// GEMM takes ceil(tiles * s / num_sms) waves of ceil(kblocks / s) K-block steps
// (~0.4 us each on one SM when the tensor pipe bounds them; ~0.75 us at 128 rows or fewer,
// where a step streams its 32 KB weight tile from HBM) plus the last tile's epilogue (~50 us for the block-closing
// epilogue, ~10 us for a plain store), and s > 1 adds a finishing pass that moves
// rows * n * (4 s + epi_bytes) bytes at ~5 TB/s.  rows is the launch's upper bound
// (the routed count is device-resident).  Every split keeps >= 1 K-block.
constexpr int kMaxSplits = 16;
int choose_splits(int tiles, int kblocks, int num_sms, long rows, long n, int epi_bytes) {
  if (tiles <= 0 || kblocks <= 1) return 1;
  double best_t = 0.0;
  int best = 1;
  for (int s = 1; s <= kMaxSplits && s <= kblocks; ++s) {
    const int kpb = (kblocks + s - 1) / s;
    const int eff = (kblocks + kpb - 1) / kpb;   // splits that own K-blocks
    if (eff != s) continue;
    const long waves = ((long)tiles * s + num_sms - 1) / num_sms;
    double t = (double)waves * kpb * (rows <= 128 ? 0.75 : 0.4);
    if (s > 1)
      t += 10.0 + (double)rows * n * (4.0 * s + epi_bytes) / 5.0e6;
    else
      t += epi_bytes > 4 ? 50.0 : 10.0;
    if (s == 1 || t < best_t * 0.97) {   // a split must win by 3%
      best_t = t;
      best = s;
    }
  }
  return best;
}

// Token counts from which the large GEMMs of a block run on CTA pairs (256-row tiles).
constexpr int kPairMinRows = 1024;

// Forward passes over every routed block run the tensor-core router's memory step in its
// history form (k_rt_hist); building with -DHERO_HISTORY_FORM=0 keeps the state form there.
#ifndef HERO_HISTORY_FORM
#define HERO_HISTORY_FORM 1
#endif

// Largest split-K partial buffer (floats) any token count up to T may ask for.
size_t splitk_ws_floats(int T, int num_sms, int nY, int K_router, int d, int I) {
  size_t most = 0;
  for (int m_t = 1; m_t <= (T + 127) / 128; ++m_t) {
    const long rows = (long)m_t * 128;
    const int rs = choose_splits(m_t * ((nY + 255) / 256), (K_router + 63) / 64, num_sms, rows, nY, 4);
    const int ds = choose_splits(m_t * (d / 256), (I + 63) / 64, num_sms, rows, d, 22);
    if (rs > 1) most = std::max(most, (size_t)rs * rows * nY);
    if (ds > 1) most = std::max(most, (size_t)ds * rows * d);
  }
  // the router contraction with the operand pair stacked along M (2T rows, K = K_router / 2)
  for (int m2 = 1; m2 <= (2 * T + 127) / 128; ++m2) {
    const long rows = (long)m2 * 128;
    const int rs2 = choose_splits(m2 * ((nY + 255) / 256), (K_router / 2 + 63) / 64, num_sms, rows, nY, 4);
    if (rs2 > 1) most = std::max(most, (size_t)rs2 * rows * nY);
  }
  return most;
}

// Upload a host matrix [rows, cols] (element type src_dt) through a device staging
// buffer into dst with the row map of launch_convert_rows.
hero_status upload_rows(hero_model* m, const void* src, hero_dtype src_dt, void* dst, long rows,
                        long cols, long grp, long grp_stride, long offset, const float* col_scale,
                        void* stage, size_t stage_elems) {
  const size_t src_es = src_dt == HERO_BF16 ? 2 : 4;
  const size_t dst_es = m->esz;
  long chunk = (long)(stage_elems / (size_t)cols);
  if (grp > 1) chunk = (chunk / grp) * grp;
  if (chunk < 1) return fail(HERO_ERR_NOMEM, "staging buffer too small for a row");
  for (long r0 = 0; r0 < rows; r0 += chunk) {
    const long nr = rows - r0 < chunk ? rows - r0 : chunk;
    CUDA_TRY(cudaMemcpy(stage, static_cast<const char*>(src) + (size_t)r0 * cols * src_es,
                        (size_t)nr * cols * src_es, cudaMemcpyHostToDevice));
    const long dst_row0 = (r0 / grp) * grp_stride;
    void* d = static_cast<char*>(dst) + (size_t)dst_row0 * cols * dst_es;
    CUDA_TRY(launch_convert_rows(stage, src_dt == HERO_BF16, d, m->bf16, nr, cols, grp, grp_stride,
                                 offset, col_scale, 0));
  }
  return HERO_OK;
}

void free_model(hero_model* m) {
  if (!m) return;
  cudaDeviceSynchronize();
  for (auto& p : m->pending) {
    cudaEventDestroy(p.e0);
    cudaEventDestroy(p.e1);
  }
  for (auto e : m->event_pool) cudaEventDestroy(e);
  for (auto e : m->ev_ready) cudaEventDestroy(e);
  for (auto e : m->ev_consumed) cudaEventDestroy(e);
  if (m->ev_kernels_done) cudaEventDestroy(m->ev_kernels_done);
  if (m->ev_fork) cudaEventDestroy(m->ev_fork);
  if (m->ev_join) cudaEventDestroy(m->ev_join);
  if (m->copy_stream) cudaStreamDestroy(m->copy_stream);
  if (m->side_stream) cudaStreamDestroy(m->side_stream);
  void* ptrs[] = {m->wgu, m->wup, m->wdown, m->w1, m->w2, m->wr, m->ffn_gain, m->router_small,
                  m->ws, m->io, m->wqkv, m->wo, m->attn_gain, m->aws, m->rope_cs, m->kv,
                  m->dec_pm, m->dec_pos, m->dec_ws, m->wdT, m->wguT, m->w1T, m->w2T, m->bws,
                  m->rt_w, m->rsm_w};
  for (void* p : ptrs)
    if (p) cudaFree(p);
  delete m;
}

}  // namespace

// ============================================================================
// C ABI
// ============================================================================

extern "C" const char* hero_last_error(void) { return g_last_error.c_str(); }

namespace {
std::atomic<uint64_t> g_wait_limit_ns{0};   // 0: the default bound
}  // namespace

uint64_t hero::wait_limit_ns() {
  const uint64_t v = g_wait_limit_ns.load(std::memory_order_relaxed);
  return v ? v : kWaitLimitNs;
}

extern "C" void hero_set_wait_limit_ns(uint64_t limit_ns) {
  g_wait_limit_ns.store(limit_ns, std::memory_order_relaxed);
}

hero_status hero::status_of_error_word(uint32_t e) {
  if (!e) return HERO_OK;
  if (e & (ERR_WAIT_PRODUCER | ERR_WAIT_MMA | ERR_WAIT_EPILOGUE | ERR_WAIT_DRAIN))
    return fail(HERO_ERR_TIMEOUT, "a device-side wait bound expired (error word 0x%x)", e);
  return fail(HERO_ERR_BAD_INDEX, "a kernel met an index outside its bounds (error word 0x%x)", e);
}

void hero::set_last_error(const char* msg) { g_last_error = msg; }

extern "C" hero_status hero_init_weights(const hero_config* cfg, const hero_weights_host* w,
                                         hero_model** out) {
  g_last_error.clear();
  if (!out) return fail(HERO_ERR_ARG, "out is NULL");
  *out = nullptr;
  hero_status s = validate_config(cfg);
  if (s != HERO_OK) return s;
  if (!w) return fail(HERO_ERR_ARG, "weights are NULL");
  const void* need[] = {w->ffn_norm_g, w->w_gate, w->w_up, w->w_down, w->ad_w1, w->ad_w2, w->eta,
                        w->r_norm_g, w->w_hd, w->w_hu, w->path_w1, w->path_b1, w->path_w2,
                        w->path_b2, w->w_q, w->w_k, w->w_v, w->w_n, w->w_c, w->th_w1, w->th_b1,
                        w->th_w2, w->th_b2, w->ps_w1, w->ps_b1, w->ps_w2, w->ps_b2};
  for (size_t i = 0; i < sizeof(need) / sizeof(need[0]); ++i)
    if (!need[i]) return fail(HERO_ERR_ARG, "weight pointer %zu is NULL", i);
  if (w->host_dtype != HERO_F32 && w->host_dtype != HERO_BF16)
    return fail(HERO_ERR_ARG, "unknown host_dtype");
  if (w->host_dtype == HERO_BF16 && cfg->dtype != HERO_BF16)
    return fail(HERO_ERR_ARG, "bf16 host weights need a bf16 model");

  int dev = 0;
  CUDA_TRY(cudaGetDevice(&dev));
  cudaDeviceProp prop;
  CUDA_TRY(cudaGetDeviceProperties(&prop, dev));
  const bool bf16 = cfg->dtype == HERO_BF16;
  if (bf16 && prop.major < 10)
    return fail(HERO_ERR_UNSUPPORTED, "bf16 models need an sm_100-family GPU (found sm_%d%d)",
                prop.major, prop.minor);
  if (bf16 && !get_encoder())
    return fail(HERO_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");

  hero_model* m = new hero_model();
  m->cfg = *cfg;
  m->device = dev;
  m->num_sms = prop.multiProcessorCount;
  m->bf16 = bf16;
  m->esz = bf16 ? 2 : 4;
  const hero_config& c = *cfg;
  const long L = c.n_layers, d = c.d_model, I = c.d_ff, r = c.d_r, dm = c.d_m;
  const long ds = c.d_h + c.d_a, nY = c.d_enc + c.d_head;
  m->np = bf16 ? (int)(d / kTcPartCols) : (int)((d + kSimtTileN - 1) / kSimtTileN);
  const hero_dtype hd = w->host_dtype;
  const size_t hes = hd == HERO_BF16 ? 2 : 4;

  auto bail = [&](hero_status st) {
    free_model(m);
    return st;
  };
#define TRY_M(expr)                      \
  do {                                   \
    hero_status st_ = (expr);            \
    if (st_ != HERO_OK) return bail(st_); \
  } while (0)
#define CUDA_M(expr)                                                                        \
  do {                                                                                      \
    cudaError_t e_ = (expr);                                                                \
    if (e_ != cudaSuccess)                                                                  \
      return bail(fail(e_ == cudaErrorMemoryAllocation ? HERO_ERR_NOMEM : HERO_ERR_CUDA,    \
                       "%s failed: %s", #expr, cudaGetErrorString(e_)));                    \
  } while (0)

  // ---- parameters ----
  const size_t es = m->esz;
  if (bf16) {
    CUDA_M(cudaMalloc(&m->wgu, (size_t)L * 2 * I * d * es));
  } else {
    CUDA_M(cudaMalloc(&m->wgu, (size_t)L * I * d * es));
    CUDA_M(cudaMalloc(&m->wup, (size_t)L * I * d * es));
  }
  CUDA_M(cudaMalloc(&m->wdown, (size_t)L * d * I * es));
  CUDA_M(cudaMalloc(&m->w1, (size_t)L * r * d * es));
  CUDA_M(cudaMalloc(&m->w2, (size_t)L * d * r * es));
  CUDA_M(cudaMalloc(&m->wr, (size_t)nY * d * es * (bf16 ? 2 : 1)));  // bf16: [W | W] for hi | lo

  size_t stage_elems = (size_t)1 << 25;  // 32 Mi elements
  void* stage = nullptr;
  CUDA_M(cudaMalloc(&stage, stage_elems * 4));
  float* gain_r = nullptr;
  auto cleanup_stage = [&] {
    if (stage) cudaFree(stage);
    if (gain_r) cudaFree(gain_r);
    stage = nullptr;
    gain_r = nullptr;
  };
  auto up = [&](const void* src, void* dst, long rows, long cols, long grp, long gstride,
                long off, const float* cs) {
    hero_status st = upload_rows(m, src, hd, dst, rows, cols, grp, gstride, off, cs, stage,
                                 stage_elems);
    return st;
  };
  hero_status st = HERO_OK;
  for (long j = 0; j < L && st == HERO_OK; ++j) {
    const char* g = static_cast<const char*>(w->w_gate) + (size_t)j * I * d * hes;
    const char* u = static_cast<const char*>(w->w_up) + (size_t)j * I * d * hes;
    if (bf16) {
      void* dst = static_cast<char*>(m->wgu) + (size_t)j * 2 * I * d * es;
      st = up(g, dst, I, d, 128, 256, 0, nullptr);
      if (st == HERO_OK) st = up(u, dst, I, d, 128, 256, 128, nullptr);
    } else {
      st = up(g, static_cast<char*>(m->wgu) + (size_t)j * I * d * es, I, d, 1, 1, 0, nullptr);
      if (st == HERO_OK)
        st = up(u, static_cast<char*>(m->wup) + (size_t)j * I * d * es, I, d, 1, 1, 0, nullptr);
    }
    if (st == HERO_OK)
      st = up(static_cast<const char*>(w->w_down) + (size_t)j * d * I * hes,
              static_cast<char*>(m->wdown) + (size_t)j * d * I * es, d, I, 1, 1, 0, nullptr);
    if (st == HERO_OK)
      st = up(static_cast<const char*>(w->ad_w1) + (size_t)j * r * d * hes,
              static_cast<char*>(m->w1) + (size_t)j * r * d * es, r, d, 1, 1, 0, nullptr);
    if (st == HERO_OK)
      st = up(static_cast<const char*>(w->ad_w2) + (size_t)j * d * r * hes,
              static_cast<char*>(m->w2) + (size_t)j * d * r * es, d, r, 1, 1, 0, nullptr);
  }
  if (st == HERO_OK) {
    // router contraction weight: rows [0, d_enc) = W_hd diag(g_r), rounded once;
    // rows [d_enc, d_enc + d_head) = first layer of f_psi.
    std::vector<float> gr = host_f32(w->r_norm_g, d, hd);
    if (cudaMalloc(&gain_r, d * sizeof(float)) != cudaSuccess ||
        cudaMemcpy(gain_r, gr.data(), d * sizeof(float), cudaMemcpyHostToDevice) != cudaSuccess)
      st = fail(HERO_ERR_CUDA, "router gain upload failed");
    // bf16 models contract it against the operand pair [hi | lo] of h_bar, so the
    // weight is stored twice along K: wr = [W | W], [nY, 2d].
    void* wr1 = m->wr;
    if (st == HERO_OK && bf16 && cudaMalloc(&wr1, (size_t)nY * d * es) != cudaSuccess)
      st = fail(HERO_ERR_NOMEM, "router weight staging allocation failed");
    if (st == HERO_OK) st = up(w->w_hd, wr1, c.d_enc, d, 1, 1, 0, gain_r);
    if (st == HERO_OK)
      st = up(w->ps_w1, static_cast<char*>(wr1) + (size_t)c.d_enc * d * es, c.d_head, d, 1, 1, 0,
              nullptr);
    if (st == HERO_OK && bf16) {
      const size_t wb = (size_t)d * es;
      if (cudaMemcpy2D(m->wr, 2 * wb, wr1, wb, wb, nY, cudaMemcpyDeviceToDevice) != cudaSuccess ||
          cudaMemcpy2D(static_cast<char*>(m->wr) + wb, 2 * wb, wr1, wb, wb, nY,
                       cudaMemcpyDeviceToDevice) != cudaSuccess)
        st = fail(HERO_ERR_CUDA, "router weight duplication failed");
    }
    if (bf16 && wr1 && wr1 != m->wr) cudaFree(wr1);
  }
  if (st == HERO_OK && cudaDeviceSynchronize() != cudaSuccess)
    st = fail(HERO_ERR_CUDA, "weight conversion failed: %s", cudaGetErrorString(cudaGetLastError()));
  cleanup_stage();
  if (st != HERO_OK) return bail(st);

  {  // LN^ffn gains and forgetting factors
    std::vector<float> gains = host_f32(w->ffn_norm_g, (size_t)L * d, hd);
    CUDA_M(cudaMalloc(&m->ffn_gain, gains.size() * sizeof(float)));
    CUDA_M(cudaMemcpy(m->ffn_gain, gains.data(), gains.size() * sizeof(float), cudaMemcpyHostToDevice));
    std::vector<float> eta = host_f32(w->eta, L, hd);
    m->rho.resize(L);
    for (long j = 0; j < L; ++j) m->rho[j] = (float)(1.0 / (1.0 + std::exp(-(double)eta[j])));
  }
  {  // shared router parameters, transposed to [in][out]; bf16 models round every
     // parameter to bf16 (the precision contract), these included
    std::vector<float> pack;
    auto params = [&](const void* src, size_t n) {
      std::vector<float> v = host_f32(src, n, hd);
      if (bf16)
        for (float& x : v) x = bf16_value(x);
      return v;
    };
    auto add_t = [&](const void* src, long rows, long cols) {  // src [rows][cols] -> [cols][rows]
      std::vector<float> v = params(src, (size_t)rows * cols);
      pack.resize((pack.size() + 3) & ~(size_t)3);  // 16-byte aligned sub-arrays
      size_t at = pack.size();
      pack.resize(at + (size_t)rows * cols);
      for (long i = 0; i < rows; ++i)
        for (long k = 0; k < cols; ++k) pack[at + (size_t)k * rows + i] = v[(size_t)i * cols + k];
      return at;
    };
    auto add = [&](const void* src, long n) {
      std::vector<float> v = params(src, n);
      pack.resize((pack.size() + 3) & ~(size_t)3);
      size_t at = pack.size();
      pack.insert(pack.end(), v.begin(), v.end());
      return at;
    };
    size_t o_hu = add_t(w->w_hu, c.d_h, c.d_enc);
    size_t o_p1 = add_t(w->path_w1, c.d_path, 6);
    size_t o_pb1 = add(w->path_b1, c.d_path);
    size_t o_p2 = add_t(w->path_w2, c.d_a, c.d_path);
    size_t o_pb2 = add(w->path_b2, c.d_a);
    // q | k | v as one [d_s][3 d_m] matrix
    pack.resize((pack.size() + 3) & ~(size_t)3);
    size_t o_qkv = pack.size();
    pack.resize(o_qkv + (size_t)ds * 3 * dm);
    {
      const void* src[3] = {w->w_q, w->w_k, w->w_v};
      for (int p = 0; p < 3; ++p) {
        std::vector<float> v = params(src[p], (size_t)dm * ds);
        for (long i = 0; i < dm; ++i)
          for (long k = 0; k < ds; ++k)
            pack[o_qkv + (size_t)k * 3 * dm + p * dm + i] = v[(size_t)i * ds + k];
      }
    }
    size_t o_n = add_t(w->w_n, dm, ds);
    size_t o_c = add_t(w->w_c, dm, dm);
    size_t o_t1 = add_t(w->th_w1, c.d_head, ds + dm + 1);
    size_t o_tb1 = add(w->th_b1, c.d_head);
    size_t o_t2 = add(w->th_w2, c.d_head);
    size_t o_tb2 = add(w->th_b2, 1);
    size_t o_pb = add(w->ps_b1, c.d_head);
    size_t o_p2w = add(w->ps_w2, c.d_head);
    size_t o_p2b = add(w->ps_b2, 1);
    CUDA_M(cudaMalloc(&m->router_small, pack.size() * sizeof(float)));
    CUDA_M(cudaMemcpy(m->router_small, pack.data(), pack.size() * sizeof(float),
                      cudaMemcpyHostToDevice));
    float* b = m->router_small;
    m->rw = RouterWeights{b + o_hu, b + o_p1, b + o_pb1, b + o_p2, b + o_pb2, b + o_qkv, b + o_n,
                          b + o_c,  b + o_t1, b + o_tb1, b + o_t2, b + o_tb2, b + o_pb, b + o_p2w,
                          b + o_p2b};
    if (bf16 && router_sm_supported(c.d_enc, c.d_head, c.d_h, c.d_a, c.d_path, dm)) {
      const RouterPackAt at{o_hu, o_p1, o_pb1, o_p2, o_pb2, o_qkv, o_n, o_c,
                            o_t1, o_tb1, o_t2, o_tb2, o_pb, o_p2w, o_p2b};
      const std::vector<uint8_t> blob = dm == 16   ? router_sm_blob<16>(pack, at)
                                        : dm == 32 ? router_sm_blob<32>(pack, at)
                                                   : router_sm_blob<64>(pack, at);
      CUDA_M(cudaMalloc(&m->rsm_w, blob.size()));
      CUDA_M(cudaMemcpy(m->rsm_w, blob.data(), blob.size(), cudaMemcpyHostToDevice));
    }
    // the router on the tensor cores (large token counts): W_hu, [W_q; W_k; W_v; W_n] and
    // W_th1 as bf16 B operands, each repeated three times along K (one copy per bf16 term
    // of the activation), f_theta's K zero-padded to a multiple of 64
    m->rtc = bf16 && c.d_enc == 256 && c.d_head == 256 && c.d_h == 48 && c.d_a == 16 &&
             c.d_path == 16 && dm <= 128 && c.max_tokens >= kPairMinRows;
    if (m->rtc) {
      const long F = ds + dm + 1;
      m->rt_kf = (int)((3 * F + 63) / 64 * 64);
      std::vector<uint16_t> whu3((size_t)c.d_h * 768), wq3((size_t)4 * dm * 3 * ds),
          th3((size_t)c.d_head * m->rt_kf, 0);
      const std::vector<float> hu = params(w->w_hu, (size_t)c.d_h * c.d_enc);
      for (long o = 0; o < c.d_h; ++o)
        for (int pp = 0; pp < 3; ++pp)
          for (long i = 0; i < 256; ++i) whu3[o * 768 + pp * 256 + i] = bf16_bits(hu[o * 256 + i]);
      const void* qs[4] = {w->w_q, w->w_k, w->w_v, w->w_n};
      for (int r4 = 0; r4 < 4; ++r4) {
        const std::vector<float> v = params(qs[r4], (size_t)dm * ds);
        for (long o = 0; o < dm; ++o)
          for (int pp = 0; pp < 3; ++pp)
            for (long i = 0; i < ds; ++i)
              wq3[((size_t)r4 * dm + o) * 3 * ds + pp * ds + i] = bf16_bits(v[o * ds + i]);
      }
      const std::vector<float> th = params(w->th_w1, (size_t)c.d_head * F);
      for (long o = 0; o < c.d_head; ++o)
        for (int pp = 0; pp < 3; ++pp)
          for (long i = 0; i < F; ++i) th3[(size_t)o * m->rt_kf + pp * F + i] = bf16_bits(th[o * F + i]);
      const size_t n_hu = whu3.size(), n_q = wq3.size(), n_th = th3.size();
      CUDA_M(cudaMalloc(&m->rt_w, (n_hu + n_q + n_th) * 2));
      uint16_t* rb = static_cast<uint16_t*>(m->rt_w);
      CUDA_M(cudaMemcpy(rb, whu3.data(), n_hu * 2, cudaMemcpyHostToDevice));
      CUDA_M(cudaMemcpy(rb + n_hu, wq3.data(), n_q * 2, cudaMemcpyHostToDevice));
      CUDA_M(cudaMemcpy(rb + n_hu + n_q, th3.data(), n_th * 2, cudaMemcpyHostToDevice));
      if (!encode_bf16_2d(&m->tm_whu3, rb, 768, c.d_h, 128) ||
          !encode_bf16_2d(&m->tm_wq3, rb + n_hu, 3 * ds, 4 * dm, 128) ||
          !encode_bf16_2d(&m->tm_th3, rb + n_hu + n_q, m->rt_kf, c.d_head, 128))
        return bail(fail(HERO_ERR_CUDA, "tensor map encoding failed"));
    }
  }

  // ---- workspace ----
  {
    const size_t Tm = (size_t)c.max_tokens;
    const long LR = c.n_layers - c.n_dense;   // routed blocks
    const bool hist_form = HERO_HISTORY_FORM && m->rtc && (dm == 64 || dm == 128) && LR > 0;
    size_t off = 0;
    struct Item {
      void** p;
      size_t bytes;
    };
    std::vector<Item> items = {
        {(void**)&m->hbar, Tm * d * 4},        {(void**)&m->delta, Tm * d * 4},
        {(void**)&m->part, Tm * m->np * 16},   {(void**)&m->Y, Tm * nY * 4 * (bf16 ? 2 : 1)},
        {(void**)&m->S, Tm * dm * dm * 4},     {(void**)&m->zeta, Tm * dm * 4},
        {(void**)&m->pst, Tm * 4},             {(void**)&m->mst, Tm * 4},
        {(void**)&m->dprev, Tm * 4},           {(void**)&m->gate, Tm * 4},
        {(void**)&m->scale_f, Tm * 4},         {(void**)&m->scale_a, Tm * 4},
        {(void**)&m->xl, Tm * d * es * (bf16 ? 2 : 1)},         {(void**)&m->u_f, Tm * d * es},
        {(void**)&m->u_a, Tm * d * es},        {(void**)&m->act, Tm * I * es},
        {(void**)&m->ah, Tm * r * es},         {(void**)&m->mask, Tm},
        {(void**)&m->idx_f, Tm * 4},           {(void**)&m->idx_a, Tm * 4},
        {(void**)&m->counts, 64},              {(void**)&m->err, 64},
        {(void**)&m->rt_enc3, m->rtc ? Tm * 768 * 2 : 0},
        {(void**)&m->rt_scal, m->rtc ? Tm * 4 * 4 : 0},
        {(void**)&m->rt_s, m->rtc ? Tm * ds * 4 : 0},
        {(void**)&m->rt_s3, m->rtc ? Tm * 3 * ds * 2 : 0},
        {(void**)&m->rt_qkvn, m->rtc ? Tm * 4 * dm * 4 : 0},
        {(void**)&m->rt_fin3, m->rtc ? Tm * (size_t)m->rt_kf * 2 : 0},
        {(void**)&m->chunk_cnt, m->rtc ? (Tm + 31) / 32 * 4 : 0},
        {(void**)&m->hist, hist_form ? Tm * (size_t)LR * 2 * dm * 4 : 0},
        {(void**)&m->hw, hist_form ? (size_t)LR * LR * 4 : 0},
        // split-K partials of the few-wave launches (router contraction, FFN down)
        {(void**)&m->splitk_ws, bf16 ? splitk_ws_floats(c.max_tokens, m->num_sms, (int)nY,
                                                        (int)(2 * d), (int)d, (int)I) * 4 : 0},
        // the router contraction beside the FFN (one 128-row tile of tokens: at most 256
        // stacked rows, at most kMaxSplits slices)
        {(void**)&m->rws, m->rsm_w ? (size_t)kMaxSplits * 256 * nY * 4 : 0},
    };
    for (auto& it : items) off += (it.bytes + 1023) & ~(size_t)1023;
    CUDA_M(cudaMalloc(&m->ws, off));
    CUDA_M(cudaMemset(m->ws, 0, off));
    m->ws_bytes = off;
    off = 0;
    for (auto& it : items) {
      *it.p = static_cast<char*>(m->ws) + off;
      off += (it.bytes + 1023) & ~(size_t)1023;
    }
    if (hist_form) {   // hw[jb L_R + i] = rho_{i+1} ... rho_{jb-1} (0-based routed blocks)
      std::vector<float> hw((size_t)LR * LR, 0.f);
      for (long jb = 0; jb < LR; ++jb) {
        double wgt = 1.0;
        for (long i = jb - 1; i >= 0; --i) {
          hw[(size_t)jb * LR + i] = (float)wgt;
          wgt *= (double)m->rho[c.n_dense + i];
        }
      }
      CUDA_M(cudaMemcpy(m->hw, hw.data(), hw.size() * 4, cudaMemcpyHostToDevice));
    } else {
      m->hist = m->hw = nullptr;
    }
  }

  // ---- tensor maps ----
  if (bf16) {
    const uint64_t Tm = (uint64_t)c.max_tokens;
    bool ok = encode_bf16_2d(&m->tm_xl, m->xl, 2 * d, Tm, 128) &&
              encode_bf16_2d(&m->tm_uf, m->u_f, d, Tm, 128) &&
              encode_bf16_2d(&m->tm_ua, m->u_a, d, Tm, 128) &&
              encode_bf16_2d(&m->tm_act, m->act, I, Tm, 128) &&
              encode_bf16_2d(&m->tm_ah, m->ah, r, Tm, 128) &&
              encode_bf16_2d(&m->tm_wr, m->wr, 2 * d, nY, 256);
    ok = ok && encode_bf16_2d(&m->tm_wr_p, m->wr, 2 * d, nY, 128);
    ok = ok && encode_bf16_2d_ld(&m->tm_xl2, m->xl, d, 2 * Tm, d, 128) &&
         encode_bf16_2d_ld(&m->tm_wr1, m->wr, d, nY, 2 * d, 256);
    if (m->rtc)
      ok = ok && encode_bf16_2d(&m->tm_enc3, m->rt_enc3, 768, Tm, 128) &&
           encode_bf16_2d(&m->tm_s3, m->rt_s3, 3 * ds, Tm, 128) &&
           encode_bf16_2d(&m->tm_fin3, m->rt_fin3, m->rt_kf, Tm, 128);
    m->tm_wgu.resize(L);
    m->tm_wd.resize(L);
    m->tm_w1.resize(L);
    m->tm_w2.resize(L);
    m->tm_wgu_p.resize(L);
    m->tm_wd_p.resize(L);
    m->tm_w1_p.resize(L);
    for (long j = 0; j < L && ok; ++j) {
      const char* wgu_j = static_cast<char*>(m->wgu) + (size_t)j * 2 * I * d * 2;
      const char* wd_j = static_cast<char*>(m->wdown) + (size_t)j * d * I * 2;
      const char* w1_j = static_cast<char*>(m->w1) + (size_t)j * r * d * 2;
      ok = encode_bf16_2d(&m->tm_wgu[j], wgu_j, d, 2 * I, 256) &&
           encode_bf16_2d(&m->tm_wd[j], wd_j, I, d, 256) &&
           encode_bf16_2d(&m->tm_w1[j], w1_j, d, r, 256) &&
           encode_bf16_2d(&m->tm_w2[j], static_cast<char*>(m->w2) + (size_t)j * d * r * 2, r, d,
                          256) &&
           encode_bf16_2d(&m->tm_wgu_p[j], wgu_j, d, 2 * I, 128) &&
           encode_bf16_2d(&m->tm_wd_p[j], wd_j, I, d, 128) &&
           encode_bf16_2d(&m->tm_w1_p[j], w1_j, d, r, 128);
    }
    if (!ok) return bail(fail(HERO_ERR_CUDA, "tensor map encoding failed"));
  }
  CUDA_M(cudaEventCreateWithFlags(&m->ev_kernels_done, cudaEventDisableTiming));
  if (m->rsm_w) {
    CUDA_M(cudaStreamCreateWithFlags(&m->side_stream, cudaStreamNonBlocking));
    CUDA_M(cudaEventCreateWithFlags(&m->ev_fork, cudaEventDisableTiming));
    CUDA_M(cudaEventCreateWithFlags(&m->ev_join, cudaEventDisableTiming));
  }
  *out = m;
  return HERO_OK;
#undef TRY_M
#undef CUDA_M
}

extern "C" void hero_free(hero_model* m) { free_model(m); }

namespace {

hero_status ensure_io(hero_model* m, size_t bytes) {
  if (m->io_bytes >= bytes) return HERO_OK;
  if (m->io) cudaFree(m->io);
  m->io = nullptr;
  m->io_bytes = 0;
  CUDA_TRY(cudaMalloc(&m->io, bytes));
  m->io_bytes = bytes;
  return HERO_OK;
}

// Router state of one forward pass (workspace for the fused stack, the caller's
// for hero_routed_block).
// hist: the history form of the memory (k_rt_hist) for a forward pass over every routed
// block from a fresh state, or nullptr (the state S, zeta).
struct BlockState {
  float *S, *zeta, *pst, *mst, *dprev;
  float* hist;
};



// Everything of block jj (layer index; routed index jr = jj - n_dense) after its
// entry (h_bar, its operand copy and the partial sums are in place): router
// contraction and router, compaction, LN_ffn, FFN and adapter branches with the
// block-closing epilogue `lo`.  HERO_FLAG_DENSE in flags runs the plain FFN block.
hero_status block_body(hero_model* m, int jj, int jr, int T, const BlockState& bs, const float* hbar,
                       const LayerOutArgs& lo, float tau, uint32_t flags, const uint8_t* mask_in_j,
                       float* gate_out_j, uint8_t* mask_out_j, int32_t* count_out_j,
                       cudaStream_t st) {
  const hero_config& c = m->cfg;
  const int L = c.n_layers, d = c.d_model, I = c.d_ff, r = c.d_r;
  const int nY = c.d_enc + c.d_head;
  const int j = jr + 1;                 // routed index (layer jj = n_dense + jr)
  const bool dense = flags & HERO_FLAG_DENSE;
  const size_t es = m->esz;
  bool chunk_counted = false;   // the router left per-32-token FFN counts (m->chunk_cnt)
  // One 128-row tile of tokens (a decoding batch): the FFN and the adapter branch run on
  // every token while the router runs on the model's second stream, on the SMs that the
  // gate/up launch leaves idle; the block-closing launch then takes each token's branch from
  // the router's decision (Eq. 3), so every output equals that of the compacted branches.
  // Bypassed tokens cost FFN FLOPs, but at one tile the FFN GEMMs are bound by their weight
  // stream, which they read whole either way.
  const int m_t0 = (T + 127) / 128;
  const int gu_units = std::min(m_t0 * ((2 * I + 255) / 256 + (r + 255) / 256), m->num_sms);
  const int side_sms = m->num_sms - gu_units;
  const int ds0 = m->bf16 ? choose_splits(m_t0 * (d / 256), (I + 63) / 64, m->num_sms,
                                          (long)m_t0 * 128, d, 22)
                          : 1;
  const bool spec_shape = !dense && m->bf16 && m->side_stream && m->rsm_w &&
                          c.router_variant == 0 && T > 0 && T <= 128 && r <= 64 && r % 8 == 0 &&
                          ds0 > 1 && side_sms >= 16;
  const bool spec = spec_shape && !(flags & HERO_FLAG_NO_SPECULATE);
  const cudaStream_t rst = spec ? m->side_stream : st;   // the router's stream
  // the router's SMs, which set its split count and tokens per CTA (and with them its fp32
  // summation order): the same with HERO_FLAG_NO_SPECULATE, so both give the same bits
  const int r_sms = spec_shape ? side_sms : m->num_sms;
  if (spec) {
    CUDA_TRY(cudaEventRecord(m->ev_fork, st));
    CUDA_TRY(cudaStreamWaitEvent(rst, m->ev_fork, 0));
  }
  if (!dense) {
    GemmArgs g{};
    g.m_dev = nullptr;
    g.m_static = T;
    g.m_max = T;
    g.N = nY;
    g.K = m->bf16 ? 2 * d : d;   // bf16: K runs over the operand pair [hi | lo]
    g.out_f32 = m->Y;
    g.ldo = nY;
    g.err = m->err;
    g.A = m->xl;
    g.B = m->wr;
    g.lda = d;
    g.ldb = d;
    const int m_t = (T + 127) / 128;
    const int rs = m->bf16 ? choose_splits(m_t * ((nY + 255) / 256), (g.K + 63) / 64, m->num_sms,
                                           (long)m_t * 128, nY, 4) : 1;
    if (rs > 1) {   // few tiles (small T): split K, then add the slices in order into Y
      g.out_f32 = m->splitk_ws;
      g.k_splits = rs;
      g.split_stride = (long)m_t * 128 * nY;
    }
    const bool pair = m->bf16 && rs == 1 && T >= kPairMinRows;
    if (pair && m->rtc && c.router_variant == 0) {
      chunk_counted = true;
      // the router on the tensor cores: five launches (RouterTcArgs)
      RouterTcArgs rt{};
      rt.T = T;
      rt.j = j;
      rt.L = L - c.n_dense;
      rt.np = m->np;
      rt.d = d;
      rt.d_h = c.d_h;
      rt.d_a = c.d_a;
      rt.d_path = c.d_path;
      rt.dm = c.d_m;
      rt.rms_eps = c.rms_eps;
      rt.eps = c.eps;
      rt.t_hist = c.t_hist;
      rt.tau = tau;
      rt.rho = m->rho[jj];
      rt.part = m->part;
      rt.dprev = bs.dprev;
      rt.pst = bs.pst;
      rt.mst = bs.mst;
      rt.S = bs.S;
      rt.zeta = bs.zeta;
      rt.hist = bs.hist;
      rt.hist_ld = (long)rt.L * 2 * c.d_m;
      rt.hw = m->hw;
      rt.w = m->rw;
      rt.enc3 = m->rt_enc3;
      rt.scal = m->rt_scal;
      rt.s = m->rt_s;
      rt.s3 = m->rt_s3;
      rt.qkvn = m->rt_qkvn;
      rt.fin3 = m->rt_fin3;
      rt.kf = m->rt_kf;
      rt.mask_in = mask_in_j;
      rt.gate = m->gate;
      rt.mask = m->mask;
      rt.gate_out = gate_out_j;
      rt.mask_out = mask_out_j;
      rt.chunk_cnt = m->chunk_cnt;
      const int ds = c.d_h + c.d_a;
      GemmArgs g1 = g;   // 1. the router contraction, encoder hidden and f_psi in the epilogue
      g1.rt = rt;
      CUDA_TRY(timed(m, HERO_K_ROUTER_GEMM, st, [&] {
        return launch_gemm_tc2(EPI_RT_ENC, m->tm_xl, m->tm_wr_p, g1, m->num_sms, st);
      }));
      auto small = [&](int N, int K) {
        GemmArgs q{};
        q.m_static = T;
        q.m_max = T;
        q.N = N;
        q.K = K;
        q.err = m->err;
        q.rt = rt;
        return q;
      };
      GemmArgs g2 = small(c.d_h, 3 * 256);   // 2. z_h = W_hu enc; path encoder; s
      CUDA_TRY(timed(m, HERO_K_ROUTER, st, [&] {
        return launch_gemm_tc2(EPI_RT_S, m->tm_enc3, m->tm_whu3, g2, m->num_sms, st);
      }));
      GemmArgs g3 = small(4 * c.d_m, 3 * ds);   // 3. q | k | v | W_n s
      g3.out_f32 = m->rt_qkvn;
      g3.ldo = 4 * c.d_m;
      CUDA_TRY(timed(m, HERO_K_ROUTER, st, [&] {
        return launch_gemm_tc2(EPI_STORE_F32, m->tm_s3, m->tm_wq3, g3, m->num_sms, st);
      }));
      CUDA_TRY(timed(m, HERO_K_ROUTER, st, [&] {   // 4.
        return rt.hist ? launch_rt_hist(rt, st) : launch_rt_mem(rt, st);
      }));
      GemmArgs g5 = small(c.d_head, m->rt_kf);   // 5. f_theta, p_hist, m_hist, g, decision
      CUDA_TRY(timed(m, HERO_K_ROUTER, st, [&] {
        return launch_gemm_tc2(EPI_RT_HEAD, m->tm_fin3, m->tm_th3, g5, m->num_sms, st);
      }));
    } else {
    // bf16, variant 0: the shared-memory router, with the operand pair stacked along M
    // (K = d, each router weight element read once per launch); the router adds token t's
    // rows 2t and 2t + 1 of every slice
    const bool stacked = m->bf16 && m->rsm_w && c.router_variant == 0;
    int rs2 = 1;
    if (stacked) {
      const int m2 = (2 * T + 127) / 128;
      rs2 = choose_splits(m2 * ((nY + 255) / 256), (d + 63) / 64, r_sms, (long)m2 * 128, nY, 4);
      g.m_static = 2 * T;
      g.m_max = 2 * T;
      g.K = d;
      g.k_splits = 0;
      g.split_stride = 0;
      g.out_f32 = m->Y;
      g.ldo = nY;
      if (rs2 > 1) {
        // beside the FFN, FFN down's slices take splitk_ws meanwhile; rws holds any split count
        g.out_f32 = spec_shape ? m->rws : m->splitk_ws;
        g.k_splits = rs2;
        g.split_stride = (long)m2 * 128 * nY;
      }
    }
    CUDA_TRY(timed(m, HERO_K_ROUTER_GEMM, rst, [&] {
      if (stacked) return launch_gemm_tc(256, EPI_STORE_F32, m->tm_xl2, m->tm_wr1, g, r_sms, rst);
      if (!m->bf16) return launch_gemm_simt(EPI_STORE_F32, g, st);
      return pair ? launch_gemm_tc2(EPI_STORE_F32, m->tm_xl, m->tm_wr_p, g, m->num_sms, st)
                  : launch_gemm_tc(256, EPI_STORE_F32, m->tm_xl, m->tm_wr, g, m->num_sms, st);
    }));

    RouterArgs ra{};
    ra.T = T;
    ra.j = j;
    ra.L = L - c.n_dense;               // L_R
    ra.np = m->np;
    ra.d = d;
    ra.d_h = c.d_h;
    ra.d_a = c.d_a;
    ra.d_enc = c.d_enc;
    ra.d_head = c.d_head;
    ra.d_path = c.d_path;
    ra.Y = g.k_splits > 1 ? g.out_f32 : m->Y;   // the router adds split-K slices as it reads
    ra.y_splits = g.k_splits > 1 ? g.k_splits : 1;
    ra.y_split_stride = g.k_splits > 1 ? g.split_stride : 0;
    ra.y_rows = stacked ? 2 : 1;
    ra.part = m->part;
    ra.dprev = bs.dprev;
    ra.pst = bs.pst;
    ra.mst = bs.mst;
    ra.S = bs.S;
    ra.zeta = bs.zeta;
    ra.rho = m->rho[jj];
    ra.w = m->rw;
    ra.rms_eps = c.rms_eps;
    ra.eps = c.eps;
    ra.t_hist = c.t_hist;
    ra.tau = tau;
    ra.mask_in = mask_in_j;
    ra.gate = m->gate;
    ra.mask = m->mask;
    ra.gate_out = gate_out_j;
    ra.mask_out = mask_out_j;
    ra.variant = c.router_variant;
    ra.wsm = c.router_variant == 0 ? m->rsm_w : nullptr;
    ra.err = m->err;
    ra.wait_ns = wait_limit_ns();
    CUDA_TRY(timed(m, HERO_K_ROUTER, rst, [&] {
      return ra.wsm ? launch_router_sm(c.d_m, ra, r_sms, rst)
                    : launch_router(c.d_m, ra, m->num_sms, st);
    }));
    }
  }
  CompactArgs ca{T, m->mask, m->gate, dense ? 1 : 0, m->idx_f, m->idx_a, m->scale_f, m->scale_a,
                 m->counts, count_out_j, dense ? gate_out_j : nullptr,
                 dense ? mask_out_j : nullptr};
  NormArgs na{T, d, m->np, m->counts, m->idx_f, m->idx_a, hbar, m->part,
              m->ffn_gain + (size_t)jj * d, c.rms_eps, m->u_f, m->u_a, (int)m->bf16};
  if (chunk_counted) ca.chunk_cnt = m->chunk_cnt;
  if (spec) {   // compaction after the router on its stream; LN_ffn of every token here
    CUDA_TRY(timed(m, HERO_K_COMPACT, rst, [&] { return launch_compact(ca, rst); }));
    CUDA_TRY(cudaEventRecord(m->ev_join, rst));
    NormArgs nall = na;
    nall.counts = nullptr;
    CUDA_TRY(timed(m, HERO_K_NORM, st, [&] { return launch_norm(nall, m->num_sms, st); }));
  } else if (T <= kRouteNormMaxT || chunk_counted) {   // compaction inside the norm's launch
    CUDA_TRY(timed(m, HERO_K_NORM, st, [&] { return launch_route_norm(ca, na, m->num_sms, st); }));
  } else {
    CUDA_TRY(timed(m, HERO_K_COMPACT, st, [&] { return launch_compact(ca, st); }));
    CUDA_TRY(timed(m, HERO_K_NORM, st, [&] { return launch_norm(na, m->num_sms, st); }));
  }

  // FFN branch: gate/up + SwiGLU, then down + scaled scatter.  The adapter branch
  // (the other token rows): W_1 with SiLU, then W_2 + scaled scatter; on bf16
  // models each adapter GEMM rides in the FFN GEMM's launch as a second problem.
  GemmArgs gu{};
  gu.m_dev = m->counts;
  gu.m_max = T;
  gu.N = m->bf16 ? 2 * I : I;
  gu.K = d;
  gu.out = m->act;
  gu.ldo = I;
  gu.err = m->err;
  gu.A = m->u_f;
  gu.lda = d;
  gu.B = static_cast<const char*>(m->wgu) + (size_t)jj * (m->bf16 ? 2 : 1) * I * d * es;
  gu.B2 = m->bf16 ? nullptr : static_cast<const char*>(m->wup) + (size_t)jj * I * d * es;
  gu.ldb = d;
  GemmArgs ad{};
  ad.m_dev = m->counts + 1;
  ad.m_max = T;
  ad.N = r;
  ad.K = d;
  ad.out = m->ah;
  ad.ldo = r;
  ad.err = m->err;
  ad.A = spec ? m->u_f : m->u_a;
  ad.lda = d;
  if (spec) {   // every token through both branches, rows in token order
    gu.m_dev = nullptr;
    gu.m_static = T;
    ad.m_dev = nullptr;
    ad.m_static = T;
  }
  ad.B = static_cast<const char*>(m->w1) + (size_t)jj * r * d * es;
  ad.ldb = d;
  GemmArgs dn{};
  dn.m_dev = m->counts;
  dn.m_max = T;
  dn.N = d;
  dn.K = I;
  dn.err = m->err;
  dn.lo = lo;
  dn.lo.idx = m->idx_f;
  dn.lo.scale = m->scale_f;
  dn.A = m->act;
  dn.lda = I;
  dn.B = static_cast<const char*>(m->wdown) + (size_t)jj * d * I * es;
  dn.ldb = I;
  if (m->bf16) {
    GemmArgs au{};   // adapter W_2: [n_a, d_r] x [d_r, d] with the closing epilogue
    au.m_dev = m->counts + 1;
    au.m_max = T;
    au.N = d;
    au.K = r;
    au.err = m->err;
    au.lo = lo;
    au.lo.idx = m->idx_a;
    au.lo.scale = m->scale_a;
    // large batches run the FFN GEMMs on CTA pairs (256-row tiles, the 2-SM MMA)
    const bool pair = T >= kPairMinRows;
    CUDA_TRY(timed(m, HERO_K_FFN_GATE_UP, st, [&] {
      if (pair)
        return dense ? launch_gemm_tc2(EPI_SWIGLU, m->tm_uf, m->tm_wgu_p[jj], gu, m->num_sms, st)
                     : launch_gemm_tc2_pair(EPI_SWIGLU, m->tm_uf, m->tm_wgu_p[jj], gu, EPI_SILU,
                                            m->tm_ua, m->tm_w1_p[jj], ad, m->num_sms, st);
      return dense ? launch_gemm_tc(256, EPI_SWIGLU, m->tm_uf, m->tm_wgu[jj], gu, m->num_sms, st)
                   : launch_gemm_tc_pair(EPI_SWIGLU, m->tm_uf, m->tm_wgu[jj], gu, EPI_SILU,
                                         spec ? m->tm_uf : m->tm_ua, m->tm_w1[jj], ad, m->num_sms,
                                         st);
    }));
    const int m_t = m_t0;
    const int ds = ds0;
    // few rows and a split FFN down: the adapter rows close in FFN down's finishing launch
    const bool adapter_in_close = !dense && T <= 256 && r <= 64 && r % 8 == 0 && ds > 1;
    if (!dense && T <= 256 && r <= 64 && !adapter_in_close) {   // few rows: the FMA-pipe kernel
      AdapterUpArgs ua{};
      ua.m_dev = m->counts + 1;
      ua.m_max = T;
      ua.d = d;
      ua.d_r = r;
      ua.ah = m->ah;
      ua.w2 = static_cast<const char*>(m->w2) + (size_t)jj * d * r * es;
      ua.bf16 = 1;
      ua.slot_cols = kTcPartCols;
      ua.lo = au.lo;
      CUDA_TRY(timed(m, HERO_K_ADAPTER_UP, st, [&] { return launch_adapter_up(ua, st); }));
    }
    // large batches: the adapter's W_2 GEMM (wide epilogue) runs after FFN down, on the
    // SMs FFN down's last wave leaves idle (pdl_mode 1 / 2: disjoint rows, inputs from
    // the gate/up launch)
    const bool adapter_after = !dense && !(T <= 256 && r <= 64);
    auto adapter_up_wide = [&](int pdl_mode) -> hero_status {
      GemmArgs aw = au;
      aw.pdl_mode = pdl_mode;
      CUDA_TRY(timed(m, HERO_K_ADAPTER_UP, st, [&] {
        return launch_gemm_tc(256, EPI_LAYER_OUT_WIDE, m->tm_ah, m->tm_w2[jj], aw, m->num_sms, st);
      }));
      return HERO_OK;
    };
    if (ds > 1) {   // few tiles (small T): split K into partials, then the closing epilogue
      GemmArgs sk = dn;
      if (spec) {
        sk.m_dev = nullptr;
        sk.m_static = T;
      }
      sk.out_f32 = m->splitk_ws;
      sk.ldo = d;
      sk.k_splits = ds;
      sk.split_stride = (long)m_t * 128 * d;
      CUDA_TRY(timed(m, HERO_K_FFN_DOWN, st, [&] {
        return launch_gemm_tc(256, EPI_STORE_F32, m->tm_act, m->tm_wd[jj], sk, m->num_sms, st);
      }));
      if (spec) CUDA_TRY(cudaStreamWaitEvent(st, m->ev_join, 0));   // the decisions
      CUDA_TRY(timed(m, HERO_K_FFN_DOWN, st, [&] {
        SplitkAdapter sa{};
        if (adapter_in_close)
          sa = SplitkAdapter{m->ah, static_cast<const char*>(m->w2) + (size_t)jj * d * r * es, r,
                             au.lo, spec ? 1 : 0};
        return launch_splitk_close(m->splitk_ws, ds, sk.split_stride, d, m->counts, T, dn.lo, sa, st);
      }));
      return adapter_after ? adapter_up_wide(0) : HERO_OK;
    }
    GemmArgs dl = dn;
    dl.pdl_mode = adapter_after ? 1 : 0;
    CUDA_TRY(timed(m, HERO_K_FFN_DOWN, st, [&] {
      return pair ? launch_gemm_tc2(EPI_LAYER_OUT, m->tm_act, m->tm_wd_p[jj], dl, m->num_sms, st)
                  : launch_gemm_tc(256, EPI_LAYER_OUT, m->tm_act, m->tm_wd[jj], dl, m->num_sms, st);
    }));
    return adapter_after ? adapter_up_wide(2) : HERO_OK;
  }
  CUDA_TRY(timed(m, HERO_K_FFN_GATE_UP, st, [&] { return launch_gemm_simt(EPI_SWIGLU, gu, st); }));
  CUDA_TRY(timed(m, HERO_K_FFN_DOWN, st, [&] { return launch_gemm_simt(EPI_LAYER_OUT, dn, st); }));
  if (!dense) {
    CUDA_TRY(timed(m, HERO_K_ADAPTER_DOWN, st, [&] { return launch_gemm_simt(EPI_SILU, ad, st); }));
    AdapterUpArgs au{};
    au.m_dev = m->counts + 1;
    au.m_max = T;
    au.d = d;
    au.d_r = r;
    au.ah = m->ah;
    au.w2 = static_cast<const char*>(m->w2) + (size_t)jj * d * r * es;
    au.bf16 = 0;
    au.slot_cols = kSimtTileN;
    au.lo = lo;
    au.lo.idx = m->idx_a;
    au.lo.scale = m->scale_a;
    CUDA_TRY(timed(m, HERO_K_ADAPTER_UP, st, [&] { return launch_adapter_up(au, st); }));
  }
  return HERO_OK;
}

// Host-resident attention stand-in fed to the stack block by block: P_k is copied
// on the model's copy stream into device slot k % 3 and the compute stream waits
// for it just before its first reader; slot k % 3 is refilled with P_{k+3} once the
// reader of P_k has run, so uploads overlap the compute of earlier blocks.
struct PFeed {
  const char* host;     // [L, T, d] in the model's operand type
  char* slots;          // 3 device slots of one block each
  size_t layer_bytes;
  const void* h0;       // host h_0, uploaded on the copy stream ahead of P_1
  void* h0_dst;
  size_t h0_bytes;
};
constexpr int kPSlots = 3;

hero_status feed_copy(hero_model* m, const PFeed& f, int k, cudaStream_t st, bool after_consume) {
  if (after_consume) CUDA_TRY(cudaStreamWaitEvent(m->copy_stream, m->ev_consumed[k - kPSlots], 0));
  CUDA_TRY(cudaMemcpyAsync(f.slots + (size_t)(k % kPSlots) * f.layer_bytes,
                           f.host + (size_t)k * f.layer_bytes, f.layer_bytes,
                           cudaMemcpyHostToDevice, m->copy_stream));
  CUDA_TRY(cudaEventRecord(m->ev_ready[k], m->copy_stream));
  (void)st;
  return HERO_OK;
}

// The per-block launch sequence on device pointers (P device-resident, or fed
// from the host through `feed`).
hero_status run_stack(hero_model* m, int T, const float* h_in, const void* P, float tau,
                      uint32_t flags, const uint8_t* mask_in, float* h_out, float* gate_out,
                      uint8_t* mask_out, int32_t* count_out, cudaStream_t st,
                      const PFeed* feed = nullptr) {
  const hero_config& c = m->cfg;
  const int L = c.n_layers, d = c.d_model;
  const bool dense = flags & HERO_FLAG_DENSE;
  const bool force = flags & HERO_FLAG_FORCE_MASK;
  const size_t es = m->esz;
  const size_t layer_elems = (size_t)T * d;
  auto p_layer = [&](int k) -> const void* {
    if (k >= L) return nullptr;
    if (feed) return feed->slots + (size_t)(k % kPSlots) * feed->layer_bytes;
    return P ? static_cast<const char*>(P) + (size_t)k * layer_elems * es : nullptr;
  };
  if (feed) {
    // h_bar and the slots may still be read by the previous call's kernels
    CUDA_TRY(cudaStreamWaitEvent(m->copy_stream, m->ev_kernels_done, 0));
    if (feed->h0)
      CUDA_TRY(cudaMemcpyAsync(feed->h0_dst, feed->h0, feed->h0_bytes, cudaMemcpyHostToDevice,
                               m->copy_stream));
    for (int k = 0; k < L && k < kPSlots; ++k) {
      hero_status s = feed_copy(m, *feed, k, st, false);
      if (s != HERO_OK) return s;
    }
  }

  for (int jj = 0; jj < L; ++jj) {
    const void* Pj = p_layer(jj);
    const void* Pn = p_layer(jj + 1);
    if (jj == 0) {
      if (feed) CUDA_TRY(cudaStreamWaitEvent(st, m->ev_ready[0], 0));
      InitArgs ia{T, d, m->np, c.d_m, h_in, Pj, (int)m->bf16, m->hbar, m->xl, (int)m->bf16,
                  m->part, m->S, m->zeta, m->pst, m->mst, m->dprev, dense ? 0 : 1};
      CUDA_TRY(timed(m, HERO_K_INIT, st, [&] { return launch_init(ia, st); }));
      if (feed) {
        CUDA_TRY(cudaEventRecord(m->ev_consumed[0], st));
        if (kPSlots < L) {
          hero_status s = feed_copy(m, *feed, kPSlots, st, true);
          if (s != HERO_OK) return s;
        }
      }
    }
    if (feed && jj + 1 < L) CUDA_TRY(cudaStreamWaitEvent(st, m->ev_ready[jj + 1], 0));
    BlockState bs{m->S, m->zeta, m->pst, m->mst, m->dprev, m->hist};
    // layers before the routing candidate set run the plain FFN block
    const int jr = jj - c.n_dense;
    const bool dense_blk = dense || jr < 0;
    LayerOutArgs lo{};
    lo.hbar = m->hbar;
    lo.delta = m->delta;
    lo.p_next = Pn;
    lo.xl = m->xl;
    lo.part = m->part;
    lo.h_out = h_out;
    lo.d = d;
    lo.np = m->np;
    lo.last = jj == L - 1;
    lo.first = jr <= 0;                       // delta_1 = 0; no delta before routing starts
    lo.p_bf16 = m->bf16;
    lo.xl_bf16 = m->bf16;
    lo.router = (!dense && jr + 1 >= 0) ? 1 : 0;   // the next block is routed
    hero_status sb = block_body(m, jj, jr, T, bs, m->hbar, lo, tau,
                                dense_blk ? (flags & ~(uint32_t)HERO_FLAG_FORCE_MASK) | HERO_FLAG_DENSE
                                          : flags,
                                force ? mask_in + (size_t)jj * T : nullptr,
                                gate_out ? gate_out + (size_t)jj * T : nullptr,
                                mask_out ? mask_out + (size_t)jj * T : nullptr,
                                count_out ? count_out + jj : nullptr, st);
    if (sb != HERO_OK) return sb;
    if (feed && jj + 1 < L) {  // P_{jj+1} has been read: refill its slot with P_{jj+4}
      CUDA_TRY(cudaEventRecord(m->ev_consumed[jj + 1], st));
      if (jj + 1 + kPSlots < L) {
        hero_status s = feed_copy(m, *feed, jj + 1 + kPSlots, st, true);
        if (s != HERO_OK) return s;
      }
    }
  }
  CUDA_TRY(cudaEventRecord(m->ev_kernels_done, st));
  return HERO_OK;
}

}  // namespace

extern "C" hero_status hero_routed_ffn_stack(hero_model* m, int64_t n_tokens, const float* h_in,
                                             const void* attn_delta, float tau_exec,
                                             uint32_t flags, const uint8_t* mask_in, float* h_out,
                                             float* gate_out, uint8_t* mask_out,
                                             int32_t* ffn_count_out, void* cuda_stream) {
  g_last_error.clear();
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  const hero_config& c = m->cfg;
  if (n_tokens < 0 || n_tokens > c.max_tokens)
    return fail(HERO_ERR_ARG, "n_tokens %lld outside [0, max_tokens=%d]", (long long)n_tokens,
                c.max_tokens);
  if (flags & ~(uint32_t)(HERO_FLAG_DENSE | HERO_FLAG_FORCE_MASK | HERO_FLAG_HOST_IO |
                          HERO_FLAG_NO_SPECULATE))
    return fail(HERO_ERR_ARG, "unknown flag bits 0x%x", flags);
  if ((flags & HERO_FLAG_DENSE) && (flags & HERO_FLAG_FORCE_MASK))
    return fail(HERO_ERR_ARG, "HERO_FLAG_DENSE and HERO_FLAG_FORCE_MASK are exclusive");
  if ((flags & HERO_FLAG_FORCE_MASK) && !mask_in && n_tokens > 0)
    return fail(HERO_ERR_ARG, "HERO_FLAG_FORCE_MASK needs mask_in");
  if (n_tokens > 0 && (!h_in || !h_out)) return fail(HERO_ERR_ARG, "h_in and h_out are required");
  if (n_tokens > 0 && (const void*)h_in == (const void*)h_out)
    return fail(HERO_ERR_ARG, "h_out must not alias h_in");
  if (!std::isfinite(tau_exec)) return fail(HERO_ERR_ARG, "tau_exec is not finite");
  cudaError_t e0 = cudaSetDevice(m->device);
  if (e0 != cudaSuccess) return fail(HERO_ERR_CUDA, "cudaSetDevice: %s", cudaGetErrorString(e0));
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const int T = (int)n_tokens;
  const int L = c.n_layers, d = c.d_model;
  const bool host = flags & HERO_FLAG_HOST_IO;

  if (T == 0) {
    if (ffn_count_out) {
      if (host)
        memset(ffn_count_out, 0, (size_t)L * 4);
      else
        CUDA_TRY(cudaMemsetAsync(ffn_count_out, 0, (size_t)L * 4, st));
    }
    return HERO_OK;
  }
  if (!host)
    return run_stack(m, T, h_in, attn_delta, tau_exec, flags, mask_in, h_out, gate_out, mask_out,
                     ffn_count_out, st);

  // Host I/O: stage inputs on the device, run, copy outputs back on the stream.
  const size_t esz = m->esz;
  const size_t p_layer_bytes = (size_t)T * d * esz;
  const size_t p_bytes = attn_delta ? (size_t)kPSlots * p_layer_bytes : 0;   // upload ring
  const size_t lt = (size_t)L * T;
  if (attn_delta && !m->copy_stream)
    CUDA_TRY(cudaStreamCreateWithFlags(&m->copy_stream, cudaStreamNonBlocking));
  while (attn_delta && (int)m->ev_ready.size() < L) {
    cudaEvent_t a = nullptr, b = nullptr;
    CUDA_TRY(cudaEventCreateWithFlags(&a, cudaEventDisableTiming));
    CUDA_TRY(cudaEventCreateWithFlags(&b, cudaEventDisableTiming));
    m->ev_ready.push_back(a);
    m->ev_consumed.push_back(b);
  }
  const size_t need = (size_t)T * d * 4 /*h_out*/ + p_bytes + lt /*mask_in*/ + lt * 4 /*gate*/ +
                      lt /*mask*/ + (size_t)L * 4 + 4096;
  hero_status s = ensure_io(m, need);
  if (s != HERO_OK) return s;
  char* p = static_cast<char*>(m->io);
  auto carve = [&](size_t bytes) {
    char* q = p;
    p += (bytes + 255) & ~(size_t)255;
    return q;
  };
  float* d_hout = reinterpret_cast<float*>(carve((size_t)T * d * 4));
  void* d_P = attn_delta ? carve(p_bytes) : nullptr;
  uint8_t* d_mask_in = (flags & HERO_FLAG_FORCE_MASK) ? reinterpret_cast<uint8_t*>(carve(lt)) : nullptr;
  float* d_gate = gate_out ? reinterpret_cast<float*>(carve(lt * 4)) : nullptr;
  uint8_t* d_mask = mask_out ? reinterpret_cast<uint8_t*>(carve(lt)) : nullptr;
  int32_t* d_cnt = ffn_count_out ? reinterpret_cast<int32_t*>(carve((size_t)L * 4)) : nullptr;
  // h_0 goes straight into the h_bar buffer (k_init adds P_1 in place): on the copy
  // stream ahead of P_1 when P is streamed, else on the compute stream.
  if (!attn_delta) CUDA_TRY(cudaMemcpyAsync(m->hbar, h_in, (size_t)T * d * 4, cudaMemcpyHostToDevice, st));
  if (d_mask_in) CUDA_TRY(cudaMemcpyAsync(d_mask_in, mask_in, lt, cudaMemcpyHostToDevice, st));
  PFeed feed{static_cast<const char*>(attn_delta), static_cast<char*>(d_P), p_layer_bytes,
             h_in, m->hbar, (size_t)T * d * 4};
  s = run_stack(m, T, m->hbar, nullptr, tau_exec, flags, d_mask_in, d_hout, d_gate, d_mask, d_cnt,
                st, attn_delta ? &feed : nullptr);
  if (s != HERO_OK) return s;
  CUDA_TRY(cudaMemcpyAsync(h_out, d_hout, (size_t)T * d * 4, cudaMemcpyDeviceToHost, st));
  if (d_gate) CUDA_TRY(cudaMemcpyAsync(gate_out, d_gate, lt * 4, cudaMemcpyDeviceToHost, st));
  if (d_mask) CUDA_TRY(cudaMemcpyAsync(mask_out, d_mask, lt, cudaMemcpyDeviceToHost, st));
  if (d_cnt) CUDA_TRY(cudaMemcpyAsync(ffn_count_out, d_cnt, (size_t)L * 4, cudaMemcpyDeviceToHost, st));
  return HERO_OK;
}

extern "C" hero_status hero_router_state_reset(hero_model* m, int64_t n_tokens,
                                               const hero_router_state* s, void* cuda_stream) {
  g_last_error.clear();
  if (!m || !s) return fail(HERO_ERR_ARG, "model or state is NULL");
  if (n_tokens < 0 || n_tokens > m->cfg.max_tokens)
    return fail(HERO_ERR_ARG, "n_tokens %lld outside [0, max_tokens=%d]", (long long)n_tokens,
                m->cfg.max_tokens);
  if (n_tokens > 0 && (!s->S || !s->zeta || !s->p_hist || !s->m_hist || !s->d_prev))
    return fail(HERO_ERR_ARG, "state pointers S, zeta, p_hist, m_hist and d_prev are required");
  CUDA_TRY(cudaSetDevice(m->device));
  CUDA_TRY(launch_state_reset(s->S, s->zeta, s->p_hist, s->m_hist, s->d_prev, (int)n_tokens,
                              m->cfg.d_m, static_cast<cudaStream_t>(cuda_stream)));
  return HERO_OK;
}

namespace {

// One block on post-attention states h_bar (layer jj, the caller's router state
// and carried h_bar_prev / delta_prev): block entry (delta, partial sums, router
// operand), then block_body writing h_out.  Arguments already validated.
hero_status routed_block_run(hero_model* m, int jj, int T, const float* h_bar, const BlockState& bs,
                             float* h_bar_prev, float* delta_prev, float tau, uint32_t flags,
                             const uint8_t* mask_in, float* h_out, float* gate_out,
                             uint8_t* mask_out, int32_t* count_out, cudaStream_t st,
                             bool entry_done = false) {
  const hero_config& c = m->cfg;
  const int jr = jj - c.n_dense;
  bool dense = flags & HERO_FLAG_DENSE;
  if (jr < 0) {   // outside the routing candidate set: the plain FFN block
    dense = true;
    flags = (flags & ~(uint32_t)HERO_FLAG_FORCE_MASK) | HERO_FLAG_DENSE;
  }
  BlockEntryArgs be{T, c.d_model, m->np, jr + 1, dense ? 0 : 1, h_bar,
                    dense ? nullptr : h_bar_prev, dense ? nullptr : delta_prev,
                    m->xl, (int)m->bf16, m->part};
  if (!entry_done)   // else the producer of h_bar closed into the entry (EPI_ATTN_ENTRY)
    CUDA_TRY(timed(m, HERO_K_INIT, st, [&] { return launch_block_entry(be, st); }));
  LayerOutArgs lo{};
  lo.hbar = const_cast<float*>(h_bar);  // read only: the block writes h_out
  lo.h_out = h_out;
  lo.part = m->part;
  lo.d = c.d_model;
  lo.np = m->np;
  lo.last = 1;
  lo.first = jr <= 0;
  lo.p_bf16 = m->bf16;
  lo.xl_bf16 = m->bf16;
  lo.router = 0;
  return block_body(m, jj, jr, T, dense ? BlockState{nullptr, nullptr, nullptr, nullptr, nullptr, nullptr} : bs,
                    h_bar, lo, tau, flags, (flags & HERO_FLAG_FORCE_MASK) ? mask_in : nullptr,
                    gate_out, mask_out, count_out, st);
}

// RoPE (cos, sin) of s * theta^(-2i/128) for positions s < rows, computed in double.
hero_status build_rope_table(hero_model* m, long rows) {
  if (rows <= m->rope_rows) return HERO_OK;
  std::vector<float> cs((size_t)rows * 64 * 2);
  for (long p = 0; p < rows; ++p)
    for (int i = 0; i < 64; ++i) {
      const double ang = (double)p * std::pow((double)m->rope_theta, -2.0 * i / 128.0);
      cs[((size_t)p * 64 + i) * 2] = (float)std::cos(ang);
      cs[((size_t)p * 64 + i) * 2 + 1] = (float)std::sin(ang);
    }
  CUDA_TRY(cudaDeviceSynchronize());   // the old table may be in use
  if (m->rope_cs) cudaFree(m->rope_cs);
  m->rope_cs = nullptr;
  m->rope_rows = 0;
  CUDA_TRY(cudaMalloc(&m->rope_cs, cs.size() * 4));
  CUDA_TRY(cudaMemcpy(m->rope_cs, cs.data(), cs.size() * 4, cudaMemcpyHostToDevice));
  m->rope_rows = rows;
  return HERO_OK;
}

// Where a sublayer's keys and values go: the workspace (nullptr) or a cache range.
struct KvTarget {
  void* k;
  void* v;
  int stride;   // positions per (sequence, head) slab
};

// Eq. 1, first line, for layer jj on B sequences of S tokens: h_bar = h + Attn(LN_attn(h)).
// With `entry`, the output projection also closes into the routed block's entry
// (h_bar written over entry->hbar = h_bar_{j-1}, delta, router operand, partials).
hero_status attention_run(hero_model* m, int jj, int B, int S, const float* h, float* h_bar,
                          cudaStream_t st, const LayerOutArgs* entry = nullptr,
                          const KvTarget* kv = nullptr) {
  const hero_config& c = m->cfg;
  const int T = B * S, d = c.d_model, H = m->n_heads, Hkv = m->n_kv_heads;
  const int nqkv = (H + 2 * Hkv) * 128;
  CUDA_TRY(timed(m, HERO_K_ATTN_PROJ, st, [&] {
    return launch_attn_norm(h, m->attn_gain + (size_t)jj * d, T, d, c.rms_eps, m->ax, st);
  }));
  GemmArgs g{};
  g.m_static = T;
  g.m_max = T;
  g.N = nqkv;
  g.K = d;
  g.ldo = nqkv;
  g.err = m->err;
  const KvTarget kt = kv ? *kv : KvTarget{m->ak, m->av, S};
  // sequences of 128 or more run the tensor-core attention, which reads v transposed
  const int S_pad = (S + 63) / 64 * 64;
  const bool tc = S >= 128 && (size_t)B * Hkv * 128 * S_pad <= m->avt_elems;
  g.rope = RopeArgs{m->aq, kt.k, (kv || !tc) ? kt.v : nullptr, m->rope_cs, nullptr, H, Hkv, S, S,
                    kt.stride, tc ? m->avt : nullptr, S_pad};
  const bool pair = T >= kPairMinRows;   // large token counts: CTA-pair tiles
  CUDA_TRY(timed(m, HERO_K_ATTN_PROJ, st, [&] {   // q, k, v with RoPE, attention layout
    return pair ? launch_gemm_tc2(EPI_QKV_ROPE, m->tm_ax, m->tm_wqkv_p[jj], g, m->num_sms, st)
                : launch_gemm_tc(256, EPI_QKV_ROPE, m->tm_ax, m->tm_wqkv[jj], g, m->num_sms, st);
  }));
  CUDA_TRY(timed(m, HERO_K_ATTN_CORE, st, [&] {
    if (tc) {
      CUtensorMap tq, tk, tv;
      if (!encode_bf16_3d(&tq, m->aq, 128, S, (uint64_t)B * H, 256, (uint64_t)S * 256) ||
          !encode_bf16_3d(&tk, kt.k, 128, S, (uint64_t)B * Hkv, 256, (uint64_t)kt.stride * 256) ||
          !encode_bf16_3d(&tv, m->avt, S, 128, (uint64_t)B * Hkv, (uint64_t)S_pad * 2,
                          (uint64_t)S_pad * 256))
        return cudaErrorInvalidValue;
      return launch_flash_tc(tq, tk, tv, B, S, H, Hkv, m->ao, m->err, st);
    }
    return launch_flash_attn(m->aq, kt.k, kt.v, B, S, H, Hkv, kt.stride, m->ao, st);
  }));
  GemmArgs o{};
  o.m_static = T;
  o.m_max = T;
  o.N = d;
  o.K = H * 128;
  o.out_f32 = h_bar;
  o.ldo = d;
  o.resid = h;
  o.err = m->err;
  if (entry) o.lo = *entry;
  CUDA_TRY(timed(m, HERO_K_ATTN_PROJ, st, [&] {
    const EpiKind e = entry ? EPI_ATTN_ENTRY : EPI_RESIDUAL;
    return pair ? launch_gemm_tc2(e, m->tm_ao, m->tm_wo_p[jj], o, m->num_sms, st)
                : launch_gemm_tc(256, e, m->tm_ao, m->tm_wo[jj], o, m->num_sms, st);
  }));
  return HERO_OK;
}

}  // namespace

extern "C" hero_status hero_routed_block(hero_model* m, int32_t block, int64_t n_tokens,
                                         const float* h_bar, const hero_router_state* s,
                                         float tau_exec, uint32_t flags, const uint8_t* mask_in,
                                         float* h_out, float* gate_out, uint8_t* mask_out,
                                         int32_t* ffn_count_out, void* cuda_stream) {
  g_last_error.clear();
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  const hero_config& c = m->cfg;
  if (block < 1 || block > c.n_layers)
    return fail(HERO_ERR_ARG, "block %d outside [1, %d]", block, c.n_layers);
  if (n_tokens < 0 || n_tokens > c.max_tokens)
    return fail(HERO_ERR_ARG, "n_tokens %lld outside [0, max_tokens=%d]", (long long)n_tokens,
                c.max_tokens);
  if (flags & ~(uint32_t)(HERO_FLAG_DENSE | HERO_FLAG_FORCE_MASK | HERO_FLAG_NO_SPECULATE))
    return fail(HERO_ERR_ARG, "hero_routed_block takes only HERO_FLAG_DENSE, HERO_FLAG_FORCE_MASK "
                              "or HERO_FLAG_NO_SPECULATE");
  if ((flags & HERO_FLAG_DENSE) && (flags & HERO_FLAG_FORCE_MASK))
    return fail(HERO_ERR_ARG, "HERO_FLAG_DENSE and HERO_FLAG_FORCE_MASK are exclusive");
  bool dense = (flags & HERO_FLAG_DENSE) || block <= c.n_dense;
  if (!std::isfinite(tau_exec)) return fail(HERO_ERR_ARG, "tau_exec is not finite");
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  if (n_tokens == 0) {
    CUDA_TRY(cudaSetDevice(m->device));
    if (ffn_count_out) CUDA_TRY(cudaMemsetAsync(ffn_count_out, 0, 4, st));
    return HERO_OK;
  }
  if (!h_bar || !h_out) return fail(HERO_ERR_ARG, "h_bar and h_out are required");
  if ((const void*)h_bar == (const void*)h_out) return fail(HERO_ERR_ARG, "h_out must not alias h_bar");
  if ((flags & HERO_FLAG_FORCE_MASK) && !mask_in)
    return fail(HERO_ERR_ARG, "HERO_FLAG_FORCE_MASK needs mask_in");
  if (!dense && (!s || !s->S || !s->zeta || !s->p_hist || !s->m_hist || !s->d_prev ||
                 !s->h_bar_prev || !s->delta_prev))
    return fail(HERO_ERR_ARG, "the router state needs all seven pointers");
  CUDA_TRY(cudaSetDevice(m->device));
  const BlockState bs = dense ? BlockState{nullptr, nullptr, nullptr, nullptr, nullptr, nullptr}
                              : BlockState{s->S, s->zeta, s->p_hist, s->m_hist, s->d_prev, nullptr};
  const hero_status sb =
      routed_block_run(m, block - 1, (int)n_tokens, h_bar, bs, dense ? nullptr : s->h_bar_prev,
                       dense ? nullptr : s->delta_prev, tau_exec, flags, mask_in, h_out, gate_out,
                       mask_out, ffn_count_out, st);
  if (sb != HERO_OK) return sb;
  CUDA_TRY(cudaEventRecord(m->ev_kernels_done, st));
  return HERO_OK;
}

extern "C" hero_status hero_attn_init(hero_model* m, const hero_attn_config* ac,
                                      const hero_attn_weights_host* w) {
  g_last_error.clear();
  if (!m || !ac || !w) return fail(HERO_ERR_ARG, "model, config and weights are required");
  if (m->attn) return fail(HERO_ERR_ARG, "the model already has its attention parameters");
  if (!m->bf16) return fail(HERO_ERR_UNSUPPORTED, "the attention sublayer needs a bf16 model");
  const hero_config& c = m->cfg;
  const long L = c.n_layers, d = c.d_model, H = ac->n_heads, Hkv = ac->n_kv_heads;
  if (H < 1 || Hkv < 1 || H % Hkv) return fail(HERO_ERR_ARG, "need H >= 1, H_kv >= 1, H_kv | H");
  if (d != 128 * H) return fail(HERO_ERR_UNSUPPORTED, "head dimension must be 128 (d = 128 H)");
  if (!(ac->rope_theta > 1.f)) return fail(HERO_ERR_ARG, "rope_theta must be > 1");
  if (!w->attn_norm_g || !w->w_q || !w->w_k || !w->w_v || !w->w_o)
    return fail(HERO_ERR_ARG, "an attention weight pointer is NULL");
  if (w->host_dtype != HERO_F32 && w->host_dtype != HERO_BF16)
    return fail(HERO_ERR_ARG, "unknown host_dtype");
  CUDA_TRY(cudaSetDevice(m->device));
  const long nqkv = (H + 2 * Hkv) * 128, Tm = c.max_tokens;
  const size_t hes = w->host_dtype == HERO_BF16 ? 2 : 4;
  CUDA_TRY(cudaMalloc(&m->wqkv, (size_t)L * nqkv * d * 2));
  CUDA_TRY(cudaMalloc(&m->wo, (size_t)L * d * d * 2));
  CUDA_TRY(cudaMalloc(&m->attn_gain, (size_t)L * d * 4));
  const size_t stage_elems = (size_t)16 << 20;
  void* stage = nullptr;
  CUDA_TRY(cudaMalloc(&stage, stage_elems * 4));
  hero_status st = HERO_OK;
  for (long j = 0; j < L && st == HERO_OK; ++j) {
    char* q = static_cast<char*>(m->wqkv) + (size_t)j * nqkv * d * 2;
    st = upload_rows(m, static_cast<const char*>(w->w_q) + (size_t)j * H * 128 * d * hes,
                     w->host_dtype, q, H * 128, d, 1, 1, 0, nullptr, stage, stage_elems);
    if (st == HERO_OK)
      st = upload_rows(m, static_cast<const char*>(w->w_k) + (size_t)j * Hkv * 128 * d * hes,
                       w->host_dtype, q, Hkv * 128, d, 1, 1, H * 128, nullptr, stage, stage_elems);
    if (st == HERO_OK)
      st = upload_rows(m, static_cast<const char*>(w->w_v) + (size_t)j * Hkv * 128 * d * hes,
                       w->host_dtype, q, Hkv * 128, d, 1, 1, (H + Hkv) * 128, nullptr, stage,
                       stage_elems);
    if (st == HERO_OK)
      st = upload_rows(m, static_cast<const char*>(w->w_o) + (size_t)j * d * d * hes, w->host_dtype,
                       static_cast<char*>(m->wo) + (size_t)j * d * d * 2, d, d, 1, 1, 0, nullptr,
                       stage, stage_elems);
  }
  cudaFree(stage);
  if (st != HERO_OK) return st;
  std::vector<float> gains = host_f32(w->attn_norm_g, (size_t)L * d, w->host_dtype);
  CUDA_TRY(cudaMemcpy(m->attn_gain, gains.data(), gains.size() * 4, cudaMemcpyHostToDevice));
  // workspace: x and o (bf16 [T,d]), the RoPE table, Q/K/V (bf16), the decoder's current
  // h and its carried delta (fp32 [T,d]; h_bar_{j-1} is carried in the model's h_bar)
  struct Item {
    void** p;
    size_t bytes;
  };
  // v transposed: sequences of S >= 128 padded to a multiple of 64 positions
  const size_t avt_elems = (size_t)Hkv * 128 * (size_t)(Tm + 63 * (Tm / 128) + 64);
  std::vector<Item> items = {
      {&m->ax, (size_t)Tm * d * 2},          {&m->ao, (size_t)Tm * d * 2},
      {&m->aq, (size_t)Tm * H * 128 * 2},
      {&m->ak, (size_t)Tm * Hkv * 128 * 2},  {&m->av, (size_t)Tm * Hkv * 128 * 2},
      {(void**)&m->hcur, (size_t)Tm * d * 4},
      {&m->avt, avt_elems * 2},
      {(void**)&m->dlprev, (size_t)Tm * d * 4}};
  size_t off = 0;
  for (auto& it : items) off += (it.bytes + 1023) & ~(size_t)1023;
  CUDA_TRY(cudaMalloc(&m->aws, off));
  off = 0;
  for (auto& it : items) {
    *it.p = static_cast<char*>(m->aws) + off;
    off += (it.bytes + 1023) & ~(size_t)1023;
  }
  m->rope_theta = ac->rope_theta;
  if (hero_status rs = build_rope_table(m, Tm); rs != HERO_OK) return rs;
  bool ok = encode_bf16_2d(&m->tm_ax, m->ax, d, Tm, 128) && encode_bf16_2d(&m->tm_ao, m->ao, d, Tm, 128);
  m->tm_wqkv.resize(L);
  m->tm_wo.resize(L);
  m->tm_wqkv_p.resize(L);
  m->tm_wo_p.resize(L);
  for (long j = 0; j < L && ok; ++j) {
    const char* wqkv_j = static_cast<char*>(m->wqkv) + (size_t)j * nqkv * d * 2;
    const char* wo_j = static_cast<char*>(m->wo) + (size_t)j * d * d * 2;
    ok = encode_bf16_2d(&m->tm_wqkv[j], wqkv_j, d, nqkv, 256) &&
         encode_bf16_2d(&m->tm_wo[j], wo_j, d, d, 256) &&
         encode_bf16_2d(&m->tm_wqkv_p[j], wqkv_j, d, nqkv, 128) &&
         encode_bf16_2d(&m->tm_wo_p[j], wo_j, d, d, 128);
  }
  if (!ok) return fail(HERO_ERR_CUDA, "tensor map encoding failed");
  m->n_heads = (int)H;
  m->n_kv_heads = (int)Hkv;
  m->avt_elems = avt_elems;
  m->attn = true;
  return HERO_OK;
}

extern "C" hero_status hero_attention_block(hero_model* m, int32_t layer, int32_t n_seqs,
                                            int32_t seq_len, const float* h, float* h_bar,
                                            void* cuda_stream) {
  g_last_error.clear();
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  if (!m->attn) return fail(HERO_ERR_ARG, "hero_attn_init has not been called");
  const hero_config& c = m->cfg;
  if (layer < 1 || layer > c.n_layers)
    return fail(HERO_ERR_ARG, "layer %d outside [1, %d]", layer, c.n_layers);
  if (n_seqs < 0 || n_seqs > 65535 || seq_len < 1 || (long)n_seqs * seq_len > c.max_tokens)
    return fail(HERO_ERR_ARG, "n_seqs x seq_len outside [0, max_tokens=%d] (n_seqs <= 65535)",
                c.max_tokens);
  if (n_seqs == 0) return HERO_OK;
  if (!h || !h_bar) return fail(HERO_ERR_ARG, "h and h_bar are required");
  if ((const void*)h == (const void*)h_bar) return fail(HERO_ERR_ARG, "h_bar must not alias h");
  CUDA_TRY(cudaSetDevice(m->device));
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const hero_status s = attention_run(m, layer - 1, n_seqs, seq_len, h, h_bar, st);
  if (s != HERO_OK) return s;
  CUDA_TRY(cudaEventRecord(m->ev_kernels_done, st));
  return HERO_OK;
}

namespace {

// The block entry that the output projection closes into (Eq. 7 bookkeeping).
LayerOutArgs entry_args(hero_model* m, int jj, uint32_t flags) {
  const int jr = jj - m->cfg.n_dense;
  LayerOutArgs entry{};
  entry.hbar = m->hbar;
  entry.delta = m->dlprev;
  entry.xl = m->xl;
  entry.part = m->part;
  entry.d = m->cfg.d_model;
  entry.np = m->np;
  entry.first = jr <= 0;
  entry.xl_bf16 = 1;
  entry.router = ((flags & HERO_FLAG_DENSE) || jr < 0) ? 0 : 1;
  return entry;
}

// Eq. 1 for one new token per cache slot b < B at position pos[b] (decoding step).
hero_status attention_decode_run(hero_model* m, int jj, int B, const int* pos, int max_pos,
                                 const float* h, cudaStream_t st, const LayerOutArgs& entry) {
  const hero_config& c = m->cfg;
  const int d = c.d_model, H = m->n_heads, Hkv = m->n_kv_heads;
  CUDA_TRY(timed(m, HERO_K_ATTN_PROJ, st, [&] {
    return launch_attn_norm(h, m->attn_gain + (size_t)jj * d, B, d, c.rms_eps, m->ax, st);
  }));
  GemmArgs g{};
  g.m_static = B;
  g.m_max = B;
  g.N = (H + 2 * Hkv) * 128;
  g.K = d;
  g.ldo = g.N;
  g.err = m->err;
  g.rope = RopeArgs{m->aq, m->kv_k(jj), m->kv_v(jj), m->rope_cs, pos, H, Hkv, 1, 1, m->kv_len};
  // few tiles at decoding sizes: split K so that every SM streams weights
  const int m_t = (B + 127) / 128;
  const long rows = (long)m_t * 128;
  auto splits_for = [&](int n, int epi_bytes) {
    int sp = choose_splits(m_t * ((n + 255) / 256), (d + 63) / 64, m->num_sms, rows, n, epi_bytes);
    while (sp > 1 && (size_t)sp * rows * n > m->dec_ws_floats) --sp;
    return sp;
  };
  const int qs = splits_for(g.N, 4);
  if (qs > 1) {
    GemmArgs sk = g;
    sk.out_f32 = m->dec_ws;
    sk.k_splits = qs;
    sk.split_stride = rows * g.N;
    CUDA_TRY(timed(m, HERO_K_ATTN_PROJ, st, [&] {
      return launch_gemm_tc(256, EPI_STORE_F32, m->tm_ax, m->tm_wqkv[jj], sk, m->num_sms, st);
    }));
    CUDA_TRY(timed(m, HERO_K_ATTN_PROJ, st, [&] {   // RoPE; q; k and v into the cache
      return launch_qkv_close(m->dec_ws, qs, sk.split_stride, B, g.rope, m->err, st);
    }));
  } else {
    CUDA_TRY(timed(m, HERO_K_ATTN_PROJ, st, [&] {   // q; k and v into the cache
      return launch_gemm_tc(256, EPI_QKV_ROPE, m->tm_ax, m->tm_wqkv[jj], g, m->num_sms, st);
    }));
  }
  CUDA_TRY(timed(m, HERO_K_ATTN_CORE, st, [&] {
    return launch_attn_decode(m->aq, m->kv_k(jj), m->kv_v(jj), pos, B, H, Hkv, m->kv_len, max_pos,
                              m->dec_pm, m->dec_pl, m->dec_po, m->ao, m->err, st);
  }));
  GemmArgs o{};
  o.m_static = B;
  o.m_max = B;
  o.N = d;
  o.K = H * 128;
  o.ldo = d;
  o.resid = h;
  o.err = m->err;
  o.lo = entry;
  const int os = splits_for(d, 22);
  if (os > 1) {
    GemmArgs sk = o;
    sk.out_f32 = m->dec_ws;
    sk.k_splits = os;
    sk.split_stride = rows * d;
    CUDA_TRY(timed(m, HERO_K_ATTN_PROJ, st, [&] {
      return launch_gemm_tc(256, EPI_STORE_F32, m->tm_ao, m->tm_wo[jj], sk, m->num_sms, st);
    }));
    CUDA_TRY(timed(m, HERO_K_ATTN_PROJ, st, [&] {
      return launch_entry_close(m->dec_ws, os, sk.split_stride, B, h, entry, st);
    }));
    return HERO_OK;
  }
  CUDA_TRY(timed(m, HERO_K_ATTN_PROJ, st, [&] {
    return launch_gemm_tc(256, EPI_ATTN_ENTRY, m->tm_ao, m->tm_wo[jj], o, m->num_sms, st);
  }));
  return HERO_OK;
}

// The decoder forward on device buffers (h_in may be m->hcur: layer 1 reads it into
// h_bar before anything writes hcur).  seq0 >= 0: the sequences are cache slots
// seq0.. and every layer's keys and values go there.  pos != nullptr: a decoding
// step (one token per cache slot, n_seqs tokens at positions pos, seq_len 1).
hero_status decoder_run(hero_model* m, int n_seqs, int seq_len, const float* h_in, float tau_exec,
                        uint32_t flags, const uint8_t* mask_in, float* h_out, float* gate_out,
                        uint8_t* mask_out, int32_t* ffn_count_out, cudaStream_t st, int seq0 = -1,
                        const int* pos = nullptr, int max_pos = 0) {
  const hero_config& c = m->cfg;
  const int L = c.n_layers, T = n_seqs * seq_len;
  if (!(flags & HERO_FLAG_DENSE))
    CUDA_TRY(launch_state_reset(m->S, m->zeta, m->pst, m->mst, m->dprev, T, c.d_m, st));
  const BlockState bs{m->S, m->zeta, m->pst, m->mst, m->dprev, m->hist};
  const float* h = h_in;
  for (int jj = 0; jj < L; ++jj) {
    // Eq. 1 with the block entry fused into the output projection: m->hbar carries
    // h_bar_{j-1} into the launch and h_bar_j out of it, m->dlprev likewise delta
    const LayerOutArgs entry = entry_args(m, jj, flags);
    hero_status s;
    if (pos) {
      s = attention_decode_run(m, jj, n_seqs, pos, max_pos, h, st, entry);
    } else if (seq0 >= 0) {
      const size_t off = (size_t)seq0 * m->n_kv_heads * m->kv_len * 128;
      const KvTarget kt{m->kv_k(jj) + off, m->kv_v(jj) + off, m->kv_len};
      s = attention_run(m, jj, n_seqs, seq_len, h, m->hbar, st, &entry, &kt);
    } else {
      s = attention_run(m, jj, n_seqs, seq_len, h, m->hbar, st, &entry);
    }
    if (s != HERO_OK) return s;
    float* out = jj == L - 1 ? h_out : m->hcur;
    s = routed_block_run(m, jj, T, m->hbar, bs, nullptr, m->dlprev, tau_exec, flags,
                         mask_in ? mask_in + (size_t)jj * T : nullptr, out,
                         gate_out ? gate_out + (size_t)jj * T : nullptr,
                         mask_out ? mask_out + (size_t)jj * T : nullptr,
                         ffn_count_out ? ffn_count_out + jj : nullptr, st, true);
    if (s != HERO_OK) return s;
    h = out;
  }
  CUDA_TRY(cudaEventRecord(m->ev_kernels_done, st));
  return HERO_OK;
}

// Argument checks shared by the decoder entry points (T tokens).  T == 0 is
// handled here: ffn_count_out is zeroed and nothing else happens.
hero_status check_decoder_args(hero_model* m, int T, const float* h_in, float tau_exec,
                               uint32_t flags, const uint8_t* mask_in, const float* h_out,
                               int32_t* ffn_count_out, void* cuda_stream) {
  const int L = m->cfg.n_layers;
  if (flags & ~(uint32_t)(HERO_FLAG_DENSE | HERO_FLAG_FORCE_MASK | HERO_FLAG_HOST_IO |
                          HERO_FLAG_NO_SPECULATE))
    return fail(HERO_ERR_ARG, "unknown flag bits 0x%x", flags);
  if ((flags & HERO_FLAG_DENSE) && (flags & HERO_FLAG_FORCE_MASK))
    return fail(HERO_ERR_ARG, "HERO_FLAG_DENSE and HERO_FLAG_FORCE_MASK are exclusive");
  if (!std::isfinite(tau_exec)) return fail(HERO_ERR_ARG, "tau_exec is not finite");
  CUDA_TRY(cudaSetDevice(m->device));
  if (T == 0) {
    if (ffn_count_out) {
      if (flags & HERO_FLAG_HOST_IO)
        memset(ffn_count_out, 0, (size_t)L * 4);
      else
        CUDA_TRY(cudaMemsetAsync(ffn_count_out, 0, (size_t)L * 4,
                                 static_cast<cudaStream_t>(cuda_stream)));
    }
    return HERO_OK;
  }
  if (!h_in || !h_out) return fail(HERO_ERR_ARG, "h_in and h_out are required");
  if ((const void*)h_in == (const void*)h_out) return fail(HERO_ERR_ARG, "h_out must not alias h_in");
  if ((flags & HERO_FLAG_FORCE_MASK) && !mask_in)
    return fail(HERO_ERR_ARG, "HERO_FLAG_FORCE_MASK needs mask_in");
  return HERO_OK;
}

// Run decoder_run on device buffers, staging host buffers first with HERO_FLAG_HOST_IO
// (h_0 straight into the decoder's running-h buffer, the decoding step's positions
// into the model's position buffer, outputs through the I/O area).
hero_status decoder_io(hero_model* m, int n_seqs, int seq_len, int seq0, const int* pos, int max_pos,
                       const float* h_in, float tau_exec, uint32_t flags, const uint8_t* mask_in,
                       float* h_out, float* gate_out, uint8_t* mask_out, int32_t* ffn_count_out,
                       cudaStream_t st) {
  const int L = m->cfg.n_layers, d = m->cfg.d_model, T = n_seqs * seq_len;
  const bool host = flags & HERO_FLAG_HOST_IO;
  flags &= ~(uint32_t)HERO_FLAG_HOST_IO;
  if (!host)
    return decoder_run(m, n_seqs, seq_len, h_in, tau_exec, flags, mask_in, h_out, gate_out,
                       mask_out, ffn_count_out, st, seq0, pos, max_pos);
  const size_t lt = (size_t)L * T;
  const size_t need = (size_t)T * d * 4 + lt /*mask_in*/ + lt * 4 + lt + (size_t)L * 4 + 4096;
  hero_status s = ensure_io(m, need);
  if (s != HERO_OK) return s;
  char* p = static_cast<char*>(m->io);
  auto carve = [&](size_t bytes) {
    char* q = p;
    p += (bytes + 255) & ~(size_t)255;
    return q;
  };
  float* d_hout = reinterpret_cast<float*>(carve((size_t)T * d * 4));
  uint8_t* d_mask_in = (flags & HERO_FLAG_FORCE_MASK) ? reinterpret_cast<uint8_t*>(carve(lt)) : nullptr;
  float* d_gate = gate_out ? reinterpret_cast<float*>(carve(lt * 4)) : nullptr;
  uint8_t* d_mask = mask_out ? reinterpret_cast<uint8_t*>(carve(lt)) : nullptr;
  int32_t* d_cnt = ffn_count_out ? reinterpret_cast<int32_t*>(carve((size_t)L * 4)) : nullptr;
  CUDA_TRY(cudaMemcpyAsync(m->hcur, h_in, (size_t)T * d * 4, cudaMemcpyHostToDevice, st));
  if (d_mask_in) CUDA_TRY(cudaMemcpyAsync(d_mask_in, mask_in, lt, cudaMemcpyHostToDevice, st));
  if (pos) {
    CUDA_TRY(cudaMemcpyAsync(m->dec_pos, pos, (size_t)n_seqs * 4, cudaMemcpyHostToDevice, st));
    pos = m->dec_pos;
  }
  s = decoder_run(m, n_seqs, seq_len, m->hcur, tau_exec, flags, d_mask_in, d_hout, d_gate, d_mask,
                  d_cnt, st, seq0, pos, max_pos);
  if (s != HERO_OK) return s;
  CUDA_TRY(cudaMemcpyAsync(h_out, d_hout, (size_t)T * d * 4, cudaMemcpyDeviceToHost, st));
  if (d_gate) CUDA_TRY(cudaMemcpyAsync(gate_out, d_gate, lt * 4, cudaMemcpyDeviceToHost, st));
  if (d_mask) CUDA_TRY(cudaMemcpyAsync(mask_out, d_mask, lt, cudaMemcpyDeviceToHost, st));
  if (d_cnt) CUDA_TRY(cudaMemcpyAsync(ffn_count_out, d_cnt, (size_t)L * 4, cudaMemcpyDeviceToHost, st));
  return HERO_OK;
}

}  // namespace

extern "C" hero_status hero_decoder_forward(hero_model* m, int32_t n_seqs, int32_t seq_len,
                                            const float* h_in, float tau_exec, uint32_t flags,
                                            const uint8_t* mask_in, float* h_out, float* gate_out,
                                            uint8_t* mask_out, int32_t* ffn_count_out,
                                            void* cuda_stream) {
  g_last_error.clear();
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  if (!m->attn) return fail(HERO_ERR_ARG, "hero_attn_init has not been called");
  const hero_config& c = m->cfg;
  if (n_seqs < 0 || n_seqs > 65535 || seq_len < 1 || (long)n_seqs * seq_len > c.max_tokens)
    return fail(HERO_ERR_ARG, "n_seqs x seq_len outside [0, max_tokens=%d] (n_seqs <= 65535)",
                c.max_tokens);
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  hero_status s = check_decoder_args(m, n_seqs * seq_len, h_in, tau_exec, flags, mask_in, h_out,
                                     ffn_count_out, cuda_stream);
  if (s != HERO_OK || n_seqs == 0) return s;
  return decoder_io(m, n_seqs, seq_len, -1, nullptr, 0, h_in, tau_exec, flags, mask_in, h_out,
                    gate_out, mask_out, ffn_count_out, st);
}

extern "C" hero_status hero_kv_cache_init(hero_model* m, int32_t max_seqs, int32_t max_len) {
  g_last_error.clear();
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  if (!m->attn) return fail(HERO_ERR_ARG, "hero_attn_init has not been called");
  if (m->kv) return fail(HERO_ERR_ARG, "the model already has a KV cache");
  if (max_seqs < 1 || max_seqs > 65535 || max_len < 1)
    return fail(HERO_ERR_ARG, "need 1 <= max_seqs <= 65535 and max_len >= 1");
  {
    const int G = m->n_heads / m->n_kv_heads;   // query heads per key/value head
    if (G != 1 && G != 2 && G != 4 && G != 8)
      return fail(HERO_ERR_UNSUPPORTED, "decoding needs 1, 2, 4 or 8 query heads per key/value head");
  }
  CUDA_TRY(cudaSetDevice(m->device));
  const hero_config& c = m->cfg;
  const size_t layer = (size_t)max_seqs * m->n_kv_heads * max_len * 128;
  const size_t bytes = (size_t)c.n_layers * 2 * layer * 2;
  cudaError_t e = cudaMalloc(&m->kv, bytes);
  if (e != cudaSuccess) {
    m->kv = nullptr;
    return fail(HERO_ERR_NOMEM, "KV cache of %zu bytes: %s", bytes, cudaGetErrorString(e));
  }
  CUDA_TRY(cudaMemset(m->kv, 0, bytes));   // never-written positions read as zeros, not NaN
  const size_t pr = (size_t)max_seqs * m->n_heads * attn_decode_chunks(max_len - 1);
  CUDA_TRY(cudaMalloc(&m->dec_pm, pr * (2 + 128) * 4));
  m->dec_pl = m->dec_pm + pr;
  m->dec_po = m->dec_pl + pr;
  CUDA_TRY(cudaMalloc(&m->dec_pos, (size_t)max_seqs * 4));
  {   // split-K slices: at most 16 splits of 128-row tiles of the wider projection
    const long rows = ((long)std::min(max_seqs, c.max_tokens) + 127) / 128 * 128;
    const long nmax = std::max((long)(m->n_heads + 2 * m->n_kv_heads) * 128, (long)c.d_model);
    m->dec_ws_floats = (size_t)16 * rows * nmax;
    CUDA_TRY(cudaMalloc(&m->dec_ws, m->dec_ws_floats * 4));
  }
  if (hero_status rs = build_rope_table(m, max_len); rs != HERO_OK) return rs;
  m->kv_seqs = max_seqs;
  m->kv_len = max_len;
  return HERO_OK;
}

extern "C" hero_status hero_decoder_prefill(hero_model* m, int32_t seq0, int32_t n_seqs,
                                            int32_t seq_len, const float* h_in, float tau_exec,
                                            uint32_t flags, const uint8_t* mask_in, float* h_out,
                                            float* gate_out, uint8_t* mask_out,
                                            int32_t* ffn_count_out, void* cuda_stream) {
  g_last_error.clear();
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  if (!m->kv) return fail(HERO_ERR_ARG, "hero_kv_cache_init has not been called");
  const hero_config& c = m->cfg;
  if (seq0 < 0 || n_seqs < 0 || (long)seq0 + n_seqs > m->kv_seqs)
    return fail(HERO_ERR_ARG, "cache slots [%d, %d) outside [0, %d)", seq0, seq0 + n_seqs, m->kv_seqs);
  if (seq_len < 1 || seq_len > m->kv_len || (long)n_seqs * seq_len > c.max_tokens)
    return fail(HERO_ERR_ARG, "seq_len %d outside [1, max_len=%d] or n_seqs x seq_len > max_tokens",
                seq_len, m->kv_len);
  hero_status s = check_decoder_args(m, n_seqs * seq_len, h_in, tau_exec, flags, mask_in, h_out,
                                     ffn_count_out, cuda_stream);
  if (s != HERO_OK || n_seqs == 0) return s;
  return decoder_io(m, n_seqs, seq_len, seq0, nullptr, 0, h_in, tau_exec, flags, mask_in, h_out,
                    gate_out, mask_out, ffn_count_out, static_cast<cudaStream_t>(cuda_stream));
}

extern "C" hero_status hero_decode_step(hero_model* m, int32_t n_seqs, const int32_t* positions,
                                        int32_t max_position, const float* h_in, float tau_exec,
                                        uint32_t flags, const uint8_t* mask_in, float* h_out,
                                        float* gate_out, uint8_t* mask_out, int32_t* ffn_count_out,
                                        void* cuda_stream) {
  g_last_error.clear();
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  if (!m->kv) return fail(HERO_ERR_ARG, "hero_kv_cache_init has not been called");
  const hero_config& c = m->cfg;
  if (n_seqs < 0 || n_seqs > m->kv_seqs || n_seqs > c.max_tokens)
    return fail(HERO_ERR_ARG, "n_seqs %d outside [0, min(max_seqs, max_tokens)]", n_seqs);
  if (max_position < 0 || max_position >= m->kv_len)
    return fail(HERO_ERR_ARG, "max_position %d outside [0, max_len=%d)", max_position, m->kv_len);
  if (n_seqs > 0 && !positions) return fail(HERO_ERR_ARG, "positions is required");
  hero_status s = check_decoder_args(m, n_seqs, h_in, tau_exec, flags, mask_in, h_out,
                                     ffn_count_out, cuda_stream);
  if (s != HERO_OK || n_seqs == 0) return s;
  return decoder_io(m, n_seqs, 1, -1, positions, max_position, h_in, tau_exec, flags, mask_in,
                    h_out, gate_out, mask_out, ffn_count_out, static_cast<cudaStream_t>(cuda_stream));
}

extern "C" hero_status hero_check_device_status(hero_model* m, void* cuda_stream) {
  g_last_error.clear();
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  CUDA_TRY(cudaStreamSynchronize(st));
  uint32_t e = 0;
  CUDA_TRY(cudaMemcpy(&e, m->err, 4, cudaMemcpyDeviceToHost));
  if (e) CUDA_TRY(cudaMemset(m->err, 0, 4));
  return status_of_error_word(e);
}

extern "C" hero_status hero_set_profiling(hero_model* m, int enable) {
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  m->profiling = enable != 0;
  return HERO_OK;
}

extern "C" hero_status hero_get_profile(hero_model* m, double* ms_out, int64_t* launches_out,
                                        int reset) {
  g_last_error.clear();
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  for (auto& p : m->pending) {
    CUDA_TRY(cudaEventSynchronize(p.e1));
    float ms = 0.f;
    CUDA_TRY(cudaEventElapsedTime(&ms, p.e0, p.e1));
    m->prof_ms[p.cls] += ms;
    m->event_pool.push_back(p.e0);
    m->event_pool.push_back(p.e1);
  }
  m->pending.clear();
  for (int k = 0; k < HERO_K_COUNT; ++k) {
    if (ms_out) ms_out[k] = m->prof_ms[k];
    if (launches_out) launches_out[k] = m->launches[k];
    if (reset) {
      m->prof_ms[k] = 0.0;
      m->launches[k] = 0;
    }
  }
  return HERO_OK;
}

extern "C" hero_status hero_gemm_bf16_check(const uint16_t* A, const uint16_t* B, float* C,
                                            int32_t M, int32_t N, int32_t K, void* cuda_stream) {
  g_last_error.clear();
  if (!A || !B || !C || M < 1 || N < 8 || K < 64 || K % 64 != 0 || N % 8 != 0)
    return fail(HERO_ERR_ARG, "need M >= 1, N >= 8 (N %% 8 == 0), K %% 64 == 0 and non-NULL pointers");
  // one error word per device, allocated with that device current
  static std::mutex mu;
  static uint32_t* err_of[64] = {};
  int dev = 0;
  CUDA_TRY(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 64) return fail(HERO_ERR_UNSUPPORTED, "device index %d above 63", dev);
  uint32_t* err = nullptr;
  {
    std::lock_guard<std::mutex> lk(mu);
    if (!err_of[dev]) {
      CUDA_TRY(cudaMalloc(&err_of[dev], 64));
      CUDA_TRY(cudaMemset(err_of[dev], 0, 64));
    }
    err = err_of[dev];
  }
  int sms = 0;
  CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  // M >= 1024 runs on CTA pairs (256-row tiles, 128-row B boxes), as the large FFN GEMMs do
  const bool pair = M >= 1024;
  CUtensorMap ta, tb;
  if (!encode_bf16_2d(&ta, A, K, M, 128) || !encode_bf16_2d(&tb, B, K, N, pair ? 128 : 256))
    return fail(HERO_ERR_CUDA, "tensor map encoding failed");
  GemmArgs g{};
  g.m_static = M;
  g.m_max = M;
  g.N = N;
  g.K = K;
  g.out_f32 = C;
  g.ldo = N;
  g.err = err;
  const cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  CUDA_TRY(pair ? launch_gemm_tc2(EPI_STORE_F32, ta, tb, g, sms, st)
                : launch_gemm_tc(256, EPI_STORE_F32, ta, tb, g, sms, st));
  // synchronous: report (and clear) what the kernel recorded in the error word
  CUDA_TRY(cudaStreamSynchronize(st));
  uint32_t e = 0;
  CUDA_TRY(cudaMemcpy(&e, err, 4, cudaMemcpyDeviceToHost));
  if (e) CUDA_TRY(cudaMemset(err, 0, 4));
  return status_of_error_word(e);
}

// ============================================================================
// Training path: backward of a routed block's branch part, L_skip's gradient
// ============================================================================

extern "C" hero_status hero_backward_init(hero_model* m) {
  g_last_error.clear();
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  if (!m->bf16) return fail(HERO_ERR_UNSUPPORTED, "the backward runs on bf16 models only");
  if (m->bw) return fail(HERO_ERR_ARG, "hero_backward_init was already called for this model");
  const hero_config& c = m->cfg;
  const size_t L = c.n_layers, d = c.d_model, I = c.d_ff, r = c.d_r, Tm = c.max_tokens;
  CUDA_TRY(cudaSetDevice(m->device));
  auto bail = [&](hero_status st) {
    void* ps[] = {m->wdT, m->wguT, m->w1T, m->w2T, m->bws};
    for (void* p : ps)
      if (p) cudaFree(p);
    m->wdT = m->wguT = m->w1T = m->w2T = m->bws = nullptr;
    return st;
  };
#define BW_CUDA(expr)                                                                        \
  do {                                                                                       \
    cudaError_t e_ = (expr);                                                                 \
    if (e_ != cudaSuccess)                                                                   \
      return bail(fail(e_ == cudaErrorMemoryAllocation ? HERO_ERR_NOMEM : HERO_ERR_CUDA,     \
                       "%s failed: %s", #expr, cudaGetErrorString(e_)));                     \
  } while (0)
  BW_CUDA(cudaMalloc(&m->wdT, L * I * d * 2));
  BW_CUDA(cudaMalloc(&m->wguT, L * 2 * I * d * 2));
  BW_CUDA(cudaMalloc(&m->w1T, L * d * r * 2));
  BW_CUDA(cudaMalloc(&m->w2T, L * d * r * 2));
  // W_down [d][I] -> [I][d]; W_gate|W_up interleaved [2I][d] -> [d][2I] (the K order of
  // the gate/up gradient rows); W_1 [d_r][d] -> [d][d_r]; W_2 [d][d_r] -> [d_r][d]
  BW_CUDA(launch_transpose_bf16(m->wdown, m->wdT, (int)d, (int)I, (int)L, 0));
  BW_CUDA(launch_transpose_bf16(m->wgu, m->wguT, (int)(2 * I), (int)d, (int)L, 0));
  BW_CUDA(launch_transpose_bf16(m->w1, m->w1T, (int)r, (int)d, (int)L, 0));
  BW_CUDA(launch_transpose_bf16(m->w2, m->w2T, (int)d, (int)r, (int)L, 0));
  m->bw_part_ld = (int)((I + 255) / 256);
  const size_t chunks = (Tm + kBwChunk - 1) / kBwChunk;
  struct Item {
    void** p;
    size_t bytes;
  };
  std::vector<Item> items = {
      {(void**)&m->bw_gu, Tm * 2 * I * 2},  {(void**)&m->bw_gf, Tm * d * 2},
      {(void**)&m->bw_ga, Tm * d * 2},      {(void**)&m->bw_da, Tm * r * 2},
      {(void**)&m->bw_rinv, Tm * 4},        {(void**)&m->bw_dgpart, Tm * m->bw_part_ld * 4},
      {(void**)&m->bw_a, Tm * r * 4},       {(void**)&m->bw_gaf, Tm * r * 4},
      {(void**)&m->bw_daf, Tm * r * 4},     {(void**)&m->bw_y2, Tm * r * 4},
      {(void**)&m->bw_duf, Tm * d * 4},     {(void**)&m->bw_dua, Tm * d * 4},
      {(void**)&m->bw_wpart, chunks * d * r * 4},
  };
  size_t off = 0;
  for (auto& it : items) off += (it.bytes + 1023) & ~(size_t)1023;
  BW_CUDA(cudaMalloc(&m->bws, off));
  BW_CUDA(cudaMemset(m->bws, 0, off));
  off = 0;
  for (auto& it : items) {
    *it.p = static_cast<char*>(m->bws) + off;
    off += (it.bytes + 1023) & ~(size_t)1023;
  }
  bool ok = encode_bf16_2d(&m->tm_bwgf, m->bw_gf, d, Tm, 128) &&
            encode_bf16_2d(&m->tm_bwga, m->bw_ga, d, Tm, 128) &&
            encode_bf16_2d(&m->tm_bwgu, m->bw_gu, 2 * I, Tm, 128) &&
            encode_bf16_2d(&m->tm_bwda, m->bw_da, r, Tm, 128);
  m->tm_wdT.resize(L);
  m->tm_wguT.resize(L);
  m->tm_w1T.resize(L);
  m->tm_w2T.resize(L);
  m->tm_wdT_p.resize(L);
  m->tm_wguT_p.resize(L);
  for (size_t j = 0; j < L && ok; ++j) {
    ok = encode_bf16_2d(&m->tm_wdT[j], static_cast<char*>(m->wdT) + j * I * d * 2, d, I, 256) &&
         encode_bf16_2d(&m->tm_wguT[j], static_cast<char*>(m->wguT) + j * 2 * I * d * 2, 2 * I, d,
                        256) &&
         encode_bf16_2d(&m->tm_wdT_p[j], static_cast<char*>(m->wdT) + j * I * d * 2, d, I, 128) &&
         encode_bf16_2d(&m->tm_wguT_p[j], static_cast<char*>(m->wguT) + j * 2 * I * d * 2, 2 * I,
                        d, 128) &&
         encode_bf16_2d(&m->tm_w1T[j], static_cast<char*>(m->w1T) + j * d * r * 2, r, d, 256) &&
         encode_bf16_2d(&m->tm_w2T[j], static_cast<char*>(m->w2T) + j * d * r * 2, d, r, 256);
  }
  if (!ok) return bail(fail(HERO_ERR_CUDA, "tensor map encoding failed"));
  BW_CUDA(cudaDeviceSynchronize());
#undef BW_CUDA
  m->bw = true;
  return HERO_OK;
}

extern "C" hero_status hero_routed_block_backward(hero_model* m, int32_t block, int64_t n_tokens,
                                                  const float* h_bar, const float* gate,
                                                  const uint8_t* mask, const float* grad_out,
                                                  uint32_t flags, float* grad_h_bar,
                                                  float* grad_gate, float* grad_w1, float* grad_w2,
                                                  void* cuda_stream) {
  g_last_error.clear();
  if (!m) return fail(HERO_ERR_ARG, "model is NULL");
  if (!m->bw) return fail(HERO_ERR_ARG, "call hero_backward_init first");
  const hero_config& c = m->cfg;
  const int L = c.n_layers, d = c.d_model, I = c.d_ff, r = c.d_r;
  if (block < 1 || block > L) return fail(HERO_ERR_ARG, "block %d outside 1..%d", block, L);
  if (flags & ~(uint32_t)HERO_FLAG_DENSE) return fail(HERO_ERR_ARG, "flags 0x%x: only HERO_FLAG_DENSE", flags);
  if (n_tokens < 0 || n_tokens > c.max_tokens)
    return fail(HERO_ERR_ARG, "n_tokens %lld outside 0..max_tokens", (long long)n_tokens);
  const bool dense = (flags & HERO_FLAG_DENSE) || block <= c.n_dense;
  if (n_tokens == 0) return HERO_OK;
  if (!h_bar || !grad_out || !grad_h_bar) return fail(HERO_ERR_ARG, "h_bar, grad_out and grad_h_bar are required");
  if (!dense && (!gate || !mask || !grad_gate || !grad_w1 || !grad_w2))
    return fail(HERO_ERR_ARG, "a routed block needs gate, mask, grad_gate, grad_w1 and grad_w2");
  if (grad_h_bar == h_bar || grad_h_bar == grad_out)
    return fail(HERO_ERR_ARG, "grad_h_bar must not alias h_bar or grad_out");
  const int T = (int)n_tokens;
  const int jj = block - 1;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  const size_t es = 2;
  CompactArgs ca{T, mask, gate, dense ? 1 : 0, m->idx_f, m->idx_a, m->scale_f, m->scale_a,
                 m->counts, nullptr, nullptr, nullptr};
  CUDA_TRY(timed(m, HERO_K_BACKWARD, st, [&] { return launch_compact(ca, st); }));
  BwPrepArgs pa{T, d, m->counts, m->idx_f, m->idx_a, h_bar, grad_out,
                m->ffn_gain + (size_t)jj * d, c.rms_eps,
                static_cast<uint16_t*>(m->u_f), static_cast<uint16_t*>(m->u_a), m->bw_gf,
                m->bw_ga, m->bw_rinv};
  CUDA_TRY(timed(m, HERO_K_BACKWARD, st, [&] { return launch_bw_prep(pa, st); }));
  // FFN rows: gate/up pre-activations (bf16), then e = G W_down with the SwiGLU backward
  // in the epilogue (in place over the pre-activations), then du = [dgate|dup] [W_g|W_u]
  GemmArgs gu{};
  gu.m_dev = m->counts;
  gu.m_max = T;
  gu.N = 2 * I;
  gu.K = d;
  gu.out = m->bw_gu;
  gu.ldo = 2 * I;
  gu.err = m->err;
  const bool pair = T >= kPairMinRows;   // large token counts: CTA-pair tiles
  CUDA_TRY(timed(m, HERO_K_BACKWARD_GEMM, st, [&] {
    return pair ? launch_gemm_tc2(EPI_STORE_BF16, m->tm_uf, m->tm_wgu_p[jj], gu, m->num_sms, st)
                : launch_gemm_tc(256, EPI_STORE_BF16, m->tm_uf, m->tm_wgu[jj], gu, m->num_sms, st);
  }));
  GemmArgs ge{};
  ge.m_dev = m->counts;
  ge.m_max = T;
  ge.N = I;
  ge.K = d;
  ge.out = m->bw_gu;
  ge.ldo = 2 * I;
  ge.err = m->err;
  ge.row_scale = m->scale_f;
  ge.row_part = m->bw_dgpart;
  ge.part_ld = m->bw_part_ld;
  CUDA_TRY(timed(m, HERO_K_BACKWARD_GEMM, st, [&] {
    return pair ? launch_gemm_tc2(EPI_BW_SWIGLU, m->tm_bwgf, m->tm_wdT_p[jj], ge, m->num_sms, st)
                : launch_gemm_tc(256, EPI_BW_SWIGLU, m->tm_bwgf, m->tm_wdT[jj], ge, m->num_sms, st);
  }));
  GemmArgs gx{};
  gx.m_dev = m->counts;
  gx.m_max = T;
  gx.N = d;
  gx.K = 2 * I;
  gx.out_f32 = m->bw_duf;
  gx.ldo = d;
  gx.err = m->err;
  CUDA_TRY(timed(m, HERO_K_BACKWARD_GEMM, st, [&] {
    return pair ? launch_gemm_tc2(EPI_STORE_F32, m->tm_bwgu, m->tm_wguT_p[jj], gx, m->num_sms, st)
                : launch_gemm_tc(256, EPI_STORE_F32, m->tm_bwgu, m->tm_wguT[jj], gx, m->num_sms, st);
  }));
  if (!dense) {
    // adapter rows: a = W_1 u and ga = G W_2 (fp32), the hidden-layer backward per row,
    // du = da W_1, and the weight gradients
    GemmArgs g1{};
    g1.m_dev = m->counts + 1;
    g1.m_max = T;
    g1.N = r;
    g1.K = d;
    g1.out_f32 = m->bw_a;
    g1.ldo = r;
    g1.err = m->err;
    CUDA_TRY(timed(m, HERO_K_BACKWARD_GEMM, st, [&] {
      return launch_gemm_tc(256, EPI_STORE_F32, m->tm_ua, m->tm_w1[jj], g1, m->num_sms, st);
    }));
    GemmArgs g2 = g1;
    g2.out_f32 = m->bw_gaf;
    CUDA_TRY(timed(m, HERO_K_BACKWARD_GEMM, st, [&] {
      return launch_gemm_tc(256, EPI_STORE_F32, m->tm_bwga, m->tm_w2T[jj], g2, m->num_sms, st);
    }));
  }
  BwRowsArgs ra{T, r, m->counts, m->idx_f, m->idx_a, m->bw_dgpart, m->bw_part_ld,
                (I + 255) / 256, m->scale_a, m->bw_a, m->bw_gaf, m->bw_daf, m->bw_da, m->bw_y2,
                dense ? nullptr : grad_gate};
  CUDA_TRY(timed(m, HERO_K_BACKWARD, st, [&] { return launch_bw_rows(ra, st); }));
  if (!dense) {
    GemmArgs g3{};
    g3.m_dev = m->counts + 1;
    g3.m_max = T;
    g3.N = d;
    g3.K = r;
    g3.out_f32 = m->bw_dua;
    g3.ldo = d;
    g3.err = m->err;
    CUDA_TRY(timed(m, HERO_K_BACKWARD_GEMM, st, [&] {
      return launch_gemm_tc(256, EPI_STORE_F32, m->tm_bwda, m->tm_w1T[jj], g3, m->num_sms, st);
    }));
    // dL/dW_2 [d, d_r] = sum over adapter rows of G[t] (1 - g) bf16(SiLU(a))^T
    BwWgradArgs w2{m->counts + 1, grad_out, m->idx_a, m->bw_y2, d, r, m->bw_wpart};
    CUDA_TRY(timed(m, HERO_K_BACKWARD, st, [&] { return launch_bw_wgrad(w2, false, T, st); }));
    CUDA_TRY(timed(m, HERO_K_BACKWARD, st, [&] {
      return launch_bw_wreduce(m->bw_wpart, m->counts + 1, T, d, r, 0, grad_w2, m->num_sms, st);
    }));
    // dL/dW_1 [d_r, d] = sum over adapter rows of da u^T (u as the forward's bf16 operand)
    BwWgradArgs w1{m->counts + 1, m->u_a, nullptr, m->bw_daf, d, r, m->bw_wpart};
    CUDA_TRY(timed(m, HERO_K_BACKWARD, st, [&] { return launch_bw_wgrad(w1, true, T, st); }));
    CUDA_TRY(timed(m, HERO_K_BACKWARD, st, [&] {
      return launch_bw_wreduce(m->bw_wpart, m->counts + 1, T, d, r, 1, grad_w1, m->num_sms, st);
    }));
  } else {
    if (grad_w1) CUDA_TRY(cudaMemsetAsync(grad_w1, 0, (size_t)r * d * 4, st));
    if (grad_w2) CUDA_TRY(cudaMemsetAsync(grad_w2, 0, (size_t)r * d * 4, st));
    if (grad_gate) CUDA_TRY(cudaMemsetAsync(grad_gate, 0, (size_t)T * 4, st));
  }
  BwOutArgs oa{T, d, m->counts, m->idx_f, m->idx_a, h_bar, grad_out,
               m->ffn_gain + (size_t)jj * d, m->bw_rinv, m->bw_duf, m->bw_dua, grad_h_bar};
  CUDA_TRY(timed(m, HERO_K_BACKWARD, st, [&] { return launch_bw_out(oa, st); }));
  (void)es;
  return HERO_OK;
}

extern "C" hero_status hero_skip_penalty_grad(int32_t n_layers, int32_t n_dense, int32_t n_seqs,
                                              int32_t seq_len, const float* gates, float alpha,
                                              float* grad_gates, void* cuda_stream) {
  g_last_error.clear();
  if (n_layers < 1 || n_dense < 0 || n_dense >= n_layers || n_seqs < 1 || seq_len < 2)
    return fail(HERO_ERR_ARG, "need n_layers >= 1, 0 <= n_dense < n_layers, n_seqs >= 1, seq_len >= 2");
  if ((int64_t)n_seqs * seq_len > INT32_MAX) return fail(HERO_ERR_ARG, "too many tokens");
  if (!gates || !grad_gates) return fail(HERO_ERR_ARG, "gates and grad_gates are required");
  if (gates == grad_gates) return fail(HERO_ERR_ARG, "grad_gates must not alias gates");
  CUDA_TRY(launch_skip_grad(gates, n_layers, n_dense, n_seqs, seq_len, alpha, grad_gates,
                            static_cast<cudaStream_t>(cuda_stream)));
  return HERO_OK;
}
