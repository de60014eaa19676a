// Internal declarations shared by the kernels and the host runtime of libhero.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/hero.h"

namespace hero {

// Launch `kernel` on `st` with programmatic stream serialisation: its launch may
// overlap the tail of the previous kernel on the stream; the kernel itself waits
// (pdl_enter) for that kernel's completion before touching memory.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args&&... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// Device error word bits (set by kernels, read by hero_check_device_status).
enum : uint32_t {
  ERR_WAIT_PRODUCER = 1u,
  ERR_WAIT_MMA = 2u,
  ERR_WAIT_EPILOGUE = 4u,
  ERR_WAIT_DRAIN = 8u,
  ERR_BAD_INDEX = 16u,
};

// Record the message hero_last_error() returns on this host thread.
void set_last_error(const char* msg);

// Status for a device error word read back by the host: HERO_ERR_TIMEOUT if any
// wait bit is set, HERO_ERR_BAD_INDEX for a bad index alone, HERO_OK for 0 (sets
// the thread's message on failure).
hero_status status_of_error_word(uint32_t e);

// Default bound on every device-side wait (nanoseconds of %globaltimer); the bound a
// launch uses is wait_limit_ns(), which hero_set_wait_limit_ns may lower (tests of the
// timeout path).  The drains that follow an expired wait (copies and tensor-core work
// still in flight must finish before the CTA frees its TMEM and exits) use their own
// fixed bound, so a tiny wait bound never shortens them.
constexpr uint64_t kWaitLimitNs = 4000000000ull;
constexpr uint64_t kDrainLimitNs = 100000000ull;
uint64_t wait_limit_ns();

// ---------------------------------------------------------------------------
// Epilogue of the two GEMMs that close a routed block (FFN down, adapter up):
// for compacted row m with token t = idx[m] and branch scale s = scale[m],
// and y = the GEMM output row,
//     h_j       = h_bar_j + s * y                        (Eq. 3)
//   if this is not the last block:
//     h_bar_{j+1} = h_j + P_{j+1}                        (Eq. 1 stand-in)
//     delta_{j+1} = h_bar_{j+1} - h_bar_j = s * y + P_{j+1}   (Eq. 7)
//   and per (token, column tile) partial sums of h_bar_{j+1}^2, delta_{j+1}^2
//   and delta_{j+1} . delta_j feed the next block's RMSNorm (Eq. 5, LN^ffn) and
//   transition features (Eqs. 7-8).  The last block writes h_j to h_out.
// ---------------------------------------------------------------------------
struct LayerOutArgs {
  const int* idx;        // [rows] compacted row -> token
  const float* scale;    // [rows] branch scale (g, 1 - g, or 1)
  float* hbar;           // [T, d] in: h_bar_j; out: h_bar_{j+1}
  float* delta;          // [T, d] in: delta_j (unless first); out: delta_{j+1}
  const void* p_next;    // [T, d] P_{j+1} (bf16 or fp32) or nullptr (= 0)
  void* xl;              // [T, d] out: h_bar_{j+1} in the GEMM operand dtype
  float* part;           // [T, np, 4] out: partial sums per column tile
  float* h_out;          // [T, d] out (last block only)
  int d;
  int np;                // partial slots per token (kTcPartCols or kSimtTileN columns each)
  int last;              // 1: write h_out only
  int first;             // 1: delta_j = 0 (do not read it)
  int p_bf16;            // P_{j+1} element type
  int xl_bf16;           // operand element type of xl
  int router;            // 0 (dense stack): skip delta and the operand copy
};

// GEMM problem description shared by the tensor-core and SIMT GEMMs.
enum EpiKind : int {
  EPI_STORE_F32 = 0,   // out_f32[m, n] = acc
  EPI_SWIGLU = 1,      // out[m, n] = SiLU(gate) * up   (gate/up column pairs)
  EPI_SILU = 2,        // out[m, n] = SiLU(acc)
  EPI_LAYER_OUT = 3,   // LayerOutArgs
  EPI_LAYER_OUT_WIDE = 4,  // the same with twice the epilogue warps, for launches whose
                           // time is the epilogue's (the adapter's rank-d_r up projection)
  EPI_RESIDUAL = 5,    // out_f32[m, n] = acc + resid[m, n]  (attention output projection)
  EPI_ATTN_ENTRY = 6,  // the same, closing into the next routed block's entry: h_bar_j =
                       // resid + acc written over lo.hbar (= h_bar_{j-1}, read first),
                       // delta_j over lo.delta, the router operand copy lo.xl and the
                       // partial sums lo.part (lo.router, lo.first as in LayerOutArgs)
  EPI_QKV_ROPE = 7,    // fused q/k/v projection: RoPE on the q and k heads, bf16 out in
                       // the attention layout (RopeArgs)
  EPI_STORE_BF16 = 8,  // out[m, n] = bf16(acc) (N a multiple of 32)
  EPI_RT_ENC = 10,     // router on the tensor cores, step 1 (RouterTcArgs): the router
                       // contraction's columns [0, 256) -> SiLU(rinv acc) as three bf16 terms,
                       // [256, 512) -> b, plus d_j and gamma from the partial sums
  EPI_RT_S = 11,       // step 2: acc = z_h = W_hu enc; the path encoder; s = [z_h; z_a]
  EPI_RT_HEAD = 12,    // step 5: acc = W_th1 [s; c; nu]; f_theta's second layer, p_hist,
                       // m_hist, g and the decision
  EPI_BW_SWIGLU = 9,   // backward of the SwiGLU product (training path): acc = e = dL/dy W_down
                       // for features n of row m; out holds the row's bf16 gate/up
                       // pre-activations in the interleaved layout and is overwritten in place
                       // by dL/dgate, dL/dup (scaled by row_scale[m] = g); row_part[m, nb] =
                       // sum over the tile's features of e * bf16(SiLU(gate) up)
};

// EPI_QKV_ROPE: columns are heads of 128 (q heads | k heads | v heads).  Row t is
// position t % S of sequence t / S, or (pos != nullptr, a decoding step) position
// pos[t] of sequence t.  Pair (i, i + 64) of a q or k head at position s turns by
// the angle s * theta^(-2i/128), whose (cos, sin) come from cs.
struct RopeArgs {
  void* q;             // bf16 [B][H][S_q][128]; a decoding step stores at index 0 (S_q = 1)
  void* k;             // bf16 [B][H_kv][S_kv][128] at the token's position
  void* v;             // bf16 [B][H_kv][S_kv][128], or nullptr (v only transposed)
  const float* cs;     // [positions >= S_kv][64][2]: cos, sin
  const int* pos;      // [B] positions of a decoding step, or nullptr
  int H, Hkv, S, S_q, S_kv;
  void* vt;            // bf16 [B][H_kv][128][S_pad]: v transposed (keys contiguous), or nullptr
  int S_pad;           // positions per row of vt (a multiple of 8)
};

struct RouterWeights {   // shared router parameters, fp32, transposed to [in][out]
  const float* w_hu_t;    // [d_enc][d_h]
  const float* path_w1_t; // [6][d_path]
  const float* path_b1;   // [d_path]
  const float* path_w2_t; // [d_path][d_a]
  const float* path_b2;   // [d_a]
  const float* w_qkv_t;   // [d_s][3 d_m]  (q | k | v)
  const float* w_n_t;     // [d_s][d_m]
  const float* w_c_t;     // [d_m][d_m]
  const float* th_w1_t;   // [d_s + d_m + 1][d_head]
  const float* th_b1;     // [d_head]
  const float* th_w2;     // [d_head]
  const float* th_b2;     // [1]
  const float* ps_b1;     // [d_head]
  const float* ps_w2;     // [d_head]
  const float* ps_b2;     // [1]
};

// The HeRo router (no ablation) at large token counts on the tensor cores.  Its small
// matrices hold bf16 values; an fp32 activation x splits exactly into three bf16 terms
// x = x_0 + x_1 + x_2 (x_0 = bf16(x), x_1 = bf16(x - x_0), x_2 = bf16(x - x_0 - x_1)), so
// with the weight matrix repeated three times along K each tensor-core product is exact and
// the sums accumulate in fp32: the precision of the fp32 FMA router.  Five launches per
// block: the router contraction with EPI_RT_ENC; W_hu with EPI_RT_S; [W_q; W_k; W_v; W_n]
// with a plain fp32 store; the memory step (k_rt_mem: memory read and write, W_c c, nu, the
// f_theta input); W_th1 with EPI_RT_HEAD.  Per-token buffers below (T rows each).
struct RouterTcArgs {
  int T, j, L, np, d, d_h, d_a, d_path, dm;
  float rms_eps, eps, t_hist, tau, rho;
  const float* part;     // [T, np, 4] partial sums of h_bar (Eqs. 5, 7-8)
  float* dprev;          // [T] in: d_{j-1} (step 1); out: d_j (step 5)
  float* pst;            // [T] p_hist
  float* mst;            // [T] m_hist
  float* S;              // [T, dm, dm]
  float* zeta;           // [T, dm]
  // history form of the memory (k_rt_hist): per token, L entries of phi(k_i) | v_i
  // (hist_ld floats per token), and the decay weights hw[(j - 1) L + i] = rho_{i+1} ... rho_{j-1}
  // of entry i seen from routed block j (1-based blocks, 0-based entries)
  float* hist;
  long hist_ld;
  const float* hw;
  RouterWeights w;
  uint16_t* enc3;        // [T, 768] bf16: the encoder hidden's three terms
  float* scal;           // [T, 4]: d_j, gamma, f_psi's second layer without bias
  float* s;              // [T, d_s] router state s (Eq. 9)
  uint16_t* s3;          // [T, 3 d_s] bf16: s's three terms
  float* qkvn;           // [T, 4 dm]: q | k | v | W_n s (Eqs. 10, 13)
  uint16_t* fin3;        // [T, kf] bf16: [s; c; nu]'s three terms, zero beyond 3 (d_s + dm + 1)
  int kf;
  const uint8_t* mask_in;
  float* gate;
  uint8_t* mask;
  float* gate_out;
  uint8_t* mask_out;
  int* chunk_cnt;        // [ceil(T / 32)] FFN decisions per 32 consecutive tokens (step 5), or nullptr
};

struct GemmArgs {
  const int* m_dev;    // device row count (nullptr: use m_static)
  int m_static;
  int m_max;           // upper bound of M (sizes the grid)
  int N, K;
  // outputs
  float* out_f32;      // EPI_STORE_F32
  void* out;           // EPI_SWIGLU / EPI_SILU: bf16 (tensor-core path) or f32
  int ldo;             // leading dimension of out / out_f32 in elements
  LayerOutArgs lo;     // EPI_LAYER_OUT
  uint32_t* err;
  // split-K (EPI_STORE_F32 only): K-blocks are cut into k_splits contiguous ranges;
  // range s stores its partial sums at out_f32 + s * split_stride
  int k_splits;        // 0 or 1: no split
  long split_stride;
  const float* resid;  // EPI_RESIDUAL: [rows, N] fp32 added to the product (ld = ldo)
  RopeArgs rope;       // EPI_QKV_ROPE
  // Programmatic dependent launch: 0 waits for the previous kernel at the start;
  // 1 also lets the next kernel launch once every CTA has taken its last tile;
  // 2 (a launch whose inputs all come from earlier kernels than the previous one,
  // writing rows the previous one does not touch) works without waiting and waits
  // for the previous kernel at its end, so the kernels after it still follow both.
  int pdl_mode;
  uint64_t wait_ns;    // bound of every mbarrier wait (set by the launcher: wait_limit_ns())
  const float* row_scale;  // EPI_BW_SWIGLU: [rows] branch scale g
  float* row_part;     // EPI_BW_SWIGLU: [rows, part_ld] per-tile sums
  int part_ld;
  RouterTcArgs rt;     // EPI_RT_*
  // SIMT path only (row-major [rows, K] operands)
  const void* A;
  const void* B;
  const void* B2;      // EPI_SWIGLU: up-projection weights (gate in B)
  int lda, ldb;
};

// Tensor-core GEMM (tcgen05 + TMA + TMEM), bf16 operands, fp32 accumulation.
// A: [rows, K] K-major; B: [N, K] K-major; 128 x 256 tiles (bn must be 256).
cudaError_t launch_gemm_tc(int bn, EpiKind epi, const CUtensorMap& tmA, const CUtensorMap& tmB,
                           const GemmArgs& args, int num_sms, cudaStream_t st);

// Grouped launch of two independent problems in one persistent kernel, the second
// problem's tiles spread evenly among the first's: (SWIGLU, SILU) = FFN gate/up
// with the adapter's down projection (disjoint rows).  The SILU problem's N (the
// adapter rank) must be a multiple of 32; a narrower-than-tile B is zero-filled
// by TMA.  (The block-closing pair, FFN down with the adapter's up projection, is
// not grouped: an adapter tile holds one of the two TMEM accumulators for a whole
// epilogue while its MMA takes under a microsecond, which stalls the FFN's MMA.)
cudaError_t launch_gemm_tc_pair(EpiKind epi0, const CUtensorMap& tmA0, const CUtensorMap& tmB0,
                                const GemmArgs& a0, EpiKind epi1, const CUtensorMap& tmA1,
                                const CUtensorMap& tmB1, const GemmArgs& a1, int num_sms,
                                cudaStream_t st);

// The same GEMM on CTA pairs (clusters of 2, the 2-SM MMA): 256 x 256 tiles, each CTA
// staging 128 rows of A and 128 rows of B per K-block.  tmB must use 128-row boxes (the
// 1-CTA kernel's B maps use 256-row boxes); A maps are the same.  No split-K.  EPI_STORE_F32,
// EPI_SWIGLU and EPI_LAYER_OUT, and the grouped (SWIGLU, SILU) launch.
cudaError_t launch_gemm_tc2(EpiKind epi, const CUtensorMap& tmA, const CUtensorMap& tmB,
                            const GemmArgs& args, int num_sms, cudaStream_t st);
cudaError_t launch_gemm_tc2_pair(EpiKind epi0, const CUtensorMap& tmA0, const CUtensorMap& tmB0,
                                 const GemmArgs& a0, EpiKind epi1, const CUtensorMap& tmA1,
                                 const CUtensorMap& tmB1, const GemmArgs& a1, int num_sms,
                                 cudaStream_t st);

// SIMT fp32 GEMM with the same epilogues (f32 models).
cudaError_t launch_gemm_simt(EpiKind epi, const GemmArgs& args, cudaStream_t st);
constexpr int kSimtTileN = 64;

// Columns per partial-sum slot of the block-closing epilogues: bf16 models (tensor
// core path) use half a 256-column tile, f32 models the SIMT tile width.
constexpr int kTcPartCols = 128;

// Attention sublayer kernels (attention.cu), head dimension 128 --------------------
cudaError_t launch_attn_norm(const float* h, const float* g, int T, int d, float eps, void* x,
                             cudaStream_t st);
// K and V hold kv_stride positions per (sequence, head) slab (>= S; the cache's max_len).
cudaError_t launch_flash_attn(const void* Q, const void* K, const void* V, int B, int S, int H,
                              int Hkv, int kv_stride, void* O, cudaStream_t st);
// Causal attention on the tcgen05 tensor cores: 3-D tensor maps (128-byte swizzle,
// boxes of 64 x 128 x 1) over Q [B H][S][128], K [B H_kv][S (stride kv_stride)][128]
// and V^T [B H_kv][128][S (stride S_pad)]; O [B S][H 128] bf16.
cudaError_t launch_flash_tc(const CUtensorMap& tmQ, const CUtensorMap& tmK, const CUtensorMap& tmV,
                            int B, int S, int H, int Hkv, void* O, uint32_t* err, cudaStream_t st);
// Decoding step: Q [B][H][128], K/V slabs of kv_stride positions, pos [B] (each <=
// max_pos < kv_stride); partials pm, pl [B][H][chunks], po [B][H][chunks][128] with
// chunks = attn_decode_chunks(max_pos); O [B][H 128] bf16.
int attn_decode_chunks(int max_pos);
cudaError_t launch_attn_decode(const void* Q, const void* K, const void* V, const int* pos, int B,
                               int H, int Hkv, int kv_stride, int max_pos, float* pm, float* pl,
                               float* po, void* O, uint32_t* err, cudaStream_t st);

// Router and bookkeeping kernels ------------------------------------------------


struct RouterArgs {
  int T, j, L, np;       // j is 1-based
  int d, d_h, d_a, d_enc, d_head, d_path;
  const float* Y;        // [T, d_enc + d_head] router contraction output, or its y_splits
                         // split-K partial slices y_split_stride floats apart (summed in
                         // slice order as they are read)
  int y_splits;
  long y_split_stride;
  int y_rows;            // rows of Y per token: 2 when the operand pair is stacked along M
                         // (rows 2t and 2t + 1 of token t, added; launch_router_sm only)
  const float* part;     // [T, np, 4]
  float* dprev;          // [T] in: d_{j-1}; out: d_j
  float* pst;            // [T] p_hist
  float* mst;            // [T] m_hist
  float* S;              // [T, d_m, d_m]
  float* zeta;           // [T, d_m]
  float rho;
  RouterWeights w;
  float rms_eps, eps, t_hist, tau;
  const uint8_t* mask_in;  // [T] decisions of this block (FORCE_MASK) or nullptr
  float* gate;           // [T]
  uint8_t* mask;         // [T]
  float* gate_out;       // [T] caller slice or nullptr
  uint8_t* mask_out;     // [T] caller slice or nullptr
  uint32_t variant;      // router ablation bits (RV_*)
  // the router's parameters as one RsmBlob (bf16 models, variant 0) for launch_router_sm,
  // else nullptr
  const void* wsm;
  uint32_t* err;         // device error word (launch_router_sm's bounded waits)
  uint64_t wait_ns;
};

// Router at small and medium token counts with all of its parameters staged in shared
// memory by one bulk copy per CTA (launch_router_sm): the widths of the Llama router
// (d_enc = d_head = 256, d_h = 48, d_a = 16, d_path = 16, so d_s = 64) and d_m <= 64,
// on bf16 models, whose router parameters are bf16 values.  Byte offsets of the blob;
// matrices are bf16, [in][out] (outputs contiguous); the vectors are fp32.
constexpr int kRsmEnc = 256, kRsmHead = 256, kRsmDh = 48, kRsmDa = 16, kRsmPath = 16,
              kRsmDs = 64;
template <int DM>
struct RsmBlob {
  static constexpr int F = kRsmDs + DM + 1;               // f_theta's input [s; c; nu]
  static constexpr int hu = 0;                            // W_hu        [256][48]
  static constexpr int q4 = hu + kRsmEnc * kRsmDh * 2;    // q|k|v|W_n   [64][4 DM]
  static constexpr int wc = q4 + kRsmDs * 4 * DM * 2;     // W_c         [DM][DM]
  static constexpr int t1 = wc + DM * DM * 2;             // W_th1       [F][256]
  static constexpr int f32 = (t1 + F * kRsmHead * 2 + 15) / 16 * 16;
  // fp32 vectors, in floats from f32
  static constexpr int p1 = 0;                            // path W_1    [6][16]
  static constexpr int pb1 = p1 + 6 * kRsmPath;           // path b_1    [16]
  static constexpr int p2 = pb1 + kRsmPath;               // path W_2    [16][16]
  static constexpr int pb2 = p2 + kRsmPath * kRsmDa;      // path b_2    [16]
  static constexpr int tb1 = pb2 + kRsmDa;                // f_theta b_1 [256]
  static constexpr int tw2 = tb1 + kRsmHead;              // f_theta w_2 [256]
  static constexpr int psb1 = tw2 + kRsmHead;             // f_psi b_1   [256]
  static constexpr int psw2 = psb1 + kRsmHead;            // f_psi w_2   [256]
  static constexpr int tb2 = psw2 + kRsmHead;             // f_theta b_2
  static constexpr int psb2 = tb2 + 1;                    // f_psi b_2
  static constexpr int nf = (psb2 + 1 + 3) / 4 * 4;
  static constexpr int bytes = f32 + nf * 4;
  static_assert(q4 % 16 == 0 && wc % 16 == 0 && t1 % 16 == 0 && bytes % 16 == 0,
                "16-byte bulk-copy regions");
};

// Router ablation bits (the values of the ABI's HERO_ROUTER_*).
enum : uint32_t { RV_NO_HISTORY = 1u, RV_NO_MEMREAD = 2u, RV_NO_AUX = 4u, RV_NO_POS = 8u };

cudaError_t launch_router(int d_m, const RouterArgs& a, int num_sms, cudaStream_t st);
// Whether launch_router_sm serves a router of these widths (RsmBlob).
bool router_sm_supported(int d_enc, int d_head, int d_h, int d_a, int d_path, int d_m);
size_t router_sm_blob_bytes(int d_m);
cudaError_t launch_router_sm(int d_m, const RouterArgs& a, int num_sms, cudaStream_t st);
// Step 4 of the tensor-core router (see RouterTcArgs): with the state S, zeta, or in the
// history form (hist, hw; d_m = 64 or 128).
cudaError_t launch_rt_mem(const RouterTcArgs& a, cudaStream_t st);
cudaError_t launch_rt_hist(const RouterTcArgs& a, cudaStream_t st);

struct InitArgs {
  int T, d, np, d_m;
  const float* h_in;     // [T, d] (may equal hbar for in-place)
  const void* p0;        // [T, d] P_1 or nullptr
  int p_bf16;
  float* hbar;
  void* xl;
  int xl_bf16;
  float* part;
  float* S;
  float* zeta;
  float* pst;
  float* mst;
  float* dprev;
  int reset_router;      // 0 in dense mode
};
cudaError_t launch_init(const InitArgs& a, cudaStream_t st);

// Entry of one routed block run on its own (hero_routed_block).
struct BlockEntryArgs {
  int T, d, np, j;       // j is 1-based
  int router;            // 0 in dense mode: only the sum of squares is needed
  const float* h_bar;    // [T, d] post-attention hidden states of this block
  float* h_bar_prev;     // [T, d] in: previous block's h_bar; out: this block's
  float* delta_prev;     // [T, d] in: previous block's delta; out: this block's
  void* xl;              // router operand copy of h_bar
  int xl_bf16;
  float* part;           // [T, np, 4]
};
cudaError_t launch_block_entry(const BlockEntryArgs& a, cudaStream_t st);
cudaError_t launch_state_reset(float* S, float* zeta, float* pst, float* mst, float* dprev, int T,
                               int dm, cudaStream_t st);

struct CompactArgs {
  int T;
  const uint8_t* mask;   // [T]
  const float* gate;     // [T]
  int dense;             // all tokens FFN, scale 1
  int* idx_f;
  int* idx_a;
  float* scale_f;
  float* scale_a;
  int* counts;           // [2] n_f, n_a
  int* count_out;        // caller slot or nullptr
  float* gate_out;       // dense mode: fill with 1 (or nullptr)
  uint8_t* mask_out;     // dense mode: fill with 1 (or nullptr)
  // launch_route_norm: the FFN decisions of each 32 consecutive tokens, counted by the
  // router's last launch (RouterTcArgs::chunk_cnt), or nullptr (a ballot scan from token 0)
  const int* chunk_cnt;
};
cudaError_t launch_compact(const CompactArgs& a, cudaStream_t st);

struct NormArgs {
  int T, d, np;
  const int* counts;     // [2] n_f, n_a; nullptr: every token's row into u_f, in token order
  const int* idx_f;
  const int* idx_a;
  const float* hbar;
  const float* part;
  const float* gain;     // [d]
  float rms_eps;
  void* u_f;             // [T, d]
  void* u_a;             // [T, d]
  int out_bf16;
};
// wpr: warps per row (each takes a contiguous d / wpr column range; wpr divides d / 4)
cudaError_t launch_norm(const NormArgs& a, int num_sms, cudaStream_t st);
// k_compact and k_norm as one launch (same outputs): T <= kRouteNormMaxT, or any T with the
// per-32-token FFN counts (CompactArgs::chunk_cnt).
constexpr int kRouteNormMaxT = 2048;
cudaError_t launch_route_norm(const CompactArgs& c, const NormArgs& a, int num_sms, cudaStream_t st);

// Adapter up-projection plus the block-closing epilogue, for the adapter rows:
// y[m, :] = W_2 ah[m, :] (rank d_r = 64 contraction), then LayerOutArgs on token
// idx[m] with scale[m] = 1 - g.  SIMT: the contraction is 2 d_r FLOP per output
// element, so the kernel is bound by the epilogue's HBM traffic.
struct AdapterUpArgs {
  const int* m_dev;     // number of adapter rows (device)
  int m_max;
  int d, d_r;
  const void* ah;       // [rows, d_r] SiLU(W_1 u), bf16 or fp32
  const void* w2;       // [d, d_r] bf16 or fp32
  int bf16;
  int slot_cols;        // columns per partial-sum slot (64 or 256)
  LayerOutArgs lo;
};
cudaError_t launch_adapter_up(const AdapterUpArgs& a, cudaStream_t st);

// Split-K finishing kernel (few-tile launches, e.g. decode): y = sum_s part[s, m, n]
// over the k_splits partial slices in slice order, then the block-closing epilogue
// (LayerOutArgs) on token idx[m] for m < *m_dev, with kTcPartCols-column partial sums.
// Decoding step: split-K q/k/v slices [splits][B][N] fp32 -> RoPE, q and cache k/v
// (RopeArgs with pos); split-K output projection slices -> the attention-entry
// epilogue (EPI_ATTN_ENTRY arithmetic; resid = h_{j-1}).
cudaError_t launch_qkv_close(const float* part, int splits, long split_stride, int B,
                             const RopeArgs& r, uint32_t* err, cudaStream_t st);
cudaError_t launch_entry_close(const float* part, int splits, long split_stride, int B,
                               const float* resid, const LayerOutArgs& lo, cudaStream_t st);
// Adapter rows closed by the same launch (bf16, few tokens): rows m_dev[0] .. m_max - 1 of
// the launch are adapter rows m - m_dev[0] (the two branches cover every token): y = W_2
// ah[row] (depth d_r, a multiple of 8, accumulated in k order as k_adapter_up does), then
// the block-closing epilogue `lo` on token lo.idx[row] with scale lo.scale[row].  ah ==
// nullptr: no adapter rows.
struct SplitkAdapter {
  const void* ah;       // bf16 [rows, d_r] SiLU(W_1 u)
  const void* w2;       // bf16 [d, d_r]
  int d_r;
  LayerOutArgs lo;
  // 1: the FFN partial rows and the rows of ah are tokens (both branches ran on every
  // token); row m of the FFN branch reads token idx_f[m]'s rows, adapter row m token idx_a[m]'s
  int by_token;
};
cudaError_t launch_splitk_close(const float* part, int splits, long split_stride, int ld,
                                const int* m_dev, int m_max, const LayerOutArgs& lo,
                                const SplitkAdapter& ad, cudaStream_t st);

// Training path: backward of a routed block's branch part (backward.cu) -------------
// Compacted rows: FFN rows 0 .. n_f - 1 (idx_f), then adapter rows (idx_a), counts [2].
struct BwPrepArgs {
  int T, d;
  const int* counts;
  const int* idx_f;
  const int* idx_a;
  const float* hbar;     // [T, d] h_bar of the block
  const float* G;        // [T, d] dL/dh
  const float* gain;     // [d] LN_ffn gain
  float rms_eps;
  uint16_t* u_f;         // [T, d] bf16 u of the FFN rows (compacted)
  uint16_t* u_a;         // [T, d] bf16 u of the adapter rows
  uint16_t* g_f;         // [T, d] bf16 G of the FFN rows
  uint16_t* g_a;         // [T, d] bf16 G of the adapter rows
  float* rinv;           // [T] 1 / rms(h_bar)
};
struct BwRowsArgs {
  int T, d_r;
  const int* counts;
  const int* idx_f;
  const int* idx_a;
  const float* dgpart;   // [T, part_ld] FFN rows: per-tile sums of e * act
  int part_ld, n_parts;
  const float* scale_a;  // [T] adapter rows: 1 - g
  const float* pre;      // [T, d_r] adapter rows: a = W_1 u
  const float* ga;       // [T, d_r] adapter rows: G W_2
  float* da_f32;         // [T, d_r] out: da
  __nv_bfloat16* da_bf16;  // [T, d_r] out: bf16(da), the input-gradient GEMM's operand
  float* y2;             // [T, d_r] out: (1 - g) bf16(SiLU(a)), the W_2 gradient's factor
  float* grad_gate;      // [T] out: dL/dg by token (nullptr: not wanted)
};
constexpr int kBwChunk = 512;   // adapter rows per weight-gradient partial
struct BwWgradArgs {
  const int* rows;       // device row count (n_a)
  const void* X;         // fp32 [tokens, N] gathered through idx, or bf16 [rows, N]
  const int* idx;
  const float* Y;        // [rows, R]
  int N, R;
  float* part;           // [chunks, N, R]
};
struct BwOutArgs {
  int T, d;
  const int* counts;
  const int* idx_f;
  const int* idx_a;
  const float* hbar;
  const float* G;
  const float* gain;
  const float* rinv;
  const float* du_f;     // [T, d] du of the FFN rows (compacted)
  const float* du_a;     // [T, d] du of the adapter rows
  float* grad_hbar;      // [T, d] out
};
cudaError_t launch_bw_prep(const BwPrepArgs& a, cudaStream_t st);
cudaError_t launch_bw_rows(const BwRowsArgs& a, cudaStream_t st);
cudaError_t launch_bw_wgrad(const BwWgradArgs& a, bool x_bf16, int max_rows, cudaStream_t st);
cudaError_t launch_bw_wreduce(const float* part, const int* rows, int max_rows, int N, int R,
                              int transposed, float* out, int num_sms, cudaStream_t st);
cudaError_t launch_bw_out(const BwOutArgs& a, cudaStream_t st);
cudaError_t launch_skip_grad(const float* gates, int L, int n_dense, int n_seqs, int seq_len,
                             float alpha, float* out, cudaStream_t st);
cudaError_t launch_transpose_bf16(const void* in, void* out, int R, int C, int batch,
                                  cudaStream_t st);

// Weight conversion: dst[map(r)] = convert(src[r]) for rows of `cols` elements.
// map(r) = (r / grp) * grp_stride + (r % grp) + offset.
cudaError_t launch_convert_rows(const void* src, int src_bf16, void* dst, int dst_bf16,
                                long rows, long cols, long grp, long grp_stride, long offset,
                                const float* col_scale, cudaStream_t st);

}  // namespace hero
