/*
 * hero.h - C ABI of the GB300 (sm_103a) implementation of HeRo's history-aware
 * routed FFN stack ("Do Dynamic Routers Need Memory? HeRo: History-Aware Routing
 * for Efficient LLM Inference", Sec. 3).
 *
 * One call runs L_R routed blocks over T independent tokens.  Each block does, per
 * token and in this order (equation numbers count the displayed equations of
 * Sec. 3: 1 dense_attention, 2 adapter, 3 ffn_route, 4 path_vector, 5 hidden
 * encoder, 6 depth features, 7-8 transition features, 9 router_state, 10 q/k/v,
 * 11 memory_read, 12 memory_update, 13 nu, 14 history head, 15 cumulative
 * history, 16 final_gate):
 *   1. memory readout  c = phi(q)^T S / (phi(q)^T zeta + eps)            Eq. 11
 *   2. router score    g = sigma(f_theta([s;c;nu]) + f_psi(h_bar))       Eqs. 4-10, 13-16
 *   3. compaction of the tokens with g >= tau_exec                        Eq. 3
 *   4. frozen SwiGLU FFN on those tokens, adapter W_2 SiLU(W_1 u) on the rest   Eqs. 2-3
 *   5. h = h_bar + g FFN(u)  or  h_bar + (1-g) Adapter(u)                 Eq. 3
 *   6. memory update   S = rho S + phi(k) v^T, zeta = rho zeta + phi(k)   Eq. 12
 * h_bar_j = h_{j-1} + P_j, where P_j (attn_delta) stands in for the dense attention
 * sublayer of Eq. 1.  Per-token memory S, zeta and path state are created and
 * zeroed inside every call (one forward pass, Sec. 3.2).
 *
 * Beyond the stack: hero_routed_block runs one block on a caller's own h_bar;
 * hero_attn_init / hero_attention_block / hero_decoder_forward add the real
 * attention sublayer of Eq. 1 (the full decoder forward); hero_kv_cache_init /
 * hero_decoder_prefill / hero_decode_step run it incrementally over a KV cache;
 * hero_backward_init / hero_routed_block_backward / hero_skip_penalty_grad give the
 * training path's gradients (Sec. 3.1, 3.3); hero_gemm_bf16_splitk_noalloc is an
 * allocation-free tensor-core GEMM.
 *
 * Conventions
 *   - Every function returns hero_status; nothing aborts or exits.  On failure
 *     hero_last_error() returns a thread-local message.
 *   - Argument errors are detected before any work is enqueued (HERO_ERR_ARG).
 *   - Tensor pointers are DEVICE memory owned by the caller unless noted (see
 *     HERO_FLAG_HOST_IO); all tensors are dense row-major.
 *   - Execution is asynchronous on the given CUDA stream (cudaStream_t, NULL =
 *     legacy default stream).  Kernels never spin without a bound: a wait that
 *     expires (4 s by default, hero_set_wait_limit_ns) sets a device error word
 *     that hero_check_device_status reports as HERO_ERR_TIMEOUT; an out-of-range
 *     index found on the device is reported as HERO_ERR_BAD_INDEX.
 *   - A model may be used by one host thread at a time.
 */
#ifndef HERO_H_
#define HERO_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  HERO_OK = 0,
  HERO_ERR_ARG = 1,          /* invalid argument; nothing was enqueued          */
  HERO_ERR_CUDA = 2,         /* a CUDA runtime call failed                      */
  HERO_ERR_NOMEM = 3,        /* device or host allocation failed                */
  HERO_ERR_UNSUPPORTED = 4,  /* shape or dtype outside what the kernels support */
  HERO_ERR_TIMEOUT = 5,      /* a device-side bounded wait expired              */
  HERO_ERR_BAD_INDEX = 6     /* a kernel met an index outside its bounds (e.g. a
                                decoding position past the cache); the offending
                                accesses were skipped                           */
} hero_status;

typedef enum { HERO_F32 = 0, HERO_BF16 = 1 } hero_dtype;

/* Shapes and constants of one routed FFN stack.
 *   n_layers   FFN layers of the stack; the last n_layers - n_dense are the routed
 *              blocks j = 1..L_R (Sec. 3.1)
 *   d_model    d, hidden width; d_ff = I, SwiGLU intermediate width
 *   d_r        adapter rank (W_1: d_r x d, W_2: d x d_r; Eq. 2)
 *   d_m        memory width (q, k, v in R^{d_m}; S is d_m x d_m per token; Sec. 3.2)
 *   d_h, d_a   widths of z^h and z^a; the router state s has d_s = d_h + d_a (Eq. 9)
 *   d_enc      inner width of the hidden encoder W_hd (Eq. 5)
 *   d_head     hidden width of f_theta and f_psi (Sec. 4.1: 256)
 *   d_path     hidden width of FFN_path (Eq. 9)
 *   max_tokens largest T a call may pass; sizes the library-owned workspace
 *   dtype      HERO_BF16: bf16 weights and GEMM operands, fp32 accumulation and
 *              fp32 residual; HERO_F32: fp32 everywhere
 *   rms_eps    RMSNorm epsilon; eps: the epsilon of Eqs. 8, 11 and 13's cosine
 *   t_hist     history temperature T_hist (Eq. 14)
 * Supported: d_m in {16, 32, 64, 128, 256}; d_s <= 128; d_enc, d_head <= 256;
 * d_path <= 64.  bf16 additionally needs d % 256 == 0, d_ff % 128 == 0 and
 * d_r % 32 == 0 (d_r <= 4096); f32 needs d % 4 == 0 and d_r <= 64. */
typedef struct {
  int32_t n_layers, d_model, d_ff, d_r, d_m;
  int32_t d_h, d_a, d_enc, d_head, d_path;
  int32_t max_tokens;
  hero_dtype dtype;
  float rms_eps, eps, t_hist;
  int32_t n_dense;   /* leading layers outside the routing candidate set (Sec. 4.1
                        placement): plain FFN blocks, scale 1, router untouched;
                        0 <= n_dense < n_layers, L_R = n_layers - n_dense */
  uint32_t router_variant;  /* 0 = HeRo; else HERO_ROUTER_* ablation bits */
} hero_config;

/* Router ablations of Sec. 4.4 (bits of hero_config.router_variant):
 *   NO_HISTORY  g = sigma(b), the local logit alone (Eq. 16 without a); memory,
 *               path features and f_theta are skipped and the router state is
 *               left untouched
 *   NO_MEMREAD  f_theta keeps s but sees c = 0 and nu = 0 (Eqs. 11, 13); the
 *               memory S, zeta is neither read nor written
 *   NO_AUX      no auxiliary path encoder: z_a = 0 in s (Eq. 9)
 *   NO_POS      routing progress r, q_rem and transition d, gamma are zeroed in
 *               x_path (Eqs. 4, 6); p_hist, m_hist remain */
enum {
  HERO_ROUTER_NO_HISTORY = 1u,
  HERO_ROUTER_NO_MEMREAD = 2u,
  HERO_ROUTER_NO_AUX = 4u,
  HERO_ROUTER_NO_POS = 8u
};

/* HOST pointers to the parameters, canonical [out, in] layouts, stacked over
 * layers where marked [L, ...].  All arrays have element type host_dtype
 * (HERO_F32: float; HERO_BF16: uint16 bf16 bit patterns, allowed only for bf16
 * models).  The library copies (and for bf16 models rounds to bf16 with
 * round-to-nearest-even) during hero_init_weights; the caller may free them on
 * return.
 *   ffn_norm_g [L,d]   gain of LN^ffn (RMSNorm)                      Eq. 1
 *   w_gate, w_up [L,I,d], w_down [L,d,I]   frozen SwiGLU FFN          Eq. 3
 *   ad_w1 [L,d_r,d], ad_w2 [L,d,d_r]       adapter                     Eq. 2
 *   eta [L]            forgetting parameters, rho_j = sigma(eta_j)    Eq. 12
 *   r_norm_g [d]       router RMSNorm gain; w_hd [d_enc,d]; w_hu [d_h,d_enc]   Eq. 5
 *   path_w1 [d_path,6], path_b1 [d_path], path_w2 [d_a,d_path], path_b2 [d_a]  Eq. 9
 *   w_q, w_k, w_v [d_m,d_s]                                            Eq. 10
 *   w_n [d_m,d_s], w_c [d_m,d_m]                                       Eq. 13
 *   th_w1 [d_head,d_s+d_m+1], th_b1 [d_head], th_w2 [1,d_head], th_b2 [1]   f_theta, Eq. 14
 *   ps_w1 [d_head,d], ps_b1 [d_head], ps_w2 [1,d_head], ps_b2 [1]          f_psi, Eq. 16
 * Shared router parameters serve every block; FFN, adapter and eta are per
 * block (Sec. 3.2). */
typedef struct {
  hero_dtype host_dtype;
  const void *ffn_norm_g, *w_gate, *w_up, *w_down, *ad_w1, *ad_w2, *eta;
  const void *r_norm_g, *w_hd, *w_hu, *path_w1, *path_b1, *path_w2, *path_b2;
  const void *w_q, *w_k, *w_v, *w_n, *w_c;
  const void *th_w1, *th_b1, *th_w2, *th_b2;
  const void *ps_w1, *ps_b1, *ps_w2, *ps_b2;
} hero_weights_host;

typedef struct hero_model hero_model; /* opaque, library-owned */

enum {
  /* Router skipped; every token runs the FFN with branch scale 1 (the dense
   * SwiGLU stack run by the same kernels).  gate_out is filled with 1,
   * mask_out with 1, ffn_count_out with T. */
  HERO_FLAG_DENSE = 1u,
  /* Decisions are read from mask_in [L,T] (nonzero = FFN); g is still computed
   * and scales the branches as in Eq. 3. */
  HERO_FLAG_FORCE_MASK = 2u,
  /* h_in, attn_delta, mask_in, h_out, gate_out, mask_out and ffn_count_out are
   * HOST pointers; the library copies them to and from the device on the stream
   * (page-locked host memory makes the copies asynchronous). */
  HERO_FLAG_HOST_IO = 4u,
  /* bf16 models, batches of at most 128 tokens (one GEMM tile of rows): by default
   * the FFN and the adapter branch run on every token while the router runs beside
   * them on a second stream, and the block-closing step takes each token's branch
   * from the router's decision (Eq. 3), with the same results.  This flag runs the
   * FFN on the routed tokens only, after the router. */
  HERO_FLAG_NO_SPECULATE = 8u
};

/* Copy, convert and repack the parameters to the current CUDA device and size
 * the workspace for cfg->max_tokens.  Synchronous.  On success *out owns all
 * device memory of the model. */
hero_status hero_init_weights(const hero_config* cfg, const hero_weights_host* w,
                              hero_model** out);

/* Run the routed FFN stack on n_tokens tokens (0 <= n_tokens <= max_tokens).
 *   h_in       [T,d] fp32 input hidden states h_0
 *   attn_delta [L,T,d] attention stand-in P_j, fp32 for f32 models, bf16 bits for
 *              bf16 models; NULL means zero
 *   tau_exec   execution threshold of Eq. 3 (g >= tau_exec runs the FFN)
 *   flags      HERO_FLAG_*
 *   mask_in    [L,T] decisions for HERO_FLAG_FORCE_MASK, else ignored (may be NULL)
 *   h_out      [T,d] fp32 output h_{L_R}; must not alias h_in
 *   gate_out   [L,T] fp32 gates g, or NULL
 *   mask_out   [L,T] uint8 decisions (1 = FFN), or NULL
 *   ffn_count_out [L] int32 number of FFN tokens per block, or NULL
 * Returns after enqueueing; outputs are valid once the stream reaches them. */
hero_status hero_routed_ffn_stack(hero_model* m, int64_t n_tokens, const float* h_in,
                                  const void* attn_delta, float tau_exec, uint32_t flags,
                                  const uint8_t* mask_in, float* h_out, float* gate_out,
                                  uint8_t* mask_out, int32_t* ffn_count_out,
                                  void* cuda_stream);

/* ---- one routed block at a time ----------------------------------------------
 * Per-token router state carried from one routed block to the next within a
 * forward pass (Sec. 3.2).  DEVICE pointers, caller-owned, T tokens.  Lets the
 * caller run its own attention sublayer between routed blocks (Eq. 1) instead of
 * the additive stand-in of hero_routed_ffn_stack. */
typedef struct {
  float* S;           /* [T, d_m, d_m] memory matrix S (Eqs. 11-12), key index first */
  float* zeta;        /* [T, d_m] normaliser zeta (Eqs. 11-12)                          */
  float* p_hist;      /* [T] history score of the previous block (Eqs. 4, 14)           */
  float* m_hist;      /* [T] cumulative history score (Eqs. 4, 15)                      */
  float* d_prev;      /* [T] ||delta|| of the previous block (Eqs. 7-8)                 */
  float* h_bar_prev;  /* [T, d] h_bar of the previous routed block (Eq. 7)              */
  float* delta_prev;  /* [T, d] delta of the previous routed block (Eq. 8)              */
} hero_router_state;

/* Start of a forward pass: S = 0, zeta = 0, p_hist = m_hist = 1, d_prev = 0
 * (Sec. 3.2; Eq. 4 initial scores).  h_bar_prev / delta_prev need no reset: block
 * 1 does not read them. */
hero_status hero_router_state_reset(hero_model* m, int64_t n_tokens, const hero_router_state* state,
                                    void* cuda_stream);

/* Block `block` (1..n_layers) on post-attention hidden states h_bar [T,d] fp32
 * (Eq. 1); blocks 1..n_dense are plain FFN blocks (state unused, may be NULL),
 * block n_dense + j is routed block j.  Reads then updates `state` (read before write,
 * Eqs. 11-12) and writes h_out [T,d] = h_bar + g FFN(u) or h_bar + (1-g)
 * Adapter(u) (Eq. 3).  flags: HERO_FLAG_DENSE or HERO_FLAG_FORCE_MASK (mask_in [T]),
 * optionally HERO_FLAG_NO_SPECULATE.
 * gate_out [T], mask_out [T], ffn_count_out [1] may be NULL.  h_out must not
 * alias h_bar.  Same error and stream conventions as hero_routed_ffn_stack;
 * host pointers are not accepted here. */
hero_status hero_routed_block(hero_model* m, int32_t block, int64_t n_tokens, const float* h_bar,
                              const hero_router_state* state, float tau_exec, uint32_t flags,
                              const uint8_t* mask_in, float* h_out, float* gate_out,
                              uint8_t* mask_out, int32_t* ffn_count_out, void* cuda_stream);

/* Release every resource of the model (NULL-safe).  Synchronizes the device. */
void hero_free(hero_model* m);

/* Message of the last failure on this host thread ("" if none). */
const char* hero_last_error(void);

/* Synchronize cuda_stream, then report what the model's kernels recorded since the
 * last check (and clear the record): HERO_ERR_TIMEOUT if any wait hit its bound
 * (the outputs of that call are incomplete), else HERO_ERR_BAD_INDEX if a kernel
 * met an out-of-range index; HERO_ERR_CUDA if the stream holds a CUDA error. */
hero_status hero_check_device_status(hero_model* m, void* cuda_stream);

/* Bound, in nanoseconds of the GPU's global timer, on every device-side wait of the
 * kernels enqueued after this call (process-wide; 0 restores the default of 4 s).
 * A wait that reaches it gives up: the kernel lets its copies and tensor-core work
 * in flight finish (a separate 100 ms bound), records the expiry in its error word
 * (reported as HERO_ERR_TIMEOUT) and returns without completing its outputs.  The
 * bound is read when a kernel is enqueued, so a captured CUDA graph keeps the bound
 * of its capture.  Meant for tests of the timeout path; lowering it in production
 * turns slow waits into failures. */
void hero_set_wait_limit_ns(uint64_t limit_ns);

/* ---- the full decoder forward: real attention in Eq. 1 -----------------------
 * Eq. 1 gives each routed block the representation after attention,
 * h_bar = h + Attn(LN_attn(h)), and keeps attention dense (Sec. 3.1).  The fused
 * stack above stands in an additive perturbation for Attn; these calls attach the
 * backbone's attention (Llama form, Sec. 4.1: RMSNorm with its own gain,
 * bias-free projections, rotate-half RoPE with inverse frequencies
 * theta^(-2i/hd), causal softmax(q k^T / sqrt(hd)) per sequence, grouped-query
 * heads: query head h reads key/value head h / (H / H_kv)) and run the whole
 * decoder.  bf16 models only; head dimension 128 (d = H * 128). */
typedef struct {
  int32_t n_heads;       /* H; d_model = 128 H                                      */
  int32_t n_kv_heads;    /* H_kv; divides H                                         */
  float rope_theta;      /* RoPE base theta                                         */
} hero_attn_config;

/* HOST pointers, canonical layouts, stacked over the model's n_layers:
 *   attn_norm_g [L,d], w_q [L,H hd,d], w_k [L,H_kv hd,d], w_v [L,H_kv hd,d],
 *   w_o [L,d,H hd]; element type host_dtype.  Copied (converted to bf16). */
typedef struct {
  hero_dtype host_dtype;
  const void *attn_norm_g, *w_q, *w_k, *w_v, *w_o;
} hero_attn_weights_host;

/* Attach the attention parameters to a bf16 model and size its attention
 * workspace for max_tokens.  HERO_ERR_UNSUPPORTED for f32 models or
 * d != 128 H; HERO_ERR_ARG for bad counts or NULL pointers.  Call once. */
hero_status hero_attn_init(hero_model* m, const hero_attn_config* c, const hero_attn_weights_host* w);

/* Eq. 1, first line, for layer `layer` (1..n_layers) on n_seqs sequences of
 * seq_len tokens, rows of h in sequence order (T = n_seqs * seq_len <=
 * max_tokens, n_seqs <= 65535): h_bar [T,d] = h + Attn(LN_attn(h)).  DEVICE pointers, fp32, must
 * not alias.  Precision: bf16 operands (LN_attn(h), q and k after RoPE, v, the
 * softmax probabilities entering P V, the attention output), fp32 accumulation
 * and softmax.  Asynchronous on cuda_stream. */
hero_status hero_attention_block(hero_model* m, int32_t layer, int32_t n_seqs, int32_t seq_len,
                                 const float* h, float* h_bar, void* cuda_stream);

/* The full decoder forward over all n_layers blocks: h_bar = h + Attn(LN_attn(h))
 * (Eq. 1), then the block's FFN routing exactly as hero_routed_block (Eqs. 2-16;
 * blocks 1..n_dense are plain FFN blocks), the router state carried in the model's
 * workspace and reset at the start.  h_in [T,d] -> h_out [T,d] fp32; tau_exec,
 * flags (HERO_FLAG_DENSE or HERO_FLAG_FORCE_MASK with mask_in [L,T], optionally
 * HERO_FLAG_HOST_IO and HERO_FLAG_NO_SPECULATE), gate_out [L,T], mask_out [L,T], ffn_count_out [L] as
 * hero_routed_ffn_stack (NULL allowed).  DEVICE pointers, or HOST pointers with
 * HERO_FLAG_HOST_IO (copied on the stream); h_out must not alias h_in.
 * n_seqs <= 65535. */
hero_status hero_decoder_forward(hero_model* m, int32_t n_seqs, int32_t seq_len, const float* h_in,
                                 float tau_exec, uint32_t flags, const uint8_t* mask_in,
                                 float* h_out, float* gate_out, uint8_t* mask_out,
                                 int32_t* ffn_count_out, void* cuda_stream);

/* ---- KV-cache decoding: the decoder's incremental form ------------------------
 * Causal attention lets a sequence grow one token at a time: a new token's
 * h_bar (Eq. 1) needs the rotated keys and values of every earlier position,
 * which the model keeps in a cache, and its routing (Eqs. 2-16) runs on that
 * token alone with a fresh router state, as every token's does.
 *
 * Allocate the cache for max_seqs sequence slots of max_len positions, all
 * layers: 2 * n_layers * max_seqs * H_kv * max_len * 128 bf16, plus the
 * split-KV partial results of the decode attention.  Needs hero_attn_init;
 * once per model (HERO_ERR_ARG on a second call); HERO_ERR_UNSUPPORTED unless
 * H / H_kv is 1, 2, 4 or 8.  Synchronous. */
hero_status hero_kv_cache_init(hero_model* m, int32_t max_seqs, int32_t max_len);

/* hero_decoder_forward on n_seqs sequences of seq_len tokens that are cache slots
 * seq0 .. seq0 + n_seqs - 1 (seq0 + n_seqs <= max_seqs, seq_len <= max_len);
 * every layer's rotated keys and values of positions 0 .. seq_len - 1 are also
 * stored in those slots.  Arguments and outputs as hero_decoder_forward. */
hero_status hero_decoder_prefill(hero_model* m, int32_t seq0, int32_t n_seqs, int32_t seq_len,
                                 const float* h_in, float tau_exec, uint32_t flags,
                                 const uint8_t* mask_in, float* h_out, float* gate_out,
                                 uint8_t* mask_out, int32_t* ffn_count_out, void* cuda_stream);

/* One decoding step: a new token for each cache slot b < n_seqs (n_seqs <=
 * max_seqs and <= max_tokens), at position positions[b] (int32 [n_seqs]); it
 * attends to positions 0 .. positions[b] - 1 of its slot (which must hold that
 * sequence's earlier keys and values) and to itself, and its key and value are
 * stored at positions[b].  max_position (host) bounds every positions[b] and
 * sizes the launch; a position outside [0, min(max_position, max_len - 1)]
 * sets the device error word (the token's cache writes are skipped; reported
 * by hero_check_device_status).  h_in [n_seqs,d] are the new tokens' inputs;
 * tau_exec, flags (HERO_FLAG_DENSE, HERO_FLAG_FORCE_MASK with mask_in
 * [L,n_seqs], HERO_FLAG_HOST_IO: h_in, positions, mask_in and the outputs are
 * host pointers; HERO_FLAG_NO_SPECULATE) and the outputs as hero_decoder_forward with T = n_seqs.
 * Precision: as hero_attention_block, except that the softmax probabilities
 * enter P V in fp32. */
hero_status hero_decode_step(hero_model* m, int32_t n_seqs, const int32_t* positions,
                             int32_t max_position, const float* h_in, float tau_exec,
                             uint32_t flags, const uint8_t* mask_in, float* h_out, float* gate_out,
                             uint8_t* mask_out, int32_t* ffn_count_out, void* cuda_stream);

/* ---- training path: gradients with the decisions fixed -------------------------
 * Sec. 3.1 keeps the routing threshold out of differentiation: the selected branch's
 * scale (g for the FFN, 1 - g for the adapter) carries the gradient to the router,
 * and Sec. 3.3 trains the adapters and the router against the language-model loss
 * plus alpha L_skip with the backbone (FFN, LN_ffn) frozen.  These calls give the
 * branch part of a routed block's backward and L_skip's gradient; the router's own
 * backward (memory recurrence, path features, heads) is not part of them.
 *
 * Build the backward's operands for a bf16 model: transposed copies of every block's
 * W_down, W_gate|W_up and adapter weights (3 d I + 2 d d_r bf16 per block) and a
 * workspace for max_tokens.  Synchronous; once per model (HERO_ERR_ARG on a second
 * call); HERO_ERR_UNSUPPORTED for f32 models. */
hero_status hero_backward_init(hero_model* m);

/* Backward of block `block` (1..n_layers) with its decisions fixed, for
 *   h = h_bar + s Branch(u),  u = LN_ffn(h_bar)                        (Eqs. 1-3)
 * s = g and Branch = FFN (SwiGLU) where mask != 0, s = 1 - g and Branch = W_2 SiLU(W_1 u)
 * (Eq. 2) elsewhere.  DEVICE pointers, fp32, row-major, T = n_tokens <= max_tokens:
 *   h_bar [T,d], gate [T] (g), mask [T] (the forward's decisions), grad_out [T,d] = dL/dh
 *   -> grad_h_bar [T,d] = dL/dh_bar (residual plus branch), grad_gate [T] = dL/dg,
 *      grad_w1 [d_r,d] = dL/dW_1, grad_w2 [d,d_r] = dL/dW_2 of this block's adapter
 *      (sums over the adapter tokens; zero when there are none).
 * HERO_FLAG_DENSE (and blocks 1..n_dense): every token through the FFN with scale 1;
 * gate, mask may be NULL and grad_gate / grad_w1 / grad_w2, if given, are zeroed.
 * Precision: bf16 GEMM operands (u and the forward's bf16 rounding points, G, the
 * SwiGLU gradients dgate|dup, da), fp32 accumulation, fp32 row-wise and weight-gradient
 * arithmetic.  grad_h_bar must not alias h_bar or grad_out.  Needs hero_backward_init.
 * Asynchronous on cuda_stream (no host synchronisation); uses the model's forward
 * workspace, so it does not overlap a forward call of the same model. */
hero_status hero_routed_block_backward(hero_model* m, int32_t block, int64_t n_tokens,
                                       const float* h_bar, const float* gate, const uint8_t* mask,
                                       const float* grad_out, uint32_t flags, float* grad_h_bar,
                                       float* grad_gate, float* grad_w1, float* grad_w2,
                                       void* cuda_stream);

/* Gradient of the skip penalty (Sec. 3.3) with respect to the gates, times alpha:
 * L_skip = 1 / (B (S - 1)) sum over sequences b and next-token positions t < S - 1 of
 * (sum_j g_{j,b,t})^2, the sum over the routed blocks j (rows n_dense.. of gates).
 * gates [n_layers, B S] (tokens in sequence order) -> grad_gates [n_layers, B S] =
 * alpha dL_skip/dg: 2 alpha / (B (S - 1)) sum_j g_{j,b,t} for t < S - 1, 0 at each
 * sequence's last position and in the dense-prefix rows.  DEVICE pointers, not
 * aliased; seq_len >= 2.  Asynchronous on cuda_stream. */
hero_status hero_skip_penalty_grad(int32_t n_layers, int32_t n_dense, int32_t n_seqs,
                                   int32_t seq_len, const float* gates, float alpha,
                                   float* grad_gates, void* cuda_stream);

/* ---- measurement ------------------------------------------------------------
 * Kernel classes of one block, for per-kernel timing. */
enum {
  HERO_K_INIT = 0,        /* first h_bar, workspace reset                     */
  HERO_K_ROUTER_GEMM = 1, /* [T x d] x [d x (d_enc+d_head)] router contraction */
  HERO_K_ROUTER = 2,      /* memory read/update, heads, gate, decision        */
  HERO_K_COMPACT = 3,     /* stable scan of the decisions into index lists    */
  HERO_K_NORM = 4,        /* LN^ffn of each token into its branch's rows      */
  HERO_K_FFN_GATE_UP = 5, /* gathered gate/up GEMM with the SwiGLU epilogue;
                             bf16 models: also the adapter W_1 GEMM (grouped) */
  HERO_K_FFN_DOWN = 6,    /* down GEMM with the scaled scatter epilogue       */
  HERO_K_ADAPTER_DOWN = 7,/* f32 models: adapter W_1 GEMM with the SiLU epilogue */
  HERO_K_ADAPTER_UP = 8,  /* adapter W_2 GEMM with the scaled scatter epilogue */
  HERO_K_ATTN_PROJ = 9,   /* LN_attn, q/k/v projection, RoPE, output projection */
  HERO_K_ATTN_CORE = 10,  /* causal softmax attention                           */
  HERO_K_BACKWARD_GEMM = 11, /* training path: the tensor-core GEMMs of a block's backward */
  HERO_K_BACKWARD = 12,   /* training path: compaction, row and reduction kernels */
  HERO_K_COUNT = 13
};

/* When enabled, every later launch of the model is bracketed by CUDA events on
 * its stream.  hero_get_profile synchronizes those events and returns, per
 * kernel class, the summed device milliseconds and the launch count since the
 * last reset (then resets when reset != 0).  Both arrays hold HERO_K_COUNT
 * entries.  The launch counters run whether or not timing is enabled. */
hero_status hero_set_profiling(hero_model* m, int enable);
hero_status hero_get_profile(hero_model* m, double* ms_out, int64_t* launches_out, int reset);

/* Building-block check of the tensor-core GEMM: C[M,N] (fp32) = A[M,K] B[N,K]^T
 * with A, B bf16 (uint16 bit patterns), DEVICE pointers, row-major, K % 64 == 0,
 * K and N multiples of 8 elements.  Not part of the routed stack's contract;
 * exposed so the GEMM core can be tested alone.  Synchronous: waits for
 * cuda_stream, then returns HERO_ERR_TIMEOUT if the kernel's wait bound expired
 * (C incomplete) or HERO_ERR_BAD_INDEX, and clears that record (one per device). */
hero_status hero_gemm_bf16_check(const uint16_t* A, const uint16_t* B, float* C, int32_t M,
                                 int32_t N, int32_t K, void* cuda_stream);

/* ---- allocation-free variant ------------------------------------------------
 * The paper has no counterpart of this entry point; it exists for callers that
 * must not allocate device memory at call time, such as a host framework that
 * owns every device allocation through its own pool, or a latency-critical loop
 * where a cudaMalloc would synchronise the device.
 *
 * C[M,N] (fp32) = A[M,K] B[N,K]^T with A, B bf16 (uint16 bit patterns), DEVICE
 * pointers owned by the caller, row-major, computed as `splits` slices of K (whole
 * 64-wide blocks) on the tensor-core GEMM kernel and added in slice order.  The
 * partial sums (splits * M * N fp32, at most 4,194,304 values = 16 MiB) and the
 * kernel's error word live in static device arrays that every GPU loading this
 * library holds until process exit.  Nothing is allocated: no cudaMalloc, no
 * cudaFree, no allocating library call.
 *   - Requires M >= 1, N % 8 == 0, K % 64 == 0, 1 <= splits <= K / 64 and
 *     splits * M * N <= 4,194,304; otherwise HERO_ERR_ARG (hero_last_error()
 *     says which limit) and nothing is enqueued.
 *   - The first call on a device resolves the static arrays' device addresses
 *     for that device (with it current); make that first call before any stream
 *     capture.
 *   - Every call shares the static arrays and the arrays keep the last call's
 *     contents; calls that overlap on the GPU (other streams, other host
 *     threads) race on them.  Serialise calls on one stream.
 *   - Asynchronous on cuda_stream like the other entry points.  An expired wait
 *     inside the GEMM (C then incomplete) is recorded in the static error word,
 *     which keeps it across calls until hero_gemm_bf16_splitk_noalloc_status reads
 *     and clears it. */
hero_status hero_gemm_bf16_splitk_noalloc(const uint16_t* A, const uint16_t* B, float* C,
                                          int32_t M, int32_t N, int32_t K, int32_t splits,
                                          void* cuda_stream);

/* Status of the allocation-free GEMM calls on the current device since the last
 * query: synchronizes cuda_stream, then returns HERO_ERR_TIMEOUT (a wait bound
 * expired in some call; its C is incomplete), HERO_ERR_BAD_INDEX or HERO_OK, and
 * clears the static error word.  Allocates nothing. */
hero_status hero_gemm_bf16_splitk_noalloc_status(void* cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* HERO_H_ */
