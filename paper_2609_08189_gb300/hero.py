"""ctypes binding of libhero (include/hero.h): argument marshalling only.

Every step of the routed FFN stack runs in the CUDA kernels of libhero.so; this
module only converts Python/PyTorch arguments into the C ABI's plain pointers and
sizes.  There is no fallback: if the library is missing or fails to load, every
entry point raises.
"""

from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional, Sequence

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libhero.so")

(HERO_OK, HERO_ERR_ARG, HERO_ERR_CUDA, HERO_ERR_NOMEM, HERO_ERR_UNSUPPORTED, HERO_ERR_TIMEOUT,
 HERO_ERR_BAD_INDEX) = range(7)
STATUS_NAMES = {0: "HERO_OK", 1: "HERO_ERR_ARG", 2: "HERO_ERR_CUDA", 3: "HERO_ERR_NOMEM",
                4: "HERO_ERR_UNSUPPORTED", 5: "HERO_ERR_TIMEOUT", 6: "HERO_ERR_BAD_INDEX"}
HERO_F32, HERO_BF16 = 0, 1
HERO_FLAG_DENSE, HERO_FLAG_FORCE_MASK, HERO_FLAG_HOST_IO, HERO_FLAG_NO_SPECULATE = 1, 2, 4, 8
HERO_ROUTER_NO_HISTORY, HERO_ROUTER_NO_MEMREAD, HERO_ROUTER_NO_AUX, HERO_ROUTER_NO_POS = 1, 2, 4, 8
KERNEL_CLASSES = ("init", "router_gemm", "router", "compact", "norm", "ffn_gate_up", "ffn_down",
                  "adapter_down", "adapter_up", "attn_proj", "attn_core", "backward_gemm",
                  "backward")
ATTN_WEIGHT_FIELDS = ("attn_norm_g", "w_q", "w_k", "w_v", "w_o")
HERO_K_COUNT = len(KERNEL_CLASSES)

WEIGHT_FIELDS = ("ffn_norm_g", "w_gate", "w_up", "w_down", "ad_w1", "ad_w2", "eta",
                 "r_norm_g", "w_hd", "w_hu", "path_w1", "path_b1", "path_w2", "path_b2",
                 "w_q", "w_k", "w_v", "w_n", "w_c", "th_w1", "th_b1", "th_w2", "th_b2",
                 "ps_w1", "ps_b1", "ps_w2", "ps_b2")


class hero_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("n_layers", "d_model", "d_ff", "d_r", "d_m", "d_h", "d_a", "d_enc", "d_head",
                 "d_path", "max_tokens")] + \
               [("dtype", ctypes.c_int), ("rms_eps", ctypes.c_float), ("eps", ctypes.c_float),
                ("t_hist", ctypes.c_float), ("n_dense", ctypes.c_int32),
                ("router_variant", ctypes.c_uint32)]


class hero_weights_host(ctypes.Structure):
    _fields_ = [("host_dtype", ctypes.c_int)] + [(n, ctypes.c_void_p) for n in WEIGHT_FIELDS]


class hero_attn_config(ctypes.Structure):
    _fields_ = [("n_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("rope_theta", ctypes.c_float)]


class hero_attn_weights_host(ctypes.Structure):
    _fields_ = [("host_dtype", ctypes.c_int)] + [(n, ctypes.c_void_p) for n in ATTN_WEIGHT_FIELDS]


STATE_FIELDS = ("S", "zeta", "p_hist", "m_hist", "d_prev", "h_bar_prev", "delta_prev")


class hero_router_state(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in STATE_FIELDS]


class HeroError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


_lib: Optional[ctypes.CDLL] = None


def load(path: Optional[str] = None) -> ctypes.CDLL:
    """Load libhero.so (raises if it is missing; build it with __graft_entry__.build())."""
    global _lib
    if _lib is not None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"libhero.so not found at {p}; run __graft_entry__.build()")
    lib = ctypes.CDLL(p)
    vp, i32, i64, f32, u32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_uint32
    lib.hero_init_weights.argtypes = [ctypes.POINTER(hero_config), ctypes.POINTER(hero_weights_host),
                                      ctypes.POINTER(vp)]
    lib.hero_init_weights.restype = ctypes.c_int
    lib.hero_routed_ffn_stack.argtypes = [vp, i64, vp, vp, f32, u32, vp, vp, vp, vp, vp, vp]
    lib.hero_routed_ffn_stack.restype = ctypes.c_int
    lib.hero_free.argtypes = [vp]
    lib.hero_free.restype = None
    lib.hero_last_error.argtypes = []
    lib.hero_last_error.restype = ctypes.c_char_p
    lib.hero_check_device_status.argtypes = [vp, vp]
    lib.hero_check_device_status.restype = ctypes.c_int
    lib.hero_set_profiling.argtypes = [vp, ctypes.c_int]
    lib.hero_set_profiling.restype = ctypes.c_int
    lib.hero_get_profile.argtypes = [vp, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(i64), ctypes.c_int]
    lib.hero_get_profile.restype = ctypes.c_int
    lib.hero_gemm_bf16_check.argtypes = [vp, vp, vp, i32, i32, i32, vp]
    lib.hero_gemm_bf16_check.restype = ctypes.c_int
    lib.hero_router_state_reset.argtypes = [vp, i64, ctypes.POINTER(hero_router_state), vp]
    lib.hero_router_state_reset.restype = ctypes.c_int
    lib.hero_routed_block.argtypes = [vp, i32, i64, vp, ctypes.POINTER(hero_router_state), f32, u32,
                                      vp, vp, vp, vp, vp, vp]
    lib.hero_routed_block.restype = ctypes.c_int
    lib.hero_attn_init.argtypes = [vp, ctypes.POINTER(hero_attn_config),
                                   ctypes.POINTER(hero_attn_weights_host)]
    lib.hero_attn_init.restype = ctypes.c_int
    lib.hero_attention_block.argtypes = [vp, i32, i32, i32, vp, vp, vp]
    lib.hero_attention_block.restype = ctypes.c_int
    lib.hero_decoder_forward.argtypes = [vp, i32, i32, vp, f32, u32, vp, vp, vp, vp, vp, vp]
    lib.hero_decoder_forward.restype = ctypes.c_int
    lib.hero_kv_cache_init.argtypes = [vp, i32, i32]
    lib.hero_kv_cache_init.restype = ctypes.c_int
    lib.hero_decoder_prefill.argtypes = [vp, i32, i32, i32, vp, f32, u32, vp, vp, vp, vp, vp, vp]
    lib.hero_decoder_prefill.restype = ctypes.c_int
    lib.hero_decode_step.argtypes = [vp, i32, vp, i32, vp, f32, u32, vp, vp, vp, vp, vp, vp]
    lib.hero_decode_step.restype = ctypes.c_int
    lib.hero_gemm_bf16_splitk_noalloc.argtypes = [vp, vp, vp, i32, i32, i32, i32, vp]
    lib.hero_gemm_bf16_splitk_noalloc.restype = ctypes.c_int
    lib.hero_gemm_bf16_splitk_noalloc_status.argtypes = [vp]
    lib.hero_gemm_bf16_splitk_noalloc_status.restype = ctypes.c_int
    lib.hero_set_wait_limit_ns.argtypes = [ctypes.c_uint64]
    lib.hero_set_wait_limit_ns.restype = None
    lib.hero_backward_init.argtypes = [vp]
    lib.hero_backward_init.restype = ctypes.c_int
    lib.hero_routed_block_backward.argtypes = [vp, i32, i64, vp, vp, vp, vp, u32, vp, vp, vp, vp, vp]
    lib.hero_routed_block_backward.restype = ctypes.c_int
    lib.hero_skip_penalty_grad.argtypes = [i32, i32, i32, i32, vp, f32, vp, vp]
    lib.hero_skip_penalty_grad.restype = ctypes.c_int
    _lib = lib
    return lib


def _check(status: int) -> None:
    if status != HERO_OK:
        raise HeroError(status, hero_last_error())


def hero_last_error() -> str:
    return load().hero_last_error().decode()


def make_config(stack_cfg, max_tokens: Optional[int] = None) -> hero_config:
    """hero_config from a synth StackConfig."""
    c = stack_cfg
    return hero_config(c.n_layers, c.d_model, c.d_ff, c.d_r, c.d_m, c.d_h, c.d_a, c.d_enc,
                       c.d_head, c.d_path, max_tokens or c.n_tokens,
                       HERO_BF16 if c.dtype == "bf16" else HERO_F32, c.rms_eps, c.eps, c.t_hist,
                       getattr(c, "n_dense", 0), getattr(c, "router_variant", 0))


def make_weights(weights: Dict[str, np.ndarray]):
    """hero_weights_host pointing into contiguous numpy arrays (kept alive by the caller)."""
    arrs = {k: np.ascontiguousarray(weights[k]) for k in WEIGHT_FIELDS}
    dts = {a.dtype for a in arrs.values()}
    if dts == {np.dtype(np.uint16)}:
        hd = HERO_BF16
    elif dts == {np.dtype(np.float32)}:
        hd = HERO_F32
    else:
        raise TypeError(f"weights must be all float32 or all uint16 bf16 bits, got {dts}")
    w = hero_weights_host(hd, *[arrs[k].ctypes.data for k in WEIGHT_FIELDS])
    return w, arrs


def hero_init_weights(cfg: hero_config, weights: Dict[str, np.ndarray]) -> int:
    w, keep = make_weights(weights)
    out = ctypes.c_void_p()
    _check(load().hero_init_weights(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(out)))
    del keep
    return out.value


def hero_routed_ffn_stack(model: int, n_tokens: int, h_in: int, attn_delta: int, tau_exec: float,
                          flags: int, mask_in: int, h_out: int, gate_out: int, mask_out: int,
                          ffn_count_out: int, cuda_stream: int) -> None:
    """Pointer-level call (ints are raw addresses, 0 for NULL)."""
    _check(load().hero_routed_ffn_stack(model, n_tokens, h_in or None, attn_delta or None,
                                        float(tau_exec), flags, mask_in or None, h_out or None,
                                        gate_out or None, mask_out or None, ffn_count_out or None,
                                        cuda_stream or None))


def make_state(ptrs: Dict[str, int]) -> hero_router_state:
    """hero_router_state from raw device addresses keyed by STATE_FIELDS (missing = NULL)."""
    return hero_router_state(*[ptrs.get(n) or None for n in STATE_FIELDS])


def hero_router_state_reset(model: int, n_tokens: int, state: hero_router_state,
                            cuda_stream: int = 0) -> None:
    _check(load().hero_router_state_reset(model, n_tokens, ctypes.byref(state), cuda_stream or None))


def hero_routed_block(model: int, block: int, n_tokens: int, h_bar: int, state: hero_router_state,
                      tau_exec: float, flags: int, mask_in: int, h_out: int, gate_out: int,
                      mask_out: int, ffn_count_out: int, cuda_stream: int) -> None:
    """One routed block on post-attention hidden states (pointer-level call)."""
    _check(load().hero_routed_block(model, block, n_tokens, h_bar or None, ctypes.byref(state),
                                    float(tau_exec), flags, mask_in or None, h_out or None,
                                    gate_out or None, mask_out or None, ffn_count_out or None,
                                    cuda_stream or None))


def hero_free(model: int) -> None:
    if model:
        load().hero_free(model)


def hero_check_device_status(model: int, cuda_stream: int = 0) -> None:
    _check(load().hero_check_device_status(model, cuda_stream or None))


def hero_set_profiling(model: int, enable: bool) -> None:
    _check(load().hero_set_profiling(model, 1 if enable else 0))


def hero_get_profile(model: int, reset: bool = True):
    ms = (ctypes.c_double * HERO_K_COUNT)()
    n = (ctypes.c_int64 * HERO_K_COUNT)()
    _check(load().hero_get_profile(model, ms, n, 1 if reset else 0))
    return {k: (ms[i], n[i]) for i, k in enumerate(KERNEL_CLASSES)}


def hero_gemm_bf16_check(A: int, B: int, C: int, M: int, N: int, K: int, cuda_stream: int = 0) -> None:
    """Synchronous; raises HeroError(HERO_ERR_TIMEOUT) if the kernel's wait bound expired."""
    _check(load().hero_gemm_bf16_check(A, B, C, M, N, K, cuda_stream or None))


def hero_backward_init(model: int) -> None:
    _check(load().hero_backward_init(model))


def hero_routed_block_backward(model: int, block: int, n_tokens: int, h_bar: int, gate: int,
                               mask: int, grad_out: int, flags: int, grad_h_bar: int,
                               grad_gate: int, grad_w1: int, grad_w2: int,
                               cuda_stream: int = 0) -> None:
    """Backward of one block's branch part with the decisions fixed (pointer-level call)."""
    _check(load().hero_routed_block_backward(model, block, n_tokens, h_bar or None, gate or None,
                                             mask or None, grad_out or None, flags,
                                             grad_h_bar or None, grad_gate or None,
                                             grad_w1 or None, grad_w2 or None,
                                             cuda_stream or None))


def hero_skip_penalty_grad(n_layers: int, n_dense: int, n_seqs: int, seq_len: int, gates: int,
                           alpha: float, grad_gates: int, cuda_stream: int = 0) -> None:
    _check(load().hero_skip_penalty_grad(n_layers, n_dense, n_seqs, seq_len, gates or None,
                                         float(alpha), grad_gates or None, cuda_stream or None))


def hero_set_wait_limit_ns(limit_ns: int) -> None:
    """Bound on device-side waits of later launches (0 restores the default 4 s)."""
    load().hero_set_wait_limit_ns(int(limit_ns))


def hero_gemm_bf16_splitk_noalloc(A: int, B: int, C: int, M: int, N: int, K: int, splits: int,
                                  cuda_stream: int = 0) -> None:
    """Split-K bf16 GEMM whose scratch lives in static device memory (no allocation)."""
    _check(load().hero_gemm_bf16_splitk_noalloc(A, B, C, M, N, K, splits, cuda_stream or None))


def hero_gemm_bf16_splitk_noalloc_status(cuda_stream: int = 0) -> None:
    """Raises if an allocation-free GEMM call since the last query recorded an error."""
    _check(load().hero_gemm_bf16_splitk_noalloc_status(cuda_stream or None))


def hero_attn_init(model: int, stack_cfg, attn_weights: Dict[str, np.ndarray]) -> None:
    """Attach the attention parameters (canonical layouts, stacked over layers)."""
    arrs = {k: np.ascontiguousarray(attn_weights[k]) for k in ATTN_WEIGHT_FIELDS}
    dts = {a.dtype for a in arrs.values()}
    if dts == {np.dtype(np.uint16)}:
        hd = HERO_BF16
    elif dts == {np.dtype(np.float32)}:
        hd = HERO_F32
    else:
        raise ValueError(f"attention weights must all be uint16 (bf16 bits) or float32, got {dts}")
    w = hero_attn_weights_host(hd, *[a.ctypes.data for a in arrs.values()])
    c = hero_attn_config(stack_cfg.n_heads, stack_cfg.n_kv_heads, stack_cfg.rope_theta)
    _check(load().hero_attn_init(model, ctypes.byref(c), ctypes.byref(w)))


def hero_attention_block(model: int, layer: int, n_seqs: int, seq_len: int, h: int, h_bar: int,
                         cuda_stream: int) -> None:
    """Eq. 1, first line, for one layer (pointer-level call)."""
    _check(load().hero_attention_block(model, layer, n_seqs, seq_len, h or None, h_bar or None,
                                       cuda_stream or None))


def hero_decoder_forward(model: int, n_seqs: int, seq_len: int, h_in: int, tau_exec: float,
                         flags: int, mask_in: int, h_out: int, gate_out: int, mask_out: int,
                         ffn_count_out: int, cuda_stream: int) -> None:
    """The full decoder forward (pointer-level call)."""
    _check(load().hero_decoder_forward(model, n_seqs, seq_len, h_in or None, float(tau_exec), flags,
                                       mask_in or None, h_out or None, gate_out or None,
                                       mask_out or None, ffn_count_out or None, cuda_stream or None))


def hero_kv_cache_init(model: int, max_seqs: int, max_len: int) -> None:
    """Allocate the model's KV cache (max_seqs slots of max_len positions, all layers)."""
    _check(load().hero_kv_cache_init(model, max_seqs, max_len))


def hero_decoder_prefill(model: int, seq0: int, n_seqs: int, seq_len: int, h_in: int,
                         tau_exec: float, flags: int, mask_in: int, h_out: int, gate_out: int,
                         mask_out: int, ffn_count_out: int, cuda_stream: int) -> None:
    """The decoder forward on cache slots seq0.., storing their keys and values."""
    _check(load().hero_decoder_prefill(model, seq0, n_seqs, seq_len, h_in or None, float(tau_exec),
                                       flags, mask_in or None, h_out or None, gate_out or None,
                                       mask_out or None, ffn_count_out or None, cuda_stream or None))


def hero_decode_step(model: int, n_seqs: int, positions: int, max_position: int, h_in: int,
                     tau_exec: float, flags: int, mask_in: int, h_out: int, gate_out: int,
                     mask_out: int, ffn_count_out: int, cuda_stream: int) -> None:
    """One decoding step: a token per cache slot b < n_seqs at positions[b]."""
    _check(load().hero_decode_step(model, n_seqs, positions or None, max_position, h_in or None,
                                   float(tau_exec), flags, mask_in or None, h_out or None,
                                   gate_out or None, mask_out or None, ffn_count_out or None,
                                   cuda_stream or None))


# ---------------------------------------------------------------------------
# PyTorch convenience layer (device tensors, current stream)
# ---------------------------------------------------------------------------

class HeroStack:
    """A loaded model plus torch-tensor calls.  PyTorch supplies memory and streams."""

    def __init__(self, stack_cfg, weights: Dict[str, np.ndarray], max_tokens: Optional[int] = None):
        self.cfg = stack_cfg
        self.max_tokens = max_tokens or stack_cfg.n_tokens
        self.model = hero_init_weights(make_config(stack_cfg, self.max_tokens), weights)

    def close(self):
        if self.model:
            hero_free(self.model)
            self.model = 0

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __call__(self, h_in, attn_delta, tau: float, flags: int = 0, mask_in=None,
                 h_out=None, gate_out=None, mask_out=None, counts_out=None, stream=None):
        """Device tensors in and out.  Returns (h_out, gate, mask, counts)."""
        import torch
        T, d = h_in.shape
        L = self.cfg.n_layers
        dev = h_in.device
        if h_out is None:
            h_out = torch.empty((T, d), dtype=torch.float32, device=dev)
        if gate_out is None:
            gate_out = torch.empty((L, T), dtype=torch.float32, device=dev)
        if mask_out is None:
            mask_out = torch.empty((L, T), dtype=torch.uint8, device=dev)
        if counts_out is None:
            counts_out = torch.empty((L,), dtype=torch.int32, device=dev)
        for t in (h_in, h_out, gate_out, mask_out, counts_out):
            assert t.is_contiguous()
        if attn_delta is not None:
            assert attn_delta.is_contiguous() and attn_delta.shape == (L, T, d)
        st = stream if stream is not None else torch.cuda.current_stream(dev)
        hero_routed_ffn_stack(self.model, T, h_in.data_ptr(),
                              attn_delta.data_ptr() if attn_delta is not None else 0,
                              tau, flags, mask_in.data_ptr() if mask_in is not None else 0,
                              h_out.data_ptr(), gate_out.data_ptr(), mask_out.data_ptr(),
                              counts_out.data_ptr(), st.cuda_stream)
        return h_out, gate_out, mask_out, counts_out

    def check(self, stream=None):
        import torch
        st = stream if stream is not None else torch.cuda.current_stream()
        hero_check_device_status(self.model, st.cuda_stream)

    def backward_init(self):
        """Transposed weight copies and workspace of the training path (hero_backward_init)."""
        hero_backward_init(self.model)

    def block_backward(self, block: int, h_bar, gate, mask, grad_out, flags: int = 0, stream=None):
        """Backward of block `block`'s branch part with its decisions fixed (device tensors).
        Returns (grad_h_bar [T, d], grad_gate [T], grad_w1 [d_r, d], grad_w2 [d, d_r])."""
        import torch
        T, d = h_bar.shape
        dev = h_bar.device
        r = self.cfg.d_r
        gh = torch.empty((T, d), dtype=torch.float32, device=dev)
        gg = torch.empty((T,), dtype=torch.float32, device=dev)
        g1 = torch.empty((r, d), dtype=torch.float32, device=dev)
        g2 = torch.empty((d, r), dtype=torch.float32, device=dev)
        for t in (h_bar, grad_out) + tuple(x for x in (gate, mask) if x is not None):
            assert t.is_contiguous()
        st = stream if stream is not None else torch.cuda.current_stream(dev)
        hero_routed_block_backward(self.model, block, T, h_bar.data_ptr(),
                                   gate.data_ptr() if gate is not None else 0,
                                   mask.data_ptr() if mask is not None else 0, grad_out.data_ptr(),
                                   flags, gh.data_ptr(), gg.data_ptr(), g1.data_ptr(), g2.data_ptr(),
                                   st.cuda_stream)
        return gh, gg, g1, g2


class HeroDecoder(HeroStack):
    """A routed stack with its attention sublayers: the full decoder forward."""

    def __init__(self, stack_cfg, weights: Dict[str, np.ndarray],
                 attn_weights: Dict[str, np.ndarray], max_tokens: Optional[int] = None):
        super().__init__(stack_cfg, weights, max_tokens)
        hero_attn_init(self.model, stack_cfg, attn_weights)

    def attention(self, layer: int, h, n_seqs: int, seq_len: int, h_bar=None, stream=None):
        """h_bar = h + Attn(LN_attn(h)) of one layer (1-based), device tensors."""
        import torch
        T, d = h.shape
        assert T == n_seqs * seq_len and h.is_contiguous()
        h_bar = h_bar if h_bar is not None else torch.empty_like(h)
        st = stream if stream is not None else torch.cuda.current_stream(h.device)
        hero_attention_block(self.model, layer, n_seqs, seq_len, h.data_ptr(), h_bar.data_ptr(),
                             st.cuda_stream)
        return h_bar

    def init_cache(self, max_seqs: int, max_len: int) -> None:
        hero_kv_cache_init(self.model, max_seqs, max_len)

    def _outs(self, T, dev, h_out, gate_out, mask_out, counts_out):
        import torch
        L, d = self.cfg.n_layers, self.cfg.d_model
        return (h_out if h_out is not None else torch.empty((T, d), dtype=torch.float32, device=dev),
                gate_out if gate_out is not None else torch.empty((L, T), dtype=torch.float32, device=dev),
                mask_out if mask_out is not None else torch.empty((L, T), dtype=torch.uint8, device=dev),
                counts_out if counts_out is not None else torch.empty((L,), dtype=torch.int32, device=dev))

    def prefill(self, h_in, tau: float, seq0: int, n_seqs: int, seq_len: int, flags: int = 0,
                mask_in=None, h_out=None, gate_out=None, mask_out=None, counts_out=None, stream=None):
        """Decoder forward on cache slots seq0 .. seq0 + n_seqs - 1, filling their cache."""
        import torch
        T = h_in.shape[0]
        assert T == n_seqs * seq_len and h_in.is_contiguous()
        outs = self._outs(T, h_in.device, h_out, gate_out, mask_out, counts_out)
        st = stream if stream is not None else torch.cuda.current_stream(h_in.device)
        hero_decoder_prefill(self.model, seq0, n_seqs, seq_len, h_in.data_ptr(), tau, flags,
                             mask_in.data_ptr() if mask_in is not None else 0,
                             *[o.data_ptr() for o in outs], st.cuda_stream)
        return outs

    def decode(self, h_in, positions, max_position: int, tau: float, flags: int = 0, mask_in=None,
               h_out=None, gate_out=None, mask_out=None, counts_out=None, stream=None):
        """One decoding step for cache slots 0 .. n - 1 (positions: device int32 [n])."""
        import torch
        n = h_in.shape[0]
        assert positions.dtype == torch.int32 and positions.numel() == n and h_in.is_contiguous()
        outs = self._outs(n, h_in.device, h_out, gate_out, mask_out, counts_out)
        st = stream if stream is not None else torch.cuda.current_stream(h_in.device)
        hero_decode_step(self.model, n, positions.data_ptr(), max_position, h_in.data_ptr(), tau,
                         flags, mask_in.data_ptr() if mask_in is not None else 0,
                         *[o.data_ptr() for o in outs], st.cuda_stream)
        return outs

    def forward(self, h_in, tau: float, n_seqs: int, seq_len: int, flags: int = 0, mask_in=None,
                h_out=None, gate_out=None, mask_out=None, counts_out=None, stream=None):
        """Device tensors in and out.  Returns (h_out, gate, mask, counts)."""
        import torch
        T, d = h_in.shape
        assert T == n_seqs * seq_len and h_in.is_contiguous()
        L = self.cfg.n_layers
        dev = h_in.device
        h_out = h_out if h_out is not None else torch.empty((T, d), dtype=torch.float32, device=dev)
        gate_out = gate_out if gate_out is not None else torch.empty((L, T), dtype=torch.float32, device=dev)
        mask_out = mask_out if mask_out is not None else torch.empty((L, T), dtype=torch.uint8, device=dev)
        counts_out = counts_out if counts_out is not None else torch.empty((L,), dtype=torch.int32, device=dev)
        st = stream if stream is not None else torch.cuda.current_stream(dev)
        hero_decoder_forward(self.model, n_seqs, seq_len, h_in.data_ptr(), tau, flags,
                             mask_in.data_ptr() if mask_in is not None else 0, h_out.data_ptr(),
                             gate_out.data_ptr(), mask_out.data_ptr(), counts_out.data_ptr(),
                             st.cuda_stream)
        return h_out, gate_out, mask_out, counts_out
