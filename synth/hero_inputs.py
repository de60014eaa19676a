"""Seeded synthetic workloads for the HeRo routed FFN stack.

This module is shared by the CUDA path's harness (bench, tests) and by the CPU
oracle.  It holds shapes, seeds and value distributions only: none of the
method's arithmetic lives here.

Workloads stand in for the paper's Llama backbones and data (Sec. 4.1: Llama-3.1-8B,
Llama-2-7B, Llama-2-13B, Tulu-3 sequences truncated to 2048 tokens): no trained
weights or datasets are available, so every tensor is drawn from a seeded
distribution with the backbone's FFN shapes.

Distributions (all i.i.d. normal, per element):
  * FFN W_gate, W_up ~ N(0, 0.02^2); W_down ~ N(0, (0.02/sqrt(2 L))^2)
  * FFN-norm gain and router RMSNorm gain: 1 + N(0, 0.02^2)
  * adapter W_1, W_2 ~ N(0, 0.02^2)
  * router projections (W_hd, W_hu, FFN_path, W_q, W_k, W_v, W_n, W_c, both heads)
    ~ N(0, 1/fan_in); biases ~ N(0, 0.1^2)
  * forgetting parameter eta_j = logit(0.98) + N(0, 0.25^2)  (rho = sigma(eta) ~ 0.98, Sec. 4.1)
  * hidden-state input h_0 ~ N(0, 1); attention stand-in P_j ~ N(0, 0.1^2)
In bf16 workloads every parameter and every P_j element is rounded to the
nearest bf16 value (round-to-nearest-even) at generation, so both sides receive
the identical bf16 numbers; h_0 stays fp32.

Random streams are keyed (seed, tensor tag, chunk) with fixed 4 Mi-element
chunks, so the values do not depend on the number of generator threads.
"""

from __future__ import annotations

import json
import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field, asdict
from typing import Dict, Optional, Sequence

import numpy as np

_CHUNK = 1 << 22


@dataclass(frozen=True)
class StackConfig:
    """Shape and workload of one routed FFN stack."""

    name: str
    n_layers: int          # L_R routed layers
    d_model: int           # d
    d_ff: int              # I, SwiGLU intermediate width
    d_r: int               # adapter rank
    d_m: int               # memory key/value width
    n_tokens: int          # T (flattened batch x sequence)
    dtype: str             # "f32" or "bf16"
    bypass: float          # target share of adapter executions (Sec. 4.1 budgets)
    d_h: int = 48          # hidden-state encoding width (Sec. 4.1: 48 of 64)
    d_a: int = 16          # path-feature encoding width (Sec. 4.1: 16 of 64)
    d_enc: int = 256       # inner width of the hidden encoder W_hd
    d_head: int = 256      # hidden width of both routing heads (Sec. 4.1)
    d_path: int = 16       # hidden width of FFN_path
    rms_eps: float = 1e-5
    eps: float = 1e-6
    t_hist: float = 0.9    # T_hist (Sec. 4.1)
    seed: int = 0
    batch: int = 1         # sequences (for reporting only; tokens are independent)
    seq_len: int = 0
    n_dense: int = 0       # leading FFN layers outside the routing candidate set (Sec. 4.1)
    router_variant: int = 0  # Sec. 4.4 router ablation bits (1 history, 2 memread, 4 aux, 8 pos)
    # attention sublayer of the full decoder forward (Eq. 1; 0 heads: the additive stand-in)
    n_heads: int = 0
    n_kv_heads: int = 0
    rope_theta: float = 10000.0
    # KV-cache decoding: a step is one new token for each of `batch` sequences at
    # position seq_len (n_tokens = batch); tau comes from the workload named here
    kv_decode_of: str = ""

    @property
    def d_s(self) -> int:
        return self.d_h + self.d_a

    def replace(self, **kw) -> "StackConfig":
        d = asdict(self)
        d.update(kw)
        return StackConfig(**d)


CONFIGS: Dict[str, StackConfig] = {
    "tiny_f32": StackConfig("tiny_f32", 4, 256, 688, 16, 16, 64, "f32", 0.27,
                            batch=1, seq_len=64),
    "llama2_7b_prefill": StackConfig("llama2_7b_prefill", 32, 4096, 11008, 64, 64, 2048,
                                     "bf16", 0.27, batch=1, seq_len=2048),
    "llama31_8b_prefill": StackConfig("llama31_8b_prefill", 32, 4096, 14336, 64, 64, 16384,
                                      "bf16", 0.2687, batch=4, seq_len=4096),
    "llama31_8b_decode": StackConfig("llama31_8b_decode", 32, 4096, 14336, 64, 64, 64,
                                     "bf16", 0.3882, batch=64, seq_len=1),
    "llama2_13b_prefill": StackConfig("llama2_13b_prefill", 40, 5120, 13824, 64, 64, 8192,
                                      "bf16", 0.27, batch=2, seq_len=4096),
    # Small bf16 stack used for full-token parity: several 128-row and 256-column tiles
    # plus ragged tails, small enough that the oracle covers every token in seconds.
    "small_bf16": StackConfig("small_bf16", 4, 512, 1024, 64, 64, 333, "bf16", 0.27,
                              batch=1, seq_len=333),
    # The paper's placement (Sec. 4.1): candidates are the latter half of the layers,
    # the adapter has d_r = 896, and the 25% budget is of all parameters of
    # Llama-3.1-8B (8.03e9): 0.25 * 8.03e9 / (16 * (3 d I - 2 d d_r)) = 74.3% of the
    # routed blocks' executions take the adapter.
    "llama31_8b_paper": StackConfig("llama31_8b_paper", 32, 4096, 14336, 896, 64, 16384, "bf16",
                                    0.7432, batch=4, seq_len=4096, n_dense=16),
    # The same placement at small shapes for full-token parity: a dense prefix, and an
    # adapter rank that is not a multiple of 64 (a ragged K tail in the tensor-core
    # up projection, a partial N tile in the down projection).
    "small_bf16_placed": StackConfig("small_bf16_placed", 4, 512, 1024, 96, 64, 333, "bf16",
                                     0.5, batch=1, seq_len=333, n_dense=2),
    # Full decoder forward (Eq. 1 with real attention): small shapes for full-token parity
    # (2 sequences of 160 tokens, 4 heads sharing 2 KV heads, head_dim 128) and
    # Llama-3.1-8B prefill shapes (32 heads, 8 KV heads, head_dim 128, RoPE base 5e5).
    "small_bf16_decoder": StackConfig("small_bf16_decoder", 4, 512, 1024, 64, 64, 320, "bf16",
                                      0.27, batch=2, seq_len=160, n_heads=4, n_kv_heads=2,
                                      rope_theta=500000.0),
    "llama31_8b_decoder": StackConfig("llama31_8b_decoder", 32, 4096, 14336, 64, 64, 16384,
                                      "bf16", 0.2687, batch=4, seq_len=4096, n_heads=32,
                                      n_kv_heads=8, rope_theta=500000.0),
    # KV-cache decoding with the same model: 64 sequences whose 4096-token prefixes are
    # in the cache, one new token each per step (T = 64 per step)
    "llama31_8b_kvdecode": StackConfig("llama31_8b_kvdecode", 32, 4096, 14336, 64, 64, 64,
                                       "bf16", 0.2687, batch=64, seq_len=4096, n_heads=32,
                                       n_kv_heads=8, rope_theta=500000.0,
                                       kv_decode_of="llama31_8b_decoder"),
}

# The 13B workload is swept over these bypass targets.
BYPASS_SWEEP_13B = (0.0, 0.27, 0.39)


# Parameter table: name -> (shape function, per-layer?, init kind, init argument).
def _shapes(c: StackConfig):
    d, I, r, L = c.d_model, c.d_ff, c.d_r, c.n_layers
    ds, dm, dh, de, dH, dp = c.d_s, c.d_m, c.d_h, c.d_enc, c.d_head, c.d_path
    return [
        # per routed block (frozen FFN + trainable adapter + forgetting parameter)
        ("ffn_norm_g", (L, d), "gain", 0.02),
        ("w_gate", (L, I, d), "normal", 0.02),
        ("w_up", (L, I, d), "normal", 0.02),
        ("w_down", (L, d, I), "normal", 0.02 / math.sqrt(2 * L)),
        ("ad_w1", (L, r, d), "normal", 0.02),
        ("ad_w2", (L, d, r), "normal", 0.02),
        ("eta", (L,), "eta", 0.25),
        # shared router parameters
        ("r_norm_g", (d,), "gain", 0.02),
        ("w_hd", (de, d), "fan_in", d),
        ("w_hu", (dh, de), "fan_in", de),
        ("path_w1", (dp, 6), "fan_in", 6),
        ("path_b1", (dp,), "normal", 0.1),
        ("path_w2", (c.d_a, dp), "fan_in", dp),
        ("path_b2", (c.d_a,), "normal", 0.1),
        ("w_q", (dm, ds), "fan_in", ds),
        ("w_k", (dm, ds), "fan_in", ds),
        ("w_v", (dm, ds), "fan_in", ds),
        ("w_n", (dm, ds), "fan_in", ds),
        ("w_c", (dm, dm), "fan_in", dm),
        ("th_w1", (dH, ds + dm + 1), "fan_in", ds + dm + 1),
        ("th_b1", (dH,), "normal", 0.1),
        ("th_w2", (1, dH), "fan_in", dH),
        ("th_b2", (1,), "normal", 0.1),
        ("ps_w1", (dH, d), "fan_in", d),
        ("ps_b1", (dH,), "normal", 0.1),
        ("ps_w2", (1, dH), "fan_in", dH),
        ("ps_b2", (1,), "normal", 0.1),
    ]


WEIGHT_NAMES = tuple(n for n, *_ in _shapes(CONFIGS["tiny_f32"]))
_TAG = {n: i + 1 for i, n in enumerate(WEIGHT_NAMES)}
_TAG_H = 101
_TAG_P = 102
_TAG_ATTN = {"attn_norm_g": 201, "w_q": 202, "w_k": 203, "w_v": 204, "w_o": 205}
ATTN_WEIGHT_NAMES = tuple(_TAG_ATTN)


def round_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest even (data encoding)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float32 (exact)."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _threads(threads: Optional[int]) -> int:
    if threads:
        return threads
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


def _fill_normal(out_flat: np.ndarray, key: Sequence[int], mean: float, std: float,
                 to_bf16: bool, threads: Optional[int]) -> None:
    """Fill out_flat (float32 or uint16 bf16 bits) with N(mean, std^2) draws.

    Chunk c of the flat tensor is drawn from default_rng([*key, c]).
    """
    n = out_flat.size
    nchunks = (n + _CHUNK - 1) // _CHUNK

    def work(c: int) -> None:
        lo, hi = c * _CHUNK, min(n, (c + 1) * _CHUNK)
        rng = np.random.default_rng([*key, c])
        v = rng.standard_normal(hi - lo, dtype=np.float32)
        if std != 1.0:
            v *= np.float32(std)
        if mean != 0.0:
            v += np.float32(mean)
        if to_bf16:
            out_flat[lo:hi] = round_to_bf16_bits(v)
        else:
            out_flat[lo:hi] = v

    nt = min(_threads(threads), nchunks)
    if nt <= 1:
        for c in range(nchunks):
            work(c)
    else:
        with ThreadPoolExecutor(nt) as ex:
            list(ex.map(work, range(nchunks)))


def generate_weights(cfg: StackConfig, threads: Optional[int] = None,
                     bf16_bits: bool = True) -> Dict[str, np.ndarray]:
    """All stack parameters, canonical [out, in] layouts, stacked over layers.

    f32 workloads return float32 arrays.  bf16 workloads return uint16 bf16 bit
    patterns when bf16_bits (the default), else the same values as float32.
    """
    out: Dict[str, np.ndarray] = {}
    is_bf16 = cfg.dtype == "bf16"
    logit98 = math.log(0.98 / 0.02)
    for name, shape, kind, arg in _shapes(cfg):
        if kind == "normal":
            mean, std = 0.0, float(arg)
        elif kind == "gain":
            mean, std = 1.0, float(arg)
        elif kind == "fan_in":
            mean, std = 0.0, 1.0 / math.sqrt(arg)
        elif kind == "eta":
            mean, std = logit98, float(arg)
        else:  # pragma: no cover
            raise ValueError(kind)
        as_bits = is_bf16 and bf16_bits
        arr = np.empty(int(np.prod(shape)), dtype=np.uint16 if as_bits else np.float32)
        _fill_normal(arr, (cfg.seed, _TAG[name]), mean, std, as_bits, threads)
        arr = arr.reshape(shape)
        if is_bf16 and not bf16_bits:
            arr = bf16_bits_to_f32(round_to_bf16_bits(arr))
        out[name] = arr
    return out


def attn_shapes(cfg: StackConfig):
    """Attention parameters per layer (Llama layout, no biases): gain of LN_attn,
    W_q [H hd, d], W_k and W_v [H_kv hd, d], W_o [d, H hd]; hd = d / H."""
    L, d, H, Hkv = cfg.n_layers, cfg.d_model, cfg.n_heads, cfg.n_kv_heads
    hd = d // H
    return [("attn_norm_g", (L, d), "gain", 0.02), ("w_q", (L, H * hd, d), "normal", 0.02),
            ("w_k", (L, Hkv * hd, d), "normal", 0.02), ("w_v", (L, Hkv * hd, d), "normal", 0.02),
            ("w_o", (L, d, H * hd), "normal", 0.02 / math.sqrt(2 * L))]


def generate_attn_weights(cfg: StackConfig, threads: Optional[int] = None) -> Dict[str, np.ndarray]:
    """Attention parameters (seed s, own stream tags), encoded like generate_weights."""
    if not cfg.n_heads:
        raise ValueError("the workload has no attention sublayer (n_heads = 0)")
    out: Dict[str, np.ndarray] = {}
    is_bf16 = cfg.dtype == "bf16"
    for name, shape, kind, arg in attn_shapes(cfg):
        mean, std = (1.0, float(arg)) if kind == "gain" else (0.0, float(arg))
        arr = np.empty(int(np.prod(shape)), dtype=np.uint16 if is_bf16 else np.float32)
        _fill_normal(arr, (cfg.seed, _TAG_ATTN[name]), mean, std, is_bf16, threads)
        out[name] = arr.reshape(shape)
    return out


def generate_h_in(cfg: StackConfig, n_tokens: Optional[int] = None,
                  threads: Optional[int] = None) -> np.ndarray:
    """Input hidden states h_0 ~ N(0,1), float32 [T, d] (seed + 2)."""
    T = cfg.n_tokens if n_tokens is None else n_tokens
    arr = np.empty(T * cfg.d_model, dtype=np.float32)
    _fill_normal(arr, (cfg.seed + 2, _TAG_H, T), 0.0, 1.0, False, threads)
    return arr.reshape(T, cfg.d_model)


def generate_attn_delta(cfg: StackConfig, n_tokens: Optional[int] = None,
                        threads: Optional[int] = None) -> np.ndarray:
    """Attention stand-in P_j ~ N(0, 0.1^2) per (layer, token, dim) (seed + 1).

    Returns [L, T, d]: uint16 bf16 bits for bf16 workloads, float32 otherwise.
    It replaces Attn(LN(h)) in Eq. 1 (dense_attention) so that h_bar_j = h_{j-1} + P_j.
    """
    T = cfg.n_tokens if n_tokens is None else n_tokens
    is_bf16 = cfg.dtype == "bf16"
    arr = np.empty(cfg.n_layers * T * cfg.d_model, dtype=np.uint16 if is_bf16 else np.float32)
    _fill_normal(arr, (cfg.seed + 1, _TAG_P, T), 0.0, 0.1, is_bf16, threads)
    return arr.reshape(cfg.n_layers, T, cfg.d_model)


def to_f64(a: np.ndarray) -> np.ndarray:
    """Decode a generated tensor (float32, or uint16 bf16 bits) to float64."""
    if a.dtype == np.uint16:
        return bf16_bits_to_f32(a).astype(np.float64)
    return np.asarray(a, dtype=np.float64)


def sample_tokens(T: int, n: int) -> np.ndarray:
    """A fixed, evenly spread token subset (includes the first and last token)."""
    if n >= T:
        return np.arange(T)
    return np.unique(np.linspace(0, T - 1, n).round().astype(np.int64))


_TAU_FILE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "tau.json")


def calibrated_tau(name: str, bypass: Optional[float] = None) -> float:
    """Execution threshold tau_exec calibrated (by the oracle) to the workload's budget."""
    with open(_TAU_FILE) as f:
        table = json.load(f)
    cfg = CONFIGS[name]
    if cfg.kv_decode_of:   # the decoding workload runs the model of its prefill workload
        return calibrated_tau(cfg.kv_decode_of, bypass)
    b = cfg.bypass if bypass is None else bypass
    key = f"{name}@{b:.4f}"
    if key not in table["tau"]:
        raise KeyError(f"no calibrated tau for {key}; run synth/calibrate_tau.py")
    return float(table["tau"][key]["tau"])
