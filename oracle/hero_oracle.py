"""Plain float64 CPU oracle of HeRo's history-aware routed FFN stack.

TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and bench.py's
cpu_baseline leg may import or run this module; the CUDA product path never
does, and this module imports nothing from the product package.

What it computes (paper "Do Dynamic Routers Need Memory? HeRo", Sec. 3):
for each routed block j = 1..L_R and each token, in the paper's order,
    h_bar   = h + P_j                                   Eq. 1 (attention stand-in)
    delta, d, gamma                                     Eqs. 7-8 (transition features)
    x_path = [r, q_rem, d, gamma, p_hist, m_hist]       Eqs. 4, 6
    z_h = W_hu SiLU(W_hd RMSNorm(h_bar))                Eq. 5
    z_a = FFN_path(x_path);  s = [z_h; z_a]             Eq. 9
    q, k, v = W_q s, W_k s, W_v s                       Eq. 10
    c = phi(q)^T S / (phi(q)^T zeta + eps)              Eq. 11 (read before write)
    nu = 0 (j = 1) | 1 - cos(W_n s, W_c c)              Eq. 13
    a = f_theta([s; c; nu]); p_hist = sigma(a/T_hist)   Eq. 14
    m_hist = m_hist * p_hist                            Eq. 15
    b = f_psi(h_bar);  g = sigma(a + b)                 Eq. 16
    S = rho S + phi(k) v^T; zeta = rho zeta + phi(k)    Eq. 12, rho = sigma(eta_j)
    u = LN_ffn(h_bar)                                   Eq. 1
    h = h_bar + g FFN(u)          if g >= tau_exec      Eq. 3
        h_bar + (1-g) Adapter(u)  otherwise             Eqs. 2-3
Equation numbers count the displayed equations of Sec. 3 in order
(1 dense_attention, 2 adapter, 3 ffn_route, 4 path_vector, 5 hidden encoder,
6 depth features, 7 transition, 8 transition_features, 9 router_state,
10 q/k/v, 11 memory_read, 12 memory_update, 13 nu, 14 history head,
15 cumulative history, 16 final_gate).

Readings where the paper is silent (each listed in the design notes):
  * FFN = Llama SwiGLU W_down(SiLU(W_gate u) * W_up u), no biases.
  * RMSNorm(h) = h / sqrt(mean(h^2) + rms_eps) * gain; the router's RMSNorm has its
    own shared gain.  FFN_path, f_theta, f_psi = Linear+bias -> SiLU -> Linear+bias;
    matrices written without a bias in the paper (W_hd, W_hu, W_q, W_k, W_v, W_n,
    W_c, W_1, W_2) have none.
  * eps = 1e-6 in Eq. 8, Eq. 11 and the cosine of Eq. 13.
  * phi(x) = ELU(x) + 1 with alpha = 1.
  * decisions: g >= tau_exec -> FFN (ties go to the FFN).
  * precision contract for bf16 workloads: values are rounded to bf16 (nearest,
    ties to even) exactly at (i) every parameter (done by the input generator),
    (ii) the operands of the router's d-wide contraction: the weight
    bf16(W_hd diag(gain_r)) for the encoder (the row scale 1/rms is applied after
    the contraction, exact in real arithmetic) and f_psi's first-layer weight;
    the activation h_bar enters both as a pair of bf16 numbers,
    hi = bf16(h_bar), lo = bf16(h_bar - hi) (16 significant bits), because a
    single bf16 rounding of the router input makes the gates of a deep stack
    drift by ~1e-3 under perturbations of 1e-7 (rounding flips cascade through
    depth), (iii) u = LN_ffn(h_bar), the FFN and adapter input, (iv) the SwiGLU
    product entering W_down, (v) the adapter hidden SiLU(W_1 u) entering W_2.
    Everything else is float64 here.  f32 workloads round nowhere.

Modes: "route" (the method), "force" (decisions taken from mask_in, g still
computed and used as branch scale), "dense" (router skipped, every token through
the FFN with scale 1: the dense SwiGLU stack).

Router ablations (Sec. 4.4, component ablations), bits of `variant`:
  NO_HISTORY  the history branch is removed: g = sigma(b), the local logit alone;
              memory, path features and f_theta are not evaluated.
  NO_MEMREAD  the history head keeps its inputs s but loses the memory: c = 0 and
              nu = 0 enter f_theta; the memory is neither read nor written.
  NO_AUX      the auxiliary path encoder is removed: z_a = 0, s = [z_h; 0].
  NO_POS      the routing progress (r, q_rem) and residual transition (d, gamma)
              features are removed from x_path (zeroed); p_hist, m_hist remain.

Placement (Sec. 4.1): only a candidate set of FFN layers is routed; the others
stay dense.  With n_dense > 0 the first n_dense layers of the stack run the plain
FFN block (scale 1, no router, router state untouched) and layers
n_dense+1 .. n_layers are the routed blocks j = 1 .. L_R, L_R = n_layers - n_dense
(the routed index j and L_R enter the path features, Eqs. 4 and 6).
"""

from __future__ import annotations

from dataclasses import dataclass
from typing import Callable, Dict, List, Optional

import numpy as np


# ---------------------------------------------------------------------------
# Elementary functions
# ---------------------------------------------------------------------------

def bf16_round(x: np.ndarray) -> np.ndarray:
    """Nearest bf16 value of each float64 element, ties to even (8 significant bits).

    Written from the bf16 format definition: 1 sign, 8 exponent and 7 fraction bits,
    the same exponent range as IEEE binary32 (subnormal spacing 2^-133).
    """
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                        # x = m * 2^e, 0.5 <= |m| < 1
    e = np.maximum(e, -125)                   # below 2^-126 the spacing stays 2^-133
    spacing = np.ldexp(1.0, e - 8)            # 8 significant bits
    with np.errstate(invalid="ignore"):
        out = np.rint(x / spacing) * spacing  # np.rint rounds half to even
    return np.where(np.isfinite(x), out, x)


def _identity(x: np.ndarray) -> np.ndarray:
    return x


def bf16_pair(x: np.ndarray) -> np.ndarray:
    """x carried as two bf16 numbers, hi = bf16(x) and lo = bf16(x - hi): 16 significant bits."""
    hi = bf16_round(x)
    return hi + bf16_round(x - hi)


def sigmoid(x: np.ndarray) -> np.ndarray:
    """Logistic function sigma(x) = 1 / (1 + exp(-x))."""
    x = np.asarray(x, dtype=np.float64)
    with np.errstate(over="ignore"):
        return 1.0 / (1.0 + np.exp(-x))


def silu(x: np.ndarray) -> np.ndarray:
    """SiLU(x) = x * sigma(x)."""
    return x * sigmoid(x)


def phi(x: np.ndarray) -> np.ndarray:
    """Positive feature map phi(x) = ELU(x) + 1 (Sec. 3.2, before Eq. 11), alpha = 1."""
    x = np.asarray(x, dtype=np.float64)
    return np.where(x > 0, x + 1.0, np.exp(np.minimum(x, 0.0)))


def rms_norm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * gain."""
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * gain


def _mlp2(x, w1, b1, w2, b2):
    """Linear+bias -> SiLU -> Linear+bias (the two-layer heads and FFN_path)."""
    return silu(x @ w1.T + b1) @ w2.T + b2


# ---------------------------------------------------------------------------
# Configuration and parameters
# ---------------------------------------------------------------------------

# Router ablation bits (Sec. 4.4); the same values as the C ABI's HERO_ROUTER_*.
NO_HISTORY, NO_MEMREAD, NO_AUX, NO_POS = 1, 2, 4, 8


@dataclass
class OracleConfig:
    n_layers: int
    d_model: int
    d_ff: int
    d_r: int
    d_m: int
    d_h: int = 48
    d_a: int = 16
    d_enc: int = 256
    d_head: int = 256
    d_path: int = 16
    rms_eps: float = 1e-5
    eps: float = 1e-6
    t_hist: float = 0.9
    dtype: str = "f32"
    n_dense: int = 0          # leading FFN layers outside the candidate set (dense)
    variant: int = 0          # router ablation bits (NO_HISTORY | NO_MEMREAD | ...)

    @staticmethod
    def from_stack(c) -> "OracleConfig":
        return OracleConfig(c.n_layers, c.d_model, c.d_ff, c.d_r, c.d_m, c.d_h, c.d_a,
                            c.d_enc, c.d_head, c.d_path, c.rms_eps, c.eps, c.t_hist, c.dtype,
                            getattr(c, "n_dense", 0), getattr(c, "router_variant", 0))


def _f64(a) -> np.ndarray:
    """Decode a parameter/input array (float32, float64, or uint16 bf16 bits) to float64."""
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


# ---------------------------------------------------------------------------
# One routed block, step by step (Sec. 3.1-3.2)
# ---------------------------------------------------------------------------

def transition_features(j: int, h_bar, h_bar_prev, delta_prev, d_prev, eps):
    """Eqs. 7-8: delta_j = h_bar_j - h_bar_{j-1} (delta_1 = 0), d_j = ||delta_j||,
    gamma_j = <delta_j, delta_{j-1}> / (d_j d_{j-1} + eps) for j > 2, else 0."""
    if j == 1:
        delta = np.zeros_like(h_bar)
    else:
        delta = h_bar - h_bar_prev
    d = np.sqrt(np.sum(delta * delta, axis=1))
    if j > 2:
        gamma = np.sum(delta * delta_prev, axis=1) / (d * d_prev + eps)
    else:
        gamma = np.zeros_like(d)
    return delta, d, gamma


def path_vector(j: int, L: int, d, gamma, p_prev, m_prev):
    """Eq. 4 with Eq. 6: [r_j, q_rem_j, d_j, gamma_j, p_hist_{j-1}, m_hist_{j-1}]."""
    T = d.shape[0]
    r = np.full(T, j / L)
    q_rem = np.full(T, (L - j) / L)
    return np.stack([r, q_rem, d, gamma, p_prev, m_prev], axis=1)


def hidden_encoder(h_bar, w, cfg: OracleConfig, R, Rx):
    """Eq. 5: z_h = W_hu SiLU(W_hd RMSNorm(h_bar)).

    RMSNorm(h) = (h * gain_r) / rms(h); the contraction is written as
    (1/rms) * (W_hd diag(gain_r)) h so that the precision contract applies to
    the operands Rx(h_bar) and R(W_hd diag(gain_r)).
    """
    rinv = 1.0 / np.sqrt(np.mean(h_bar * h_bar, axis=1) + cfg.rms_eps)
    w_enc = R(w["w_hd"] * w["r_norm_g"][None, :])
    pre = rinv[:, None] * (Rx(h_bar) @ w_enc.T)
    return silu(pre) @ w["w_hu"].T


def path_encoder(x_path, w):
    """Eq. 9, first line: z_a = FFN_path(x_path) (Linear+bias, SiLU, Linear+bias)."""
    return _mlp2(x_path, w["path_w1"], w["path_b1"], w["path_w2"], w["path_b2"])


def memory_read(fq, S, zeta, eps):
    """Eq. 11: c = phi(q)^T S / (phi(q)^T zeta + eps), S[t] indexed [key m, value n]."""
    num = np.einsum("tm,tmn->tn", fq, S)
    den = np.einsum("tm,tm->t", fq, zeta)
    return num / (den + eps)[:, None]


def memory_write(S, zeta, fk, v, rho):
    """Eq. 12: S = rho S + phi(k) v^T;  zeta = rho zeta + phi(k)."""
    S_new = rho * S + np.einsum("tm,tn->tmn", fk, v)
    zeta_new = rho * zeta + fk
    return S_new, zeta_new


def history_dissimilarity(j: int, s, c, w, eps):
    """Eq. 13: nu_1 = 0; for j > 1, nu_j = 1 - cos(W_n s, W_c c)."""
    if j == 1:
        return np.zeros(s.shape[0])
    a = s @ w["w_n"].T
    b = c @ w["w_c"].T
    cos = np.sum(a * b, axis=1) / (np.linalg.norm(a, axis=1) * np.linalg.norm(b, axis=1) + eps)
    return 1.0 - cos


def history_head(s, c, nu, w):
    """Eq. 14, first part: a = f_theta([s; c; nu]) (scalar per token)."""
    x = np.concatenate([s, c, nu[:, None]], axis=1)
    return _mlp2(x, w["th_w1"], w["th_b1"], w["th_w2"], w["th_b2"])[:, 0]


def local_head(h_bar, w, Rx):
    """Eq. 16, first part: b = f_psi(h_bar); its first layer reads the operand Rx(h_bar)."""
    return _mlp2(Rx(h_bar), w["ps_w1"], w["ps_b1"], w["ps_w2"], w["ps_b2"])[:, 0]


def swiglu_ffn(u, wl, R):
    """Frozen FFN (Llama SwiGLU): W_down (SiLU(W_gate u) * W_up u)."""
    act = R(silu(u @ wl["w_gate"].T) * (u @ wl["w_up"].T))
    return act @ wl["w_down"].T


def adapter(u, wl, R):
    """Eq. 2: Adapter(u) = W_2 SiLU(W_1 u)."""
    return R(silu(u @ wl["ad_w1"].T)) @ wl["ad_w2"].T


# ---------------------------------------------------------------------------
# The attention sublayer of Eq. 1 (the full decoder forward)
# ---------------------------------------------------------------------------
# Readings (the paper keeps the backbone's attention, Sec. 3.1, and names Llama
# backbones, Sec. 4.1): Llama attention without biases; LN_attn is RMSNorm with
# its own gain; RoPE in the rotate-half form, inverse frequencies
# theta^(-2i/hd); causal softmax(q k^T / sqrt(hd)) per sequence; grouped-query
# heads (query head h reads key/value head h // (H / H_kv)).  Precision points
# for bf16 workloads: x = LN_attn(h), q and k after RoPE, v, the softmax
# probabilities entering P V, and the attention output entering W_o.

def rope_cos_sin(seq_len: int, hd: int, theta: float):
    """cos and sin tables [S, hd/2] of RoPE (position p, frequency theta^(-2i/hd))."""
    inv = theta ** (-np.arange(0, hd, 2, dtype=np.float64) / hd)
    ang = np.arange(seq_len, dtype=np.float64)[:, None] * inv[None, :]
    return np.cos(ang), np.sin(ang)


def apply_rope(x, cos, sin):
    """Rotate-half RoPE on x [..., S, hd]: each pair (x_i, x_{i+hd/2}) is rotated by
    position p times frequency i."""
    h = x.shape[-1] // 2
    x1, x2 = x[..., :h], x[..., h:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)


def attention_sublayer(h, wa, n_heads: int, n_kv_heads: int, theta: float, n_seqs: int,
                       seq_len: int, rms_eps: float, R=None):
    """Eq. 1, first line: h_bar = h + Attn(LN_attn(h)) on n_seqs sequences of seq_len
    tokens (rows of h in sequence order).  wa: attn_norm_g [d], w_q [H hd, d],
    w_k / w_v [H_kv hd, d], w_o [d, H hd] (float64)."""
    R = R or _identity
    T, d = h.shape
    hd = d // n_heads
    x = R(rms_norm(h, wa["attn_norm_g"], rms_eps))
    shape = lambda a, nh: a.reshape(n_seqs, seq_len, nh, hd).transpose(0, 2, 1, 3)
    q = shape(x @ wa["w_q"].T, n_heads)
    k = shape(x @ wa["w_k"].T, n_kv_heads)
    v = shape(x @ wa["w_v"].T, n_kv_heads)
    cos, sin = rope_cos_sin(seq_len, hd, theta)
    q, k, v = R(apply_rope(q, cos, sin)), R(apply_rope(k, cos, sin)), R(v)
    group = n_heads // n_kv_heads
    k = np.repeat(k, group, axis=1)
    v = np.repeat(v, group, axis=1)
    scores = q @ k.transpose(0, 1, 3, 2) / np.sqrt(hd)                   # [B, H, S, S]
    scores = np.where(np.tril(np.ones((seq_len, seq_len), dtype=bool)), scores, -np.inf)
    scores = scores - scores.max(axis=-1, keepdims=True)
    p = np.exp(scores)
    p = R(p / p.sum(axis=-1, keepdims=True))
    o = R(p @ v).transpose(0, 2, 1, 3).reshape(T, n_heads * hd)
    return h + o @ wa["w_o"].T


def attention_rows(h_seq, rows, wa, n_heads: int, n_kv_heads: int, theta: float,
                   rms_eps: float, R=None):
    """attention_sublayer restricted to query positions `rows` of ONE sequence h_seq
    [S, d] (keys and values of all its positions): h_bar[rows].  The same steps in
    the same order, for checking long sequences on a sample of positions."""
    R = R or _identity
    S, d = h_seq.shape
    hd = d // n_heads
    rows = np.asarray(rows)
    last = int(rows.max()) + 1                                   # causal: keys < last suffice
    x = R(rms_norm(h_seq[:last], wa["attn_norm_g"], rms_eps))
    cos, sin = rope_cos_sin(last, hd, theta)
    q = (x[rows] @ wa["w_q"].T).reshape(len(rows), n_heads, hd).transpose(1, 0, 2)
    k = (x @ wa["w_k"].T).reshape(last, n_kv_heads, hd).transpose(1, 0, 2)
    v = (x @ wa["w_v"].T).reshape(last, n_kv_heads, hd).transpose(1, 0, 2)
    q = R(apply_rope(q, cos[rows], sin[rows]))
    k, v = R(apply_rope(k, cos, sin)), R(v)
    group = n_heads // n_kv_heads
    k = np.repeat(k, group, axis=0)
    v = np.repeat(v, group, axis=0)
    scores = q @ k.transpose(0, 2, 1) / np.sqrt(hd)                   # [H, rows, last]
    scores = np.where(np.arange(last)[None, None, :] <= rows[None, :, None], scores, -np.inf)
    scores = scores - scores.max(axis=-1, keepdims=True)
    p = np.exp(scores)
    p = R(p / p.sum(axis=-1, keepdims=True))
    o = R(p @ v).transpose(1, 0, 2).reshape(len(rows), n_heads * hd)
    return h_seq[rows] + o @ wa["w_o"].T


# ---------------------------------------------------------------------------
# The stack
# ---------------------------------------------------------------------------

_LAYER_KEYS = ("ffn_norm_g", "w_gate", "w_up", "w_down", "ad_w1", "ad_w2")
_SHARED_KEYS = ("r_norm_g", "w_hd", "w_hu", "path_w1", "path_b1", "path_w2", "path_b2",
                "w_q", "w_k", "w_v", "w_n", "w_c", "th_w1", "th_b1", "th_w2", "th_b2",
                "ps_w1", "ps_b1", "ps_w2", "ps_b2")


def routed_ffn_stack(cfg: OracleConfig, weights: Dict[str, np.ndarray], h_in, attn_delta,
                     tau: float, mode: str = "route", mask_in=None,
                     branch_scale: str = "gate", record: bool = False,
                     hooks: Optional[Dict[str, Callable]] = None,
                     attn: Optional[Callable] = None) -> Dict[str, object]:
    """Run the routed FFN stack on tokens h_in [T, d].

    attn_delta: [L, T, d] attention stand-in (None = zero).
    attn: optional callable (layer index from 0, h) -> h_bar that replaces the stand-in
    with a real attention sublayer (the full decoder forward; attn_delta is ignored).
    mode: "route" | "force" (mask_in [L, T] gives decisions; rows of the dense
    prefix are ignored) | "dense".
    branch_scale: "gate" (Eq. 3: g and 1 - g) or "one" (unscaled branches).
    Returns h_out [T, d], gate [L, T], mask [L, T] (uint8), counts [L] (FFN tokens)
    and, if record, per-layer intermediates under "layers".
    """
    if mode not in ("route", "force", "dense"):
        raise ValueError(mode)
    if mode == "force" and mask_in is None:
        raise ValueError("force mode needs mask_in")
    R = bf16_round if cfg.dtype == "bf16" else _identity
    Rx = bf16_pair if cfg.dtype == "bf16" else _identity   # router activation operand
    hk = hooks or {}
    L = cfg.n_layers
    n_dense = cfg.n_dense
    if not 0 <= n_dense < L:
        raise ValueError("need 0 <= n_dense < n_layers")
    L_R = L - n_dense                                               # routed blocks
    h = _f64(h_in)
    T = h.shape[0]
    w = {k: _f64(weights[k]) for k in _SHARED_KEYS}
    eta = _f64(weights["eta"])

    S = np.zeros((T, cfg.d_m, cfg.d_m))
    zeta = np.zeros((T, cfg.d_m))
    p_prev = np.ones(T)            # p_hist_{l_0} = 1
    m_prev = np.ones(T)            # m_hist_{l_0} = 1
    h_bar_prev = None
    delta_prev = None
    d_prev = np.zeros(T)
    gates = np.zeros((L, T))
    masks = np.zeros((L, T), dtype=np.uint8)
    counts = np.zeros(L, dtype=np.int64)
    layers: List[Dict[str, np.ndarray]] = []

    for layer in range(1, L + 1):
        wl = {k: _f64(weights[k][layer - 1]) for k in _LAYER_KEYS}
        if attn is not None:
            h_bar = attn(layer - 1, h)                              # Eq. 1
        else:
            P = 0.0 if attn_delta is None else _f64(attn_delta[layer - 1])
            h_bar = h + P                                           # Eq. 1 stand-in
        rec: Dict[str, np.ndarray] = {"h_bar": h_bar}
        j = layer - n_dense                                         # routed index (Sec. 4.1)
        dense_layer = mode == "dense" or j < 1
        if dense_layer:
            g = np.ones(T)
            decide = np.ones(T, dtype=bool)
        elif cfg.variant & NO_HISTORY:                              # ablation: local logit
            b = local_head(h_bar, w, Rx)                            # Eq. 16
            g = sigmoid(b)
            if mode == "route":
                decide = g >= tau
            else:
                decide = np.asarray(mask_in[layer - 1]).astype(bool)
            if record:
                rec.update(b=b)
        else:
            delta, d, gamma = transition_features(j, h_bar, h_bar_prev, delta_prev,
                                                  d_prev, cfg.eps)
            x_path = path_vector(j, L_R, d, gamma, p_prev, m_prev)
            if cfg.variant & NO_POS:                                # ablation: no progress /
                x_path[:, :4] = 0.0                                 # transition features
            z_h = hidden_encoder(h_bar, w, cfg, R, Rx)
            z_a = path_encoder(x_path, w)
            if cfg.variant & NO_AUX:                                # ablation: no path encoder
                z_a = np.zeros_like(z_a)
            s = np.concatenate([z_h, z_a], axis=1)                 # Eq. 9
            q = s @ w["w_q"].T                                      # Eq. 10
            k = s @ w["w_k"].T
            v = s @ w["w_v"].T
            fq = hk.get("phi", phi)(q)
            fk = hk.get("phi", phi)(k)
            if cfg.variant & NO_MEMREAD:                            # ablation: no memory access
                c = np.zeros((T, cfg.d_m))
                nu = np.zeros(T)
            else:
                c = memory_read(fq, S, zeta, cfg.eps)               # Eq. 11 (before write)
                nu = history_dissimilarity(j, s, c, w, cfg.eps)     # Eq. 13
            a = history_head(s, c, nu, w)                           # Eq. 14
            p = sigmoid(a / cfg.t_hist)
            m = m_prev * p                                          # Eq. 15
            b = local_head(h_bar, w, Rx)                            # Eq. 16
            g = sigmoid(a + b)
            if "gate" in hk:                                        # test hook: g override
                g = hk["gate"](layer, g)
            rho = sigmoid(eta[layer - 1])
            if not cfg.variant & NO_MEMREAD:
                S, zeta = memory_write(S, zeta, fk, v, rho)         # Eq. 12
            if mode == "route":
                decide = g >= tau                                   # Eq. 3 threshold
            else:
                decide = np.asarray(mask_in[layer - 1]).astype(bool)
            if record:
                rec.update(delta=delta, d=d, gamma=gamma, x_path=x_path, z_h=z_h, z_a=z_a,
                           s=s, q=q, k=k, v=v, c=c, nu=nu, a=a, b=b, p=p, m=m,
                           S=S.copy(), zeta=zeta.copy(), rho=np.float64(rho))
            h_bar_prev, delta_prev, d_prev = h_bar, delta, d
            p_prev, m_prev = p, m

        u = R(rms_norm(h_bar, wl["ffn_norm_g"], cfg.rms_eps))       # Eq. 1, u = LN_ffn(h_bar)
        if dense_layer or branch_scale == "one":
            sf = np.ones(T)
            sa = np.ones(T)
        else:
            sf, sa = g, 1.0 - g
        h_new = h_bar.copy()
        F = np.nonzero(decide)[0]
        A = np.nonzero(~decide)[0]
        if F.size:
            h_new[F] += sf[F, None] * swiglu_ffn(u[F], wl, R)       # Eq. 3, g >= tau
        if A.size:
            h_new[A] += sa[A, None] * adapter(u[A], wl, R)          # Eq. 3, g < tau
        gates[layer - 1] = g
        masks[layer - 1] = decide.astype(np.uint8)
        counts[layer - 1] = F.size
        if record:
            rec.update(g=g, mask=decide.copy(), u=u, h=h_new)
            layers.append(rec)
        h = h_new

    out: Dict[str, object] = {"h_out": h, "gate": gates, "mask": masks, "counts": counts}
    if record:
        out["layers"] = layers
    return out


def decoder_forward(cfg: OracleConfig, weights, attn_weights, h_in, tau: float, n_heads: int,
                    n_kv_heads: int, theta: float, n_seqs: int, seq_len: int, **kw):
    """The full decoder forward: each block's h_bar comes from the attention sublayer
    (Eq. 1) instead of the stand-in; everything else as routed_ffn_stack."""
    R = bf16_round if cfg.dtype == "bf16" else _identity
    wa_all = {k: _f64(v) for k, v in attn_weights.items()}

    def attn(j, h):
        wa = {k: v[j] for k, v in wa_all.items()}
        return attention_sublayer(h, wa, n_heads, n_kv_heads, theta, n_seqs, seq_len,
                                  cfg.rms_eps, R)

    return routed_ffn_stack(cfg, weights, h_in, None, tau, attn=attn, **kw)


def bypass_fraction(masks: np.ndarray, n_dense: int = 0) -> float:
    """Share of the routed blocks' FFN executions replaced by the adapter:
    sum_j n_a,j / (L_R T), over the routed blocks only (rows n_dense.. of masks)."""
    m = np.asarray(masks)[n_dense:]
    return float(1.0 - m.mean()) if m.size else 0.0


# ---------------------------------------------------------------------------
# Training objective (Sec. 3.3), for gradient checks of the training path
# ---------------------------------------------------------------------------

# Parameters the training path optimises (Sec. 3.3: the backbone - FFN, its norm gain
# and attention - is frozen; adapters, state encoders, depth memory and router heads
# are trained).
TRAINABLE = ("ad_w1", "ad_w2", "eta", "r_norm_g", "w_hd", "w_hu", "path_w1", "path_b1",
             "path_w2", "path_b2", "w_q", "w_k", "w_v", "w_n", "w_c", "th_w1", "th_b1",
             "th_w2", "th_b2", "ps_w1", "ps_b1", "ps_w2", "ps_b2")


def skip_penalty(gates, n_seqs: int, seq_len: int, n_dense: int = 0) -> float:
    """L_skip (Sec. 3.3): for each sequence and each of its seq_len - 1 next-token
    positions, the square of the token's summed gates over the routed blocks, averaged
    over B (T - 1).  gates [L, n_seqs seq_len], tokens in sequence order; rows of the
    dense prefix carry no gate."""
    g = np.asarray(gates, dtype=np.float64)[n_dense:]
    g = g.reshape(g.shape[0], n_seqs, seq_len)[:, :, :seq_len - 1]
    return float(np.sum(np.sum(g, axis=0) ** 2) / (n_seqs * (seq_len - 1)))


def training_loss(cfg: OracleConfig, weights, h_in, attn_delta, mask, G, alpha: float,
                  n_seqs: int, seq_len: int, hooks=None) -> float:
    """L = <G, h_out> + alpha L_skip with the decisions fixed to mask [L, T]: the
    threshold of Eq. 3 is not differentiated, the selected branch's scale g or 1 - g
    carries the gradient to the router (Sec. 3.1).  G [T, d] is a synthetic upstream
    gradient standing in for dL_LM / dh_out (no language-model head or data)."""
    out = routed_ffn_stack(cfg, weights, h_in, attn_delta, 0.0, mode="force", mask_in=mask,
                           hooks=hooks)
    return float(np.sum(np.asarray(G, dtype=np.float64) * out["h_out"])) + \
        alpha * skip_penalty(out["gate"], n_seqs, seq_len, cfg.n_dense)


def directional_derivative(f: Callable[[float], float], h: float) -> float:
    """Central difference (f(h) - f(-h)) / 2h of a function of the step along a direction."""
    return (f(h) - f(-h)) / (2.0 * h)


def silu_grad(x: np.ndarray) -> np.ndarray:
    """d SiLU / dx = sigma(x) (1 + x (1 - sigma(x)))."""
    s = sigmoid(x)
    return s * (1.0 + x * (1.0 - s))


def rms_norm_backward(x, gain, eps: float, du):
    """Gradient of u = RMSNorm(x) gain with respect to x, given du (last axis):
    r = (mean(x^2) + eps)^(-1/2), u = x r gain, so
    dx = r (du gain) - x r^3 mean(x (du gain))."""
    r = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)
    dg = du * gain
    return r * dg - x * r ** 3 * np.mean(x * dg, axis=-1, keepdims=True)


def block_branch_backward(h_bar, g, decide, G, wl, rms_eps: float):
    """Backward of the branch part of a routed block with its decisions fixed (Eq. 3,
    Eq. 2, the SwiGLU FFN and LN_ffn), for the training path (Sec. 3.3: the backbone
    is frozen, the adapter trains, and the selected branch's scale g or 1 - g carries
    the gradient to the router):
        h_out = h_bar + s * Branch(u),  u = LN_ffn(h_bar),
        s = g, Branch = FFN for decide; s = 1 - g, Branch = Adapter otherwise,
    given G = dL/dh_out [T, d].  Returns dL/dh_bar (residual plus branch path),
    dL/dg [T], and dL/dW_1 [d_r, d], dL/dW_2 [d, d_r] of the adapter.  float64, no
    rounding (the f32 model)."""
    G = np.asarray(G, dtype=np.float64)
    T, d = h_bar.shape
    u = rms_norm(h_bar, wl["ffn_norm_g"], rms_eps)
    du = np.zeros((T, d))
    dg = np.zeros(T)
    dW1 = np.zeros_like(wl["ad_w1"])
    dW2 = np.zeros_like(wl["ad_w2"])
    F = np.nonzero(decide)[0]
    A = np.nonzero(~np.asarray(decide, dtype=bool))[0]
    if F.size:   # h += g W_down (SiLU(W_gate u) * W_up u)
        uf = u[F]
        gate, up = uf @ wl["w_gate"].T, uf @ wl["w_up"].T
        y = (silu(gate) * up) @ wl["w_down"].T
        dg[F] = np.sum(G[F] * y, axis=1)
        dy = g[F, None] * G[F]
        dact = dy @ wl["w_down"]
        dgate = dact * up * silu_grad(gate)
        dup = dact * silu(gate)
        du[F] = dgate @ wl["w_gate"] + dup @ wl["w_up"]
    if A.size:   # h += (1 - g) W_2 SiLU(W_1 u)
        ua = u[A]
        a = ua @ wl["ad_w1"].T
        hid = silu(a)
        y = hid @ wl["ad_w2"].T
        dg[A] = -np.sum(G[A] * y, axis=1)
        dy = (1.0 - g[A])[:, None] * G[A]
        dW2 = dy.T @ hid
        da = (dy @ wl["ad_w2"]) * silu_grad(a)
        dW1 = da.T @ ua
        du[A] = da @ wl["ad_w1"]
    dh_bar = G + rms_norm_backward(h_bar, wl["ffn_norm_g"], rms_eps, du)
    return {"dh_bar": dh_bar, "dg": dg, "dW1": dW1, "dW2": dW2}


def skip_penalty_grad(gates, n_seqs: int, seq_len: int, n_dense: int = 0):
    """d L_skip / d g [L, T]: 2 / (B (T - 1)) times the token's summed routed gates at its
    next-token positions, 0 at a sequence's last position and in dense-prefix rows."""
    g = np.asarray(gates, dtype=np.float64)
    out = np.zeros_like(g)
    tot = g[n_dense:].sum(axis=0)
    pos = np.arange(g.shape[1]) % seq_len
    out[n_dense:] = np.where(pos < seq_len - 1, 2.0 / (n_seqs * (seq_len - 1)) * tot, 0.0)[None, :]
    return out
