"""Gradients of the training objective (Sec. 3.3) by reverse-mode differentiation.

Test infrastructure, like the rest of oracle/: only tests/ may import it.

A float64 PyTorch restatement of the routed stack (oracle/hero_oracle.py,
routed_ffn_stack) for the f32 model (no rounding), with the decisions fixed as the
training path fixes them (the threshold of Eq. 3 is not differentiated; the selected
branch's scale g or 1 - g carries the gradient to the router, Sec. 3.1).  The
parameters are leaf tensors, so autograd gives dL/dtheta for every trainable tensor
(adapters, state encoders, depth memory, router heads) and dL/dh_in, for

    L = <G, h_out> + alpha L_skip,

G a synthetic upstream gradient standing in for dL_LM/dh_out.  The restatement follows
the same equations in the same order as the NumPy oracle; tests pin its forward to the
NumPy oracle's and its gradients to central differences of the NumPy objective, so a
GPU backward can be compared with these gradients element by element.
"""

from __future__ import annotations

from typing import Dict, Iterable, Tuple

import numpy as np
import torch

from oracle import hero_oracle as ho


def _t(a) -> torch.Tensor:
    return torch.as_tensor(ho._f64(a))


def _silu(x):
    return x * torch.sigmoid(x)


def _phi(x):
    """ELU(x) + 1 (Sec. 3.2)."""
    return torch.where(x > 0, x + 1.0, torch.exp(torch.clamp(x, max=0.0)))


def _rms_norm(x, gain, eps):
    return x / torch.sqrt(torch.mean(x * x, dim=-1, keepdim=True) + eps) * gain


def _mlp2(x, w1, b1, w2, b2):
    return _silu(x @ w1.T + b1) @ w2.T + b2


def stack_loss_and_grads(cfg: ho.OracleConfig, weights: Dict[str, np.ndarray], h_in, attn_delta,
                         mask, G, alpha: float, n_seqs: int, seq_len: int,
                         wrt: Iterable[str] = ho.TRAINABLE + ("h_in",)
                         ) -> Tuple[float, Dict[str, np.ndarray]]:
    """L and its gradients with respect to `wrt` (parameter names, and "h_in").
    mask [L, T] fixes the decisions; attn_delta [L, T, d] (None = zero)."""
    if cfg.dtype != "f32" or cfg.variant:
        raise ValueError("the restatement covers the f32 model without ablations")
    wrt = tuple(wrt)
    P = {k: _t(v).requires_grad_(k in wrt) for k, v in weights.items()}
    h = _t(h_in).requires_grad_("h_in" in wrt)
    L, n_dense = cfg.n_layers, cfg.n_dense
    L_R = L - n_dense
    T = h.shape[0]
    S = torch.zeros((T, cfg.d_m, cfg.d_m), dtype=torch.float64)
    zeta = torch.zeros((T, cfg.d_m), dtype=torch.float64)
    p_prev = torch.ones(T, dtype=torch.float64)
    m_prev = torch.ones(T, dtype=torch.float64)
    h_bar_prev = delta_prev = None
    d_prev = torch.zeros(T, dtype=torch.float64)
    gates = []
    x = h
    for layer in range(1, L + 1):
        wl = {k: P[k][layer - 1] for k in ("ffn_norm_g", "w_gate", "w_up", "w_down", "ad_w1", "ad_w2")}
        h_bar = x + (0.0 if attn_delta is None else _t(attn_delta[layer - 1]))   # Eq. 1 stand-in
        j = layer - n_dense
        decide = torch.as_tensor(np.asarray(mask[layer - 1]).astype(bool))
        if j < 1:                                       # dense prefix: the plain FFN block
            g = torch.ones(T, dtype=torch.float64)
            decide = torch.ones(T, dtype=torch.bool)
        else:
            if j == 1:                                  # Eqs. 7-8
                delta = torch.zeros_like(h_bar)
                d = torch.zeros(T, dtype=torch.float64)
            else:
                delta = h_bar - h_bar_prev
                d = torch.sqrt(torch.sum(delta * delta, dim=1))
            gamma = (torch.sum(delta * delta_prev, dim=1) / (d * d_prev + cfg.eps) if j > 2
                     else torch.zeros(T, dtype=torch.float64))
            x_path = torch.stack([torch.full((T,), j / L_R, dtype=torch.float64),
                                  torch.full((T,), (L_R - j) / L_R, dtype=torch.float64),
                                  d, gamma, p_prev, m_prev], dim=1)          # Eqs. 4, 6
            rinv = 1.0 / torch.sqrt(torch.mean(h_bar * h_bar, dim=1) + cfg.rms_eps)
            pre = rinv[:, None] * (h_bar @ (P["w_hd"] * P["r_norm_g"][None, :]).T)
            z_h = _silu(pre) @ P["w_hu"].T                                     # Eq. 5
            z_a = _mlp2(x_path, P["path_w1"], P["path_b1"], P["path_w2"], P["path_b2"])
            s = torch.cat([z_h, z_a], dim=1)                                    # Eq. 9
            q, k, v = s @ P["w_q"].T, s @ P["w_k"].T, s @ P["w_v"].T            # Eq. 10
            fq, fk = _phi(q), _phi(k)
            c = torch.einsum("tm,tmn->tn", fq, S) / (torch.einsum("tm,tm->t", fq, zeta) + cfg.eps)[:, None]
            if j == 1:                                                          # Eq. 13
                nu = torch.zeros(T, dtype=torch.float64)
            else:
                an, bc = s @ P["w_n"].T, c @ P["w_c"].T
                nu = 1.0 - torch.sum(an * bc, dim=1) / (
                    torch.linalg.norm(an, dim=1) * torch.linalg.norm(bc, dim=1) + cfg.eps)
            a = _mlp2(torch.cat([s, c, nu[:, None]], dim=1), P["th_w1"], P["th_b1"], P["th_w2"],
                      P["th_b2"])[:, 0]                                         # Eq. 14
            p = torch.sigmoid(a / cfg.t_hist)
            m = m_prev * p                                                      # Eq. 15
            b = _mlp2(h_bar, P["ps_w1"], P["ps_b1"], P["ps_w2"], P["ps_b2"])[:, 0]   # Eq. 16
            g = torch.sigmoid(a + b)
            rho = torch.sigmoid(P["eta"][layer - 1])
            S = rho * S + torch.einsum("tm,tn->tmn", fk, v)                     # Eq. 12
            zeta = rho * zeta + fk
            h_bar_prev, delta_prev, d_prev = h_bar, delta, d
            p_prev, m_prev = p, m
            gates.append(g)
        u = _rms_norm(h_bar, wl["ffn_norm_g"], cfg.rms_eps)
        ffn = (_silu(u @ wl["w_gate"].T) * (u @ wl["w_up"].T)) @ wl["w_down"].T
        ad = _silu(u @ wl["ad_w1"].T) @ wl["ad_w2"].T
        x = h_bar + torch.where(decide[:, None], g[:, None] * ffn, (1.0 - g)[:, None] * ad)  # Eq. 3
    loss = torch.sum(_t(G) * x)
    if gates:                                                                   # L_skip
        gs = torch.stack(gates).reshape(len(gates), n_seqs, seq_len)[:, :, :seq_len - 1]
        loss = loss + alpha * torch.sum(torch.sum(gs, dim=0) ** 2) / (n_seqs * (seq_len - 1))
    loss.backward()
    grads = {k: P[k].grad.numpy().copy() for k in wrt if k != "h_in"}
    if "h_in" in wrt:
        grads["h_in"] = h.grad.numpy().copy()
    return float(loss.detach()), grads
