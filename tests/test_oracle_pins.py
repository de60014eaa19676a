"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each check compares the oracle with something other than itself: a library
routine (torch's bf16 conversion, F.rms_norm, F.silu, F.elu), a textbook stack
(dense SwiGLU, Houlsby adapter), a closed form (the memory as an explicit
weighted sum, the second-block read, transition features of a branch-free
stack, the zero-router gate), invariants (ranges, token independence,
causality of decisions by brute force over all paths) and an independent
per-token pure-Python restatement on tiny shapes.  The last group plants
plausible mistakes in the oracle and shows that a pin catches each one.
"""

import math
import struct

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import hero_oracle as ho
from synth import hero_inputs as hi

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _tiny(dtype="f32", **kw):
    base = hi.CONFIGS["tiny_f32"] if dtype == "f32" else hi.CONFIGS["small_bf16"]
    return base.replace(**kw) if kw else base


def _inputs(cfg):
    return hi.generate_weights(cfg), hi.generate_h_in(cfg), hi.generate_attn_delta(cfg)


def _w64(w):
    return {k: hi.to_f64(v) for k, v in w.items()}


def _t(x):
    return torch.as_tensor(np.asarray(x, dtype=np.float64))


def _tbf16(x: torch.Tensor) -> torch.Tensor:
    """Library bf16 rounding (torch) of a float64 tensor, through float32."""
    return x.to(torch.float32).to(torch.bfloat16).to(torch.float64)


# ---------------------------------------------------------------------------
# Elementary functions against library routines
# ---------------------------------------------------------------------------

def test_bf16_round_matches_torch():
    rng = np.random.default_rng(5)
    x = np.concatenate([rng.standard_normal(200000) * 10.0 ** rng.integers(-30, 30, 200000),
                        [0.0, -0.0, 1.0, -1.0, 3.0e38, 1e-40, -1e-42]])
    x32 = x.astype(np.float32).astype(np.float64)      # f32-representable: no double rounding
    # exact ties between two bf16 neighbours must go to the even one
    ties = (np.arange(1, 2000, dtype=np.float64) * 2.0 + 1.0) * 2.0 ** -8 + 1.0
    for v in (x32, ties, -ties):
        ref = torch.tensor(v, dtype=torch.float32).to(torch.bfloat16).to(torch.float64).numpy()
        np.testing.assert_array_equal(ho.bf16_round(v), ref)


def test_bf16_pair_is_a_16_bit_split():
    """hi = bf16(x), lo = bf16(x - hi): both bf16 (torch agrees), |x - (hi + lo)| <= 2^-16 |x|."""
    rng = np.random.default_rng(7)
    x = (rng.standard_normal(100000) * 10.0 ** rng.integers(-5, 5, 100000)).astype(np.float32)
    x = x.astype(np.float64)
    pair = ho.bf16_pair(x)
    hi = torch.tensor(x, dtype=torch.float32).to(torch.bfloat16).to(torch.float64)
    lo = (torch.tensor(x) - hi).to(torch.float32).to(torch.bfloat16).to(torch.float64)
    np.testing.assert_array_equal(pair, (hi + lo).numpy())
    assert np.all(np.abs(x - pair) <= 2.0 ** -16 * np.abs(x))


def test_elementwise_functions_match_torch():
    x = np.linspace(-30, 30, 10001)
    np.testing.assert_allclose(ho.sigmoid(x), torch.sigmoid(_t(x)).numpy(), rtol=1e-15, atol=1e-300)
    np.testing.assert_allclose(ho.silu(x), F.silu(_t(x)).numpy(), rtol=1e-14, atol=1e-300)
    # torch forms ELU(x) + 1 as expm1(x) + 1, which cancels for x << 0: absolute bound
    np.testing.assert_allclose(ho.phi(x), (F.elu(_t(x)) + 1.0).numpy(), rtol=1e-15, atol=1e-15)
    g = np.linspace(0.5, 1.5, 64)
    hbar = np.random.default_rng(1).standard_normal((7, 64)) * 3
    np.testing.assert_allclose(ho.rms_norm(hbar, g, 1e-5),
                               F.rms_norm(_t(hbar), (64,), _t(g), 1e-5).numpy(), rtol=1e-14)


# ---------------------------------------------------------------------------
# P1 / P1': dense stack and adapter stack against textbook restatements
# ---------------------------------------------------------------------------

def _textbook_dense(cfg, w, h, P, bf16):
    """Textbook residual SwiGLU stack h_j = h_{j-1} + P_j + W_d(SiLU(W_g u) * W_u u)."""
    r = _tbf16 if bf16 else (lambda x: x)
    W = _w64(w)
    x = _t(h)
    for j in range(cfg.n_layers):
        hb = x + _t(hi.to_f64(P[j]))
        u = r(F.rms_norm(hb, (cfg.d_model,), _t(W["ffn_norm_g"][j]), cfg.rms_eps))
        act = r(F.silu(u @ _t(W["w_gate"][j]).T) * (u @ _t(W["w_up"][j]).T))
        x = hb + act @ _t(W["w_down"][j]).T
    return x.numpy()


def _textbook_adapter(cfg, w, h, P, bf16):
    """Houlsby bottleneck-adapter stack h_j = h_{j-1} + P_j + W_2 SiLU(W_1 u)."""
    r = _tbf16 if bf16 else (lambda x: x)
    W = _w64(w)
    x = _t(h)
    for j in range(cfg.n_layers):
        hb = x + _t(hi.to_f64(P[j]))
        u = r(F.rms_norm(hb, (cfg.d_model,), _t(W["ffn_norm_g"][j]), cfg.rms_eps))
        x = hb + r(F.silu(u @ _t(W["ad_w1"][j]).T)) @ _t(W["ad_w2"][j]).T
    return x.numpy()


def check_dense(cfg):
    w, h, P = _inputs(cfg)
    out = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P, 0.5, mode="dense")
    ref = _textbook_dense(cfg, w, h, P, cfg.dtype == "bf16")
    return np.max(np.abs(out["h_out"] - ref)) / np.max(np.abs(ref)), out


def test_p1_dense_equals_textbook_swiglu_stack_f32():
    err, out = check_dense(_tiny())
    assert err < 1e-13
    assert (out["mask"] == 1).all() and (out["gate"] == 1).all()


def test_p1_dense_equals_textbook_swiglu_stack_bf16():
    # torch rounds float64 -> bf16 through float32; rare double-rounding cases move
    # single elements by one bf16 step, hence the looser bound.
    err, _ = check_dense(_tiny("bf16"))
    assert err < 1e-4


def check_adapter_stack(cfg):
    w, h, P = _inputs(cfg)
    zeros = np.zeros((cfg.n_layers, cfg.n_tokens), dtype=np.uint8)
    out = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P, 0.5, mode="force",
                              mask_in=zeros, branch_scale="one")
    ref = _textbook_adapter(cfg, w, h, P, cfg.dtype == "bf16")
    return np.max(np.abs(out["h_out"] - ref)) / np.max(np.abs(ref))


def test_p1p_all_adapter_equals_houlsby_stack():
    assert check_adapter_stack(_tiny()) < 1e-13
    assert check_adapter_stack(_tiny("bf16")) < 1e-4


# ---------------------------------------------------------------------------
# Eq. 3: branch choice and gate scaling, layer by layer
# ---------------------------------------------------------------------------

def check_branch_scaling(cfg, tau):
    w, h, P = _inputs(cfg)
    W = _w64(w)
    out = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P, tau, record=True)
    worst = 0.0
    for j, rec in enumerate(out["layers"]):
        hb = _t(rec["h_bar"])
        g = _t(rec["g"])[:, None]
        u = F.rms_norm(hb, (cfg.d_model,), _t(W["ffn_norm_g"][j]), cfg.rms_eps)
        ffn = (F.silu(u @ _t(W["w_gate"][j]).T) * (u @ _t(W["w_up"][j]).T)) @ _t(W["w_down"][j]).T
        ada = F.silu(u @ _t(W["ad_w1"][j]).T) @ _t(W["ad_w2"][j]).T
        m = torch.as_tensor(rec["g"] >= tau)[:, None]
        assert (m[:, 0].numpy() == rec["mask"]).all()
        ref = torch.where(m, hb + g * ffn, hb + (1 - g) * ada)
        worst = max(worst, float((ref - _t(rec["h"])).abs().max()))
    return worst, out


def test_eq3_branch_choice_and_scaling():
    cfg = _tiny()
    worst, out = check_branch_scaling(cfg, hi.calibrated_tau("tiny_f32"))
    assert worst < 1e-13
    assert 0 < out["mask"].sum() < out["mask"].size


# ---------------------------------------------------------------------------
# P2 / P3: the depth memory against closed forms
# ---------------------------------------------------------------------------

def _phi_t(x):
    return (F.elu(_t(x)) + 1.0).numpy()


def check_memory_closed_form(cfg, eta=None):
    w, h, P = _inputs(cfg)
    if eta is not None:
        w = dict(w)
        w["eta"] = np.full(cfg.n_layers, eta, dtype=np.float32)
    out = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P, 0.4, record=True)
    lay = out["layers"]
    eta64 = hi.to_f64(w["eta"])
    rho = 1.0 / (1.0 + np.exp(-eta64))
    worst_S = worst_c = 0.0
    for j in range(len(lay)):
        # S_j = sum_{i<=j} (prod_{m=i+1..j} rho_m) phi(k_i) v_i^T ; zeta likewise
        S = np.zeros_like(lay[j]["S"])
        Z = np.zeros_like(lay[j]["zeta"])
        for i in range(j + 1):
            decay = np.prod(rho[i + 1:j + 1])
            fk = _phi_t(lay[i]["k"])
            S += decay * fk[:, :, None] * lay[i]["v"][:, None, :]
            Z += decay * fk
        worst_S = max(worst_S, np.max(np.abs(S - lay[j]["S"])) / (np.max(np.abs(S)) + 1e-300),
                      np.max(np.abs(Z - lay[j]["zeta"])) / np.max(np.abs(Z)))
        # c_j reads S_{j-1}: a weighted sum of v_1..v_{j-1}
        fq = _phi_t(lay[j]["q"])
        num = np.zeros_like(lay[j]["c"])
        den = np.zeros(fq.shape[0])
        for i in range(j):
            wgt = np.prod(rho[i + 1:j]) * np.sum(fq * _phi_t(lay[i]["k"]), axis=1)
            num += wgt[:, None] * lay[i]["v"]
            den += wgt
        c = num / (den + cfg.eps)[:, None]
        worst_c = max(worst_c, np.max(np.abs(c - lay[j]["c"])))
    return worst_S, worst_c, out


def test_p2_memory_equals_explicit_weighted_sum():
    ws, wc, out = check_memory_closed_form(_tiny())
    assert ws < 1e-12 and wc < 1e-12
    ws, wc, _ = check_memory_closed_form(_tiny("bf16"))
    assert ws < 1e-12 and wc < 1e-12


def test_p2_rho_one_is_causal_linear_attention():
    """With rho = 1 the read is Katharopoulos causal linear attention over depth."""
    cfg = _tiny()
    w, h, P = _inputs(cfg)
    w = dict(w)
    w["eta"] = np.full(cfg.n_layers, 60.0, dtype=np.float32)   # sigma(60) == 1.0 in float64
    out = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P, 0.4, record=True)
    lay = out["layers"]
    q = torch.stack([_t(l["q"]) for l in lay], 1)               # [T, L, dm]
    k = torch.stack([_t(l["k"]) for l in lay], 1)
    v = torch.stack([_t(l["v"]) for l in lay], 1)
    fq, fk = F.elu(q) + 1, F.elu(k) + 1
    kv = torch.cumsum(fk[..., :, None] * v[..., None, :], dim=1)  # inclusive prefix sums
    ks = torch.cumsum(fk, dim=1)
    kv = torch.cat([torch.zeros_like(kv[:, :1]), kv[:, :-1]], 1)   # strictly earlier blocks
    ks = torch.cat([torch.zeros_like(ks[:, :1]), ks[:, :-1]], 1)
    c = torch.einsum("tlm,tlmn->tln", fq, kv) / (torch.einsum("tlm,tlm->tl", fq, ks) + cfg.eps)[..., None]
    got = torch.stack([_t(l["c"]) for l in lay], 1)
    assert float((c - got).abs().max()) < 1e-12


def check_second_block(cfg):
    w, h, P = _inputs(cfg)
    out = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P, 0.4, record=True)
    l1, l2 = out["layers"][0], out["layers"][1]
    x = np.sum(_phi_t(l2["q"]) * _phi_t(l1["k"]), axis=1)
    c2 = l1["v"] * (x / (x + cfg.eps))[:, None]
    return max(np.max(np.abs(l1["c"])), np.max(np.abs(c2 - l2["c"]))), out


def test_p3_first_and_second_block_reads():
    err, out = check_second_block(_tiny())
    assert err < 1e-13
    l1 = out["layers"][0]
    assert (l1["nu"] == 0).all() and (l1["d"] == 0).all() and (l1["gamma"] == 0).all()
    assert (out["layers"][1]["gamma"] == 0).all()


# ---------------------------------------------------------------------------
# P4: ranges and recurrences
# ---------------------------------------------------------------------------

def test_p4_ranges_and_recurrences():
    cfg = _tiny()
    w, h, P = _inputs(cfg)
    out = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P,
                              hi.calibrated_tau("tiny_f32"), record=True)
    m_acc = np.ones(cfg.n_tokens)
    for j, l in enumerate(out["layers"], start=1):
        xp = l["x_path"]
        assert np.allclose(xp[:, 0] + xp[:, 1], 1.0)
        assert np.allclose(xp[:, 0], j / cfg.n_layers)
        m_acc = m_acc * l["p"]
        np.testing.assert_allclose(l["m"], m_acc, rtol=1e-14)
        assert ((l["p"] > 0) & (l["p"] < 1)).all() and ((l["g"] > 0) & (l["g"] < 1)).all()
        assert (np.abs(l["gamma"]) <= 1).all() and ((l["nu"] >= 0) & (l["nu"] <= 2)).all()
        assert (l["zeta"] > 0).all()
        if j > 1:
            assert np.allclose(xp[:, 4], out["layers"][j - 2]["p"])
            assert np.allclose(xp[:, 5], out["layers"][j - 2]["m"])
        else:
            assert (xp[:, 4] == 1).all() and (xp[:, 5] == 1).all()


# ---------------------------------------------------------------------------
# Closed forms with designed parameters
# ---------------------------------------------------------------------------

def check_transition_closed_form(cfg):
    """Branch-free stack (W_down = W_2 = 0): h_bar_j - h_bar_{j-1} = P_j exactly."""
    w, h, _ = _inputs(cfg)
    w = dict(w)
    w["w_down"] = np.zeros_like(w["w_down"])
    w["ad_w2"] = np.zeros_like(w["ad_w2"])
    rng = np.random.default_rng(3)
    P = np.empty((cfg.n_layers, cfg.n_tokens, cfg.d_model))
    P[0] = rng.standard_normal(P[0].shape) * 0.1
    for j in range(1, cfg.n_layers):            # correlated so that gamma is far from 0
        P[j] = 0.8 * P[j - 1] * (-1) ** j + 0.2 * rng.standard_normal(P[0].shape) * 0.1
    out = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P, 0.4, record=True)
    worst = 0.0
    for j, l in enumerate(out["layers"], start=1):
        if j == 1:
            d_ref = np.zeros(cfg.n_tokens)
            g_ref = np.zeros(cfg.n_tokens)
        else:
            d_ref = np.linalg.norm(P[j - 1], axis=1)
            if j > 2:
                g_ref = np.sum(P[j - 1] * P[j - 2], axis=1) / (
                    d_ref * np.linalg.norm(P[j - 2], axis=1) + cfg.eps)
            else:
                g_ref = np.zeros(cfg.n_tokens)
        worst = max(worst, np.max(np.abs(l["d"] - d_ref)), np.max(np.abs(l["gamma"] - g_ref)))
    return worst, out


def test_transition_features_closed_form():
    worst, out = check_transition_closed_form(_tiny())
    assert worst < 1e-12
    assert np.abs(out["layers"][2]["gamma"]).mean() > 0.5


def test_zero_router_closed_form():
    """All router matrices zero, biases kept: every quantity has a closed form."""
    cfg = _tiny()
    w, h, P = _inputs(cfg)
    w = dict(w)
    for k in ("w_hd", "w_hu", "path_w1", "path_w2", "w_q", "w_k", "w_v", "w_n", "w_c",
              "th_w1", "th_w2", "ps_w1", "ps_w2"):
        w[k] = np.zeros_like(w[k])
    out = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P, 0.5, record=True)
    bt2, bp2 = float(w["th_b2"][0]), float(w["ps_b2"][0])
    p = 1 / (1 + math.exp(-bt2 / cfg.t_hist))
    for j, l in enumerate(out["layers"], start=1):
        np.testing.assert_allclose(l["g"], 1 / (1 + math.exp(-(bt2 + bp2))), rtol=1e-14)
        np.testing.assert_allclose(l["p"], p, rtol=1e-14)
        np.testing.assert_allclose(l["m"], p ** j, rtol=1e-13)
        np.testing.assert_allclose(l["s"][:, cfg.d_h:], np.broadcast_to(w["path_b2"], (cfg.n_tokens, cfg.d_a)))
        assert (l["s"][:, :cfg.d_h] == 0).all() and (l["c"] == 0).all()
        np.testing.assert_allclose(l["nu"], 0.0 if j == 1 else 1.0)
        np.testing.assert_allclose(l["zeta"], sum(np.prod(1 / (1 + np.exp(-hi.to_f64(w["eta"][i + 1:j]))))
                                                  for i in range(j)), rtol=1e-13)


# ---------------------------------------------------------------------------
# P5: brute force over every forced path (causality of decisions)
# ---------------------------------------------------------------------------

def check_path_brute_force(cfg, tau):
    w, h, P = _inputs(cfg)
    oc = ho.OracleConfig.from_stack(cfg)
    free = ho.routed_ffn_stack(oc, w, h, P, tau)
    L, T = cfg.n_layers, cfg.n_tokens
    consistent = np.zeros((2 ** L, T), dtype=bool)
    for pi in range(2 ** L):
        path = np.array([(pi >> j) & 1 for j in range(L)], dtype=np.uint8)
        forced = ho.routed_ffn_stack(oc, w, h, P, tau, mode="force",
                                     mask_in=np.repeat(path[:, None], T, axis=1))
        consistent[pi] = ((forced["gate"] >= tau) == path[:, None].astype(bool)).all(axis=0)
    n_consistent = consistent.sum(axis=0)
    chosen = np.argmax(consistent, axis=0)
    free_code = sum(free["mask"][j].astype(np.int64) << j for j in range(L))
    return n_consistent, chosen, free_code


def test_p5_unique_self_consistent_path_is_the_free_run():
    n, chosen, free_code = check_path_brute_force(_tiny(), hi.calibrated_tau("tiny_f32"))
    assert (n == 1).all()
    assert (chosen == free_code).all()
    assert len(np.unique(free_code)) > 3


# ---------------------------------------------------------------------------
# P6: token independence;  P7: budget
# ---------------------------------------------------------------------------

def test_p6_token_independence():
    cfg = _tiny()
    w, h, P = _inputs(cfg)
    oc = ho.OracleConfig.from_stack(cfg)
    tau = hi.calibrated_tau("tiny_f32")
    full = ho.routed_ffn_stack(oc, w, h, P, tau)
    perm = np.random.default_rng(0).permutation(cfg.n_tokens)
    permuted = ho.routed_ffn_stack(oc, w, h[perm], P[:, perm], tau)
    np.testing.assert_array_equal(permuted["h_out"], full["h_out"][perm])
    np.testing.assert_array_equal(permuted["mask"], full["mask"][:, perm])
    sub = np.arange(5, 40, 3)
    part = ho.routed_ffn_stack(oc, w, h[sub], P[:, sub], tau)
    np.testing.assert_allclose(part["h_out"], full["h_out"][sub], rtol=1e-14, atol=1e-14)
    np.testing.assert_array_equal(part["mask"], full["mask"][:, sub])


def test_p7_budget_tiny():
    cfg = _tiny()
    w, h, P = _inputs(cfg)
    out = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P,
                              hi.calibrated_tau("tiny_f32"))
    assert abs(ho.bypass_fraction(out["mask"]) - cfg.bypass) <= 1.0 / (cfg.n_layers * cfg.n_tokens)
    np.testing.assert_array_equal(out["counts"], out["mask"].sum(axis=1))


# ---------------------------------------------------------------------------
# P8: independent per-token, per-element pure-Python restatement (tiny shapes)
# ---------------------------------------------------------------------------

def _bf16_bits(x: float) -> float:
    """Scalar round-to-nearest-even to bf16 from the float64 bit pattern: keep the sign,
    the 11 exponent bits and the top 7 of the 52 fraction bits, rounding on the 45
    dropped bits (ties to an even kept part; a carry moves into the exponent).
    Independent of the oracle's frexp-based bf16_round; normal bf16 range only."""
    if x == 0.0:
        return x
    b = struct.unpack("<Q", struct.pack("<d", x))[0]
    sign, mag = b & (1 << 63), b & ((1 << 63) - 1)
    assert (mag >> 52) >= 1023 - 126, "bf16 subnormals are outside these tests"
    keep, rest = mag >> 45, mag & ((1 << 45) - 1)
    if rest > (1 << 44) or (rest == (1 << 44) and keep & 1):
        keep += 1
    return struct.unpack("<d", struct.pack("<Q", sign | (keep << 45)))[0]


def _py_stack(cfg, W, h_in, P, tau, n_dense=0, variant=0, bf16=False):
    """Per-token loops over scalars, written from Sec. 3 without numpy linear algebra.
    The first n_dense layers are plain FFN blocks (Sec. 4.1 placement); the rest are
    routed blocks j = 1 .. L - n_dense.  variant: the Sec. 4.4 ablations, bits
    1 = w/o History (g from the local logit), 2 = w/o MemRead (c = 0, nu = 0, no
    memory), 4 = w/o Aux State (z_a = 0), 8 = w/o Pos State (r, q_rem, d, gamma = 0).
    bf16: the bf16 models' precision contract (parameters already bf16 values), a
    bf16 rounding r() at exactly these points: the router contraction's weight
    r(W_hd[o][i] g_r[i]) with its 1/rms row scale applied after the sum; the router's
    d-wide activation (encoder and f_psi's first layer) as the pair r(x) + r(x - r(x));
    u = LN_ffn(h_bar); the SwiGLU product; the adapter hidden SiLU(W_1 u)."""
    L, d = cfg.n_layers, cfg.d_model
    LR = L - n_dense
    r = _bf16_bits if bf16 else (lambda x: x)

    def pair(x):
        hi_ = r(x)
        return hi_ + r(x - hi_)

    def mv(M, x):
        return [sum(M[o][i] * x[i] for i in range(len(x))) for o in range(len(M))]

    def ffn(layer, u):
        gt, up = mv(W["w_gate"][layer - 1], u), mv(W["w_up"][layer - 1], u)
        return mv(W["w_down"][layer - 1], [r(sl(x) * z) for x, z in zip(gt, up)])

    def adp(layer, u):
        return mv(W["ad_w2"][layer - 1], [r(sl(x)) for x in mv(W["ad_w1"][layer - 1], u)])

    def ln_ffn(layer, hb):
        rf = math.sqrt(sum(x * x for x in hb) / d + cfg.rms_eps)
        return [r(hb[i] / rf * W["ffn_norm_g"][layer - 1][i]) for i in range(d)]

    def f_psi(hb):
        xp = [pair(x) for x in hb] if bf16 else hb
        hl = [sl(x + b) for x, b in zip(mv(W["ps_w1"], xp), W["ps_b1"])]
        return sum(x * y for x, y in zip(W["ps_w2"][0], hl)) + W["ps_b2"][0]

    def encoder_pre(hb):
        rms = math.sqrt(sum(x * x for x in hb) / d + cfg.rms_eps)
        if not bf16:
            nr = [hb[i] / rms * W["r_norm_g"][i] for i in range(d)]
            return mv(W["w_hd"], nr)
        xp = [pair(x) for x in hb]
        return [sum(r(W["w_hd"][o][i] * W["r_norm_g"][i]) * xp[i] for i in range(d)) / rms
                for o in range(len(W["w_hd"]))]

    def sg(x):
        return 1.0 / (1.0 + math.exp(-x))

    def sl(x):
        return x * sg(x)

    def ph(x):
        return x + 1.0 if x > 0 else math.exp(x)

    out_h, out_g = [], []
    for t in range(len(h_in)):
        h = list(h_in[t])
        dm = cfg.d_m
        S = [[0.0] * dm for _ in range(dm)]
        Z = [0.0] * dm
        p_prev = m_prev = 1.0
        hb_prev = dl_prev = None
        d_prev = 0.0
        gs = []
        for layer in range(1, L + 1):
            hb = [h[i] + P[layer - 1][t][i] for i in range(d)]
            if layer <= n_dense:
                y = ffn(layer, ln_ffn(layer, hb))
                h = [hb[i] + y[i] for i in range(d)]
                gs.append(1.0)
                continue
            j = layer - n_dense
            if variant & 1:                                    # w/o History
                g = sg(f_psi(hb))
                u = ln_ffn(layer, hb)
                if g >= tau:
                    y = ffn(layer, u)
                    h = [hb[i] + g * y[i] for i in range(d)]
                else:
                    y = adp(layer, u)
                    h = [hb[i] + (1 - g) * y[i] for i in range(d)]
                gs.append(g)
                continue
            if j == 1:
                dl = [0.0] * d
            else:
                dl = [hb[i] - hb_prev[i] for i in range(d)]
            dd = math.sqrt(sum(x * x for x in dl))
            gam = 0.0
            if j > 2:
                gam = sum(dl[i] * dl_prev[i] for i in range(d)) / (dd * d_prev + cfg.eps)
            zh = mv(W["w_hu"], [sl(x) for x in encoder_pre(hb)])
            xp = [j / LR, (LR - j) / LR, dd, gam, p_prev, m_prev]
            if variant & 8:                                    # w/o Pos State
                xp = [0.0, 0.0, 0.0, 0.0, p_prev, m_prev]
            hid = [sl(x + b) for x, b in zip(mv(W["path_w1"], xp), W["path_b1"])]
            za = [x + b for x, b in zip(mv(W["path_w2"], hid), W["path_b2"])]
            if variant & 4:                                    # w/o Aux State
                za = [0.0] * len(za)
            s = zh + za
            q, k, v = mv(W["w_q"], s), mv(W["w_k"], s), mv(W["w_v"], s)
            fq, fk = [ph(x) for x in q], [ph(x) for x in k]
            den = sum(fq[m] * Z[m] for m in range(dm)) + cfg.eps
            c = [sum(fq[m] * S[m][n] for m in range(dm)) / den for n in range(dm)]
            if variant & 2:                                    # w/o MemRead
                c = [0.0] * dm
                nu = 0.0
            elif j == 1:
                nu = 0.0
            else:
                a1, b1 = mv(W["w_n"], s), mv(W["w_c"], c)
                na = math.sqrt(sum(x * x for x in a1))
                nb = math.sqrt(sum(x * x for x in b1))
                nu = 1.0 - sum(x * y for x, y in zip(a1, b1)) / (na * nb + cfg.eps)
            hh = [sl(x + b) for x, b in zip(mv(W["th_w1"], s + c + [nu]), W["th_b1"])]
            a = sum(x * y for x, y in zip(W["th_w2"][0], hh)) + W["th_b2"][0]
            p = sg(a / cfg.t_hist)
            m = m_prev * p
            g = sg(a + f_psi(hb))
            rho = sg(W["eta"][layer - 1])
            for mm in range(dm):
                for n in range(dm):
                    S[mm][n] = rho * S[mm][n] + fk[mm] * v[n]
                Z[mm] = rho * Z[mm] + fk[mm]
            if variant & 2:                                    # the memory stays empty
                S = [[0.0] * dm for _ in range(dm)]
                Z = [0.0] * dm
            u = ln_ffn(layer, hb)
            if g >= tau:
                y = ffn(layer, u)
                h = [hb[i] + g * y[i] for i in range(d)]
            else:
                y = adp(layer, u)
                h = [hb[i] + (1 - g) * y[i] for i in range(d)]
            gs.append(g)
            hb_prev, dl_prev, d_prev, p_prev, m_prev = hb, dl, dd, p, m
        out_h.append(h)
        out_g.append(gs)
    return np.array(out_h), np.array(out_g).T


def test_p8_loop_restatement_tiny_shapes():
    cfg = hi.StackConfig("micro", 3, 8, 12, 4, 4, 6, "f32", 0.3, d_h=3, d_a=2, d_enc=5,
                         d_head=6, d_path=3, seed=11)
    w, h, P = _inputs(cfg)
    W = {k: hi.to_f64(v).tolist() for k, v in w.items()}
    oc = ho.OracleConfig.from_stack(cfg)
    base = ho.routed_ffn_stack(oc, w, h, P, 0.0, record=True)
    tau = float(np.median(base["gate"]))                  # a mix of both branches
    got = ho.routed_ffn_stack(oc, w, h, P, tau)
    ref_h, ref_g = _py_stack(cfg, W, hi.to_f64(h).tolist(), hi.to_f64(P).tolist(), tau)
    np.testing.assert_allclose(got["gate"], ref_g, rtol=0, atol=1e-12)
    np.testing.assert_allclose(got["h_out"], ref_h, rtol=0, atol=1e-12)
    assert 0 < got["mask"].sum() < got["mask"].size


@pytest.mark.parametrize("variant", [1, 2, 4, 8, 4 | 8, 2 | 4 | 8])
def test_p8_router_ablations_restatement(variant):
    """Sec. 4.4 component ablations against the independent loop restatement."""
    cfg = hi.StackConfig("micro", 4, 8, 12, 4, 4, 6, "f32", 0.3, d_h=3, d_a=2, d_enc=5,
                         d_head=6, d_path=3, seed=13)
    w, h, P = _inputs(cfg)
    W = {k: hi.to_f64(v).tolist() for k, v in w.items()}
    oc = ho.OracleConfig.from_stack(cfg)
    oc.variant = variant
    base = ho.routed_ffn_stack(oc, w, h, P, 0.0)
    tau = float(np.median(base["gate"]))
    got = ho.routed_ffn_stack(oc, w, h, P, tau, record=True)
    ref_h, ref_g = _py_stack(cfg, W, hi.to_f64(h).tolist(), hi.to_f64(P).tolist(), tau,
                             variant=variant)
    np.testing.assert_allclose(got["gate"], ref_g, rtol=0, atol=1e-12)
    np.testing.assert_allclose(got["h_out"], ref_h, rtol=0, atol=1e-12)
    full = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P, tau)
    assert np.max(np.abs(full["gate"] - got["gate"])) > 1e-6   # the ablation changes g
    if variant & 2:                                           # no memory read or write
        for rec in got["layers"]:
            assert not rec["S"].any() and not rec["c"].any() and not rec["nu"].any()


def test_p8_placement_dense_prefix_restatement():
    """Sec. 4.1 placement: the first n_dense FFN layers stay dense, the candidate
    layers after them are routed blocks j = 1 .. L_R with their own L_R."""
    cfg = hi.StackConfig("micro", 5, 8, 12, 4, 4, 6, "f32", 0.3, d_h=3, d_a=2, d_enc=5,
                         d_head=6, d_path=3, seed=12)
    w, h, P = _inputs(cfg)
    W = {k: hi.to_f64(v).tolist() for k, v in w.items()}
    oc = ho.OracleConfig.from_stack(cfg)
    oc.n_dense = 2
    base = ho.routed_ffn_stack(oc, w, h, P, 0.0)
    tau = float(np.median(base["gate"][2:]))
    got = ho.routed_ffn_stack(oc, w, h, P, tau)
    ref_h, ref_g = _py_stack(cfg, W, hi.to_f64(h).tolist(), hi.to_f64(P).tolist(), tau, n_dense=2)
    np.testing.assert_allclose(got["gate"], ref_g, rtol=0, atol=1e-12)
    np.testing.assert_allclose(got["h_out"], ref_h, rtol=0, atol=1e-12)
    assert (got["mask"][:2] == 1).all() and 0 < got["mask"][2:].sum() < got["mask"][2:].size
    assert ho.bypass_fraction(got["mask"], n_dense=2) == 1.0 - got["mask"][2:].mean()


def test_bf16_bits_rounding_matches_torch():
    """The restatement's own bf16 rounding against torch's conversion (values that are
    float32-representable, so torch's path through float32 rounds once) and exact ties."""
    rng = np.random.default_rng(9)
    x = (rng.standard_normal(3000) * 10.0 ** rng.integers(-20, 20, 3000)).astype(np.float32)
    ties = (np.arange(1, 300, dtype=np.float64) * 2.0 + 1.0) * 2.0 ** -8 + 1.0
    for v in (x.astype(np.float64), ties, -ties):
        ref = torch.tensor(v, dtype=torch.float32).to(torch.bfloat16).to(torch.float64).numpy()
        got = np.array([_bf16_bits(float(a)) for a in v])
        np.testing.assert_array_equal(got, ref)


def _micro_bf16(seed=17, n_layers=3):
    cfg = hi.StackConfig("micro", n_layers, 8, 12, 4, 4, 6, "bf16", 0.3, d_h=3, d_a=2, d_enc=5,
                         d_head=6, d_path=3, seed=seed)
    w, h, P = _inputs(cfg)
    W = {k: hi.to_f64(v).tolist() for k, v in w.items()}
    oc = ho.OracleConfig.from_stack(cfg)
    tau = float(np.median(ho.routed_ffn_stack(oc, w, h, P, 0.0)["gate"]))   # both branches
    return cfg, oc, w, h, P, W, tau


def _bf16_restatement_agrees(oc, w, h, P, W, tau, cfg, n_dense=0):
    got = ho.routed_ffn_stack(oc, w, h, P, tau)
    ref_h, ref_g = _py_stack(cfg, W, hi.to_f64(h).tolist(), hi.to_f64(P).tolist(), tau,
                             n_dense=n_dense, bf16=True)
    return (np.max(np.abs(got["gate"] - ref_g)) <= 1e-12 and
            np.max(np.abs(got["h_out"] - ref_h)) <= 1e-12, got)


@pytest.mark.parametrize("n_dense", [0, 1])
def test_p8_bf16_precision_contract_restatement(n_dense):
    """The bf16 models' rounding points (router weight W_hd diag(g_r), the router's
    activation pair in the encoder and in f_psi, u, the SwiGLU product, the adapter
    hidden) in the oracle's bf16 mode equal the per-element restatement, which takes
    them from the contract with its own bf16 rounding; and the rounding matters (the
    unrounded stack differs)."""
    cfg, oc, w, h, P, W, tau = _micro_bf16(n_layers=3 + n_dense)
    oc.n_dense = n_dense
    ok, got = _bf16_restatement_agrees(oc, w, h, P, W, tau, cfg, n_dense)
    assert ok
    m = got["mask"][n_dense:]
    assert 0 < m.sum() < m.size                      # both branches exercised
    unrounded = ho.routed_ffn_stack(ho.OracleConfig(**{**oc.__dict__, "dtype": "f32"}), w, h, P, tau,
                                    mode="force", mask_in=got["mask"])
    assert np.max(np.abs(unrounded["h_out"] - got["h_out"])) > 1e-7   # far above 1e-12


def test_bf16_planted_mistakes_are_caught(monkeypatch):
    """Each plausible slip in the bf16 contract makes the restatement disagree."""
    cfg, oc, w, h, P, W, tau = _micro_bf16()
    assert _bf16_restatement_agrees(oc, w, h, P, W, tau, cfg)[0]
    plants = {
        # f_psi reads a single bf16 rounding of h_bar instead of the pair
        "local_head": lambda f: (lambda hb, ww, Rx: f(hb, ww, ho.bf16_round)),
        # the encoder weight W_hd diag(g_r) left unrounded
        "hidden_encoder": lambda f: (lambda hb, ww, c, R, Rx: f(hb, ww, c, ho._identity, Rx)),
        # the SwiGLU product enters W_down unrounded
        "swiglu_ffn": lambda f: (lambda u, wl, R: f(u, wl, ho._identity)),
        # the adapter hidden enters W_2 unrounded
        "adapter": lambda f: (lambda u, wl, R: f(u, wl, ho._identity)),
    }
    for name, make in plants.items():
        with monkeypatch.context() as mp:
            mp.setattr(ho, name, make(getattr(ho, name)))
            assert not _bf16_restatement_agrees(oc, w, h, P, W, tau, cfg)[0], name


def _py_attention(h, wa, H, Hkv, theta, n_seqs, S, eps, bf16):
    """Eq. 1's attention sublayer per element (Llama form), bf16 rounding r() at LN_attn(h),
    q and k after RoPE, v, the normalised probabilities and the attention output."""
    r = _bf16_bits if bf16 else (lambda x: x)
    T, d = len(h), len(h[0])
    hd = d // H
    half = hd // 2

    def mv(M, x):
        return [sum(M[o][i] * x[i] for i in range(len(x))) for o in range(len(M))]

    x = []
    for t in range(T):
        rms = math.sqrt(sum(v * v for v in h[t]) / d + eps)
        x.append([r(h[t][i] / rms * wa["attn_norm_g"][i]) for i in range(d)])
    Q, K, V = [mv(wa["w_q"], xt) for xt in x], [mv(wa["w_k"], xt) for xt in x], \
        [mv(wa["w_v"], xt) for xt in x]

    def rope(vec, pos):
        out = list(vec)
        for i in range(half):
            ang = pos * theta ** (-2.0 * i / hd)
            c, sn = math.cos(ang), math.sin(ang)
            out[i] = vec[i] * c - vec[i + half] * sn
            out[i + half] = vec[i + half] * c + vec[i] * sn
        return out

    out = []
    for t in range(T):
        b, pos = divmod(t, S)
        o = []
        for hh in range(H):
            kv = hh // (H // Hkv)
            q = [r(z) for z in rope(Q[t][hh * hd:(hh + 1) * hd], pos)]
            sc = []
            for p2 in range(pos + 1):
                t2 = b * S + p2
                k = [r(z) for z in rope(K[t2][kv * hd:(kv + 1) * hd], p2)]
                sc.append(sum(qi * ki for qi, ki in zip(q, k)) / math.sqrt(hd))
            mx = max(sc)
            e = [math.exp(z - mx) for z in sc]
            tot = sum(e)
            pr_ = [r(z / tot) for z in e]
            for c in range(hd):
                o.append(r(sum(pr_[p2] * r(V[b * S + p2][kv * hd + c]) for p2 in range(pos + 1))))
        y = mv(wa["w_o"], o)
        out.append([h[t][i] + y[i] for i in range(d)])
    return np.array(out)


@pytest.mark.parametrize("bf16", [False, True])
def test_attention_restatement_with_precision_points(bf16, monkeypatch):
    """attention_sublayer (f32, and bf16 at R28's rounding points) equals the per-element
    restatement on micro shapes; a planted slip (q and k rounded before RoPE as well) is
    caught."""
    rng = np.random.default_rng(21)
    n_seqs, S, H, Hkv, d, theta = 2, 5, 4, 2, 16, 500000.0
    h = rng.standard_normal((n_seqs * S, d))
    wa = {"attn_norm_g": 1 + 0.02 * rng.standard_normal(d),
          "w_q": 0.3 * rng.standard_normal((d, d)), "w_k": 0.3 * rng.standard_normal((d // 2, d)),
          "w_v": 0.3 * rng.standard_normal((d // 2, d)), "w_o": 0.3 * rng.standard_normal((d, d))}
    if bf16:
        wa = {k: ho.bf16_round(v) for k, v in wa.items()}
    R = ho.bf16_round if bf16 else None
    got = ho.attention_sublayer(h, wa, H, Hkv, theta, n_seqs, S, 1e-5, R)
    ref = _py_attention(h.tolist(), {k: v.tolist() for k, v in wa.items()}, H, Hkv, theta, n_seqs,
                        S, 1e-5, bf16)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)
    if bf16:
        orig = ho.apply_rope
        monkeypatch.setattr(ho, "apply_rope", lambda x, c, s_: orig(ho.bf16_round(x), c, s_))
        planted = ho.attention_sublayer(h, wa, H, Hkv, theta, n_seqs, S, 1e-5, R)
        assert np.max(np.abs(planted - ref)) > 1e-9


# ---------------------------------------------------------------------------
# Planted mistakes: each plausible slip in the oracle is caught by a pin
# ---------------------------------------------------------------------------

def test_planted_mistakes_are_caught(monkeypatch):
    cfg = _tiny()
    tau = hi.calibrated_tau("tiny_f32")

    def caught(check):
        try:
            return not check()
        except AssertionError:
            return True

    # 1. phi without the +1 (plain ELU): the second-block closed form fails
    with monkeypatch.context() as mp:
        mp.setattr(ho, "phi", lambda x: np.where(x > 0, x, np.exp(np.minimum(x, 0)) - 1))
        assert caught(lambda: check_second_block(cfg)[0] < 1e-13)
    # 2. forgetting applied to the new term instead of the old state
    with monkeypatch.context() as mp:
        mp.setattr(ho, "memory_write",
                   lambda S, z, fk, v, rho: (S + rho * np.einsum("tm,tn->tmn", fk, v), z + rho * fk))
        assert caught(lambda: max(check_memory_closed_form(cfg)[:2]) < 1e-12)
    # 3. write before read: c_j would see the current block's own state
    orig_read = ho.memory_read

    def read_after_write(fq, S, zeta, eps):
        return orig_read(fq, S + 1.0, zeta + 1.0, eps)
    with monkeypatch.context() as mp:
        mp.setattr(ho, "memory_read", read_after_write)
        assert caught(lambda: check_second_block(cfg)[0] < 1e-13)
    # 4. transition against two blocks back
    orig_tf = ho.transition_features

    def tf_wrong_sign(j, hb, hbp, dp, d_prev, eps):
        delta, d, gamma = orig_tf(j, hb, hbp, dp, d_prev, eps)
        return delta, d, -gamma
    with monkeypatch.context() as mp:
        mp.setattr(ho, "transition_features", tf_wrong_sign)
        assert caught(lambda: check_transition_closed_form(cfg)[0] < 1e-12)
    # 5. gate and up projections swapped in the SwiGLU
    with monkeypatch.context() as mp:
        mp.setattr(ho, "swiglu_ffn", lambda u, wl, R: R(silu_swapped(u, wl)) @ wl["w_down"].T)
        assert caught(lambda: check_dense(cfg)[0] < 1e-13)
    # 6. adapter hidden without its activation
    with monkeypatch.context() as mp:
        mp.setattr(ho, "adapter", lambda u, wl, R: (u @ wl["ad_w1"].T) @ wl["ad_w2"].T)
        assert caught(lambda: check_adapter_stack(cfg) < 1e-13)
    # 7. branch scale swapped (FFN scaled by 1 - g)
    orig_stack = ho.routed_ffn_stack

    def swapped(*a, **k):
        out = orig_stack(*a, **k)
        for rec in out.get("layers", []):
            rec["g"] = 1.0 - rec["g"]
        return out
    with monkeypatch.context() as mp:
        mp.setattr(ho, "routed_ffn_stack", swapped)
        assert caught(lambda: check_branch_scaling(cfg, tau)[0] < 1e-13)
    # 8. decision threshold inverted: brute force no longer finds the free run
    def inverted(*a, **k):
        out = orig_stack(*a, **k)
        if k.get("mode", "route") == "route":
            out["mask"] = 1 - out["mask"]
        return out
    with monkeypatch.context() as mp:
        mp.setattr(ho, "routed_ffn_stack", inverted)
        n, chosen, free_code = check_path_brute_force(cfg, tau)
        assert not (chosen == free_code).all()


def silu_swapped(u, wl):
    return ho.silu(u @ wl["w_up"].T) * (u @ wl["w_gate"].T)


# ---------------------------------------------------------------------------
# The attention sublayer of the full decoder forward (Eq. 1)
# ---------------------------------------------------------------------------

def _attn_inputs(seq_len=24, n_seqs=2, H=4, Hkv=2, d=64, seed=5):
    cfg = hi.StackConfig("attn_micro", 2, d, 96, 8, 8, n_seqs * seq_len, "f32", 0.3,
                         d_h=4, d_a=4, d_enc=8, d_head=8, d_path=4, seed=seed, batch=n_seqs,
                         seq_len=seq_len, n_heads=H, n_kv_heads=Hkv, rope_theta=500000.0)
    wa = {k: hi.to_f64(v)[0] for k, v in hi.generate_attn_weights(cfg).items()}
    return cfg, wa, hi.to_f64(hi.generate_h_in(cfg))


def test_rope_rotation_properties():
    """RoPE rotates each (x_i, x_{i+hd/2}) pair: norms are kept, position 0 is the
    identity, and q.k depends only on the position difference."""
    rng = np.random.default_rng(0)
    hd, S = 16, 40
    cos, sin = ho.rope_cos_sin(S, hd, 10000.0)
    q, k = rng.standard_normal((S, hd)), rng.standard_normal((S, hd))
    rq = ho.apply_rope(q, cos, sin)
    np.testing.assert_allclose(rq[0], q[0], rtol=0, atol=1e-15)
    np.testing.assert_allclose(np.linalg.norm(rq, axis=1), np.linalg.norm(q, axis=1), rtol=1e-13)
    qq = np.repeat(q[:1], S, axis=0)
    kk = np.repeat(k[:1], S, axis=0)
    dots = np.sum(ho.apply_rope(qq, cos, sin)[5:] * ho.apply_rope(kk, cos, sin)[:-5], axis=1)
    np.testing.assert_allclose(dots, dots[0], rtol=1e-11)   # positions (m, m-5) for every m
    # the frequency of pair i is theta^(-2i/hd): pair 0 turns by one radian per position
    np.testing.assert_allclose(cos[:, 0], np.cos(np.arange(S)), atol=1e-15)


def test_attention_matches_torch_sdpa():
    """Projection, causal softmax attention with grouped KV heads, output projection and
    residual against torch's scaled_dot_product_attention (float64, no rounding)."""
    cfg, wa, h = _attn_inputs()
    B, S, H, Hkv, d = cfg.batch, cfg.seq_len, cfg.n_heads, cfg.n_kv_heads, cfg.d_model
    hd = d // H
    got = ho.attention_sublayer(h, wa, H, Hkv, cfg.rope_theta, B, S, cfg.rms_eps)
    x = F.rms_norm(_t(h), (d,), _t(wa["attn_norm_g"]), cfg.rms_eps)
    sh = lambda a, nh: a.reshape(B, S, nh, hd).transpose(1, 2)
    q = sh(x @ _t(wa["w_q"]).T, H)
    k = sh(x @ _t(wa["w_k"]).T, Hkv)
    v = sh(x @ _t(wa["w_v"]).T, Hkv)
    cos, sin = ho.rope_cos_sin(S, hd, cfg.rope_theta)
    q = _t(ho.apply_rope(q.numpy(), cos, sin))
    k = _t(ho.apply_rope(k.numpy(), cos, sin))
    k = k.repeat_interleave(H // Hkv, dim=1)
    v = v.repeat_interleave(H // Hkv, dim=1)
    o = F.scaled_dot_product_attention(q, k, v, is_causal=True)
    ref = _t(h) + o.transpose(1, 2).reshape(B * S, H * hd) @ _t(wa["w_o"]).T
    np.testing.assert_allclose(got, ref.numpy(), rtol=0, atol=1e-12)


def test_attention_is_causal_and_per_sequence():
    cfg, wa, h = _attn_inputs()
    B, S = cfg.batch, cfg.seq_len
    run = lambda x: ho.attention_sublayer(x, wa, cfg.n_heads, cfg.n_kv_heads, cfg.rope_theta, B, S,
                                          cfg.rms_eps)
    base = run(h)
    h2 = h.copy()
    h2[S + 10] += 1.0                     # token 10 of the second sequence
    out = run(h2)
    changed = np.nonzero(np.abs(out - base).max(axis=1) > 1e-12)[0]
    assert changed.min() == S + 10 and changed.max() < 2 * S   # itself and later tokens only
    assert (changed >= S + 10).all()


def test_attention_single_token_is_value_path():
    """A one-token sequence attends only to itself: h_bar = h + W_o [v of its KV head]."""
    cfg, wa, h = _attn_inputs(seq_len=1, n_seqs=6)
    H, Hkv, d = cfg.n_heads, cfg.n_kv_heads, cfg.d_model
    hd = d // H
    got = ho.attention_sublayer(h, wa, H, Hkv, cfg.rope_theta, 6, 1, cfg.rms_eps)
    x = F.rms_norm(_t(h), (d,), _t(wa["attn_norm_g"]), cfg.rms_eps).numpy()
    v = (x @ wa["w_v"].T).reshape(6, Hkv, hd)
    o = np.repeat(v, H // Hkv, axis=1).reshape(6, H * hd)
    np.testing.assert_allclose(got, h + o @ wa["w_o"].T, rtol=0, atol=1e-12)


def test_attention_rows_equals_full_sublayer():
    """The sampled-position form (used to check long sequences) equals the full one."""
    cfg, wa, h = _attn_inputs(seq_len=40, n_seqs=1)
    full = ho.attention_sublayer(h, wa, cfg.n_heads, cfg.n_kv_heads, cfg.rope_theta, 1, 40,
                                 cfg.rms_eps, ho.bf16_round)
    rows = np.array([0, 7, 19, 39])
    got = ho.attention_rows(h, rows, wa, cfg.n_heads, cfg.n_kv_heads, cfg.rope_theta, cfg.rms_eps,
                            ho.bf16_round)
    np.testing.assert_allclose(got, full[rows], rtol=0, atol=1e-12)


def test_rope_is_complex_rotation():
    """RoPE in its complex form (RoFormer): the pair (x_i, x_{i+hd/2}) read as
    z = x_i + i x_{i+hd/2} is multiplied by exp(i s theta^(-2i/hd)) at position s."""
    rng = np.random.default_rng(1)
    hd, S, theta = 16, 12, 500000.0
    x = rng.standard_normal((S, hd))
    cos, sin = ho.rope_cos_sin(S, hd, theta)
    got = ho.apply_rope(x, cos, sin)
    z = x[:, :hd // 2] + 1j * x[:, hd // 2:]
    ang = np.arange(S)[:, None] * theta ** (-2.0 * np.arange(hd // 2)[None, :] / hd)
    w = z * np.exp(1j * ang)
    np.testing.assert_allclose(got, np.concatenate([w.real, w.imag], axis=1), rtol=0, atol=1e-13)


# ---------------------------------------------------------------------------
# Training objective (Sec. 3.3): the pins a training path's gradients are checked with
# ---------------------------------------------------------------------------

def test_skip_penalty_gradient_closed_form():
    """d L_skip / d g_{j,b,t} = 2 / (B (T - 1)) sum_j' g_{j',b,t} for the T - 1
    next-token positions, 0 at a sequence's last position and for dense-prefix rows."""
    rng = np.random.default_rng(3)
    n_dense, L, B, S = 1, 4, 2, 5
    g = rng.uniform(0.05, 0.95, size=(L, B * S))
    base = ho.skip_penalty(g, B, S, n_dense)
    for j in range(L):
        for t in range(B * S):
            e = np.zeros_like(g)
            e[j, t] = 1.0
            fd = ho.directional_derivative(lambda hh: ho.skip_penalty(g + hh * e, B, S, n_dense), 1e-6)
            pos = t % S
            want = 0.0 if (j < n_dense or pos == S - 1) else \
                2.0 / (B * (S - 1)) * g[n_dense:, t].sum()
            assert abs(fd - want) < 1e-8, (j, t, fd, want)
    assert base == pytest.approx(np.sum(g[n_dense:].reshape(L - n_dense, B, S)[:, :, :S - 1].sum(0) ** 2)
                                 / (B * (S - 1)), rel=1e-15)


def _training_inputs():
    cfg = hi.CONFIGS["tiny_f32"]
    oc = ho.OracleConfig.from_stack(cfg)
    w, h, P = hi.generate_weights(cfg), hi.generate_h_in(cfg), hi.generate_attn_delta(cfg)
    free = ho.routed_ffn_stack(oc, w, h, P, hi.calibrated_tau(cfg.name))
    G = np.random.default_rng(5).standard_normal(h.shape)
    return cfg, oc, w, h, P, free["mask"], G


def test_last_block_gate_gradient_closed_form():
    """Eq. 3 with the decision fixed: in the last block g scales only the selected
    branch, so dL/dg_{L,t} = <G_t, FFN(u_t)> (FFN token) or -<G_t, Adapter(u_t)>
    (adapter token), plus alpha times L_skip's term - checked against central
    differences of the whole objective with g_{L,t} perturbed."""
    cfg, oc, w, h, P, mask, G = _training_inputs()
    B, S, alpha = 2, 32, 0.3
    rec = ho.routed_ffn_stack(oc, w, h, P, 0.0, mode="force", mask_in=mask, record=True)
    u = rec["layers"][-1]["u"]
    wl = {k: ho._f64(w[k][-1]) for k in ("w_gate", "w_up", "w_down", "ad_w1", "ad_w2")}
    L = cfg.n_layers
    ffn_t = int(np.nonzero(mask[-1])[0][0])
    ad_t = int(np.nonzero(mask[-1] == 0)[0][0])
    for t in sorted({ffn_t, ad_t, S - 1, S}):
        def f(hh, t=t):
            def hook(layer, g):
                if layer != L:
                    return g
                g = g.copy()
                g[t] += hh
                return g
            return ho.training_loss(oc, w, h, P, mask, G, alpha, B, S, hooks={"gate": hook})
        fd = ho.directional_derivative(f, 1e-5)
        if mask[-1, t]:
            branch = ho.swiglu_ffn(u[t:t + 1], wl, ho._identity)[0]
            want = float(G[t] @ branch)
        else:
            branch = ho.adapter(u[t:t + 1], wl, ho._identity)[0]
            want = -float(G[t] @ branch)
        if t % S != S - 1:
            want += alpha * 2.0 / (B * (S - 1)) * float(rec["gate"][:, t].sum())
        assert abs(fd - want) <= 1e-6 * max(1.0, abs(want)), (t, fd, want)


@pytest.mark.parametrize("key", ho.TRAINABLE)
def test_training_loss_is_smooth_along_each_trainable_tensor(key):
    """With the decisions fixed the objective is differentiable in every trainable
    tensor: central differences at h and h/2 agree to the O(h^2) truncation, and the
    derivative is nonzero (every trained tensor reaches the loss)."""
    cfg, oc, w, h, P, mask, G = _training_inputs()
    B, S, alpha = 2, 32, 0.3
    base = w[key].astype(np.float64)
    V = np.random.default_rng(100 + ho.TRAINABLE.index(key)).standard_normal(base.shape)
    scale = max(float(np.sqrt(np.mean(base ** 2))), 1e-3)

    def f(hh):
        w2 = dict(w)
        w2[key] = base + hh * scale * V
        return ho.training_loss(oc, w2, h, P, mask, G, alpha, B, S)

    d1 = ho.directional_derivative(f, 1e-4)
    d2 = ho.directional_derivative(f, 5e-5)
    assert abs(d1) > 1e-9, key
    assert abs(d1 - d2) <= 1e-5 * max(1.0, abs(d1)), (key, d1, d2)


@pytest.mark.parametrize("n_dense", [0, 1])
def test_decoder_forward_is_the_stack_fed_its_attention_updates(n_dense):
    """decoder_forward wires Eq. 1: replaying routed_ffn_stack with the additive input
    P_j = h_bar_j - h_{j-1} taken from the decoder run's own records reproduces its
    outputs, gates and decisions exactly (f32 model, free-running; with and without a
    dense prefix)."""
    cfg = hi.StackConfig("dec_micro", 3, 256, 96, 8, 8, 2 * 20, "f32", 0.3, d_h=4, d_a=4,
                         d_enc=8, d_head=8, d_path=4, seed=7, batch=2, seq_len=20,
                         n_heads=2, n_kv_heads=1, rope_theta=500000.0, n_dense=n_dense)
    oc = ho.OracleConfig.from_stack(cfg)
    w, wa = hi.generate_weights(cfg), hi.generate_attn_weights(cfg)
    h0 = hi.to_f64(hi.generate_h_in(cfg))
    first = ho.decoder_forward(oc, w, wa, h0, 0.5, 2, 1, cfg.rope_theta, 2, 20)
    tau = float(np.median(first["gate"][n_dense]))
    dec = ho.decoder_forward(oc, w, wa, h0, tau, 2, 1, cfg.rope_theta, 2, 20, record=True)
    hs = [h0] + [rec["h"] for rec in dec["layers"]]
    P = np.stack([rec["h_bar"] - hs[j] for j, rec in enumerate(dec["layers"])])
    stack = ho.routed_ffn_stack(oc, w, h0, P, tau)
    np.testing.assert_array_equal(stack["mask"], dec["mask"])
    np.testing.assert_allclose(stack["gate"], dec["gate"], rtol=0, atol=1e-13)
    np.testing.assert_allclose(stack["h_out"], dec["h_out"], rtol=0, atol=1e-12)
    assert 0 < dec["mask"][n_dense:].mean() < 1


def test_block_branch_backward_matches_central_differences():
    """block_branch_backward against central differences of the forward branch
    combination (LN_ffn, SwiGLU FFN or adapter, scale g or 1 - g, residual), for every
    returned gradient: h_bar and g element-wise on a sample, W_1 and W_2 along random
    directions."""
    cfg = hi.CONFIGS["tiny_f32"]
    w = hi.generate_weights(cfg)
    wl = {k: ho._f64(w[k][1]) for k in ("ffn_norm_g", "w_gate", "w_up", "w_down", "ad_w1", "ad_w2")}
    rng = np.random.default_rng(11)
    T, d = 24, cfg.d_model
    h_bar = rng.standard_normal((T, d))
    g = rng.uniform(0.1, 0.9, T)
    decide = rng.random(T) < 0.6
    G = rng.standard_normal((T, d))

    def loss(hb=h_bar, gg=g, wl_=wl):
        u = ho.rms_norm(hb, wl_["ffn_norm_g"], cfg.rms_eps)
        out = hb.copy()
        F, A = np.nonzero(decide)[0], np.nonzero(~decide)[0]
        out[F] += gg[F, None] * ho.swiglu_ffn(u[F], wl_, ho._identity)
        out[A] += (1 - gg[A])[:, None] * ho.adapter(u[A], wl_, ho._identity)
        return float(np.sum(G * out))

    bw = ho.block_branch_backward(h_bar, g, decide, G, wl, cfg.rms_eps)
    eps = 1e-6
    for t, c in [(0, 0), (3, 17), (5, 200), (int(np.nonzero(~decide)[0][0]), 33)]:
        e = np.zeros_like(h_bar)
        e[t, c] = 1.0
        fd = ho.directional_derivative(lambda hh: loss(hb=h_bar + hh * e), eps)
        assert abs(fd - bw["dh_bar"][t, c]) <= 1e-6 * max(1.0, abs(fd)), (t, c, fd, bw["dh_bar"][t, c])
    for t in range(T):
        e = np.zeros(T)
        e[t] = 1.0
        fd = ho.directional_derivative(lambda hh: loss(gg=g + hh * e), eps)
        assert abs(fd - bw["dg"][t]) <= 1e-6 * max(1.0, abs(fd)), t
    for key, gk in (("ad_w1", "dW1"), ("ad_w2", "dW2")):
        V = rng.standard_normal(wl[key].shape)

        def f(hh, key=key, V=V):
            wl2 = dict(wl)
            wl2[key] = wl[key] + hh * V
            return loss(wl_=wl2)
        fd = ho.directional_derivative(f, eps)
        assert abs(fd - float(np.sum(bw[gk] * V))) <= 1e-6 * max(1.0, abs(fd)), key


def test_skip_penalty_grad_matches_differences():
    rng = np.random.default_rng(4)
    n_dense, L, B, S = 2, 5, 3, 4
    g = rng.uniform(0.05, 0.95, size=(L, B * S))
    grad = ho.skip_penalty_grad(g, B, S, n_dense)
    V = rng.standard_normal(g.shape)
    fd = ho.directional_derivative(lambda hh: ho.skip_penalty(g + hh * V, B, S, n_dense), 1e-6)
    assert abs(fd - float(np.sum(grad * V))) < 1e-8


def test_autograd_restatement_matches_the_oracle_and_central_differences():
    """oracle/hero_autograd.py restates the stack in PyTorch float64 for reverse-mode
    gradients.  Its objective equals the NumPy oracle's, and its gradient along a
    random direction of every trainable tensor (and of h_in) equals the NumPy
    objective's central difference; on a placement with a dense prefix as well."""
    from oracle import hero_autograd as hg
    for n_dense in (0, 1):
        cfg = hi.CONFIGS["tiny_f32"].replace(n_dense=n_dense)
        oc = ho.OracleConfig.from_stack(cfg)
        w, h, P = hi.generate_weights(cfg), hi.generate_h_in(cfg), hi.generate_attn_delta(cfg)
        mask = ho.routed_ffn_stack(oc, w, h, P, hi.calibrated_tau("tiny_f32"))["mask"]
        G = np.random.default_rng(5).standard_normal(h.shape)
        B, S, alpha = 2, 32, 0.3
        loss, grads = hg.stack_loss_and_grads(oc, w, h, P, mask, G, alpha, B, S)
        ref = ho.training_loss(oc, w, h, P, mask, G, alpha, B, S)
        assert abs(loss - ref) <= 1e-12 * max(1.0, abs(ref))
        rng = np.random.default_rng(8 + n_dense)
        for key in ho.TRAINABLE + ("h_in",):
            base = ho._f64(h) if key == "h_in" else w[key].astype(np.float64)
            V = rng.standard_normal(base.shape)
            scale = max(float(np.sqrt(np.mean(base ** 2))), 1e-3)

            def f(hh, key=key, base=base, V=V, scale=scale):
                if key == "h_in":
                    return ho.training_loss(oc, w, base + hh * scale * V, P, mask, G, alpha, B, S)
                w2 = dict(w)
                w2[key] = base + hh * scale * V
                return ho.training_loss(oc, w2, h, P, mask, G, alpha, B, S)
            fd = ho.directional_derivative(f, 1e-5)
            an = float(np.sum(grads[key] * scale * V))
            assert abs(fd - an) <= 1e-6 * max(1.0, abs(fd)), (n_dense, key, fd, an)
