"""GPU parity of the full decoder forward: the attention sublayer of Eq. 1 (LN_attn,
q/k/v projections, RoPE, causal grouped-query softmax attention, output projection
with the residual) and the routed blocks fed by it.

Attention parity compares the attention update h_bar - h row by row:
max_t ||(x - h)_t - (y - h)_t||_inf / ||(y - h)_t||_inf below 2e-2 (the bf16 hidden
state bound), both sides rounding the same operands to bf16 (LN_attn(h), q and k
after RoPE, v, the probabilities entering P V, the attention output).  The CUDA
path rounds exp(s - running max) before the division by the row sum (the
FlashAttention schedule), the oracle the normalised probability: one bf16 rounding
of the same magnitude either way.

Free-running decoder comparisons extend the near-boundary rule of the stack tests:
a token whose decision flips near tau_exec changes its own later states AND, through
attention, those of every later position of its sequence, so those positions are
dropped from the next block on.
"""

import numpy as np
import pytest

from oracle import hero_oracle as ho
from synth import hero_inputs as hi
from tests import parity as pr

pytestmark = pytest.mark.gpu

H_TOL = pr.H_TOL["bf16"]


@pytest.fixture(scope="module")
def hero():
    import torch
    assert torch.cuda.is_available()
    from paper_2609_08189_gb300 import build, hero as H
    build.build()
    H.load()
    return H


def _dev(a):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda")


def _attn_layer(wa, j):
    return {k: ho._f64(v[j]) for k, v in wa.items()}


def _attn_err(x, y, h):
    return float(np.max(pr.rel_err_rows(x - h, y - h)))


# ------------------------------------------------------------------------------
# the attention sublayer alone
# ------------------------------------------------------------------------------

# S >= 128 runs the tensor-core kernel (128-row query tiles, K and transposed V tiles
# of 128 keys), shorter sequences the mma.sync kernel (64-row tiles)
SHAPES = [(2, 160), (1, 1), (5, 1), (3, 77), (1, 64), (1, 300), (4, 65), (0, 8), (1, 128),
          (2, 256), (3, 130), (1, 511)]


@pytest.fixture(scope="module")
def small_decoder(hero):
    cfg = hi.CONFIGS["small_bf16_decoder"]
    w, wa = hi.generate_weights(cfg), hi.generate_attn_weights(cfg)
    dec = hero.HeroDecoder(cfg, w, wa, max_tokens=512)
    yield cfg, w, wa, dec
    dec.close()


@pytest.mark.parametrize("n_seqs,seq_len", SHAPES)
def test_attention_block_parity(small_decoder, n_seqs, seq_len):
    """Every layer, several sequence shapes: ragged query/key tiles (77, 65, 130, 160,
    300, 511), whole tiles (64, 128, 256), single-token sequences (the score is the
    token with itself: o = v), and no sequences."""
    import torch
    cfg, _, wa, dec = small_decoder
    T = n_seqs * seq_len
    h = hi.generate_h_in(cfg.replace(n_tokens=max(T, 1)))[:T]
    hd = _dev(h)
    for layer in range(1, cfg.n_layers + 1):
        got = dec.attention(layer, hd, n_seqs, seq_len)
        torch.cuda.synchronize()
        dec.check()
        if T == 0:
            continue
        ref = ho.attention_sublayer(ho._f64(h), _attn_layer(wa, layer - 1), cfg.n_heads,
                                    cfg.n_kv_heads, cfg.rope_theta, n_seqs, seq_len, cfg.rms_eps,
                                    ho.bf16_round)
        err = _attn_err(got.cpu().numpy().astype(np.float64), ref, ho._f64(h))
        print(n_seqs, seq_len, layer, err)
        assert err < H_TOL, (layer, err)


def test_attention_is_causal_and_per_sequence(small_decoder):
    """Changing the last token of sequence 0 changes no other row of h_bar; changing a
    token of sequence 1 leaves sequence 0 alone (bit for bit)."""
    import torch
    cfg, _, _, dec = small_decoder
    B, S = 2, 160
    h = hi.generate_h_in(cfg)[:B * S].copy()
    base = dec.attention(1, _dev(h), B, S).cpu().numpy()
    h2 = h.copy()
    h2[S - 1] *= 1.5
    h2[S + 10] += 0.25
    out = dec.attention(1, _dev(h2), B, S).cpu().numpy()
    torch.cuda.synchronize()
    np.testing.assert_array_equal(out[:S - 1], base[:S - 1])
    np.testing.assert_array_equal(out[S:S + 10], base[S:S + 10])
    assert np.any(out[S - 1] != base[S - 1]) and np.any(out[S + 10:] != base[S + 10:])


def test_attention_full_size_sampled(hero):
    """Llama-3.1-8B attention shapes in the bench's launch configuration (4 sequences
    of 4096 tokens, 32 query heads on 8 key/value heads): one layer, sampled query
    positions of two sequences against the oracle's per-position form (all keys of
    the sequence)."""
    import torch
    base = hi.CONFIGS["llama31_8b_decoder"]
    cfg = base.replace(name="llama31_8b_decoder_2l", n_layers=2)
    w, wa = hi.generate_weights(cfg), hi.generate_attn_weights(cfg)
    dec = hero.HeroDecoder(cfg, w, wa)
    del w
    B, S = cfg.batch, cfg.seq_len
    h = hi.generate_h_in(cfg)
    got = dec.attention(1, _dev(h), B, S)
    torch.cuda.synchronize()
    dec.check()
    rows = np.array([0, 1, 63, 64, 65, 127, 1000, 2047, 2048, 4095])
    wa0 = _attn_layer(wa, 0)
    for b in (0, B - 1):
        hs = ho._f64(h[b * S:(b + 1) * S])
        ref = ho.attention_rows(hs, rows, wa0, cfg.n_heads, cfg.n_kv_heads, cfg.rope_theta,
                                cfg.rms_eps, ho.bf16_round)
        x = got[torch.as_tensor(b * S + rows, device="cuda")].cpu().numpy().astype(np.float64)
        err = _attn_err(x, ref, hs[rows])
        print("seq", b, "err", err)
        assert err < H_TOL, (b, err)
    dec.close()
    torch.cuda.empty_cache()


# ------------------------------------------------------------------------------
# the decoder forward
# ------------------------------------------------------------------------------

def compare_decoder_free(gpu: pr.GpuRun, ref, n_seqs: int, seq_len: int,
                         pos: np.ndarray = None, boundary: float = pr.BOUNDARY) -> pr.Report:
    """compare_free with attention contamination: a near-boundary flip of the token at
    position p of sequence b at block j drops positions >= p of sequence b from
    block j + 1 on (the token itself from block j on).  pos: position of each compared
    row in its sequence (default: rows are the whole batch in order)."""
    g_ref, m_ref = ref["gate"], ref["mask"]
    L, T = g_ref.shape
    seq = np.arange(T) // seq_len if pos is None else np.repeat(np.arange(n_seqs), T // n_seqs)
    pos = np.arange(T) % seq_len if pos is None else pos
    rep = pr.Report(T)
    alive = np.ones(T, dtype=bool)
    for j in range(L):
        near = np.abs(g_ref[j] - ref["tau"]) < boundary
        mism = gpu.mask[j] != m_ref[j]
        far = alive & mism & ~near
        rep.mask_mismatch_far += int(far.sum())
        dropped = alive & mism & near
        rep.boundary_tokens += [int(t) for t in np.nonzero(dropped)[0]]
        if alive.any():
            rep.gate_err = max(rep.gate_err, float(np.max(np.abs(gpu.gate[j][alive] - g_ref[j][alive]))))
        alive &= ~mism
        for t in np.nonzero(dropped)[0]:
            alive &= ~((seq == seq[t]) & (pos >= pos[t]))
    if alive.any():
        rep.h_err = float(np.max(pr.rel_err_rows(gpu.h_out[alive], ref["h_out"][alive])))
    rep.compared_h = int(alive.sum())
    return rep


def _run_decoder(dec, h, tau, n_seqs, seq_len, flags=0, mask_in=None, rows=None):
    import torch
    mi = _dev(mask_in) if mask_in is not None else None
    h_out, g, m, c = dec.forward(_dev(h), tau, n_seqs, seq_len, flags=flags, mask_in=mi)
    torch.cuda.synchronize()
    dec.check()
    sel = slice(None) if rows is None else torch.as_tensor(rows, device="cuda")
    return pr.GpuRun(h_out[sel].cpu().numpy().astype(np.float64),
                     g[:, sel].cpu().numpy().astype(np.float64), m[:, sel].cpu().numpy(),
                     c.cpu().numpy())


def _oracle_decoder(cfg, w, wa, h, tau, n_seqs, seq_len, **kw):
    out = ho.decoder_forward(ho.OracleConfig.from_stack(cfg), w, wa, h, tau, cfg.n_heads,
                             cfg.n_kv_heads, cfg.rope_theta, n_seqs, seq_len, **kw)
    out["tau"] = tau
    return out


def test_decoder_forward_parity(small_decoder, hero):
    """All tokens of 2 sequences of 160 through 4 blocks: free-running, forced with the
    oracle's decisions, and dense."""
    cfg, w, wa, dec = small_decoder
    B, S = cfg.batch, cfg.seq_len
    tau = hi.calibrated_tau(cfg.name)
    h = hi.generate_h_in(cfg)
    ref = _oracle_decoder(cfg, w, wa, h, tau, B, S)
    gpu = _run_decoder(dec, h, tau, B, S)
    rep = compare_decoder_free(gpu, ref, B, S)
    print("free", rep, "bypass", 1 - gpu.mask.mean(), "oracle", 1 - ref["mask"].mean())
    assert rep.mask_mismatch_far == 0, rep
    assert rep.gate_err < pr.GATE_TOL, rep
    assert rep.compared_h >= 0.8 * rep.n_tokens, rep
    assert rep.h_err < H_TOL, rep
    np.testing.assert_array_equal(gpu.counts, gpu.mask.sum(axis=1))
    assert 0 < gpu.mask.sum() < gpu.mask.size
    forced = _run_decoder(dec, h, tau, B, S, flags=hero.HERO_FLAG_FORCE_MASK, mask_in=ref["mask"])
    frep = pr.compare_forced(forced, ref)
    print("forced", frep)
    assert frep.mask_mismatch_far == 0
    assert frep.gate_err < pr.GATE_TOL and frep.h_err < H_TOL, frep
    dense = _run_decoder(dec, h, tau, B, S, flags=hero.HERO_FLAG_DENSE)
    dref = _oracle_decoder(cfg, w, wa, h, tau, B, S, mode="dense")
    derr = float(np.max(pr.rel_err_rows(dense.h_out, dref["h_out"])))
    print("dense", derr)
    assert derr < H_TOL
    assert (dense.mask == 1).all() and (dense.counts == B * S).all()


def test_decoder_matches_caller_driven_blocks(small_decoder, hero):
    """hero_decoder_forward equals the caller-driven form: hero_attention_block, then
    hero_routed_block with a caller-held router state.  The same arithmetic except
    the order of the fp32 sums behind the block entry's norms (the decoder's output
    projection sums per 128-column slot, k_block_entry per row), so decisions agree
    exactly and gates and states to 1e-4, ten times inside the oracle bound."""
    import torch
    cfg, w, wa, dec = small_decoder
    B, S = cfg.batch, cfg.seq_len
    T, L, d, dm = B * S, cfg.n_layers, cfg.d_model, cfg.d_m
    tau = hi.calibrated_tau(cfg.name)
    h0 = _dev(hi.generate_h_in(cfg))
    h_out, g, m, _ = dec.forward(h0, tau, B, S)
    f = dict(device="cuda", dtype=torch.float32)
    ts = {"S": torch.zeros((T, dm, dm), **f), "zeta": torch.zeros((T, dm), **f),
          "p_hist": torch.ones((T,), **f), "m_hist": torch.ones((T,), **f),
          "d_prev": torch.zeros((T,), **f), "h_bar_prev": torch.zeros((T, d), **f),
          "delta_prev": torch.zeros((T, d), **f)}
    state = hero.make_state({k: v.data_ptr() for k, v in ts.items()})
    stream = torch.cuda.current_stream().cuda_stream
    gs = torch.empty((L, T), **f)
    ms = torch.empty((L, T), device="cuda", dtype=torch.uint8)
    hero.hero_router_state_reset(dec.model, T, state, stream)
    x = h0
    for j in range(1, L + 1):
        hb = dec.attention(j, x, B, S)
        x = torch.empty_like(hb)
        hero.hero_routed_block(dec.model, j, T, hb.data_ptr(), state, tau, 0, 0, x.data_ptr(),
                               gs[j - 1].data_ptr(), ms[j - 1].data_ptr(), 0, stream)
    torch.cuda.synchronize()
    dec.check()
    gerr = float((gs - g).abs().max())
    err = float(np.max(pr.rel_err_rows(x.cpu().numpy().astype(np.float64),
                                       h_out.cpu().numpy().astype(np.float64))))
    print("caller-driven vs fused: mask equal", bool((ms == m).all()), "gate", gerr, "h", err)
    np.testing.assert_array_equal(ms.cpu().numpy(), m.cpu().numpy())
    assert gerr < 1e-4 and err < 1e-4, (gerr, err)


def test_decoder_full_size_prefix(hero):
    """Llama-3.1-8B decoder shapes, the bench's launch configuration (4 x 4096 tokens,
    32 routed blocks, 32 query heads on 8 key/value heads): the first positions of every sequence depend on
    nothing after them (causal attention, per-token routing), so the oracle run on
    those prefixes alone gives their exact expected values inside the full run."""
    import torch
    cfg = hi.CONFIGS["llama31_8b_decoder"]
    B, S, P = cfg.batch, cfg.seq_len, 24
    tau = hi.calibrated_tau(cfg.name)
    w, wa = hi.generate_weights(cfg), hi.generate_attn_weights(cfg)
    h = hi.generate_h_in(cfg)
    dec = hero.HeroDecoder(cfg, w, wa)
    rows = (np.arange(B)[:, None] * S + np.arange(P)[None, :]).reshape(-1)
    gpu_all = _run_decoder(dec, h, tau, B, S)
    np.testing.assert_array_equal(gpu_all.counts, gpu_all.mask.sum(axis=1))
    assert 0.0 < 1 - gpu_all.mask.mean() < 1.0
    gpu = pr.GpuRun(gpu_all.h_out[rows], gpu_all.gate[:, rows], gpu_all.mask[:, rows], gpu_all.counts)
    ref = _oracle_decoder(cfg, w, wa, h[rows], tau, B, P)
    bound = pr.free_run_gate_bound("llama31_8b_prefill")
    rep = compare_decoder_free(gpu, ref, B, P, boundary=bound)
    print("full-size prefix", rep, "bypass", 1 - gpu_all.mask.mean())
    assert rep.mask_mismatch_far == 0, rep
    assert rep.gate_err < bound, rep
    assert rep.compared_h >= 0.5 * rep.n_tokens, rep
    assert rep.h_err < H_TOL, rep
    dec.close()
    del gpu_all
    torch.cuda.empty_cache()


def test_decoder_rejects_bad_shapes(small_decoder, hero):
    cfg, _, _, dec = small_decoder
    import torch
    h = torch.zeros((8, cfg.d_model), device="cuda")
    with pytest.raises(hero.HeroError):
        hero.hero_attention_block(dec.model, 0, 1, 8, h.data_ptr(), h.data_ptr() + 4, 0)
    with pytest.raises(hero.HeroError):
        hero.hero_attention_block(dec.model, 1, 1, 8, h.data_ptr(), h.data_ptr(), 0)
    with pytest.raises(hero.HeroError):
        hero.hero_attention_block(dec.model, 1, 1, 513, h.data_ptr(), h.data_ptr() + 4, 0)
    with pytest.raises(hero.HeroError):
        hero.hero_decoder_forward(dec.model, 1, 8, h.data_ptr(), float("nan"), 0, 0,
                                  h.data_ptr() + 4, 0, 0, 0, 0)
