"""GPU parity of KV-cache decoding (the decoder's incremental form of Eq. 1).

A decoding step's token at position p of a sequence sees the keys and values of
positions 0..p-1 (from the cache, written by the prefill or earlier steps) and its
own; its routing is its own.  So its expected result is the oracle's decoder
forward over that sequence's first p tokens followed by the new token, last row.
Forced-mask runs feed the oracle's decisions (prefill and step) and compare every
value; free-running runs compare decisions and values of the tokens whose
sequence saw no near-boundary flip.  Tolerances as the decoder forward tests.
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


def _dev(a, dtype=None):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(a)).to("cuda")
    return t if dtype is None else t.to(dtype)


def _np(t):
    return t.cpu().numpy()


@pytest.fixture(scope="module")
def small(hero):
    cfg = hi.CONFIGS["small_bf16_decoder"]
    w, wa = hi.generate_weights(cfg), hi.generate_attn_weights(cfg)
    dec = hero.HeroDecoder(cfg, w, wa, max_tokens=256)
    dec.init_cache(max_seqs=4, max_len=64)
    yield cfg, w, wa, dec
    dec.close()


def _oracle(cfg, w, wa, h, tau, n_seqs, seq_len, **kw):
    out = ho.decoder_forward(ho.OracleConfig.from_stack(cfg), w, wa, h, tau, cfg.n_heads,
                             cfg.n_kv_heads, cfg.rope_theta, n_seqs, seq_len, **kw)
    out["tau"] = tau
    return out


def _step_refs(cfg, w, wa, tau, h0, B, S, new_rows, pos):
    """Oracle of a decoding step: per sequence b the forward over its first pos[b]
    prefill tokens followed by the new tokens new_rows[k][b] (k = 0.. steps so far);
    returns the last row's h_out, gate [L] and mask [L] per sequence."""
    outs = []
    for b in range(B):
        rows = [h0[b * S:b * S + pos[b]]] + [nr[b:b + 1] for nr in new_rows]
        seq = np.concatenate(rows, axis=0)
        r = _oracle(cfg, w, wa, seq, tau, 1, seq.shape[0])
        outs.append((r["h_out"][-1], r["gate"][:, -1], r["mask"][:, -1]))
    return (np.stack([o[0] for o in outs]), np.stack([o[1] for o in outs], axis=1),
            np.stack([o[2] for o in outs], axis=1))


def test_decode_steps_forced_match_oracle(small, hero):
    """Prefill 3 sequences of 40 (forced to the oracle's decisions), then two decoding
    steps at ragged positions (40, 17, 33), then +1: each step's token against the
    oracle's forward over its prefix and the new tokens."""
    import torch
    cfg, w, wa, dec = small
    B, S = 3, 40
    tau = hi.calibrated_tau(cfg.name)
    h0 = hi.generate_h_in(cfg.replace(n_tokens=B * S))
    ref_pre = _oracle(cfg, w, wa, h0, tau, B, S)
    dec.prefill(_dev(h0), tau, 0, B, S, flags=hero.HERO_FLAG_FORCE_MASK,
                mask_in=_dev(np.ascontiguousarray(ref_pre["mask"])))
    pos = np.array([40, 17, 33])
    new_rows = []
    for step in range(2):
        hn = hi.generate_h_in(cfg.replace(n_tokens=B, seed=11 + step))
        new_rows.append(hn)
        # the oracle's prefix stops at the step's position: earlier steps are part of it
        p0 = pos - step
        h_ref, g_ref, m_ref = _step_refs(cfg, w, wa, tau, h0, B, S, new_rows, p0)
        h_out, g, m, c = dec.decode(_dev(hn), _dev(pos.astype(np.int32)), int(pos.max()), tau,
                                    flags=hero.HERO_FLAG_FORCE_MASK,
                                    mask_in=_dev(np.ascontiguousarray(m_ref)))
        torch.cuda.synchronize()
        dec.check()
        gerr = float(np.max(np.abs(_np(g).astype(np.float64) - g_ref)))
        herr = float(np.max(pr.rel_err_rows(_np(h_out).astype(np.float64), h_ref)))
        print("step", step, "pos", pos, "gate", gerr, "h", herr)
        np.testing.assert_array_equal(_np(m), m_ref)
        np.testing.assert_array_equal(_np(c), m_ref.sum(axis=1))
        assert gerr < pr.GATE_TOL and herr < H_TOL, (gerr, herr)
        pos = pos + 1


def test_decode_free_running(small, hero):
    """Free-running prefill and step: decisions equal the oracle's except within 1e-3
    of tau; a sequence with such a flip in its prefix is not compared."""
    import torch
    cfg, w, wa, dec = small
    B, S = 4, 48
    tau = hi.calibrated_tau(cfg.name)
    h0 = hi.generate_h_in(cfg.replace(n_tokens=B * S, seed=5))
    ref_pre = _oracle(cfg, w, wa, h0, tau, B, S)
    _, _, m_pre, _ = dec.prefill(_dev(h0), tau, 0, B, S)
    torch.cuda.synchronize()
    m_pre = _np(m_pre)
    pos = np.array([48, 47, 1, 30])
    hn = hi.generate_h_in(cfg.replace(n_tokens=B, seed=17))
    h_ref, g_ref, m_ref = _step_refs(cfg, w, wa, tau, h0, B, S, [hn], pos)
    h_out, g, m, _ = dec.decode(_dev(hn), _dev(pos.astype(np.int32)), int(pos.max()), tau)
    torch.cuda.synchronize()
    dec.check()
    g, m, h_out = _np(g).astype(np.float64), _np(m), _np(h_out).astype(np.float64)
    compared = 0
    for b in range(B):
        pre = slice(b * S, b * S + pos[b])
        flips = m_pre[:, pre] != ref_pre["mask"][:, pre]
        near = np.abs(ref_pre["gate"][:, pre] - tau) < pr.BOUNDARY
        assert not (flips & ~near).any(), b
        if flips.any():
            continue
        own = m[:, b] != m_ref[:, b]
        assert not (own & ~(np.abs(g_ref[:, b] - tau) < pr.BOUNDARY)).any(), b
        if own.any():
            continue
        compared += 1
        assert np.max(np.abs(g[:, b] - g_ref[:, b])) < pr.GATE_TOL
        assert pr.rel_err_rows(h_out[b:b + 1], h_ref[b:b + 1])[0] < H_TOL
    assert compared >= 3, compared


def test_decode_step_repeats_prefill_rows(small, hero):
    """A step whose token is the prefill's token at the same position reproduces the
    prefill's result for it (same keys and values, same routing)."""
    import torch
    cfg, w, wa, dec = small
    B, S = 4, 50
    tau = hi.calibrated_tau(cfg.name)
    h0 = hi.generate_h_in(cfg.replace(n_tokens=B * S, seed=3))
    h_pre, g_pre, m_pre, _ = dec.prefill(_dev(h0), tau, 0, B, S)
    torch.cuda.synchronize()
    pos = np.array([49, 0, 25, 63 - 14])
    rows = np.arange(B) * S + pos
    h_out, g, m, _ = dec.decode(_dev(h0[rows]), _dev(pos.astype(np.int32)), 49, tau)
    torch.cuda.synchronize()
    dec.check()
    hp, gp, mp = _np(h_pre)[rows], _np(g_pre)[:, rows], _np(m_pre)[:, rows]
    np.testing.assert_array_equal(_np(m), mp)
    assert float(np.max(np.abs(_np(g) - gp))) < pr.GATE_TOL
    assert float(np.max(pr.rel_err_rows(_np(h_out).astype(np.float64), hp.astype(np.float64)))) < H_TOL


def test_decode_rejects_and_reports(small, hero):
    """Argument errors come back before any work; a position past max_position is
    reported through the device error word (its cache writes stay in bounds)."""
    import torch
    cfg, _, _, dec = small
    h = torch.zeros((2, cfg.d_model), device="cuda")
    out = torch.zeros_like(h)
    pos = torch.tensor([3, 4], dtype=torch.int32, device="cuda")
    for args in [(2, pos.data_ptr(), 64), (2, pos.data_ptr(), -1), (5, pos.data_ptr(), 10),
                 (2, 0, 10)]:
        with pytest.raises(hero.HeroError) as e:
            hero.hero_decode_step(dec.model, args[0], args[1], args[2], h.data_ptr(), 0.3, 0, 0,
                                  out.data_ptr(), 0, 0, 0, 0)
        assert e.value.status == hero.HERO_ERR_ARG
    with pytest.raises(hero.HeroError):
        hero.hero_decoder_prefill(dec.model, 3, 2, 8, h.data_ptr(), 0.3, 0, 0, out.data_ptr(), 0, 0, 0, 0)
    bad = torch.tensor([3, 9], dtype=torch.int32, device="cuda")
    dec.decode(h, bad, 5, 0.3)
    with pytest.raises(hero.HeroError) as e:
        dec.check()
    assert e.value.status == hero.HERO_ERR_BAD_INDEX   # not taken for an expired wait
    dec.decode(h, pos, 5, 0.3)        # the model stays usable
    dec.check()


def test_decode_full_size(hero):
    """Llama-3.1-8B shapes: 8 cache slots with a 4096-token prefill (two prefill calls
    of 4 x 4096), then one step for all 8 slots at positions up to 4095 whose tokens
    repeat prefill tokens (the prefill's results for them, which the prefix test checks
    against the oracle), and one step at position 20 after a 20-token prefill, both
    forced to the oracle's decisions, checked against the oracle's 21-token forward."""
    import torch
    cfg = hi.CONFIGS["llama31_8b_decoder"]
    B, S = cfg.batch, cfg.seq_len
    tau = hi.calibrated_tau(cfg.name)
    w, wa = hi.generate_weights(cfg), hi.generate_attn_weights(cfg)
    h0 = hi.generate_h_in(cfg)
    dec = hero.HeroDecoder(cfg, w, wa)
    dec.init_cache(max_seqs=2 * B, max_len=S + 8)
    pre = [dec.prefill(_dev(h0), tau, seq0, B, S) for seq0 in (0, B)]
    torch.cuda.synchronize()
    h_pre, g_pre, m_pre = _np(pre[0][0]), _np(pre[0][1]), _np(pre[0][2])
    pos = np.array([4095, 0, 17, 2048, 4095, 4094, 1000, 3])
    rows = (np.arange(2 * B) % B) * S + pos
    h_out, g, m, _ = dec.decode(_dev(h0[rows]), _dev(pos.astype(np.int32)), 4095, tau)
    torch.cuda.synchronize()
    dec.check()
    # the two paths round different operands (the prefill's P V takes bf16 probabilities,
    # the step's fp32) and 32 blocks amplify that like an fp32-level perturbation of h_0:
    # the free-running full-depth bound applies
    # the free-running full-depth bound applies to gates, and a decision may differ only
    # where the prefill's gate lies within that bound of tau (that token is then dropped)
    bound = pr.free_run_gate_bound("llama31_8b_prefill")
    gs, ms_, hs = _np(g).astype(np.float64), _np(m), _np(h_out).astype(np.float64)
    gp, mp, hp = g_pre[:, rows].astype(np.float64), m_pre[:, rows], h_pre[rows].astype(np.float64)
    alive = np.ones(len(rows), dtype=bool)
    gerr = 0.0
    for j in range(cfg.n_layers):
        flip = ms_[j] != mp[j]
        assert not (flip & alive & ~(np.abs(gp[j] - tau) < bound)).any(), j
        gerr = max(gerr, float(np.max(np.abs(gs[j] - gp[j])[alive], initial=0.0)))
        alive &= ~flip
    herr = float(np.max(pr.rel_err_rows(hs[alive], hp[alive])))
    print("full-size step vs prefill rows: gate", gerr, "h", herr, "compared", int(alive.sum()))
    assert alive.sum() >= 6 and gerr < bound and herr < H_TOL
    # slot 0 refilled with a 20-token prefill forced to the oracle's decisions, then a
    # new token at position 20, against the oracle's 21-token forward
    hn = hi.generate_h_in(cfg.replace(n_tokens=1, seed=23))
    seq = np.concatenate([h0[:20], hn], axis=0)
    ref = _oracle(cfg, w, wa, seq, tau, 1, 21)
    dec.prefill(_dev(h0[:20]), tau, 0, 1, 20, flags=hero.HERO_FLAG_FORCE_MASK,
                mask_in=_dev(np.ascontiguousarray(ref["mask"][:, :20])))
    h1, g1, m1, _ = dec.decode(_dev(hn), _dev(np.array([20], dtype=np.int32)), 20, tau,
                               flags=hero.HERO_FLAG_FORCE_MASK,
                               mask_in=_dev(np.ascontiguousarray(ref["mask"][:, -1:])))
    torch.cuda.synchronize()
    dec.check()
    gerr = float(np.max(np.abs(_np(g1)[:, 0] - ref["gate"][:, -1])))
    herr = float(pr.rel_err_rows(_np(h1).astype(np.float64), ref["h_out"][-1:])[0])
    print("full-size step at 20: gate", gerr, "h", herr)
    assert gerr < pr.free_run_gate_bound("llama31_8b_prefill") and herr < H_TOL
    dec.close()
    torch.cuda.empty_cache()


def test_host_io_and_graph_capture(small, hero):
    """The decoder forward and a decoding step through host buffers (HERO_FLAG_HOST_IO)
    equal the device-buffer calls bit for bit, and a decoding step captured in a CUDA
    graph replays to the eager result (device-resident positions: no host sync)."""
    import torch
    cfg, w, wa, dec = small
    B, S, d, L = 3, 40, cfg.d_model, cfg.n_layers
    tau = hi.calibrated_tau(cfg.name)
    h0 = hi.generate_h_in(cfg.replace(n_tokens=B * S, seed=9))
    ref = dec.forward(_dev(h0), tau, B, S)
    torch.cuda.synchronize()
    hp = torch.from_numpy(h0).pin_memory()
    ho_ = torch.empty((B * S, d)).pin_memory()
    gp = torch.empty((L, B * S)).pin_memory()
    mp = torch.empty((L, B * S), dtype=torch.uint8).pin_memory()
    cp = torch.empty((L,), dtype=torch.int32).pin_memory()
    stream = torch.cuda.current_stream().cuda_stream
    hero.hero_decoder_forward(dec.model, B, S, hp.data_ptr(), tau, hero.HERO_FLAG_HOST_IO, 0,
                              ho_.data_ptr(), gp.data_ptr(), mp.data_ptr(), cp.data_ptr(), stream)
    torch.cuda.synchronize()
    dec.check()
    assert torch.equal(ho_, ref[0].cpu()) and torch.equal(gp, ref[1].cpu()) and torch.equal(mp, ref[2].cpu())
    assert torch.equal(cp, ref[3].cpu())
    # a prefill, then the same step through device buffers, host buffers and a graph
    dec.prefill(_dev(h0), tau, 0, B, S)
    hn = hi.generate_h_in(cfg.replace(n_tokens=B, seed=31))
    pos = np.array([40, 12, 39], dtype=np.int32)
    outs = [torch.empty((B, d), device="cuda"), torch.empty((L, B), device="cuda"),
            torch.empty((L, B), dtype=torch.uint8, device="cuda"),
            torch.empty((L,), dtype=torch.int32, device="cuda")]
    hn_d, pos_d = _dev(hn), _dev(pos)
    dec.decode(hn_d, pos_d, 40, tau, h_out=outs[0], gate_out=outs[1], mask_out=outs[2],
               counts_out=outs[3])
    torch.cuda.synchronize()
    eager = [o.clone() for o in outs]
    hp2 = torch.from_numpy(hn).pin_memory()
    pp = torch.from_numpy(pos).pin_memory()
    ho2 = torch.empty((B, d)).pin_memory()
    cp2 = torch.empty((L,), dtype=torch.int32).pin_memory()
    hero.hero_decode_step(dec.model, B, pp.data_ptr(), 40, hp2.data_ptr(), tau, hero.HERO_FLAG_HOST_IO,
                          0, ho2.data_ptr(), 0, 0, cp2.data_ptr(), stream)
    torch.cuda.synchronize()
    assert torch.equal(ho2, eager[0].cpu()) and torch.equal(cp2, eager[3].cpu())
    for o in outs:
        o.zero_()
    graph = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream()
    cap.wait_stream(torch.cuda.current_stream())
    with torch.cuda.graph(graph, stream=cap):
        dec.decode(hn_d, pos_d, 40, tau, h_out=outs[0], gate_out=outs[1], mask_out=outs[2],
                   counts_out=outs[3], stream=cap)
    torch.cuda.current_stream().wait_stream(cap)
    graph.replay()
    torch.cuda.synchronize()
    dec.check()
    for a_, b_ in zip(outs, eager):
        assert torch.equal(a_, b_)
