"""GPU parity of single routed blocks (hero_routed_block).

Teacher-forced parity: block j of the CUDA path is fed the oracle's own state
before block j (memory S, zeta, p_hist, m_hist, d_{j-1}, h_bar_{j-1}, delta_{j-1})
and its post-attention input h_bar_j, runs once, and is compared with the oracle's
block j: gates, decisions, h_j and the updated state.  Each block is compared in
isolation, so the bf16 rounding cascade through depth (see the free-running
tests) does not enter and the stated bounds apply block by block at full size.
Also: chaining hero_routed_block over all blocks reproduces hero_routed_ffn_stack.
"""

import numpy as np
import pytest

from oracle import hero_oracle as ho
from synth import hero_inputs as hi
from tests import parity as pr

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def hero():
    import torch
    assert torch.cuda.is_available()
    from paper_2609_08189_gb300 import build, hero as H
    build.build()
    H.load()
    return H


def _state_tensors(T, d, dm):
    import torch
    f = dict(device="cuda", dtype=torch.float32)
    return {"S": torch.zeros((T, dm, dm), **f), "zeta": torch.zeros((T, dm), **f),
            "p_hist": torch.ones((T,), **f), "m_hist": torch.ones((T,), **f),
            "d_prev": torch.zeros((T,), **f), "h_bar_prev": torch.zeros((T, d), **f),
            "delta_prev": torch.zeros((T, d), **f)}


def _ptrs(ts):
    return {k: v.data_ptr() for k, v in ts.items()}


TF = [("tiny_f32", None, None), ("small_bf16", None, None), ("small_bf16_placed", None, None),
      ("llama2_7b_prefill", None, 32), ("llama31_8b_prefill", None, 32),
      ("llama31_8b_decode", None, 32), ("llama2_13b_prefill", 0.27, 16),
      ("llama2_13b_prefill", 0.0, 16), ("llama2_13b_prefill", 0.39, 16),
      ("llama31_8b_paper", None, 16)]


@pytest.mark.parametrize("name,bypass,n_sample", TF)
def test_teacher_forced_blocks(hero, name, bypass, n_sample):
    import torch
    inp = pr.inputs(name, bypass=bypass)
    cfg = inp.cfg
    rows = np.arange(cfg.n_tokens) if n_sample is None else hi.sample_tokens(cfg.n_tokens, n_sample)
    T, d, dm, L = len(rows), cfg.d_model, cfg.d_m, cfg.n_layers
    ref = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), inp.weights, inp.h[rows],
                              inp.P[:, rows], inp.tau, record=True)
    lay = ref["layers"]
    st = hero.HeroStack(cfg, inp.weights, max_tokens=T)
    ts = _state_tensors(T, d, dm)
    state = hero.make_state(_ptrs(ts))
    g = torch.empty(T, device="cuda")
    m = torch.empty(T, device="cuda", dtype=torch.uint8)
    h_out = torch.empty((T, d), device="cuda")
    cnt = torch.empty(1, device="cuda", dtype=torch.int32)
    stream = torch.cuda.current_stream().cuda_stream
    tol_h = pr.H_TOL[cfg.dtype]
    worst_g = worst_h = worst_S = 0.0
    far = 0
    f32 = lambda a: torch.as_tensor(np.ascontiguousarray(a, dtype=np.float32), device="cuda")
    nd = cfg.n_dense          # layers 1..nd are plain FFN blocks (placement)
    for j in range(1, L + 1):
        jr = j - nd
        if jr == 1:
            hero.hero_router_state_reset(st.model, T, state, stream)
        elif jr > 1:
            prev = lay[j - 2]
            ts["S"].copy_(f32(prev["S"]))
            ts["zeta"].copy_(f32(prev["zeta"]))
            ts["p_hist"].copy_(f32(prev["p"]))
            ts["m_hist"].copy_(f32(prev["m"]))
            ts["d_prev"].copy_(f32(prev["d"]))
            ts["h_bar_prev"].copy_(f32(prev["h_bar"]))
            ts["delta_prev"].copy_(f32(prev["delta"]))
        cur = lay[j - 1]
        hb = f32(cur["h_bar"])
        mask_in = torch.as_tensor(cur["mask"].astype(np.uint8), device="cuda")
        hero.hero_routed_block(st.model, j, T, hb.data_ptr(), state, inp.tau,
                               hero.HERO_FLAG_FORCE_MASK, mask_in.data_ptr(), h_out.data_ptr(),
                               g.data_ptr(), m.data_ptr(), cnt.data_ptr(), stream)
        torch.cuda.synchronize()
        st.check()
        gg = g.cpu().numpy().astype(np.float64)
        worst_g = max(worst_g, float(np.max(np.abs(gg - cur["g"]))))
        worst_h = max(worst_h, float(np.max(pr.rel_err_rows(h_out.cpu().numpy().astype(np.float64),
                                                            cur["h"]))))
        # the free decision the GPU would take agrees with the oracle's away from the boundary
        dec = gg >= inp.tau
        far += int(np.sum((dec != cur["mask"]) & (np.abs(cur["g"] - inp.tau) >= pr.BOUNDARY)))
        assert int(cnt.item()) == int(cur["mask"].sum())
        if jr >= 1:
            Sg = ts["S"].cpu().numpy().astype(np.float64)
            worst_S = max(worst_S, float(np.max(np.abs(Sg - cur["S"])) /
                                         (np.max(np.abs(cur["S"])) + 1e-30)))
    print(name, "teacher-forced: gate", worst_g, "h", worst_h, "S", worst_S)
    assert far == 0
    assert worst_g < pr.GATE_TOL
    assert worst_h < tol_h
    assert worst_S < (1e-5 if cfg.dtype == "f32" else 1e-3)
    st.close()


@pytest.mark.parametrize("name", ["tiny_f32", "small_bf16", "small_bf16_placed"])
def test_block_chain_equals_fused_stack(hero, name):
    """Blocks run one by one (attention stand-in added by the caller) == the fused stack."""
    import torch
    inp = pr.inputs(name)
    cfg = inp.cfg
    T, d, L = cfg.n_tokens, cfg.d_model, cfg.n_layers
    st = hero.HeroStack(cfg, inp.weights)
    fused = pr.run_gpu(st, inp)
    ts = _state_tensors(T, d, cfg.d_m)
    state = hero.make_state(_ptrs(ts))
    stream = torch.cuda.current_stream().cuda_stream
    h = torch.from_numpy(inp.h).cuda()
    if inp.P.dtype == np.uint16:
        P = torch.from_numpy(inp.P.astype(np.int32) << 16).cuda().view(torch.float32)
    else:
        P = torch.from_numpy(inp.P).cuda()
    g = torch.empty((L, T), device="cuda")
    m = torch.empty((L, T), device="cuda", dtype=torch.uint8)
    hero.hero_router_state_reset(st.model, T, state, stream)
    for j in range(1, L + 1):
        hb = h + P[j - 1]                    # the caller's "attention" output
        h = torch.empty_like(hb)
        hero.hero_routed_block(st.model, j, T, hb.data_ptr(), state, inp.tau, 0, 0, h.data_ptr(),
                               g[j - 1].data_ptr(), m[j - 1].data_ptr(), 0, stream)
    torch.cuda.synchronize()
    st.check()
    np.testing.assert_array_equal(m.cpu().numpy(), fused.mask)
    assert np.max(np.abs(g.cpu().numpy() - fused.gate)) < 1e-5
    assert np.max(pr.rel_err_rows(h.cpu().numpy().astype(np.float64), fused.h_out)) < 1e-4
    st.close()


def test_block_argument_errors(hero):
    import torch
    inp = pr.inputs("tiny_f32")
    st = hero.HeroStack(inp.cfg, inp.weights)
    state = hero.make_state({})
    x = torch.zeros((4, inp.cfg.d_model), device="cuda")
    y = torch.zeros_like(x)
    for block in (0, inp.cfg.n_layers + 1):
        with pytest.raises(hero.HeroError) as e:
            hero.hero_routed_block(st.model, block, 4, x.data_ptr(), state, 0.5, 0, 0, y.data_ptr(),
                                   0, 0, 0, 0)
        assert e.value.status == hero.HERO_ERR_ARG
    with pytest.raises(hero.HeroError) as e:   # routed mode needs the state
        hero.hero_routed_block(st.model, 1, 4, x.data_ptr(), state, 0.5, 0, 0, y.data_ptr(), 0, 0, 0, 0)
    assert e.value.status == hero.HERO_ERR_ARG
    with pytest.raises(hero.HeroError):        # host I/O is not accepted per block
        hero.hero_routed_block(st.model, 1, 4, x.data_ptr(), state, 0.5, hero.HERO_FLAG_HOST_IO, 0,
                               y.data_ptr(), 0, 0, 0, 0)
    # dense mode needs no state
    hero.hero_routed_block(st.model, 1, 4, x.data_ptr(), state, 0.5, hero.HERO_FLAG_DENSE, 0,
                           y.data_ptr(), 0, 0, 0, 0)
    torch.cuda.synchronize()
    st.check()
    st.close()


def test_teacher_forced_blocks_tensor_core_router(hero):
    """From 1024 tokens, when the router contraction does not split K, the router runs on the
    tensor cores (five launches; the router's small matrices as bf16 B operands, each fp32
    activation split into three bf16 terms, so every product is exact and the sums accumulate
    in fp32).  At Llama-3.1-8B shapes that needs about 8192 tokens, more than the oracle runs
    in seconds; tokens are independent, so 32 sampled tokens, each with its oracle state before
    every block, are repeated 256 times to fill 8192 rows.  Teacher-forced over 4 blocks:
    every row against its token's oracle values, with the stated bounds, and the 256 copies
    of a token bitwise equal."""
    import torch
    base = hi.CONFIGS["llama31_8b_prefill"]
    cfg = base.replace(n_layers=4)
    w = hi.generate_weights(cfg)
    rows = hi.sample_tokens(cfg.n_tokens, 32)
    h = hi.generate_h_in(cfg)[rows]
    P = hi.generate_attn_delta(cfg)[:, rows]
    tau = hi.calibrated_tau(base.name)
    rep = 256
    T, d, dm, L = len(rows) * rep, cfg.d_model, cfg.d_m, cfg.n_layers
    ref = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P, tau, record=True)
    lay = ref["layers"]
    st = hero.HeroStack(cfg.replace(n_tokens=T), w, max_tokens=T)
    ts = _state_tensors(T, d, dm)
    state = hero.make_state(_ptrs(ts))
    g = torch.empty(T, device="cuda")
    m = torch.empty(T, device="cuda", dtype=torch.uint8)
    h_out = torch.empty((T, d), device="cuda")
    cnt = torch.empty(1, device="cuda", dtype=torch.int32)
    stream = torch.cuda.current_stream().cuda_stream
    tile = lambda a: np.tile(np.asarray(a), (rep,) + (1,) * (np.ndim(a) - 1))
    f32 = lambda a: torch.as_tensor(np.ascontiguousarray(tile(a), dtype=np.float32), device="cuda")
    worst_g = worst_h = worst_S = 0.0
    far = 0
    for j in range(1, L + 1):
        if j == 1:
            hero.hero_router_state_reset(st.model, T, state, stream)
        else:
            prev = lay[j - 2]
            for key, src in (("S", "S"), ("zeta", "zeta"), ("p_hist", "p"), ("m_hist", "m"),
                             ("d_prev", "d"), ("h_bar_prev", "h_bar"), ("delta_prev", "delta")):
                ts[key].copy_(f32(prev[src]))
        cur = lay[j - 1]
        mask_in = torch.as_tensor(tile(cur["mask"].astype(np.uint8)), device="cuda")
        hero.hero_routed_block(st.model, j, T, f32(cur["h_bar"]).data_ptr(), state, tau,
                               hero.HERO_FLAG_FORCE_MASK, mask_in.data_ptr(), h_out.data_ptr(),
                               g.data_ptr(), m.data_ptr(), cnt.data_ptr(), stream)
        torch.cuda.synchronize()
        st.check()
        gg = g.cpu().numpy().astype(np.float64).reshape(rep, -1)
        hh = h_out.cpu().numpy().astype(np.float64).reshape(rep, len(rows), d)
        Sg = ts["S"].cpu().numpy().astype(np.float64).reshape(rep, len(rows), dm, dm)
        for arr in (gg, hh, Sg):   # the copies of a token agree bitwise
            assert (arr == arr[:1]).all()
        worst_g = max(worst_g, float(np.max(np.abs(gg[0] - cur["g"]))))
        worst_h = max(worst_h, float(np.max(pr.rel_err_rows(hh[0], cur["h"]))))
        far += int(np.sum(((gg[0] >= tau) != cur["mask"]) & (np.abs(cur["g"] - tau) >= pr.BOUNDARY)))
        worst_S = max(worst_S, float(np.max(np.abs(Sg[0] - cur["S"])) / np.max(np.abs(cur["S"]))))
    print("tensor-core router, teacher-forced at", T, "rows: gate", worst_g, "h", worst_h, "S", worst_S)
    assert far == 0
    assert worst_g < pr.GATE_TOL
    assert worst_h < pr.H_TOL["bf16"]
    assert worst_S < 1e-3
    st.close()


def test_history_form_stack_equals_block_chain(hero):
    """The fused stack runs the tensor-core router's memory step in its history form (the
    unrolled recurrence of Eq. 12 over the token's earlier (phi(k_i), v_i)); the block API
    keeps the state S.  Same inputs at Llama-3.1-8B shapes, 8192 tokens, 4 blocks (the
    tensor-core path in both), the stack's decisions forced on the block chain.

    The two paths form h_bar's partial sums in different kernels, so gates start a few ulp
    apart (block 1 has no history: below 1e-6) and a few tokens amplify that through depth,
    about 3x per block in the mean.  With the state form in the stack too (a build with
    -DHERO_HISTORY_FORM=0) the differences are the same: max 4.1e-4 and mean 1.3e-6 at
    block 4, against 4.8e-4 and 1.4e-6 with the history form.  A wrong decay weight or
    history entry would move every token's c, so the per-block mean gate difference is held
    to 1e-5 and the maximum to the free-running drift bound."""
    import torch
    base = hi.CONFIGS["llama31_8b_prefill"]
    T = 8192
    cfg = base.replace(n_layers=4, n_tokens=T)
    inp = pr.Inputs(cfg, hi.generate_weights(cfg), hi.generate_h_in(cfg), hi.generate_attn_delta(cfg),
                    hi.calibrated_tau(base.name))
    d, dm, L = cfg.d_model, cfg.d_m, cfg.n_layers
    st = hero.HeroStack(cfg, inp.weights, max_tokens=T)
    fused = pr.run_gpu(st, inp)
    ts = _state_tensors(T, d, dm)
    state = hero.make_state(_ptrs(ts))
    stream = torch.cuda.current_stream().cuda_stream
    h = torch.from_numpy(inp.h).cuda()
    P = torch.from_numpy(inp.P.astype(np.int32) << 16).cuda().view(torch.float32)
    forced = torch.from_numpy(fused.mask.astype(np.uint8)).cuda()
    g = torch.empty((L, T), device="cuda")
    m = torch.empty((L, T), device="cuda", dtype=torch.uint8)
    hero.hero_router_state_reset(st.model, T, state, stream)
    for j in range(1, L + 1):
        hb = h + P[j - 1]
        h = torch.empty_like(hb)
        hero.hero_routed_block(st.model, j, T, hb.data_ptr(), state, inp.tau,
                               hero.HERO_FLAG_FORCE_MASK, forced[j - 1].data_ptr(), h.data_ptr(),
                               g[j - 1].data_ptr(), m[j - 1].data_ptr(), 0, stream)
    torch.cuda.synchronize()
    st.check()
    gd = np.abs(g.cpu().numpy().astype(np.float64) - fused.gate)
    eh = pr.rel_err_rows(h.cpu().numpy().astype(np.float64), fused.h_out)
    print("history form vs state form, per block: max", gd.max(axis=1), "mean", gd.mean(axis=1),
          "h max", eh.max(), "h median", np.median(eh))
    assert gd[0].max() < 1e-6
    assert (gd.mean(axis=1) < 1e-5).all()
    assert gd.max() < pr.free_run_gate_bound("llama31_8b_prefill")
    assert np.median(eh) < 1e-5
    st.close()
