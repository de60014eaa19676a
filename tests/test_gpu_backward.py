"""GPU parity of the training path (Sec. 3.1, Sec. 3.3): the backward of a routed
block's branch part with its decisions fixed (hero_routed_block_backward) and the
skip penalty's gradient (hero_skip_penalty_grad), against the oracle's
block_branch_backward and skip_penalty_grad (float64, pinned by central differences).

Bounds (bf16 models; the oracle takes the bf16 parameters and fp32 inputs in float64
with no intermediate rounding, while the GPU rounds its GEMM operands to bf16 with
fp32 accumulation):
  * dL/dh_bar: per token ||x_t - y_t||_inf / ||y_t||_inf below 2e-2 (the hidden-state
    bound of bf16 workloads);
  * dL/dg, dL/dW_1, dL/dW_2: max |x - y| below 2e-2 max |y| (the same relative bound
    taken over the whole output, since single entries can be near zero).
"""

import numpy as np
import pytest

from oracle import hero_oracle as ho
from synth import hero_inputs as hi
from tests import parity as pr

pytestmark = pytest.mark.gpu

REL = 2e-2
_LAYER_KEYS = ("ffn_norm_g", "w_gate", "w_up", "w_down", "ad_w1", "ad_w2")


@pytest.fixture(scope="module")
def hero():
    import torch
    assert torch.cuda.is_available()
    from paper_2609_08189_gb300 import build, hero as H
    build.build()
    H.load()
    return H


def _wl(weights, j):
    return {k: ho._f64(weights[k][j - 1]) for k in _LAYER_KEYS}


def _dev(a, dtype=None):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(a))
    return t.cuda() if dtype is None else t.to(dtype).cuda()


def _run(st, j, h_bar, g, mask, G, flags=0):
    import torch
    out = st.block_backward(j, _dev(h_bar), None if g is None else _dev(g),
                            None if mask is None else _dev(mask), _dev(G), flags=flags)
    torch.cuda.synchronize()
    st.check()
    return [o.cpu().numpy().astype(np.float64) for o in out]


def _rel_max(x, y):
    return float(np.max(np.abs(x - y)) / max(np.max(np.abs(y)), 1e-30))


def _compare(got, ref, rows=None, check_w=True):
    gh, gg, g1, g2 = got
    sel = slice(None) if rows is None else rows
    eh = float(np.max(pr.rel_err_rows(gh[sel], ref["dh_bar"])))
    eg = _rel_max(gg[sel], ref["dg"])
    assert eh < REL, eh
    assert eg < REL, eg
    if check_w:
        e1, e2 = _rel_max(g1, ref["dW1"]), _rel_max(g2, ref["dW2"])
        assert e1 < REL and e2 < REL, (e1, e2)
        return eh, eg, e1, e2
    return eh, eg


@pytest.fixture(scope="module")
def small(hero):
    inp = pr.inputs("small_bf16")
    cfg = inp.cfg
    ref = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), inp.weights, inp.h, inp.P, inp.tau,
                              record=True)
    st = hero.HeroStack(cfg, inp.weights)
    st.backward_init()
    G = np.random.default_rng(31).standard_normal((cfg.n_tokens, cfg.d_model)).astype(np.float32)
    yield inp, ref, st, G
    st.close()


def test_block_backward_small_every_block(small):
    """Every block of the small bf16 stack, all 333 tokens, teacher-forced: the block's
    h_bar, g and decisions come from the oracle's forward."""
    inp, ref, st, G = small
    for j in range(1, inp.cfg.n_layers + 1):
        lay = ref["layers"][j - 1]
        hb = lay["h_bar"].astype(np.float32)
        g = lay["g"].astype(np.float32)
        mask = lay["mask"].astype(np.uint8)
        assert 0 < mask.sum() < mask.size
        exp = ho.block_branch_backward(hb.astype(np.float64), g.astype(np.float64),
                                       mask.astype(bool), G, _wl(inp.weights, j), inp.cfg.rms_eps)
        errs = _compare(_run(st, j, hb, g, mask, G), exp)
        print("block", j, "errors dh_bar, dg, dW1, dW2:", errs)


@pytest.mark.parametrize("path", [0, 1])
def test_block_backward_single_branch(small, path):
    """All tokens on one branch: the other branch's rows are empty (n_a = 0 gives zero
    adapter gradients)."""
    inp, ref, st, G = small
    lay = ref["layers"][1]
    hb, g = lay["h_bar"].astype(np.float32), lay["g"].astype(np.float32)
    mask = np.full(inp.cfg.n_tokens, path, dtype=np.uint8)
    exp = ho.block_branch_backward(hb.astype(np.float64), g.astype(np.float64), mask.astype(bool),
                                   G, _wl(inp.weights, 2), inp.cfg.rms_eps)
    got = _run(st, 2, hb, g, mask, G)
    if path == 1:
        assert not got[2].any() and not got[3].any()
        _compare(got, exp, check_w=False)
    else:
        _compare(got, exp)


@pytest.mark.parametrize("T", [1, 2, 129])
def test_block_backward_ragged_token_counts(small, T):
    inp, ref, st, G = small
    lay = ref["layers"][2]
    hb, g = lay["h_bar"][:T].astype(np.float32), lay["g"][:T].astype(np.float32)
    mask = lay["mask"][:T].astype(np.uint8)
    if T == 2:
        mask = np.array([1, 0], dtype=np.uint8)
    exp = ho.block_branch_backward(hb.astype(np.float64), g.astype(np.float64), mask.astype(bool),
                                   G[:T], _wl(inp.weights, 3), inp.cfg.rms_eps)
    got = _run(st, 3, hb, g, mask, G[:T])
    _compare(got, exp, check_w=bool((mask == 0).any()))


def test_block_backward_dense_flag(small, hero):
    """HERO_FLAG_DENSE: every token through the FFN with scale 1 (a dense block's
    backward); dL/dg and the adapter gradients come back zero."""
    inp, ref, st, G = small
    lay = ref["layers"][0]
    hb = lay["h_bar"].astype(np.float32)
    T = inp.cfg.n_tokens
    exp = ho.block_branch_backward(hb.astype(np.float64), np.ones(T), np.ones(T, dtype=bool), G,
                                   _wl(inp.weights, 1), inp.cfg.rms_eps)
    gh, gg, g1, g2 = _run(st, 1, hb, None, None, G, flags=hero.HERO_FLAG_DENSE)
    assert float(np.max(pr.rel_err_rows(gh, exp["dh_bar"]))) < REL
    assert not gg.any() and not g1.any() and not g2.any()


def test_block_backward_is_deterministic(small):
    inp, ref, st, G = small
    lay = ref["layers"][3]
    args = (lay["h_bar"].astype(np.float32), lay["g"].astype(np.float32),
            lay["mask"].astype(np.uint8), G)
    a, b = _run(st, 4, *args), _run(st, 4, *args)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


def test_block_backward_argument_errors(hero, small):
    import torch
    inp, ref, st, G = small
    T, d = 8, inp.cfg.d_model
    x = torch.zeros((T, d), device="cuda")
    y = torch.zeros_like(x)
    g = torch.zeros(T, device="cuda")
    m = torch.zeros(T, device="cuda", dtype=torch.uint8)
    w = torch.zeros(inp.cfg.d_r * d, device="cuda")
    call = lambda mod, blk, gh, fl=0: hero.hero_routed_block_backward(
        mod, blk, T, x.data_ptr(), g.data_ptr(), m.data_ptr(), y.data_ptr(), fl, gh, g.data_ptr(),
        w.data_ptr(), w.data_ptr(), 0)
    for blk in (0, inp.cfg.n_layers + 1):
        with pytest.raises(hero.HeroError) as e:
            call(st.model, blk, torch.empty_like(x).data_ptr())
        assert e.value.status == hero.HERO_ERR_ARG
    with pytest.raises(hero.HeroError) as e:        # grad_h_bar aliases h_bar
        call(st.model, 1, x.data_ptr())
    assert e.value.status == hero.HERO_ERR_ARG
    with pytest.raises(hero.HeroError) as e:        # unknown flag
        call(st.model, 1, torch.empty_like(x).data_ptr(), 2)
    assert e.value.status == hero.HERO_ERR_ARG
    other = hero.HeroStack(inp.cfg, inp.weights)
    with pytest.raises(hero.HeroError) as e:        # hero_backward_init not called
        call(other.model, 1, torch.empty_like(x).data_ptr())
    assert e.value.status == hero.HERO_ERR_ARG
    other.close()
    with pytest.raises(hero.HeroError) as e:        # a second init
        st.backward_init()
    assert e.value.status == hero.HERO_ERR_ARG
    f32 = pr.inputs("tiny_f32")
    fm = hero.HeroStack(f32.cfg, f32.weights)
    with pytest.raises(hero.HeroError) as e:
        fm.backward_init()
    assert e.value.status == hero.HERO_ERR_UNSUPPORTED
    fm.close()


@pytest.mark.parametrize("name,T", [("llama31_8b_prefill", 4000), ("llama2_13b_prefill", 2500)])
def test_block_backward_llama_shapes(hero, name, T):
    """Llama FFN shapes (d, I, d_r of the workload; two blocks of it, block 2 tested) on
    T tokens (not a multiple of the 128-row tile): dL/dh_bar and dL/dg on an evenly
    spread token sample (tokens are independent once the decisions are fixed), the
    adapter's weight gradients over all adapter tokens (the oracle's adapter part alone)."""
    cfg = hi.CONFIGS[name].replace(n_layers=2, n_tokens=T)
    w = hi.generate_weights(cfg)
    rng = np.random.default_rng(41)
    hb = rng.standard_normal((T, cfg.d_model)).astype(np.float32)
    g = rng.uniform(0.05, 0.95, T).astype(np.float32)
    mask = (g >= 0.3).astype(np.uint8)
    G = rng.standard_normal((T, cfg.d_model)).astype(np.float32)
    st = hero.HeroStack(cfg, w)
    st.backward_init()
    got = _run(st, 2, hb, g, mask, G)
    st.close()
    wl = _wl(w, 2)
    rows = hi.sample_tokens(T, 48)
    exp = ho.block_branch_backward(hb[rows].astype(np.float64), g[rows].astype(np.float64),
                                   mask[rows].astype(bool), G[rows], wl, cfg.rms_eps)
    _compare(got, exp, rows=rows, check_w=False)
    A = np.nonzero(mask == 0)[0]
    expw = ho.block_branch_backward(hb[A].astype(np.float64), g[A].astype(np.float64),
                                    np.zeros(len(A), dtype=bool), G[A], wl, cfg.rms_eps)
    e1, e2 = _rel_max(got[2], expw["dW1"]), _rel_max(got[3], expw["dW2"])
    print(name, "dW1", e1, "dW2", e2, "adapter rows", len(A))
    assert e1 < REL and e2 < REL


@pytest.mark.parametrize("n_dense,n_seqs,seq_len", [(0, 3, 7), (1, 2, 5), (0, 1, 2)])
def test_skip_penalty_grad(hero, n_dense, n_seqs, seq_len):
    import torch
    L = 4
    T = n_seqs * seq_len
    gates = np.random.default_rng(5).uniform(0, 1, (L, T)).astype(np.float32)
    out = torch.full((L, T), float("nan"), device="cuda")
    gd = _dev(gates)
    hero.hero_skip_penalty_grad(L, n_dense, n_seqs, seq_len, gd.data_ptr(), 0.3, out.data_ptr(),
                                torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    ref = 0.3 * ho.skip_penalty_grad(gates.astype(np.float64), n_seqs, seq_len, n_dense)
    np.testing.assert_allclose(out.cpu().numpy(), ref, rtol=1e-6, atol=1e-7)
    with pytest.raises(hero.HeroError) as e:    # one-token sequences have no next-token term
        hero.hero_skip_penalty_grad(L, 0, T, 1, gd.data_ptr(), 0.3, out.data_ptr(), 0)
    assert e.value.status == hero.HERO_ERR_ARG
