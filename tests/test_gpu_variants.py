"""GPU parity of the router ablations (Sec. 4.4) and of memory widths d_m = 32, 128, 256.

Each ablation bit (HERO_ROUTER_NO_HISTORY, _NO_MEMREAD, _NO_AUX, _NO_POS) and the
widest memory of the paper's memory-dimension ablation run through the CUDA path
and are compared with the float64 oracle run with the same switch: free-running
(decisions near the threshold excluded, as in the other free-running tests) and
forced-mask (the oracle's decisions fed to the GPU).  tau is the median of the
oracle's first-block gates (the first block does not depend on tau), so both
branches are exercised.
"""

import numpy as np
import pytest

from oracle import hero_oracle as ho
from synth import hero_inputs as hi
from tests import parity as pr

pytestmark = pytest.mark.gpu

VARIANTS = [ho.NO_HISTORY, ho.NO_MEMREAD, ho.NO_AUX, ho.NO_POS, ho.NO_AUX | ho.NO_POS]
CASES = ([(name, v, None) for name in ("tiny_f32", "small_bf16") for v in VARIANTS] +
         [("tiny_f32", 0, 256), ("small_bf16", 0, 256), ("small_bf16", ho.NO_MEMREAD, 256),
          # the small-token-count router splits a token's memory step over warps; these
          # widths take whole-row iterations of 4 and 16 rows per warp
          ("small_bf16", 0, 32), ("small_bf16", 0, 128)])


@pytest.fixture(scope="module")
def hero():
    import torch
    assert torch.cuda.is_available()
    from paper_2609_08189_gb300 import build, hero as H
    build.build()
    H.load()
    return H


def _inputs(name, variant, d_m):
    base = hi.CONFIGS[name]
    kw = {"router_variant": variant}
    if d_m:
        kw["d_m"] = d_m
    cfg = base.replace(name=f"{name}_v{variant}_m{d_m or base.d_m}", **kw)
    w, h, P = hi.generate_weights(cfg), hi.generate_h_in(cfg), hi.generate_attn_delta(cfg)
    first = ho.routed_ffn_stack(ho.OracleConfig.from_stack(cfg), w, h, P, 0.5)
    tau = float(np.median(first["gate"][0]))   # block 1's gates do not depend on tau
    return pr.Inputs(cfg, w, h, P, tau)


@pytest.mark.parametrize("name,variant,d_m", CASES)
def test_router_variant_parity(hero, name, variant, d_m):
    inp = _inputs(name, variant, d_m)
    cfg = inp.cfg
    st = hero.HeroStack(cfg, inp.weights)
    tol_h = pr.H_TOL[cfg.dtype]
    gpu = pr.run_gpu(st, inp)
    ref = pr.run_oracle(inp)
    rep = pr.compare_free(gpu, ref, tol_h)
    print(cfg.name, "free", rep, "bypass", 1 - gpu.mask.mean())
    assert rep.mask_mismatch_far == 0, rep
    assert rep.gate_err < pr.GATE_TOL, rep
    assert len(rep.boundary_tokens) <= max(1, 0.02 * rep.n_tokens), rep
    assert rep.compared_h >= 0.9 * rep.n_tokens, rep
    assert rep.h_err < tol_h, rep
    np.testing.assert_array_equal(gpu.counts, gpu.mask.sum(axis=1))
    assert 0 < gpu.mask.sum() < gpu.mask.size          # both branches taken
    forced = pr.run_gpu(st, inp, flags=hero.HERO_FLAG_FORCE_MASK, mask_in=ref["mask"])
    frep = pr.compare_forced(forced, ref)
    print(cfg.name, "forced", frep)
    assert frep.mask_mismatch_far == 0
    assert frep.gate_err < pr.GATE_TOL and frep.h_err < tol_h
    st.close()


def test_variant_changes_the_router(hero):
    """The switch reaches the kernel: the ablated router's gates differ from HeRo's."""
    full = _inputs("small_bf16", 0, None)
    abl = _inputs("small_bf16", ho.NO_HISTORY, None)
    g_full = pr.run_gpu(hero.HeroStack(full.cfg, full.weights), full).gate[0]
    g_abl = pr.run_gpu(hero.HeroStack(abl.cfg, abl.weights), abl).gate[0]
    assert np.max(np.abs(g_full - g_abl)) > 1e-3
