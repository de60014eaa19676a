"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Small workloads compare every token; the full-size workloads run all T tokens on
the GPU in the bench's launch configuration and compare an evenly spread token
sample with the oracle run on exactly those tokens (tokens are independent
through the stack, P6 of the oracle pins).
"""

import numpy as np
import pytest

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


def _stack(H, inp, max_tokens=None):
    return H.HeroStack(inp.cfg, inp.weights, max_tokens=max_tokens)


def _assert_free(rep, tol_h, max_boundary_frac=0.02, gate_tol=pr.GATE_TOL):
    assert rep.mask_mismatch_far == 0, rep
    assert rep.gate_err < gate_tol, rep
    assert len(rep.boundary_tokens) <= max(1, max_boundary_frac * rep.n_tokens), rep
    assert rep.compared_h >= 0.9 * rep.n_tokens, rep
    assert rep.h_err < tol_h, rep


# ------------------------------------------------------------------------------
# the tensor-core GEMM alone
# ------------------------------------------------------------------------------

@pytest.mark.parametrize("M,N,K", [(1, 256, 64), (128, 512, 128), (129, 264, 4096), (333, 512, 1024),
                                   (1000, 768, 256)])
def test_gemm_building_block(hero, M, N, K):
    import torch
    g = torch.Generator(device="cuda").manual_seed(M * 7 + N + K)
    A = torch.randn(M, K, device="cuda", generator=g).to(torch.bfloat16)
    B = torch.randn(N, K, device="cuda", generator=g).to(torch.bfloat16)
    C = torch.full((M, N), float("nan"), device="cuda")
    hero.hero_gemm_bf16_check(A.data_ptr(), B.data_ptr(), C.data_ptr(), M, N, K,
                              torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    ref = A.double() @ B.double().T
    err = (C.double() - ref).abs().max().item()
    assert err <= 1e-5 * K ** 0.5 * ref.abs().max().item() + 1e-6, err


# ------------------------------------------------------------------------------
# full-token parity on small workloads
# ------------------------------------------------------------------------------

@pytest.mark.parametrize("name", ["tiny_f32", "small_bf16", "small_bf16_placed"])
def test_free_running(hero, name):
    inp = pr.inputs(name)
    st = _stack(hero, inp)
    gpu = pr.run_gpu(st, inp)
    ref = pr.run_oracle(inp)
    rep = pr.compare_free(gpu, ref, pr.H_TOL[inp.cfg.dtype])
    print(name, rep)
    _assert_free(rep, pr.H_TOL[inp.cfg.dtype])
    np.testing.assert_array_equal(gpu.counts, gpu.mask.sum(axis=1))
    bypass = 1 - gpu.mask[inp.cfg.n_dense:].mean()          # routed blocks only
    assert abs(bypass - inp.cfg.bypass) < 0.03
    st.close()


@pytest.mark.parametrize("name", ["tiny_f32", "small_bf16", "small_bf16_placed"])
def test_forced_mask(hero, name):
    inp = pr.inputs(name)
    st = _stack(hero, inp)
    ref = pr.run_oracle(inp)
    gpu = pr.run_gpu(st, inp, flags=hero.HERO_FLAG_FORCE_MASK, mask_in=ref["mask"])
    rep = pr.compare_forced(gpu, ref)
    print(name, rep)
    assert rep.mask_mismatch_far == 0
    assert rep.gate_err < pr.GATE_TOL
    assert rep.h_err < pr.H_TOL[inp.cfg.dtype]
    st.close()


@pytest.mark.parametrize("name", ["tiny_f32", "small_bf16", "small_bf16_placed"])
def test_dense(hero, name):
    inp = pr.inputs(name)
    st = _stack(hero, inp)
    ref = pr.run_oracle(inp, mode="dense")
    gpu = pr.run_gpu(st, inp, flags=hero.HERO_FLAG_DENSE)
    assert (gpu.mask == 1).all() and (gpu.gate == 1).all()
    assert (gpu.counts == inp.cfg.n_tokens).all()
    err = np.max(pr.rel_err_rows(gpu.h_out, ref["h_out"]))
    assert err < pr.H_TOL[inp.cfg.dtype], err
    st.close()


@pytest.mark.parametrize("name,path", [("tiny_f32", 0), ("tiny_f32", 1), ("small_bf16", 0),
                                       ("small_bf16", 1)])
def test_single_branch_everywhere(hero, name, path):
    """Forced all-adapter and all-FFN paths (one branch empty at every block)."""
    inp = pr.inputs(name)
    L, T = inp.cfg.n_layers, inp.cfg.n_tokens
    mask = np.full((L, T), path, dtype=np.uint8)
    st = _stack(hero, inp)
    ref = pr.run_oracle(inp, mode="force", mask_in=mask)
    gpu = pr.run_gpu(st, inp, flags=hero.HERO_FLAG_FORCE_MASK, mask_in=mask)
    assert (gpu.counts == path * T).all()
    assert np.max(np.abs(gpu.gate - ref["gate"])) < pr.GATE_TOL
    assert np.max(pr.rel_err_rows(gpu.h_out, ref["h_out"])) < pr.H_TOL[inp.cfg.dtype]
    st.close()


@pytest.mark.parametrize("T", [1, 2, 127, 129])
def test_ragged_token_counts(hero, T):
    """Fewer tokens than the model was sized for, including a single token."""
    inp = pr.inputs("small_bf16")
    st = _stack(hero, inp)
    rows = np.arange(T)
    gpu = pr.run_gpu(st, inp, n_tokens=T)
    ref = pr.run_oracle(inp, rows=rows)
    rep = pr.compare_free(gpu, ref, pr.H_TOL["bf16"])
    _assert_free(rep, pr.H_TOL["bf16"], max_boundary_frac=0.5)
    st.close()


@pytest.mark.parametrize("T", [200, 700, 1100, 2049, 4096])
def test_router_paths_by_token_count(hero, T):
    """The router's kernel follows the token count (bf16, the small_bf16 widths, whose router
    has the Llama widths); every token against the oracle, free-running:
      200   the router with its parameters in shared memory, 2 tokens per CTA
      700   the same, 8 tokens per CTA
      1100  8 tokens per CTA, compaction inside the norm's launch
      2049  16 tokens per CTA, the separate compaction (past 2048 tokens)
      4096  the router contraction no longer splits K: the router on the tensor cores, its
            memory step in the history form (small_bf16 has d = 512)."""
    inp = pr.inputs("small_bf16", cfg=hi.CONFIGS["small_bf16"].replace(n_tokens=T))
    st = _stack(hero, inp)
    gpu = pr.run_gpu(st, inp)
    ref = pr.run_oracle(inp)
    rep = pr.compare_free(gpu, ref, pr.H_TOL["bf16"])
    print(T, rep)
    _assert_free(rep, pr.H_TOL["bf16"])
    st.close()


@pytest.mark.parametrize("d_m", [16, 32, 128])
def test_tensor_core_router_memory_widths(hero, d_m):
    """The router on the tensor cores at other memory widths (small_bf16 widths, 4096 tokens:
    the router contraction does not split): the fused stack (state form for d_m = 16 and 32,
    history form for 128) against the oracle on every token, free-running; and the block
    chain (hero_routed_block, state form) with the stack's decisions forced against the
    stack."""
    import torch
    T = 4096
    cfg = hi.CONFIGS["small_bf16"].replace(n_tokens=T, d_m=d_m)
    inp = pr.inputs("small_bf16", cfg=cfg)
    st = _stack(hero, inp)
    gpu = pr.run_gpu(st, inp)
    ref = pr.run_oracle(inp)
    rep = pr.compare_free(gpu, ref, pr.H_TOL["bf16"])
    print(d_m, rep)
    _assert_free(rep, pr.H_TOL["bf16"])
    d, L = cfg.d_model, cfg.n_layers
    f = dict(device="cuda", dtype=torch.float32)
    ts = {"S": torch.zeros((T, d_m, d_m), **f), "zeta": torch.zeros((T, d_m), **f),
          "p_hist": torch.ones((T,), **f), "m_hist": torch.ones((T,), **f),
          "d_prev": torch.zeros((T,), **f), "h_bar_prev": torch.zeros((T, d), **f),
          "delta_prev": torch.zeros((T, d), **f)}
    state = hero.make_state({k: v.data_ptr() for k, v in ts.items()})
    stream = torch.cuda.current_stream().cuda_stream
    h = torch.from_numpy(inp.h).cuda()
    P = torch.from_numpy(inp.P.astype(np.int32) << 16).cuda().view(torch.float32)
    forced = torch.from_numpy(gpu.mask.astype(np.uint8)).cuda()
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
    gd = np.abs(g.cpu().numpy().astype(np.float64) - gpu.gate)
    print(d_m, "block chain vs stack: gate max", gd.max(), "mean", gd.mean())
    assert gd.mean() < 1e-5 and gd.max() < pr.GATE_TOL
    st.close()


def test_zero_tokens_and_argument_errors(hero):
    import torch
    inp = pr.inputs("tiny_f32")
    st = _stack(hero, inp)
    counts = torch.full((inp.cfg.n_layers,), 7, dtype=torch.int32, device="cuda")
    hero.hero_routed_ffn_stack(st.model, 0, 0, 0, inp.tau, 0, 0, 0, 0, 0, counts.data_ptr(), 0)
    torch.cuda.synchronize()
    assert (counts == 0).all()
    x = torch.zeros((inp.cfg.n_tokens, inp.cfg.d_model), device="cuda")
    with pytest.raises(hero.HeroError) as e:   # T above max_tokens
        hero.hero_routed_ffn_stack(st.model, inp.cfg.n_tokens + 1, x.data_ptr(), 0, 0.5, 0, 0,
                                   x.data_ptr() + 4, 0, 0, 0, 0)
    assert e.value.status == hero.HERO_ERR_ARG
    with pytest.raises(hero.HeroError) as e:   # aliasing in/out
        hero.hero_routed_ffn_stack(st.model, 4, x.data_ptr(), 0, 0.5, 0, 0, x.data_ptr(), 0, 0, 0, 0)
    assert e.value.status == hero.HERO_ERR_ARG
    st.check()
    st.close()


def test_host_io_matches_device_path(hero):
    """HERO_FLAG_HOST_IO (host buffers, copies inside the call) == device buffers."""
    import torch
    inp = pr.inputs("small_bf16")
    st = _stack(hero, inp)
    dev = pr.run_gpu(st, inp)
    L, T, d = inp.cfg.n_layers, inp.cfg.n_tokens, inp.cfg.d_model
    h = torch.from_numpy(inp.h).pin_memory()
    P = torch.from_numpy(inp.P).pin_memory()
    h_out = torch.empty((T, d), dtype=torch.float32).pin_memory()
    g = torch.empty((L, T), dtype=torch.float32).pin_memory()
    m = torch.empty((L, T), dtype=torch.uint8).pin_memory()
    c = torch.empty((L,), dtype=torch.int32).pin_memory()
    hero.hero_routed_ffn_stack(st.model, T, h.data_ptr(), P.data_ptr(), inp.tau,
                               hero.HERO_FLAG_HOST_IO, 0, h_out.data_ptr(), g.data_ptr(),
                               m.data_ptr(), c.data_ptr(), torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(h_out.numpy(), dev.h_out.astype(np.float32))
    np.testing.assert_array_equal(m.numpy(), dev.mask)
    np.testing.assert_array_equal(c.numpy(), dev.counts)
    st.close()


# ------------------------------------------------------------------------------
# full-size workloads, sampled tokens
# ------------------------------------------------------------------------------

FULL = [("llama2_7b_prefill", None, 64), ("llama31_8b_prefill", None, 64),
        ("llama31_8b_decode", None, 64), ("llama2_13b_prefill", 0.27, 32),
        ("llama2_13b_prefill", 0.0, 32), ("llama2_13b_prefill", 0.39, 32),
        ("llama31_8b_paper", None, 32)]


@pytest.mark.parametrize("name,bypass,n_sample", FULL)
def test_full_size_sampled(hero, name, bypass, n_sample):
    import torch
    inp = pr.inputs(name, bypass=bypass)
    cfg = inp.cfg
    rows = hi.sample_tokens(cfg.n_tokens, n_sample)
    st = _stack(hero, inp)
    gpu_all = pr.run_gpu(st, inp)          # all T tokens, bench launch configuration
    gpu = pr.GpuRun(gpu_all.h_out[rows], gpu_all.gate[:, rows], gpu_all.mask[:, rows], gpu_all.counts)
    ref = pr.run_oracle(inp, rows=rows)
    bound = pr.free_run_gate_bound(name)
    rep = pr.compare_free(gpu, ref, pr.H_TOL["bf16"], boundary=bound)
    print(name, rep, "bypass", 1 - gpu_all.mask.mean())
    _assert_free(rep, pr.H_TOL["bf16"], max_boundary_frac=0.1, gate_tol=bound)
    # whole-workload properties: counts agree with decisions, bypass near the budget
    np.testing.assert_array_equal(gpu_all.counts, gpu_all.mask.sum(axis=1))
    target = cfg.bypass if bypass is None else bypass
    assert (gpu_all.mask[:cfg.n_dense] == 1).all()           # dense prefix (placement)
    assert abs((1 - gpu_all.mask[cfg.n_dense:].mean()) - target) < 0.05
    # forced mode on the sample: the GPU follows the oracle's decisions
    mask_in = gpu_all.mask.copy()
    mask_in[:, rows] = ref["mask"]
    forced = pr.run_gpu(st, inp, flags=hero.HERO_FLAG_FORCE_MASK, mask_in=mask_in, rows=rows)
    frep = pr.compare_forced(forced, ref)
    print(name, "forced", frep)
    assert frep.gate_err < pr.free_run_gate_bound(name) and frep.h_err < pr.H_TOL["bf16"]
    st.close()
    del gpu_all
    torch.cuda.empty_cache()


@pytest.mark.parametrize("name", ["small_bf16", "llama31_8b_decode"])
def test_cuda_graph_replay_matches_eager(hero, name):
    """One stack call captured into a CUDA graph replays to the eager result, bit for bit
    (no host synchronisation inside the call; the decode shape runs the split-K GEMMs)."""
    import torch
    inp = pr.inputs(name)
    cfg = inp.cfg
    T, d, L = cfg.n_tokens, cfg.d_model, cfg.n_layers
    st = _stack(hero, inp)
    dev = torch.device("cuda")
    h = torch.from_numpy(np.ascontiguousarray(inp.h)).to(dev)
    P = torch.from_numpy(np.ascontiguousarray(inp.P)).to(dev)
    outs = [torch.empty((T, d), device=dev), torch.empty((L, T), device=dev),
            torch.empty((L, T), dtype=torch.uint8, device=dev),
            torch.empty((L,), dtype=torch.int32, device=dev)]
    st(h, P, inp.tau, h_out=outs[0], gate_out=outs[1], mask_out=outs[2], counts_out=outs[3])
    torch.cuda.synchronize()
    eager = [o.clone() for o in outs]
    for o in outs:
        o.zero_()
    graph = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream()
    cap.wait_stream(torch.cuda.current_stream())
    with torch.cuda.graph(graph, stream=cap):
        st(h, P, inp.tau, h_out=outs[0], gate_out=outs[1], mask_out=outs[2], counts_out=outs[3],
           stream=cap)
    torch.cuda.current_stream().wait_stream(cap)
    for o in outs:
        o.zero_()
    graph.replay()
    graph.replay()
    torch.cuda.synchronize()
    st.check()
    for a, b in zip(outs, eager):
        assert torch.equal(a, b)
    if T <= 128:   # the speculative branches (every token through both) against the compacted
        st(h, P, inp.tau, flags=hero.HERO_FLAG_NO_SPECULATE, h_out=outs[0], gate_out=outs[1],
           mask_out=outs[2], counts_out=outs[3])
        torch.cuda.synchronize()
        st.check()
        for a, b in zip(outs, eager):
            assert torch.equal(a, b)
    st.close()


@pytest.mark.parametrize("T", [1, 37, 64, 128])
def test_speculative_branches_equal_compacted(hero, T):
    """Batches of one 128-row tile run the FFN and the adapter branch on every token while
    the router runs on a second stream, and the closing launch takes each token's branch from
    the decision; HERO_FLAG_NO_SPECULATE runs the FFN on the routed tokens after the router.
    Each GEMM row depends on its own operand row only and the K order is the same, so h_out,
    g, the decisions and the counts agree bit for bit; the speculative run also against the
    oracle on every token, free-running (small_bf16 widths; from 37 tokens)."""
    inp = pr.inputs("small_bf16", cfg=hi.CONFIGS["small_bf16"].replace(n_tokens=T))
    st = _stack(hero, inp)
    a = pr.run_gpu(st, inp)
    b = pr.run_gpu(st, inp, flags=hero.HERO_FLAG_NO_SPECULATE)
    np.testing.assert_array_equal(a.h_out, b.h_out)
    np.testing.assert_array_equal(a.gate, b.gate)
    np.testing.assert_array_equal(a.mask, b.mask)
    np.testing.assert_array_equal(a.counts, b.counts)
    np.testing.assert_array_equal(a.counts, a.mask.sum(axis=1))
    if T > 1:   # one token: the near-boundary rule may leave nothing to compare
        ref = pr.run_oracle(inp)
        rep = pr.compare_free(a, ref, pr.H_TOL["bf16"])
        print(T, rep, "bypass", 1 - a.mask.mean())
        _assert_free(rep, pr.H_TOL["bf16"])
    st.close()
